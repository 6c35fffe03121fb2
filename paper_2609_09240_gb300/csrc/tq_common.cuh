// tq_common.cuh - device-side helpers shared by the CUDA kernels of the
// packed ternary linear layer (format constants, fp16 bit helpers, the
// kernel-side problem descriptor).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "tq.h"

namespace tq {

constexpr int kGroup = TQ_GROUP;            // trits per group along K
constexpr int kGroupBytes = TQ_GROUP_BYTES;  // 25 full bytes + 1 tail byte
constexpr int kFullBytes = 25;
constexpr int kTailTrits = 3;
// Tail byte of an all-zero group: digits (1,1,1) plus the two pad digits 1.
constexpr int kZeroByte = 121;  // 1 + 3 + 9 + 27 + 81

__host__ __device__ inline int64_t row_bytes_of(int K) {
  int64_t raw = (int64_t)(K / kGroup) * kGroupBytes;
  return (raw + 15) / 16 * 16;
}
__host__ __device__ inline int sal_words_of(int K) { return (K / kGroup + 31) / 32; }

// Kernel-side descriptor of one projection (copied by value into launch
// parameters; all pointers are device pointers).
struct Problem {
  const uint8_t *plane1;
  const uint32_t *sal;
  const int32_t *rowptr;
  const uint8_t *plane2;
  const __half *s1;
  const __half *off;
  const __half *s2;
  const __half *x;  // [M][K]
  void *y;          // [M][N] fp16 or fp32
  unsigned char *wsB;  // workspace: activation slots of this problem
  float *wsCS;         // workspace: per-group C and S of this problem
  const int32_t *p2idx;  // optional second-plane index (tq_plane2_index), or null
  int32_t y2_off;      // workspace bytes from wsB: second-plane partial sums [N][M] (M <= 8 path)
  int32_t map_off;     // workspace bytes from wsB: 128-byte tensor map of plane 1 (M <= 8 path)
  int32_t N, K;
  int32_t tile_begin;  // first global tile index of this problem
  int32_t nnz;         // plane-2 records (rowptr[N]); indices are clamped below it
  __host__ __device__ float *y2() const { return reinterpret_cast<float *>(wsB + y2_off); }
  __host__ __device__ void *map() const { return wsB + map_off; }
};

struct BatchParams {
  int32_t count;        // problems in prob[]
  int32_t M;            // tokens (rows of every x)
  int32_t total_tiles;  // sum of tiles over problems
  int32_t out_f32;      // y is fp32 (else fp16)
  int32_t g4_split;     // M <= 2: target groups per work unit of a 256-row tile (0: whole tiles)
  int32_t general;      // nonzero: the general decode kernels even for M <= 2 (the one-group-per-lane
                        // kernel's operands are then not in the workspace)
  int32_t g4_only;      // nonzero: only the one-group-per-lane kernels read the activation operands
                        // (the prep kernel writes no general-layout fragments or C/S)
  Problem prob[TQ_MAX_BATCH];
};

// One problem of an element-wise call as the API hands it to the kernels
// (tq_ew.cu): the weight, x, the fp32 plane-1 result, y and the views of
// the plane-1 pass in the workspace.
struct EwCall {
  const tq_ew_weight *w;
  const uint16_t *x;
  float *ydense;
  void *y;
  uint16_t *s1v, *offv;
  uint32_t *salv;
  int32_t *rpv;
};

}  // namespace tq
