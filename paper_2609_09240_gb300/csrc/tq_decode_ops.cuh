// tq_decode_ops.cuh - device helpers shared by the decode-path kernels
// (M <= 16 tokens): the shared-memory window layout around the lane-
// replicated byte table, the bounded wait with a CTA-wide abort flag, the
// byte -> MMA-operand table word and its PRMT/LOP3 helpers, asynchronous
// copies and the m16n8k16 MMA wrappers.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

#include "tq_common.cuh"
#include "tq_sm100.cuh"

namespace tq {
namespace mm {

constexpr int kLutBytes = 65536;  // 256 byte values x 256 B (32 lanes x 4 B used)
constexpr uint32_t kLutShared = 65536;  // shared-window address of the table
constexpr uint32_t kDynShared = 1024;   // shared-window offset of dynamic smem
constexpr int kDynBytes = 232448;       // whole opt-in shared memory of a CTA
constexpr int kArena1 = (int)(kLutShared - kDynShared);   // below the table
constexpr int kArena2 = kDynBytes - kArena1 - kLutBytes;  // above the table

// Bounded wait on an mbarrier phase that also gives up when another role of
// the CTA has raised the abort flag; a wait that runs out sets the timeout
// bit of the device status word and raises the flag itself.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, volatile int32_t *abort_) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1;; ++i) {
    // sleep in the wait rather than spin: the waiting warps share the
    // issue slots with the decoding warps
    if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if ((i & 7u) == 0) {
      if (*abort_) return false;
      if (global_ns() - t0 > kWaitLimitNs) break;
    }
  }
  atomicOr(&g_tq_device_status, kStatusTimeout);
  *abort_ = 1;
  return false;
}

// Table word of a byte value v = sum_i d_i 3^i (digits d_i = trit + 1): the
// fp16 pair (4 + d0 + d2/4, 4 + d1 + d3/4); invalid bytes (243..255) map to
// the exponent pattern alone.  w_prime() turns it into (16 + d2, 16 + d3)
// with one LOP3, and the fifth MMA slot of a byte is 4 + v/256 (the byte put
// under the exponent byte 0x44 by one PRMT).
__host__ __device__ __forceinline__ uint32_t lut_word(int v) {
  uint32_t w = 0x44004400u;
  if (v <= 242) {
    const uint32_t d0 = v % 3, d1 = (v / 3) % 3, d2 = (v / 9) % 3, d3 = (v / 27) % 3;
    w |= (d0 << 8) | (d2 << 6) | (d1 << 24) | (d3 << 22);
  }
  return w;
}

// Fills the lane-replicated table: entry v in words 64 v .. 64 v + 31 (the
// copy of lane l at word 64 v + l), written as 16-byte stores, each thread
// computing an entry once per four copies.
__device__ __forceinline__ void lut_fill_replicated(uint32_t *lut, int tid, int nthreads) {
  for (int i = tid; i < 256 * 8; i += nthreads) {
    const uint32_t w = lut_word(i >> 3);
    reinterpret_cast<uint4 *>(lut + (i >> 3) * 64)[i & 7] = make_uint4(w, w, w, w);
  }
}

// The low (hi = false) or high fp16 of a word, as float.
template <bool HI>
__device__ __forceinline__ float half_of(uint32_t w) {
  const __half2 h = *reinterpret_cast<const __half2 *>(&w);
  return HI ? __high2float(h) : __low2float(h);
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t s) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(s));
  return d;
}
// The table is constant after set-up: an ordinary (reorderable) load.
__device__ __forceinline__ uint32_t lut_load(uint32_t addr) {
  uint32_t w;
  asm("ld.shared.u32 %0, [%1];" : "=r"(w) : "r"(addr));
  return w;
}
__device__ __forceinline__ uint32_t w_prime(uint32_t w) {
  uint32_t d;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(d) : "r"(w), "n"(0x00C000C0), "n"(0x4C004C00));
  return d;
}

// 16-byte asynchronous global -> shared copies (completion tracked per
// thread in commit groups).
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// D += A * B, m16n8k16, fp16 in, fp32 accumulate.
__device__ __forceinline__ void mma16816(float *d, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// D = A * B (zero accumulator in).
__device__ __forceinline__ void mma16816_z(float *d, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                           uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%10,%10,%10,%10};"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(0.f));
}

}  // namespace mm

// Operand layout of the one-group-per-lane decode kernel for M <= 2 tokens
// (tq_gemv_g4.cu), written by the prep kernel.  A stage is SG groups of a
// 256-row tile: SG = 8 for one token (lane c of a row owns groups 2c and
// 2c + 1, the MMA's 8 columns are the stage's 8 groups), SG = 4 for two
// tokens (lane c owns group c, columns 2c + t are its two tokens).  Each
// stage has two activation-slot slices (the two groups of a lane, or its
// two tokens): per slice, 16-byte chunks [pair jp][lane position c] holding
// b0, b1 of the lane's MMAs 2 jp and 2 jp + 1; then per stage the C/S block
// [c] x (C_a, C_b, S_a, S_b) floats of the two slices.  Per problem the
// slots of all stages come first, then the C/S blocks.
namespace g4 {
constexpr int kRows = 256;  // tile rows
constexpr int kMaxM = 2;    // most tokens of the one-group-per-lane kernel
__host__ __device__ constexpr int stage_groups(int M) { return M == 1 ? 8 : 4; }
__host__ __device__ constexpr int words(int SG) { return SG == 8 ? 13 : 7; }  // window words per lane and row
__host__ __device__ constexpr int pairs(int SG) { return (5 * words(SG) + 1) / 2; }  // 16-byte chunks per slice
__host__ __device__ constexpr int slice_bytes(int SG) { return pairs(SG) * 64; }
constexpr int kCSStage = 64;
__host__ __device__ constexpr int nstages(int K, int SG) { return (K / kGroup + SG - 1) / SG; }
__host__ __device__ inline int64_t pad256(int64_t b) { return (b + 255) / 256 * 256; }
__host__ __device__ inline int64_t b_bytes(int M, int K) {
  return (int64_t)nstages(K, stage_groups(M)) * 2 * slice_bytes(stage_groups(M));
}
__host__ __device__ inline int64_t cs_bytes(int M, int K) { return (int64_t)nstages(K, stage_groups(M)) * kCSStage; }
// Whether a batch runs the one-group-per-lane kernel.
__host__ __device__ inline bool takes(const BatchParams &bp) { return bp.M >= 1 && bp.M <= kMaxM && !bp.general; }
// Split tiles (several CTAs per tile): one arrival counter per (tile,
// decode warp), after the C/S blocks.
constexpr int kMaxWarps = 16;
__host__ __device__ inline int64_t ticket_bytes(int N) { return (int64_t)((N + kRows - 1) / kRows) * kMaxWarps * 4; }
}  // namespace g4
}  // namespace tq
