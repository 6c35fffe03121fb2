// tq_gemv_g4.cu - decode-path linear for M <= 2 tokens, one group per lane.
//
// What is computed is the decode path's sum (per-group reading of the
// paper's eq. W-hat, "Model and Representation"; packed execution as in
// "Direct Packed Execution"):
//   y[m][n] = sum_g ( s1[n,g] * P1[n,g,m] + off[n,g] * S[g,m] ) + y2[n][m],
// with P1 = sum_{k in g} T1[n,k] x[m,k], S = sum_{k in g} x[m,k] and y2 the
// second plane's s2 * P2 sums, written before this kernel runs.
//
// Layout of the work.  A stage is 4 consecutive groups (104 packed bytes of
// a row) of a 256-row tile.  Lane (g, c) of a warp (g = lane / 4,
// c = lane % 4) owns group c of the stage for the rows of its MMA fragment
// (rows g and g + 8 of each of the warp's two m16 tiles): the 7 aligned
// words that cover that group's 26 bytes (2 bytes of a neighbouring group
// ride along with zero activations).  In one m16n8k16 MMA every lane of a
// row therefore contributes products of a different group, and the MMA's 8
// columns keep them apart: column 2c collects group c for token 0 and
// column 2c + 1 group c for token 1.  Lane (g', c) holds the activation
// slots of column g' (B's column), real when g' = 2c + token and zero
// otherwise, so each column receives exactly its group's products; the
// accumulator fragment of lane (g, c) then holds rows g, g + 8 x columns
// 2c, 2c + 1, which are exactly the lane's own group and tokens, and every
// lane applies its own s1 / off.  Compared with one group at a time (the
// general decode kernel), no MMA slot is spent on the padding of 26-byte
// groups to 32-byte windows, and the per-group epilogue runs on all lanes.
//
// Operand encoding (five MMA slots per packed byte): the byte v = sum_i d_i
// 3^i (d_i = trit + 1) gives, through the lane-replicated table, W = (4 +
// d0 + d2/4, 4 + d1 + d3/4), then W' = (16 + d2, 16 + d3) by one LOP3 and
// the fifth slot 4 + v/256 by one PRMT for two bytes; the activation slots
// written by the prep kernel make the MMA return const + sum_i d_i x_i, and
// the accumulator starts at -const (C), so that it ends at sum_i t_i x_i.
// A word of 4 bytes gives 10 registers (W, W' of each byte, then the two
// fifth-slot words), i.e. 5 MMAs per m16 tile; 7 words give 35.
//
// Roles: warps 0..7 decode and multiply 32 rows each; warp 8 moves every
// stage into a ring of 4 shared-memory slots: the tile's plane-1 bytes (one
// 2-D tensor copy of 112 bytes x 256 rows: stages start on a 16-byte
// boundary, so odd stages are copied from 8 bytes earlier), the activation
// slots and C / S of the stage (bulk copies) and s1 / off (tensor copies of
// the 8-group box that holds the stage, or plain loads when rows of scales
// are not whole 16-byte units).  Every wait is bounded (tq_sm100.cuh).
#include <cuda.h>

#include "tq_common.cuh"
#include "tq_decode_ops.cuh"
#include "tq_sm100.cuh"

namespace tq {
namespace g4 {

using mm::kArena1;
using mm::kArena2;
using mm::kDynBytes;
using mm::kDynShared;
using mm::kLutBytes;
using mm::kLutShared;

constexpr int kStageBytes = 104;  // plane-1 bytes per row per stage (kStageG = 4 groups, lane c owns group c)
constexpr int kBox = 112;         // bytes per row copied per stage (and the shared row stride)
constexpr int kWords = 7;         // window words per lane and row
static_assert(kBPairs * 2 >= 5 * kWords, "activation chunks cover the 35 MMAs of a stage");
constexpr int kWarpsD = 8, kWarpProd = 8, kThreads = 9 * 32;
constexpr int kNS = 4;            // stage slots
constexpr int kP1Slot = kRows * kBox;    // 28672
constexpr int kSOHalf = kRows * 16;      // s1 (then off): 8 groups of fp16 per row
constexpr int kSOSlot = 2 * kSOHalf;
// arena 1 (below the table): plane-1 slots 0 and 1, barriers, the zero
// activation block, the C/S slots
constexpr int kOffBars = 2 * kP1Slot;
constexpr int kOffZero = kOffBars + 256;
constexpr int kOffCS = kOffZero + kBTok;
constexpr int kEnd1 = kOffCS + kNS * kCSStage;
static_assert(kEnd1 <= kArena1, "arena 1 overflow");
// arena 2 (above the table): plane-1 slots 2 and 3, s1/off slots, activation slots
constexpr int kOffSO = 2 * kP1Slot;
constexpr int kOffB = kOffSO + kNS * kSOSlot;
__host__ __device__ constexpr int used2(int MB) { return kOffB + kNS * kBTok * MB; }
static_assert(used2(2) <= kArena2, "arena 2 overflow");

struct Bars {
  uint64_t full[kNS], empty[kNS];
  int32_t abort_;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

// Schedule: CTA c processes global 256-row tiles [cta_tile[c], cta_tile[c+1]).
struct Sched {
  int32_t cta_tile[257];
};

// Iterates (tile, stage) in the CTA's order; tiles are numbered over the
// problems in order, ceil(N / 256) each.
struct Walk {
  const BatchParams *bp;
  int tile, t_end, pi, tb, s, nst;
  __device__ void locate() {
    for (;;) {
      const int T = (bp->prob[pi].N + kRows - 1) / kRows;
      if (tile < tb + T) break;
      tb += T;
      ++pi;
    }
    nst = nstages(bp->prob[pi].K);
    s = 0;
  }
  __device__ Walk(const BatchParams *b, int t0, int t1) : bp(b), tile(t0), t_end(t1), pi(0), tb(0), s(0), nst(0) {
    if (tile < t_end) locate();
  }
  __device__ bool valid() const { return tile < t_end; }
  __device__ const Problem &P() const { return bp->prob[pi]; }
  __device__ int n0() const { return (tile - tb) * kRows; }
  __device__ bool last_stage() const { return s + 1 == nst; }
  __device__ void next() {
    if (++s < nst) return;
    if (++tile < t_end) locate();
  }
};

// The 10 operand registers of one packed word: W, W' of bytes 0..3, then
// the fifth-slot words of bytes (0, 1) and (2, 3).
__device__ __forceinline__ void decode_word(uint32_t x, uint32_t tag, uint32_t *a) {
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint32_t w = mm::lut_load(mm::prmt(x, tag, 0x7604u | (k << 4)));
    a[2 * k] = w;
    a[2 * k + 1] = mm::w_prime(w);
  }
  a[8] = mm::prmt(x, 0x44444444u, 0x4140u);
  a[9] = mm::prmt(x, 0x44444444u, 0x4342u);
}

__device__ __forceinline__ float half_at(const unsigned char *p) {
  return __half2float(*reinterpret_cast<const __half *>(p));
}

// Workspace addresses of a problem's activation slots and C/S (after the
// general decode path's 512-byte map slot).
__device__ __forceinline__ const unsigned char *ws_b(const Problem &P) {
  return P.wsB + P.map_off + 512;
}
__device__ __forceinline__ const unsigned char *ws_cs(const Problem &P, int MB) {
  return ws_b(P) + pad256(b_bytes(MB, P.K));
}

template <bool F32, int MB>
__global__ void __launch_bounds__(kThreads, 1)
    gemv_g4_kernel(const __grid_constant__ BatchParams bp, const __grid_constant__ Sched sc) {
  extern __shared__ __align__(1024) unsigned char dyn[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (smem_u32(dyn) != kDynShared) {
    // the table address trick needs the dynamic window right after the
    // reserved 1 KiB of shared memory; anything else is reported
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  // offsets (from dyn) of the slots of stage buffer b
  constexpr int kA2 = kArena1 + kLutBytes;
  auto p1_off = [](int b) -> int { return b < 2 ? b * kP1Slot : kA2 + (b - 2) * kP1Slot; };
  Bars *bars = reinterpret_cast<Bars *>(dyn + kOffBars);
  volatile int32_t *abort_ = &bars->abort_;

  // ---- one-time set-up: the lane-replicated table, the zero block, barriers
  {
    uint32_t *lut = reinterpret_cast<uint32_t *>(dyn + kArena1);
    for (int i = tid; i < 256 * 32; i += kThreads) lut[(i >> 5) * 64 + (i & 31)] = mm::lut_word(i >> 5);
    for (int i = tid; i < kBTok / 16; i += kThreads)
      reinterpret_cast<uint4 *>(dyn + kOffZero)[i] = make_uint4(0u, 0u, 0u, 0u);
  }
  if (tid == 0) {
    for (int i = 0; i < kNS; ++i) {
      mbar_init(&bars->full[i], 1 + 32);  // the producer's expect-tx arrival + its 32 lanes' arrivals
      mbar_init(&bars->empty[i], kWarpsD);
    }
    bars->abort_ = 0;
    mbar_fence_init();
  }
  __syncthreads();
  const int t_begin = sc.cta_tile[blockIdx.x], t_end = sc.cta_tile[blockIdx.x + 1];

  if (warp < kWarpsD) {
    // ============================================================ decode
    const int g = lane >> 2, c = lane & 3;
    const uint32_t tag = kLutShared | ((uint32_t)lane << 2);
    // first window word of group c in the stage row: bytes 0, 26, 52, 78
    // start in words 0, 6, 13, 19
    const int wb = 4 * ((c * 13) >> 1);
    const int rA = 32 * warp + g;  // rows rA, rA + 8 (tile 0) and rA + 16, rA + 24 (tile 1)
    // activation slots: this lane's column is token g & 1 of group g >> 1
    const bool realB = ((g >> 1) == c) && ((g & 1) < MB);
    float y[2][2][MB];
#pragma unroll
    for (int t = 0; t < 2; ++t)
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int k = 0; k < MB; ++k) y[t][h][k] = 0.f;
    uint32_t buf = 0, phase = 0;
    for (Walk w(&bp, t_begin, t_end); w.valid(); w.next()) {
      const bool ok = __all_sync(0xffffffffu, mm::wait_or_abort(&bars->full[buf], phase, abort_));
      if (!ok) break;
      const int s = w.s;
      const unsigned char *p1 = dyn + p1_off((int)buf) + 8 * (s & 1) + wb + rA * kBox;
      const unsigned char *bq =
          dyn + (realB ? kA2 + kOffB + (int)buf * kBTok * MB + (g & 1) * kBTok + c * 16 : kOffZero);
      const float4 cs = *reinterpret_cast<const float4 *>(dyn + kOffCS + (int)buf * kCSStage + c * 16);
      // accumulators start at -C (token 0 in columns 2c, token 1 in 2c + 1)
      float d0[4] = {-cs.x, -cs.y, -cs.x, -cs.y}, d1[4] = {-cs.x, -cs.y, -cs.x, -cs.y};
#pragma unroll
      for (int i = 0; i < kWords; ++i) {
        const uint32_t x0 = *reinterpret_cast<const uint32_t *>(p1 + 4 * i);
        const uint32_t x1 = *reinterpret_cast<const uint32_t *>(p1 + 8 * kBox + 4 * i);
        const uint32_t x2 = *reinterpret_cast<const uint32_t *>(p1 + 16 * kBox + 4 * i);
        const uint32_t x3 = *reinterpret_cast<const uint32_t *>(p1 + 24 * kBox + 4 * i);
        uint32_t a0[10], a1[10], a2[10], a3[10];
        decode_word(x0, tag, a0);
        decode_word(x1, tag, a1);
        decode_word(x2, tag, a2);
        decode_word(x3, tag, a3);
#pragma unroll
        for (int m = 0; m < 5; ++m) {
          const int j = 5 * i + m;
          const uint4 q = *reinterpret_cast<const uint4 *>(bq + (j >> 1) * 64);
          const uint32_t b0 = (j & 1) ? q.z : q.x, b1 = (j & 1) ? q.w : q.y;
          mm::mma16816(d0, a0[2 * m], a1[2 * m], a0[2 * m + 1], a1[2 * m + 1], b0, b1);
          mm::mma16816(d1, a2[2 * m], a3[2 * m], a2[2 * m + 1], a3[2 * m + 1], b0, b1);
        }
      }
      // s1 / off of (row, group c): the stage's groups sit at 4 (s & 1) in
      // the 8-group rows of the slot
      {
        const unsigned char *so = dyn + kA2 + kOffSO + (int)buf * kSOSlot + 2 * (4 * (s & 1) + c);
#pragma unroll
        for (int t = 0; t < 2; ++t) {
          const float *d = t ? d1 : d0;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int r = rA + 16 * t + 8 * h;
            const float s1 = half_at(so + r * 16), of = half_at(so + kSOHalf + r * 16);
            y[t][h][0] = fmaf(s1, d[2 * h], fmaf(of, cs.z, y[t][h][0]));
            if (MB > 1) y[t][h][MB - 1] = fmaf(s1, d[2 * h + 1], fmaf(of, cs.w, y[t][h][MB - 1]));
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->empty[buf]);
      if (w.last_stage()) {
        // sum the four groups' lanes of each row, add the second plane, write y
#pragma unroll
        for (int t = 0; t < 2; ++t)
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int k = 0; k < MB; ++k) {
              float v = y[t][h][k];
              v += __shfl_xor_sync(0xffffffffu, v, 1);
              v += __shfl_xor_sync(0xffffffffu, v, 2);
              y[t][h][k] = v;
            }
        const Problem &P = w.P();
        const int n = w.n0() + rA + 16 * (c >> 1) + 8 * (c & 1);  // lane c writes (tile c >> 1, half c & 1)
        if (n < P.N) {
#pragma unroll
          for (int k = 0; k < MB; ++k) {
            float v = c == 0 ? y[0][0][k] : c == 1 ? y[0][1][k] : c == 2 ? y[1][0][k] : y[1][1][k];
            if (P.nnz > 0) v += P.y2()[(int64_t)n * MB + k];
            if (F32)
              static_cast<float *>(P.y)[(int64_t)k * P.N + n] = v;
            else
              static_cast<__half *>(P.y)[(int64_t)k * P.N + n] = __float2half_rn(v);
          }
        }
#pragma unroll
        for (int t = 0; t < 2; ++t)
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int k = 0; k < MB; ++k) y[t][h][k] = 0.f;
      }
      if (++buf == (uint32_t)kNS) buf = 0, phase ^= 1u;
    }
  } else if (warp == kWarpProd) {
    // ========================================================== producer
    uint32_t buf = 0, phase = 0, q = 0;
    int map_pi = -1;
    for (Walk w(&bp, t_begin, t_end); w.valid(); w.next(), ++q) {
      const Problem &P = w.P();
      const int s = w.s, n0 = w.n0();
      const int G = P.K / kGroup;
      int ok = 1;
      if (lane == 0) ok = mm::wait_or_abort(&bars->empty[buf], phase ^ 1u, abort_) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;  // uniform across the warp
      uint64_t *full = &bars->full[buf];
      // s1 / off go by tensor copies when their rows are whole 16-byte units
      // (the prep kernel then built their maps), else by plain loads
      const bool so_map = (G % 8 == 0) && ((((uintptr_t)P.s1) | ((uintptr_t)P.off)) & 15u) == 0;
      unsigned char *so = dyn + kA2 + kOffSO + (int)buf * kSOSlot;
      const unsigned char *maps = static_cast<const unsigned char *>(P.map());
      if (lane == 0) {
        if (w.pi != map_pi) {
          // the problem's tensor maps, written by the prep kernel
          asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps) : "memory");
          if (so_map) {
            asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps + 128) : "memory");
            asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps + 256) : "memory");
          }
          map_pi = w.pi;
        }
        mbar_arrive_expect_tx(full, (uint32_t)(kP1Slot + kBTok * MB + kCSStage) + (so_map ? (uint32_t)kSOSlot : 0u));
        // the stage's 104 bytes of the tile's 256 rows, from the 16-byte
        // boundary at or before them (rows past N and bytes past the row's
        // end arrive as zeros)
        asm volatile(
            "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                smem_u32(dyn + p1_off((int)buf))),
            "l"(maps), "r"(kStageBytes * s - 8 * (s & 1)), "r"(n0), "r"(smem_u32(full))
            : "memory");
        bulk_g2s(dyn + kA2 + kOffB + (int)buf * kBTok * MB, ws_b(P) + (int64_t)s * kBTok * MB, kBTok * MB, full);
        bulk_g2s(dyn + kOffCS + (int)buf * kCSStage, ws_cs(P, MB) + (int64_t)s * kCSStage, kCSStage, full);
        if (so_map) {
          // the 8-group box holding the stage, for s1 and for off
          asm volatile(
              "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                  smem_u32(so)),
              "l"(maps + 128), "r"(8 * (s >> 1)), "r"(n0), "r"(smem_u32(full))
              : "memory");
          asm volatile(
              "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                  smem_u32(so + kSOHalf)),
              "l"(maps + 256), "r"(8 * (s >> 1)), "r"(n0), "r"(smem_u32(full))
              : "memory");
        }
      }
      __syncwarp();
      if (!so_map) {
        // the stage's 4 groups of s1 and off (zeros past G or N), at 4 (s & 1)
        // of each row's 8-group slot
        const int rows = min(kRows, P.N - n0);
        __half *d1 = reinterpret_cast<__half *>(so), *d2 = reinterpret_cast<__half *>(so + kSOHalf);
        for (int r = lane; r < rows; r += 32) {
          const int64_t o = (int64_t)(n0 + r) * G;
#pragma unroll
          for (int gg = 0; gg < kStageG; ++gg) {
            const int gi = kStageG * s + gg;
            d1[r * 8 + 4 * (s & 1) + gg] = gi < G ? P.s1[o + gi] : __float2half_rn(0.f);
            d2[r * 8 + 4 * (s & 1) + gg] = gi < G ? P.off[o + gi] : __float2half_rn(0.f);
          }
        }
      }
      mbar_arrive(full);  // the lanes' arrivals (the barrier counts 1 + 32)
      if (++buf == (uint32_t)kNS) buf = 0, phase ^= 1u;
    }
    // drain: every issued copy lands before the CTA exits (waited on even
    // after an abort; bounded by the wall-time limit)
    if (lane == 0) {
      for (uint32_t k = (q > (uint32_t)kNS ? q - kNS : 0); k < q; ++k) mbar_wait(&bars->full[k % kNS], (k / kNS) & 1u);
    }
  }
  __syncthreads();
}

}  // namespace g4

TQ_STATUS_ACCESSOR(read_status_gemv_g4)

int g4_rows_per_tile() { return g4::kRows; }
int64_t g4_workspace_bytes(int M, int K) {
  return g4::pad256(g4::b_bytes(M, K)) + g4::pad256(g4::cs_bytes(K));
}

// The M <= 2 decode kernel over a batch whose prep (activation slots, maps,
// y2) and second plane have been launched on the same stream.
cudaError_t launch_gemv_g4(const BatchParams &bp, int num_sms, cudaStream_t s) {
  thread_local g4::Sched sc;
  if (bp.M < 1 || bp.M > 2) return cudaErrorInvalidValue;
  const int ctas = min(num_sms, 256);
  int64_t total_cost = 0;
  for (int i = 0; i < bp.count; ++i)
    total_cost += (int64_t)((bp.prob[i].N + g4::kRows - 1) / g4::kRows) * (bp.prob[i].K / kGroup);
  // contiguous tile ranges of about equal cost (tiles x groups)
  int c = 0, tile = 0;
  int64_t run = 0;
  sc.cta_tile[0] = 0;
  for (int i = 0; i < bp.count; ++i) {
    const int tiles_i = (bp.prob[i].N + g4::kRows - 1) / g4::kRows;
    const int64_t cost = bp.prob[i].K / kGroup;
    for (int t = 0; t < tiles_i; ++t, ++tile) {
      const int64_t mid2 = 2 * run + cost;
      while (c < ctas - 1 && mid2 * ctas >= 2 * total_cost * (int64_t)(c + 1)) sc.cta_tile[++c] = tile;
      run += cost;
    }
  }
  while (c < ctas) sc.cta_tile[++c] = tile;
  auto kern = bp.M == 1 ? (bp.out_f32 ? g4::gemv_g4_kernel<true, 1> : g4::gemv_g4_kernel<false, 1>)
                        : (bp.out_f32 ? g4::gemv_g4_kernel<true, 2> : g4::gemv_g4_kernel<false, 2>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, g4::kDynBytes);
  if (e != cudaSuccess) return e;
  kern<<<ctas, g4::kThreads, g4::kDynBytes, s>>>(bp, sc);
  return cudaGetLastError();
}

}  // namespace tq
