// tq_prefill.cu - prefill-path linear (M > 16 tokens): the packed weights are
// dequantized tile by tile into shared memory and contracted with tcgen05
// MMAs (fp16 operands, fp32 accumulators in tensor memory).
//
// What is computed (the paper's eq. W-hat per group, "Model and
// Representation"; weight-only A16): y[m][n] = sum_k x[m][k] W[n][k] with
//   W[n][k] = s1[n,g] t1[n,k] + off[n,g] + sal[n,g] s2[j(n,g)] t2[n,k],  g = k / 128,
// each W element rounded once to fp16 (x is fp16), fp32 accumulation.
//
// prefill2_kernel: a 128-row x 512-token output tile per CTA (or 256
// tokens for narrow grids), weights as the MMA's M operand; x tiles and
// per-group plane-1 windows arrive by tensor copies, 16 warps decode the
// weight tiles into shared memory, one thread issues the MMAs (see its
// comment).
// Weight decode: a byte's five digits d (trit + 1) select among the row's
// three fp16 values off - s1, off, off + s1 held in two registers; a
// 243-entry table gives, per digit, the PRMT selector nibbles of its value,
// so two weights cost one PRMT.  Every wait is bounded.
#include <cuda.h>

#include <algorithm>
#include <cudaTypedefs.h>

#include "tq_common.cuh"
#include "tq_sm100.cuh"

namespace tq {
namespace pf {

constexpr int BK = 128;          // K per group

__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, volatile int32_t *abort_) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1;; ++i) {
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

// Selector entry of a byte value: byte i (i < 5) = the PRMT nibbles (2 d_i,
// 2 d_i + 1) that pick value d_i from {v0 | v1 << 16, v2 | v2 << 16}.
__device__ __forceinline__ uint64_t sel_entry(int v) {
  uint64_t e = 0;
  if (v > 242) v = 121;  // invalid bytes decode as all-zero trits (not produced by tq_pack)
  for (int i = 0; i < 5; ++i) {
    const int d = v % 3;
    v /= 3;
    e |= (uint64_t)((2 * d) | ((2 * d + 1) << 4)) << (8 * i);
  }
  return e;
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t s) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(s));
  return d;
}

// One weight row's data for one group, loaded a group ahead of its decode:
// the raw aligned words of its 26 bytes and of its plane-2 record, s1, off,
// s2, and whether the group is salient.
struct RowGroup {
  uint32_t r8[7], q8[7];
  unsigned short s1, of, s2;
  bool odd, rodd, salient;
};

// the 7 words of a 26-byte run, byte 0 first, from its raw aligned words
__device__ __forceinline__ void realign(const uint32_t *r8, bool odd, uint32_t *rw) {
#pragma unroll
  for (int i = 0; i < 7; ++i) rw[i] = odd ? __funnelshift_r(r8[i], i < 6 ? r8[i + 1] : 0u, 16) : r8[i];
}

// 5 NP fp16x2 words from byte pairs P0 .. P0 + NP - 1 of a 26-byte run
// (word i = trits 10 P0 + 2i, + 1).
template <int P0, int NP>
__device__ __forceinline__ void decode_pairs(const uint32_t *rw, uint32_t v01, uint32_t v22, const uint64_t *sel,
                                             uint32_t *out) {
#pragma unroll
  for (int q = 0; q < NP; ++q) {
    const int p = P0 + q;
    const int ba = 2 * p, bb = 2 * p + 1;
    const uint32_t va = (rw[ba >> 2] >> (8 * (ba & 3))) & 0xffu;
    const uint32_t vb = (rw[bb >> 2] >> (8 * (bb & 3))) & 0xffu;
    const uint64_t ta = sel[va], tb = sel[vb];
    const uint32_t ta_lo = (uint32_t)ta, ta_hi = (uint32_t)(ta >> 32);
    const uint32_t tb_lo = (uint32_t)tb, tb_hi = (uint32_t)(tb >> 32);
    out[5 * q] = prmt(v01, v22, ta_lo);
    out[5 * q + 1] = prmt(v01, v22, ta_lo >> 16);
    out[5 * q + 2] = prmt(v01, v22, prmt(ta_hi, tb_lo, 0x0040u));
    out[5 * q + 3] = prmt(v01, v22, tb_lo >> 8);
    out[5 * q + 4] = prmt(v01, v22, prmt(tb_lo, tb_hi, 0x0043u));
  }
}

// Quarter Q of a group's 128 weights of one row (16 words, K = 32 Q .. 32 Q
// + 31): s1 t1 + off, plus s2 t2 when any row of the warp is salient.
// Quarter Q decodes byte pairs 3 Q .. 3 Q + 3 (trits 30 Q .. 30 Q + 39) and
// keeps words Q .. Q + 15.
template <int Q>
__device__ __forceinline__ void decode_row_quarter(const RowGroup &cur, const uint64_t *sel, uint32_t *wv) {
  constexpr int P0 = 3 * Q, W0 = Q;
  const float s1 = __half2float(__ushort_as_half(cur.s1)), of = __half2float(__ushort_as_half(cur.of));
  uint32_t rw[7];
  realign(cur.r8, cur.odd, rw);
  const __half h0 = __float2half_rn(of - s1), h1 = __float2half_rn(of), h2 = __float2half_rn(of + s1);
  const uint32_t v01 = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
  const uint32_t v22 = (uint32_t)__half_as_ushort(h2) * 0x00010001u;
  uint32_t w1[20];
  decode_pairs<P0, 4>(rw, v01, v22, sel, w1);
#pragma unroll
  for (int i = 0; i < 16; ++i) wv[i] = w1[W0 + i];
  if (__any_sync(0xffffffffu, cur.salient)) {
    const float s2 = __half2float(__ushort_as_half(cur.s2));
    uint32_t rec[7];
    realign(cur.q8, cur.rodd, rec);
    const __half q0 = __float2half_rn(-s2), q2 = __float2half_rn(s2);
    const uint32_t u01 = (uint32_t)__half_as_ushort(q0);  // (-s2, 0)
    const uint32_t u22 = (uint32_t)__half_as_ushort(q2) * 0x00010001u;
    uint32_t w2[20];
    decode_pairs<P0, 4>(rec, u01, u22, sel, w2);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const __half2 x = *reinterpret_cast<const __half2 *>(&wv[i]);
      const __half2 y = *reinterpret_cast<const __half2 *>(&w2[W0 + i]);
      const __half2 z = __hadd2(x, y);
      wv[i] = *reinterpret_cast<const uint32_t *>(&z);
    }
  }
}

// Core-matrix offset of (row, K element e) in a tile of 8-row groups x 16
// core matrices along K.
__device__ __forceinline__ int cm_off(int row, int e) { return ((row >> 3) * 16 + (e >> 3)) * 128 + (row & 7) * 16; }

// ------------------------------------------------------------------------
// prefill2_kernel: a 128-row x (256 TT)-token output tile per CTA, weights
// as the MMA's M operand (M = 128), tokens as N = 256 per token half.
//  * warps 0..15 (thread r + 128 q = quarter q of weight row n0 + r): decode
//    each group's 32 weights of their quarter row into a 2-slot ring of
//    weight tiles (32 KiB, the no-swizzle K-major core-matrix layout, 16
//    core matrices along K), from the group's plane-1 window (a tensor copy
//    of 48 bytes per row by warp 16's lane 1, 2-slot ring);
//  * warp 16 (lane 0): the x tiles, 256 TT tokens x 64 K per stage (TT
//    2-D tensor copies of 256 tokens with 128-byte swizzling, the K-major
//    layout the MMA reads through a swizzled descriptor), into a 2-slot
//    ring, two stages per group;
//  * warp 17 (one thread): per stage 4 TT MMAs (M = 128 rows, N = 256
//    tokens, K = 16; token half t into tensor-memory columns 256 t ..);
//  * at the end warps 0..15 read the accumulators and write y.
// A decoded weight tile serves 256 TT tokens and 8 TT MMAs: with TT = 2
// every weight is decoded once per 512 tokens.  Needs a tensor map of x
// that the host encodes (x 16-byte aligned, K a multiple of 128).
constexpr int BR2 = 128;                 // weight rows per CTA
constexpr int BT2 = 256;                 // tokens per MMA (N) and per token half
constexpr int XK2 = 64;                  // K per x stage
constexpr int kXHalf2 = BT2 * XK2 * 2;   // 32 KiB: one token half of an x stage
constexpr int kWTile2 = BR2 * BK * 2;    // 32 KiB
constexpr int kPRow2 = 48;                 // plane-1 window per row: the 16-byte units covering a group
constexpr int kPSlot2 = BR2 * kPRow2;      // 6 KiB
constexpr int NW2 = 2, NX2 = 2, NP2 = 2;
constexpr int kDecWarps2 = 16, kWarpProd2 = 16, kWarpMma2 = 17;
constexpr int kThreads2 = 18 * 32;
constexpr uint32_t kTmemCols2 = 512;
template <int TT>
struct Lay2 {
  static constexpr int kXStage = TT * kXHalf2;
  static constexpr int oW = 0;
  static constexpr int oX = NW2 * kWTile2;
  static constexpr int oP = oX + NX2 * kXStage;
  static constexpr int oSel = oP + NP2 * kPSlot2;
  static constexpr int oBar = oSel + 256 * 8;
  static constexpr int kSmem = oBar + 256;
  static_assert(kSmem <= 232448, "prefill2 shared memory");
};

// The problems of one launch (one projection, or a batch of them sharing
// M): each problem's tensor maps of x and plane 1 and its first tile in the
// launch's 1-D grid (tiles problem by problem, row tile major, token tile
// minor; the host puts the problems with the longest K first, so that the
// block scheduler starts the longest tiles first and back-fills the waves).
constexpr int kPfMaxBatch = 16;
struct PfBatch {
  CUtensorMap xmap[kPfMaxBatch];
  CUtensorMap pmap[kPfMaxBatch];
  Problem prob[kPfMaxBatch];
  int32_t tile_begin[kPfMaxBatch + 1];
  int32_t count, mtiles;  // problems; token tiles per problem
};
static_assert(sizeof(PfBatch) <= 32764, "prefill launch parameters");

struct Bars2 {
  uint64_t xfull[NX2], xempty[NX2], wfull[NW2], wempty[NW2], pfull[NP2], pempty[NP2], done;
  uint32_t tmem_slot;
  int32_t abort_;
};
static_assert(sizeof(Bars2) <= 256, "prefill2 barriers");

template <bool F32, int TT>
__global__ void __launch_bounds__(kThreads2, 1)
    prefill2_kernel(const __grid_constant__ PfBatch B, int M) {
  using L = Lay2<TT>;
  extern __shared__ __align__(1024) unsigned char smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // this CTA's problem and tile
  int pi = 0;
  while (pi + 1 < B.count && B.tile_begin[pi + 1] <= (int)blockIdx.x) ++pi;
  const Problem &P = B.prob[pi];
  const CUtensorMap *xmap = &B.xmap[pi], *pmap = &B.pmap[pi];
  const int local = (int)blockIdx.x - B.tile_begin[pi];
  const int m0 = (local % B.mtiles) * (TT * BT2), n0 = (local / B.mtiles) * BR2;
  const int N = P.N, G = P.K / kGroup;
  uint64_t *sel = reinterpret_cast<uint64_t *>(smem + L::oSel);
  Bars2 *bars = reinterpret_cast<Bars2 *>(smem + L::oBar);
  volatile int32_t *abort_ = &bars->abort_;
  for (int i = tid; i < 256; i += kThreads2) sel[i] = sel_entry(i);
  if (tid == 0) {
    for (int i = 0; i < NX2; ++i) {
      mbar_init(&bars->xfull[i], 1);  // the producer's expect-tx arrival
      mbar_init(&bars->xempty[i], 1);
    }
    for (int i = 0; i < NW2; ++i) {
      mbar_init(&bars->wfull[i], kDecWarps2 * 32);
      mbar_init(&bars->wempty[i], 1);
    }
    for (int i = 0; i < NP2; ++i) {
      mbar_init(&bars->pfull[i], 1);           // the producer's expect-tx arrival
      mbar_init(&bars->pempty[i], kDecWarps2);  // one arrival per decoder warp
    }
    mbar_init(&bars->done, 1);
    bars->abort_ = 0;
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(&bars->tmem_slot, kTmemCols2);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_slot;

  if (warp < kDecWarps2) {
    // ======================================================= weight decode
    // Thread r + 128 q = quarter q of row n0 + r.  The group's packed bytes
    // come from the plane-1 window ring (one tensor copy per group: 48 bytes
    // of each row, from the 16-byte unit that holds the group's first byte);
    // s1 / off (8 groups per load where rows allow), salience and the
    // plane-2 record are loaded by the thread one group ahead.
    const int r = tid & (BR2 - 1), qq = tid >> 7;  // quarter qq of row r (warp-uniform)
    const int n = n0 + r;
    const bool valid = n < N;
    const int W = sal_words_of(P.K);
    const uint32_t *salrow = P.sal + (int64_t)(valid ? n : 0) * W;
    int64_t j = (valid && P.nnz > 0) ? P.rowptr[n] : 0;
    uint32_t salw = (valid && P.nnz > 0) ? __ldg(salrow) : 0u;
    const bool vec8 = (G % 8) == 0 && ((((uintptr_t)P.s1) | ((uintptr_t)P.off)) & 15u) == 0;
    const unsigned short *s1h = reinterpret_cast<const unsigned short *>(P.s1) + (int64_t)(valid ? n : 0) * G;
    const unsigned short *ofh = reinterpret_cast<const unsigned short *>(P.off) + (int64_t)(valid ? n : 0) * G;
    uint4 s1v = make_uint4(0u, 0u, 0u, 0u), ofv = make_uint4(0u, 0u, 0u, 0u);
    // everything of group g but its plane-1 bytes
    auto fetch = [&](int g, RowGroup &nx) {
      if (vec8) {
        if ((g & 7) == 0 && valid) {
          s1v = __ldg(reinterpret_cast<const uint4 *>(s1h + g));
          ofv = __ldg(reinterpret_cast<const uint4 *>(ofh + g));
        }
        const int k = g & 7;
        const uint32_t ws1 = k < 2 ? s1v.x : k < 4 ? s1v.y : k < 6 ? s1v.z : s1v.w;
        const uint32_t wof = k < 2 ? ofv.x : k < 4 ? ofv.y : k < 6 ? ofv.z : ofv.w;
        nx.s1 = (unsigned short)((k & 1) ? ws1 >> 16 : ws1);
        nx.of = (unsigned short)((k & 1) ? wof >> 16 : wof);
      } else {
        nx.s1 = valid ? __ldg(s1h + g) : (unsigned short)0;
        nx.of = valid ? __ldg(ofh + g) : (unsigned short)0;
      }
      if ((g & 31) == 0 && g > 0 && valid && P.nnz > 0) salw = __ldg(salrow + (g >> 5));
      nx.salient = (salw >> (g & 31)) & 1u;
      nx.s2 = 0;
      nx.rodd = false;
#pragma unroll
      for (int i = 0; i < 7; ++i) nx.q8[i] = 0x79797979u;
      if (nx.salient) {
        const int64_t jj = j < P.nnz ? j : P.nnz - 1;
        const int64_t off0 = jj * kGroupBytes;
        nx.rodd = (off0 & 3) != 0;  // plane 2 is 16-byte aligned: records start 0 or 2 bytes into a word
        const uint32_t *rs = reinterpret_cast<const uint32_t *>(P.plane2 + off0 - (nx.rodd ? 2 : 0));
#pragma unroll
        for (int i = 0; i < 6; ++i) nx.q8[i] = __ldg(rs + i);
        nx.q8[6] = nx.rodd ? __ldg(rs + 6) : (uint32_t)__ldg(reinterpret_cast<const uint16_t *>(rs + 6));
        nx.s2 = __ldg(reinterpret_cast<const unsigned short *>(P.s2) + jj);
        ++j;
      }
    };
    RowGroup nx;
    fetch(0, nx);
    for (int g = 0; g < G; ++g) {
      const int s = g % NW2, ps = g % NP2;
      if (g >= NW2 && !__all_sync(0xffffffffu, wait_or_abort(&bars->wempty[s], ((uint32_t)(g / NW2) & 1u) ^ 1u, abort_)))
        break;
      if (!__all_sync(0xffffffffu, wait_or_abort(&bars->pfull[ps], (uint32_t)(g / NP2) & 1u, abort_))) break;
      RowGroup cur = nx;
      {
        // the row's 7 words of group g: the window's words from (26 g mod 16) / 4 on
        const uint4 *pw = reinterpret_cast<const uint4 *>(smem + L::oP + ps * kPSlot2 + r * kPRow2);
        const uint4 a0 = pw[0], a1 = pw[1], a2 = pw[2];
        const uint32_t w[12] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w, a2.x, a2.y, a2.z, a2.w};
        const int q = ((kGroupBytes * g) & 15) >> 2;
        uint32_t t[10];
#pragma unroll
        for (int i = 0; i < 10; ++i) t[i] = (q & 2) ? w[i + 2] : w[i];
#pragma unroll
        for (int i = 0; i < 7; ++i) cur.r8[i] = (q & 1) ? t[i + 1] : t[i];
        cur.odd = g & 1;  // the group starts 2 bytes into its first word
      }
      if (g + 1 < G) fetch(g + 1, nx);
      uint32_t wv[16];
      if (qq == 0)
        decode_row_quarter<0>(cur, sel, wv);
      else if (qq == 1)
        decode_row_quarter<1>(cur, sel, wv);
      else if (qq == 2)
        decode_row_quarter<2>(cur, sel, wv);
      else
        decode_row_quarter<3>(cur, sel, wv);
      unsigned char *Wt = smem + L::oW + s * kWTile2;
#pragma unroll
      for (int kc = 0; kc < 4; ++kc)
        *reinterpret_cast<uint4 *>(Wt + cm_off(r, (4 * qq + kc) * 8)) =
            make_uint4(wv[4 * kc], wv[4 * kc + 1], wv[4 * kc + 2], wv[4 * kc + 3]);
      fence_proxy_async_smem();  // the MMA reads these stores through the async proxy
      mbar_arrive(&bars->wfull[s]);
      // the window is released once the stores that depend on its words have
      // issued (releasing right after the loads would let the next tensor copy
      // overwrite words a lane has not received yet)
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->pempty[ps]);
    }
  } else if (warp == kWarpProd2) {
    // ===================================== x tiles (lane 0), plane-1 windows (lane 1)
    if (lane == 1) {
      uint32_t issued = 0;
      for (int g = 0; g < G; ++g) {
        const int sl = g % NP2;
        if (g >= NP2 && !wait_or_abort(&bars->pempty[sl], ((uint32_t)(g / NP2) & 1u) ^ 1u, abort_)) break;
        mbar_arrive_expect_tx(&bars->pfull[sl], (uint32_t)(BR2 * kPRow2));
        // bytes from the 16-byte unit holding the group's first byte; rows n0 ..
        asm volatile(
            "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                smem_u32(smem + L::oP + sl * kPSlot2)),
            "l"(pmap), "r"((kGroupBytes * g) & ~15), "r"(n0), "r"(smem_u32(&bars->pfull[sl]))
            : "memory");
        ++issued;
      }
      for (uint32_t k = (issued > (uint32_t)NP2 ? issued - NP2 : 0); k < issued; ++k)
        mbar_wait(&bars->pfull[k % NP2], (k / NP2) & 1u);
    }
    if (lane == 0) {
      uint32_t issued = 0;
      for (int xs = 0; xs < 2 * G; ++xs) {
        const int sl = xs % NX2;
        if (xs >= NX2 && !wait_or_abort(&bars->xempty[sl], ((uint32_t)(xs / NX2) & 1u) ^ 1u, abort_)) break;
        mbar_arrive_expect_tx(&bars->xfull[sl], (uint32_t)L::kXStage);
        // K = 64 xs .., tokens m0 + 256 t .. (tokens past M arrive as zeros)
#pragma unroll
        for (int t = 0; t < TT; ++t)
          asm volatile(
              "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                  smem_u32(smem + L::oX + sl * L::kXStage + t * kXHalf2)),
              "l"(xmap), "r"(xs * XK2), "r"(m0 + t * BT2), "r"(smem_u32(&bars->xfull[sl]))
              : "memory");
        ++issued;
      }
      // every issued copy lands before the CTA exits (bounded)
      for (uint32_t k = (issued > (uint32_t)NX2 ? issued - NX2 : 0); k < issued; ++k)
        mbar_wait(&bars->xfull[k % NX2], (k / NX2) & 1u);
    }
  } else if (warp == kWarpMma2 && lane == 0) {
    // ================================================================= MMA
    const uint32_t idesc = idesc_f16_f32(128, BT2);
    bool ok = true;
    for (int g = 0; g < G && ok; ++g) {
      const int s = g % NW2;
      if (!wait_or_abort(&bars->wfull[s], (uint32_t)(g / NW2) & 1u, abort_)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t Wb = smem_u32(smem + L::oW + s * kWTile2);
      for (int h = 0; h < 2; ++h) {
        const int xs = 2 * g + h, sl = xs % NX2;
        if (!wait_or_abort(&bars->xfull[sl], (uint32_t)(xs / NX2) & 1u, abort_)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t Xb = smem_u32(smem + L::oX + sl * L::kXStage);
#pragma unroll
        for (int kk = 0; kk < XK2 / 16; ++kk) {
          const uint64_t adesc = smem_desc(Wb + (4 * h + kk) * 256, 128, 2048);
          const uint32_t acc = (g > 0 || h > 0 || kk > 0) ? 1u : 0u;
#pragma unroll
          for (int t = 0; t < TT; ++t)
            mma_smemA(tmem + (uint32_t)(t * BT2), adesc, smem_desc_sw128(Xb + t * kXHalf2 + kk * 32), idesc, acc);
        }
        mma_commit(&bars->xempty[sl]);
      }
      if (ok) mma_commit(&bars->wempty[s]);
    }
    if (ok) mma_commit(&bars->done);
  }

  // ================================================================ epilogue
  __syncwarp();
  if (warp < kDecWarps2) {
    const bool ok = __all_sync(0xffffffffu, wait_or_abort(&bars->done, 0u, abort_));
    tc_fence_after();
    if (ok) {
      // 16 warps: tensor-memory lane quarter q (rows 32 q ..), then a
      // quarter of the 256 TT token columns
      const int q = warp & 3, part = warp >> 2;  // 0..3
      const int cb = part * (TT * BT2 / 4), ce = cb + TT * BT2 / 4;
      const int n = n0 + 32 * q + lane;
#pragma unroll 1
      for (int c0 = cb; c0 < ce; c0 += 8) {
        uint32_t v[8];
        tmem_ld8(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)c0, v);
        tmem_wait_ld();
        if (n < N) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int m = m0 + c0 + i;
            if (m < M) {
              if (F32)
                static_cast<float *>(P.y)[(int64_t)m * N + n] = __uint_as_float(v[i]);
              else
                static_cast<__half *>(P.y)[(int64_t)m * N + n] = __float2half_rn(__uint_as_float(v[i]));
            }
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols2);
  }
}

}  // namespace pf

TQ_STATUS_ACCESSOR(read_status_prefill)

// x [M][K] fp16 as a 2-D tensor, box 64 (K) x 256 (tokens), 128-byte
// swizzling.  false when the driver's encoder is unavailable or refuses.
static bool encode_x_map(const void *x, int M, int K, CUtensorMap *out) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = [] {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      fn = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }();
  if (!encode) return false;
  cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)M};
  cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  cuuint32_t box[2] = {(cuuint32_t)pf::XK2, (cuuint32_t)pf::BT2};
  cuuint32_t estr[2] = {1, 1};
  return encode(out, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(x), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// plane 1 [N][row bytes] as a 2-D byte tensor, box 48 bytes x `rows` rows.
static bool encode_p_map(const void *plane1, int N, int K, int rows, CUtensorMap *out) {
  static PFN_cuTensorMapEncodeTiled_v12000 encode = [] {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      fn = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }();
  if (!encode) return false;
  const int64_t rb = row_bytes_of(K);
  cuuint64_t dims[2] = {(cuuint64_t)rb, (cuuint64_t)N};
  cuuint64_t strides[1] = {(cuuint64_t)rb};
  cuuint32_t box[2] = {(cuuint32_t)pf::kPRow2, (cuuint32_t)rows};
  cuuint32_t estr[2] = {1, 1};
  return encode(out, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(plane1), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// One launch over `count` (<= kPfMaxBatch) problems sharing M: 512-token
// tiles (each weight decoded once per 512 tokens) unless the tokens fit one
// 256-token tile or twice as many 256-token CTAs still fit in one wave.
static cudaError_t launch_prefill_group(const Problem *probs, int count, int M, bool f32, cudaStream_t s) {
  thread_local pf::PfBatch B;  // large: kept off the stack
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t rows = 0;
  for (int i = 0; i < count; ++i) rows += (probs[i].N + pf::BR2 - 1) / pf::BR2;
  const int mt512 = (M + 2 * pf::BT2 - 1) / (2 * pf::BT2);
  const bool wide = M > pf::BT2 && (int64_t)mt512 * rows * 2 > sms;
  B.mtiles = wide ? mt512 : (M + pf::BT2 - 1) / pf::BT2;
  // problems with the longest K first (their tiles take the longest)
  int order[pf::kPfMaxBatch];
  for (int i = 0; i < count; ++i) order[i] = i;
  std::stable_sort(order, order + count, [&](int a, int b) { return probs[a].K > probs[b].K; });
  B.count = count;
  B.tile_begin[0] = 0;
  for (int k = 0; k < count; ++k) {
    const Problem &P = probs[order[k]];
    if (!encode_x_map(P.x, M, P.K, &B.xmap[k]) || !encode_p_map(P.plane1, P.N, P.K, pf::BR2, &B.pmap[k]))
      return cudaErrorNotSupported;  // the driver's tensor-map encoder is unavailable or refused the shapes
    B.prob[k] = P;
    B.tile_begin[k + 1] = B.tile_begin[k] + (P.N + pf::BR2 - 1) / pf::BR2 * B.mtiles;
  }
  auto kern = wide ? (f32 ? pf::prefill2_kernel<true, 2> : pf::prefill2_kernel<false, 2>)
                   : (f32 ? pf::prefill2_kernel<true, 1> : pf::prefill2_kernel<false, 1>);
  const int smem = wide ? pf::Lay2<2>::kSmem : pf::Lay2<1>::kSmem;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  kern<<<B.tile_begin[count], pf::kThreads2, smem, s>>>(B, M);
  return cudaGetLastError();
}

cudaError_t launch_prefill(const Problem &P, int M, bool f32, cudaStream_t s) {
  return launch_prefill_group(&P, 1, M, f32, s);
}

// A batch of problems sharing M > 16, kPfMaxBatch per launch.
cudaError_t launch_prefill_batched(const Problem *probs, int count, int M, bool f32, cudaStream_t s) {
  for (int i = 0; i < count; i += pf::kPfMaxBatch) {
    const cudaError_t e = launch_prefill_group(probs + i, std::min(pf::kPfMaxBatch, count - i), M, f32, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace tq
