// tq_gemv_g4.cu - decode-path linear for M <= 2 tokens, one group per lane.
//
// What is computed is the decode path's sum (per-group reading of the
// paper's eq. W-hat, "Model and Representation"; packed execution as in
// "Direct Packed Execution"):
//   y[m][n] = sum_g ( s1[n,g] * P1[n,g,m] + off[n,g] * S[g,m] ) + y2[n][m],
// with P1 = sum_{k in g} T1[n,k] x[m,k], S = sum_{k in g} x[m,k] and y2 the
// second plane's s2 * P2 sums, written before this kernel runs.
//
// Layout of the work.  A stage is SG consecutive groups of a 256-row tile.
// Lane (g, c) of a warp (g = lane / 4, c = lane % 4) owns, for the rows of
// its MMA fragment (rows g and g + 8 of each of the warp's m16 tiles), the
// aligned window words covering its groups:
//  * one token, SG = 8: groups 2c and 2c + 1, the 13 words (52 bytes) at
//    byte 52c of the stage row;
//  * two tokens, SG = 4: group c, the 7 words that cover its 26 bytes (2
//    bytes of a neighbouring group ride along with zero activations).
// In one m16n8k16 MMA every lane of a row therefore contributes products of
// different groups, and the MMA's 8 columns keep them apart: column 2c + h
// collects the lane position c's slice h (its group 2c + h for one token,
// token h of its group for two).  Lane (g', c) holds the activation slots of
// column g' (B's column): real when g' = 2c + h, zero otherwise, so each
// column receives exactly its own products; the accumulator fragment of
// lane (g, c) then holds rows g, g + 8 x columns 2c, 2c + 1, which are
// exactly the lane's own slices, and every lane applies its own s1 / off.
// Compared with one group at a time (the general decode kernel), no MMA slot
// is spent on padding 26-byte groups to 32-byte windows, and the per-group
// epilogue runs on all lanes.
//
// Operand encoding (five MMA slots per packed byte): the byte v = sum_i d_i
// 3^i (d_i = trit + 1) gives, through the lane-replicated table, W = (4 +
// d0 + d2/4, 4 + d1 + d3/4), then W' = (16 + d2, 16 + d3) by one LOP3 and
// the fifth slot 4 + v/256 by one PRMT for two bytes; the activation slots
// written by the prep kernel make the MMA return const + sum_i d_i x_i, and
// the accumulator starts at -const (C), so that it ends at sum_i t_i x_i.
// A word of 4 bytes gives 10 registers (W, W' of each byte, then the two
// fifth-slot words), i.e. 5 MMAs per m16 tile.
//
// Roles: the decode warps multiply their rows; the last warp moves every
// stage into a ring of shared-memory slots (2 of 8 groups or 4 of 4
// groups): the tile's plane-1 bytes (one 2-D tensor copy per stage, 208 x
// 256 bytes; with 4-group stages 112 x 256, odd stages copied from 8 bytes
// before their 16-byte-misaligned start), the stage's activation slots and
// C / S (bulk copies) and s1 / off (tensor copies of the 8-group box that
// holds the stage, or plain loads when rows of scales are not whole 16-byte
// units).  Every wait is bounded (tq_sm100.cuh).
#include <cuda.h>

#include <algorithm>

#include "tq_common.cuh"
#include "tq_decode_ops.cuh"
#include "tq_p2_tile.cuh"
#include "tq_sm100.cuh"

namespace tq {
namespace g4 {

using mm::kArena1;
using mm::kArena2;
using mm::kDynBytes;
using mm::kDynShared;
using mm::kLutBytes;
using mm::kLutShared;

// decode warps and m16 tiles per decode warp (x 16 = 256 rows): sixteen
// warps of one tile each, with the activation loads of the lanes that hold
// zero columns left out (measured 0.542 ms per Qwen3-8B step against 0.557
// for eight warps of two tiles sharing each load, and 0.554 for sixteen
// warps loading on every lane)
constexpr int kWD1 = 16, kTL1 = 1;
constexpr int kWD2 = 16, kTL2 = 1;
constexpr int kA2 = kArena1 + kLutBytes;  // dynamic-smem offset of arena 2 (above the table)

// Shared-memory layout of the stage ring for SG groups per stage.
//  Arena 1 (below the table): the first N1 plane-1 slots, the barriers, the
//  zero activation block and the C/S slots.  Arena 2 (above the table): the
//  other plane-1 slots, the s1/off slots (s1 then off, 8 groups of fp16 per
//  row) and the activation slots (two slices per stage).
//  Bank placement of the 16-byte activation loads: such a load is served a
//  quarter-warp at a time, and quarter q (lanes g = 2q, 2q + 1) holds the
//  real slots of lane position q: slice 0 in 16-byte bank group q of a
//  128-byte line, slice 1 (kSlice apart) in group q + 4, so the two never
//  share banks.  The lanes of zero columns load nothing (their registers
//  stay zero) and the zero block is not read; it keeps the C/S slots at
//  the offset measured fastest (without it the one-token step took 0.25 %
//  longer).
template <int SG>
struct Cfg {
  static constexpr int kStageBytes = 26 * SG;              // plane-1 bytes per row per stage
  static constexpr int kBox = SG == 8 ? 208 : 112;         // bytes per row copied (and the shared row stride)
  static constexpr int kWords = words(SG);                 // window words per lane and row
  static constexpr int kPairs = pairs(SG);
  static constexpr int kSliceG = slice_bytes(SG);          // one slice in the workspace
  static constexpr int kSlice = kSliceG + (kSliceG % 128 == 64 ? 0 : 64);  // in shared memory
  static constexpr int kNS = SG == 8 ? 2 : 4;              // stage slots
  static constexpr int kN1 = SG == 8 ? 1 : 2;              // plane-1 slots in arena 1
  static constexpr int kP1Slot = kRows * kBox;
  static constexpr int kSOHalf = kRows * 16;
  static constexpr int kSOSlot = 2 * kSOHalf;
  static constexpr int kOffBars = kN1 * kP1Slot;
  static constexpr int kOffZero = kOffBars + 256;
  static constexpr int kZeroBytes = kSliceG + 128;
  static constexpr int kOffCS = kOffZero + kZeroBytes;
  static constexpr int kEnd1 = kOffCS + kNS * kCSStage;
  static constexpr int kOffSO = (kNS - kN1) * kP1Slot;     // in arena 2
  static constexpr int kOffB = kOffSO + kNS * kSOSlot;
  static constexpr int kEnd2 = kOffB + kNS * 2 * kSlice;
  static_assert(kEnd1 <= kArena1, "arena 1 overflow");
  static_assert(kEnd2 <= kArena2, "arena 2 overflow");
  static_assert(kSlice % 128 == 64 && (2 * kSlice) % 128 == 0, "slice bank placement");
  static_assert(2 * kPairs >= 5 * kWords, "activation chunks cover the MMAs of a stage");
  __device__ static int p1_off(int b) { return b < kN1 ? b * kP1Slot : kA2 + (b - kN1) * kP1Slot; }
};

struct Bars {
  uint64_t full[4], empty[4];
  int32_t abort_;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

// Schedule: CTA c processes global work units [cta_unit[c], cta_unit[c+1]).
// A unit is one 256-row tile's stages [k nst / u, (k + 1) nst / u), the
// tile cut into u = min(nst, ceil(G / split)) parts for a target of `split`
// groups per unit (split = 0: u = 1, whole tiles); units are numbered over
// the problems in order, tile-major.
struct Sched {
  int32_t cta_unit[257];
  int32_t split;
};
__host__ __device__ inline int unit_parts(int K, int SG, int split) {
  const int G = K / kGroup, nst = nstages(K, SG);
  return split > 0 ? min(nst, max(1, (G + split - 1) / split)) : 1;
}

template <int SG>
struct Walk {
  const BatchParams *bp;
  int split, unit, u_end, pi, ub, u, nst, tile, s, s_end;
  __device__ int parts(int p) const { return unit_parts(bp->prob[p].K, SG, split); }
  __device__ void locate() {
    for (;;) {
      const int U = (bp->prob[pi].N + kRows - 1) / kRows * parts(pi);
      if (unit < ub + U) break;
      ub += U;
      ++pi;
    }
    u = parts(pi);
    nst = nstages(bp->prob[pi].K, SG);
    const int local = unit - ub, k = local % u;
    tile = local / u;
    s = k * nst / u;
    s_end = (k + 1) * nst / u;
  }
  __device__ Walk(const BatchParams *b, int sp, int u0, int u1)
      : bp(b), split(sp), unit(u0), u_end(u1), pi(0), ub(0), u(1), nst(0), tile(0), s(0), s_end(0) {
    if (unit < u_end) locate();
  }
  __device__ bool valid() const { return unit < u_end; }
  __device__ const Problem &P() const { return bp->prob[pi]; }
  __device__ int n0() const { return tile * kRows; }
  __device__ bool last_stage() const { return s + 1 == s_end; }  // of this unit
  __device__ bool shared_tile() const { return u > 1; }
  __device__ void next() {
    if (++s < s_end) return;
    if (++unit < u_end) locate();
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

// The activation registers of an MMA pair: a 16-byte shared-memory load by
// the lanes that hold real slots; the other lanes leave r as it is (zero
// from the start of the kernel), so no register needs clearing.
__device__ __forceinline__ void ld_b_real(uint32_t (&r)[4], const unsigned char *addr, bool real) {
  asm volatile(
      "{\n.reg .pred p;\nsetp.ne.b32 p, %5, 0;\n@p ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];\n}"
      : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3])
      : "r"(smem_u32(addr)), "r"((uint32_t)real));
}
constexpr int kBSets = 4;  // activation register sets (pairs p, p + 1, ... in rotation)

// Workspace addresses of a problem's activation slots and C/S (after the
// general decode path's 512-byte map slot).
__device__ __forceinline__ const unsigned char *ws_b(const Problem &P) { return P.wsB + P.map_off + 512; }
__device__ __forceinline__ const unsigned char *ws_cs(const Problem &P, int MB) {
  return ws_b(P) + pad256(b_bytes(MB, P.K));
}
__device__ __forceinline__ int32_t *ws_tickets(const Problem &P, int MB) {
  return reinterpret_cast<int32_t *>(const_cast<unsigned char *>(ws_cs(P, MB)) + pad256(cs_bytes(MB, P.K)));
}

// Set-up shared by the kernels below: the lane-replicated table, the zero
// activation block, the stage barriers.
template <int SG, int WD>
__device__ __forceinline__ void setup_cta(unsigned char *dyn, int tid, int nthreads) {
  using C = Cfg<SG>;
  Bars *bars = reinterpret_cast<Bars *>(dyn + C::kOffBars);
  uint32_t *lut = reinterpret_cast<uint32_t *>(dyn + kArena1);
  mm::lut_fill_replicated(lut, tid, nthreads);
  for (int i = tid; i < C::kZeroBytes / 16; i += nthreads)
    reinterpret_cast<uint4 *>(dyn + C::kOffZero)[i] = make_uint4(0u, 0u, 0u, 0u);
  if (tid == 0) {
    for (int i = 0; i < C::kNS; ++i) {
      mbar_init(&bars->full[i], 1 + 32);  // the producer's expect-tx arrival + its 32 lanes' arrivals
      mbar_init(&bars->empty[i], WD);
    }
    bars->abort_ = 0;
    mbar_fence_init();
  }
}

// One stage in slot buf for a decode warp: the MMAs of its TL m16 tiles
// over the stage's window words, then s1 / off of the lane's groups added to
// y[tile][half][token].  (rA: the warp's first row of the lane; wb: the
// lane's first window byte; realB: whether the lane holds real activation
// slots; tag: table base | lane * 4.)
template <int MB, int SG, int TL>
__device__ __forceinline__ void decode_stage(const unsigned char *dyn, int buf, int s, int rA, int wb, int c, int g,
                                             bool realB, uint32_t tag, uint32_t (&bz)[kBSets][4], float (&y)[TL][2][MB]) {
  using C = Cfg<SG>;
  const int shift = SG == 8 ? 0 : 8 * (s & 1);  // odd 4-group stages are copied from 8 bytes early
  const unsigned char *p1 = dyn + C::p1_off(buf) + shift + wb + rA * C::kBox;
  const unsigned char *bq =
      dyn + (realB ? kA2 + C::kOffB + (buf * 2 + (g & 1)) * C::kSlice + c * 16 : C::kOffZero + 16 * ((g >> 1) + 2));
  const float4 cs = *reinterpret_cast<const float4 *>(dyn + C::kOffCS + buf * kCSStage + c * 16);
  // accumulators start at -C (slice 0 in columns 2c, slice 1 in 2c + 1)
  // one accumulator chain per MMA position m of a word (five chains), so
  // that an MMA waits for the result of the one five places earlier only
  // (0.500 ms per Qwen3-8B step, against 0.513 with two chains by word and
  // 0.517 with one; ten chains exceed the 96 registers a thread may hold
  // with 17 warps, five of them on one scheduler)
  float d2[TL][5][4];
#pragma unroll
  for (int t = 0; t < TL; ++t) {
    d2[t][0][0] = d2[t][0][2] = -cs.x, d2[t][0][1] = d2[t][0][3] = -cs.y;
#pragma unroll
    for (int k = 1; k < 5; ++k) d2[t][k][0] = d2[t][k][1] = d2[t][k][2] = d2[t][k][3] = 0.f;
  }
#pragma unroll
  for (int i = 0; i < C::kWords; ++i) {
    uint32_t a[TL][2][10];
#pragma unroll
    for (int t = 0; t < TL; ++t)
#pragma unroll
      for (int h = 0; h < 2; ++h)
        decode_word(*reinterpret_cast<const uint32_t *>(p1 + (16 * t + 8 * h) * C::kBox + 4 * i), tag, a[t][h]);
#pragma unroll
    for (int m = 0; m < 5; ++m) {
      const int j = 5 * i + m;
      // lanes of zero columns keep zero registers (no shared-memory
      // traffic); the registers are never cleared, as a predicated load into
      // a fresh value would cost a clearing move per MMA (one token: 0.518
      // ms per Qwen3-8B step against 0.541; two tokens: 0.626 against 0.640
      // with the zero lanes loading a zero block)
      uint32_t b0, b1;
      {
        uint32_t(&r)[4] = bz[(j >> 1) % kBSets];
        if ((j & 1) == 0) ld_b_real(r, bq + (j >> 1) * 64, realB);
        b0 = (j & 1) ? r[2] : r[0], b1 = (j & 1) ? r[3] : r[1];
      }
#pragma unroll
      for (int t = 0; t < TL; ++t)
        mm::mma16816(d2[t][m], a[t][0][2 * m], a[t][1][2 * m], a[t][0][2 * m + 1], a[t][1][2 * m + 1], b0, b1);
    }
  }
  float d[TL][4];
#pragma unroll
  for (int t = 0; t < TL; ++t)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      d[t][e] = d2[t][0][e];
#pragma unroll
      for (int k = 1; k < 5; ++k) d[t][e] += d2[t][k][e];
    }
  // s1 / off of (row, the lane's groups): the slot holds 8 groups per row
  // (both halves of an 8-group stage; an odd 4-group stage's at 4)
  const unsigned char *so = dyn + kA2 + C::kOffSO + buf * C::kSOSlot;
#pragma unroll
  for (int t = 0; t < TL; ++t) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = rA + 16 * t + 8 * h;
      if (SG == 8) {
        // groups 2c, 2c + 1 (columns 2c, 2c + 1) of the one token
        const __half2 s1 = *reinterpret_cast<const __half2 *>(so + r * 16 + 4 * c);
        const __half2 of = *reinterpret_cast<const __half2 *>(so + C::kSOHalf + r * 16 + 4 * c);
        float v = fmaf(__low2float(of), cs.z, y[t][h][0]);
        v = fmaf(__high2float(of), cs.w, v);
        v = fmaf(__low2float(s1), d[t][2 * h], v);
        y[t][h][0] = fmaf(__high2float(s1), d[t][2 * h + 1], v);
      } else {
        // group c, tokens 0 and 1 (columns 2c, 2c + 1)
        const int gl = 2 * (4 * (s & 1) + c);
        const float s1 = __half2float(*reinterpret_cast<const __half *>(so + r * 16 + gl));
        const float of = __half2float(*reinterpret_cast<const __half *>(so + C::kSOHalf + r * 16 + gl));
        y[t][h][0] = fmaf(s1, d[t][2 * h], fmaf(of, cs.z, y[t][h][0]));
        y[t][h][MB - 1] = fmaf(s1, d[t][2 * h + 1], fmaf(of, cs.w, y[t][h][MB - 1]));
      }
    }
  }
}

// The sum over the four lane positions of each row (every lane of a quad
// then holds it).
template <int MB, int TL>
__device__ __forceinline__ void quad_sum(float (&y)[TL][2][MB]) {
#pragma unroll
  for (int t = 0; t < TL; ++t)
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int k = 0; k < MB; ++k) {
        float v = y[t][h][k];
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 2);
        y[t][h][k] = v;
      }
}

// The producer's copies of stage s of the tile at row n0 of problem P into
// slot buf (after the slot's empty wait), ending with the lanes' arrivals on
// its full barrier.  map_pi: the problem whose tensor maps were last
// acquired (the fence is needed once per problem).
template <int MB, int SG>
__device__ __forceinline__ void produce_stage(unsigned char *dyn, Bars *bars, int buf, const Problem &P, int pi,
                                              int &map_pi, int s, int n0, int lane) {
  using C = Cfg<SG>;
  constexpr int kNSl = SG == 8 ? 2 : MB;
  const int G = P.K / kGroup;
  uint64_t *full = &bars->full[buf];
  // s1 / off go by tensor copies when their rows are whole 16-byte units
  // (the prep kernel then built their maps), else by asynchronous copies or
  // plain loads
  const bool so_map = (G % 8 == 0) && ((((uintptr_t)P.s1) | ((uintptr_t)P.off)) & 15u) == 0;
  unsigned char *so = dyn + kA2 + C::kOffSO + buf * C::kSOSlot;
  const unsigned char *maps = static_cast<const unsigned char *>(P.map());
  const int g8 = SG == 8 ? s : s >> 1;  // the 8-group box holding the stage
  if (lane == 0) {
    if (pi != map_pi) {
      // the problem's tensor maps, written by the prep kernel
      asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps) : "memory");
      if (so_map) {
        asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps + 128) : "memory");
        asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps + 256) : "memory");
      }
      map_pi = pi;
    }
    mbar_arrive_expect_tx(full, (uint32_t)(C::kP1Slot + kNSl * C::kSliceG + kCSStage) +
                                    (so_map ? (uint32_t)C::kSOSlot : 0u));
    // the stage's plane-1 bytes of the tile's 256 rows from the 16-byte
    // boundary at or before them (rows past N and bytes past the row's end
    // arrive as zeros)
    const int x = SG == 8 ? C::kStageBytes * s : C::kStageBytes * s - 8 * (s & 1);
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_u32(dyn + C::p1_off(buf))),
        "l"(maps), "r"(x), "r"(n0), "r"(smem_u32(full))
        : "memory");
#pragma unroll
    for (int sl = 0; sl < kNSl; ++sl)
      bulk_g2s(dyn + kA2 + C::kOffB + (buf * 2 + sl) * C::kSlice, ws_b(P) + ((int64_t)s * 2 + sl) * C::kSliceG,
               C::kSliceG, full);
    bulk_g2s(dyn + C::kOffCS + buf * kCSStage, ws_cs(P, MB) + (int64_t)s * kCSStage, kCSStage, full);
    if (so_map) {
      asm volatile(
          "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
              smem_u32(so)),
          "l"(maps + 128), "r"(8 * g8), "r"(n0), "r"(smem_u32(full))
          : "memory");
      asm volatile(
          "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
              smem_u32(so + C::kSOHalf)),
          "l"(maps + 256), "r"(8 * g8), "r"(n0), "r"(smem_u32(full))
          : "memory");
    }
  }
  __syncwarp();
  const int col0 = SG == 8 ? 0 : 4 * (s & 1);  // the stage's first column in the 8-group slot rows
  if (!so_map && G % 4 == 0 && ((((uintptr_t)P.s1) | ((uintptr_t)P.off)) & 7u) == 0) {
    // rows of scales in whole 8-byte units (G a multiple of 4): 8-byte
    // asynchronous copies of each 4-group half of the stage (zero-filled
    // past G or N); each lane's arrival waits for its own copies
    const int rows = min(kRows, P.N - n0);
    for (int r = lane; r < kRows; r += 32) {
#pragma unroll
      for (int hh = 0; hh < SG / 4; ++hh) {
        const int gi = SG * s + 4 * hh;
        const bool real = r < rows && gi < G;
        const int64_t o = real ? (int64_t)(n0 + r) * G + gi : 0;
        const uint32_t dst = smem_u32(so + r * 16 + 2 * (col0 + 4 * hh));
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(P.s1 + o), "r"(real ? 8 : 0)
                     : "memory");
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst + C::kSOHalf), "l"(P.off + o),
                     "r"(real ? 8 : 0)
                     : "memory");
      }
    }
    cp_async_mbar_arrive_noinc(full);  // the lane's arrival, once its copies have landed
  } else {
    if (!so_map) {
      // other shapes: the stage's groups of s1 and off one by one (zeros
      // past G or N) at their place in each row's 8-group slot
      const int rows = min(kRows, P.N - n0);
      __half *d1 = reinterpret_cast<__half *>(so), *d2 = reinterpret_cast<__half *>(so + C::kSOHalf);
      for (int r = lane; r < rows; r += 32) {
        const int64_t o = (int64_t)(n0 + r) * G;
#pragma unroll
        for (int gg = 0; gg < SG; ++gg) {
          const int gi = SG * s + gg;
          d1[r * 8 + col0 + gg] = gi < G ? P.s1[o + gi] : __float2half_rn(0.f);
          d2[r * 8 + col0 + gg] = gi < G ? P.off[o + gi] : __float2half_rn(0.f);
        }
      }
    }
    mbar_arrive(full);  // the lanes' arrivals (the barrier counts 1 + 32)
  }
}

// WD decode warps with TL m16 tiles each (WD x TL x 16 = 256 rows), and one
// producer warp; SG groups per stage (8 for one token, 4 for two).
template <bool F32, int MB, int SG, int WD, int TL>
__global__ void __launch_bounds__((WD + 1) * 32, 1)
    gemv_g4_kernel(const __grid_constant__ BatchParams bp, const __grid_constant__ Sched sc) {
  using C = Cfg<SG>;
  static_assert(WD * TL * 16 == kRows && WD <= kMaxWarps, "decode warps cover the tile");
  static_assert((SG == 8 && MB == 1) || (SG == 4 && MB == 2), "stage shape per token count");
  constexpr int kNS = C::kNS;
  extern __shared__ __align__(1024) unsigned char dyn[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (smem_u32(dyn) != kDynShared) {
    // the table address trick needs the dynamic window right after the
    // reserved 1 KiB of shared memory; anything else is reported
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  Bars *bars = reinterpret_cast<Bars *>(dyn + C::kOffBars);
  volatile int32_t *abort_ = &bars->abort_;
  setup_cta<SG, WD>(dyn, tid, (WD + 1) * 32);
  __syncthreads();
  // everything below reads what the prep and second-plane kernels wrote
  grid_dep_wait();
  // a programmatically launched successor (the next call's prep kernel)
  // may be scheduled now; it waits for this grid before touching memory
  grid_dep_launch_next();
  const int t_begin = sc.cta_unit[blockIdx.x], t_end = sc.cta_unit[blockIdx.x + 1];

  if (warp < WD) {
    // ============================================================ decode
    // warp w owns rows rA + 16 t and rA + 16 t + 8 of its TL m16 tiles t
    const int g = lane >> 2, c = lane & 3;
    const uint32_t tag = kLutShared | ((uint32_t)lane << 2);
    // first window word of the lane's groups in the stage row: 8-group
    // stages at byte 52c; 4-group stages the word holding byte 26c (words
    // 0, 6, 13, 19)
    const int wb = SG == 8 ? 52 * c : 4 * ((c * 13) >> 1);
    const int rA = 16 * TL * warp + g;
    // activation slots: this lane's column is slice g & 1 of lane position g >> 1
    const bool realB = ((g >> 1) == c) && ((g & 1) < (SG == 8 ? 2 : MB));
    float y[TL][2][MB];
#pragma unroll
    for (int t = 0; t < TL; ++t)
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int k = 0; k < MB; ++k) y[t][h][k] = 0.f;
    uint32_t bz[kBSets][4] = {};  // activation registers (zero-column lanes: zero throughout)
    uint32_t buf = 0, phase = 0;
    for (Walk<SG> w(&bp, sc.split, t_begin, t_end); w.valid(); w.next()) {
      const bool ok = __all_sync(0xffffffffu, mm::wait_or_abort(&bars->full[buf], phase, abort_));
      if (!ok) break;
      decode_stage<MB, SG, TL>(dyn, (int)buf, w.s, rA, wb, c, g, realB, tag, bz, y);
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->empty[buf]);
      if (w.last_stage()) {
        // sum the four lane positions of each row, add the second plane,
        // write y: the quad's rows (t, h) go to lanes c = (2 t + h) mod 4
        quad_sum<MB, TL>(y);
        const Problem &P = w.P();
        auto store = [&](int n, int k, float v) {
          if (F32)
            static_cast<float *>(P.y)[(int64_t)k * P.N + n] = v;
          else
            static_cast<__half *>(P.y)[(int64_t)k * P.N + n] = __float2half_rn(v);
        };
        if (!w.shared_tile()) {
          // the whole tile was this CTA's: write y (+ the second plane)
#pragma unroll
          for (int t = 0; t < TL; ++t)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int n = w.n0() + rA + 16 * t + 8 * h;
              if (((2 * t + h) & 3) == c && n < P.N) {
#pragma unroll
                for (int k = 0; k < MB; ++k) store(n, k, y[t][h][k] + (P.nnz > 0 ? P.y2()[(int64_t)n * MB + k] : 0.f));
              }
            }
        } else {
          // a share of the tile's stages: add the partial sums into y2 (fp32
          // atomics, zeroed by the prep kernel); the last of the tile's
          // units to arrive for this warp's rows writes them
#pragma unroll
          for (int t = 0; t < TL; ++t)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int n = w.n0() + rA + 16 * t + 8 * h;
              if (((2 * t + h) & 3) == c && n < P.N) {
#pragma unroll
                for (int k = 0; k < MB; ++k) atomicAdd(P.y2() + (int64_t)n * MB + k, y[t][h][k]);
              }
            }
          __threadfence();
          __syncwarp();
          int last = 0;
          if (lane == 0) last = atomicAdd(ws_tickets(P, MB) + w.tile * kMaxWarps + warp, 1) == w.u - 1;
          if (__shfl_sync(0xffffffffu, last, 0)) {
            __threadfence();
#pragma unroll
            for (int t = 0; t < TL; ++t)
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const int n = w.n0() + rA + 16 * t + 8 * h;
                if (((2 * t + h) & 3) == c && n < P.N) {
#pragma unroll
                  for (int k = 0; k < MB; ++k) store(n, k, __ldcg(P.y2() + (int64_t)n * MB + k));
                }
              }
          }
        }
#pragma unroll
        for (int t = 0; t < TL; ++t)
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int k = 0; k < MB; ++k) y[t][h][k] = 0.f;
      }
      if (++buf == (uint32_t)kNS) buf = 0, phase ^= 1u;
    }
  } else if (warp == WD) {
    // ========================================================== producer
    uint32_t buf = 0, phase = 0, q = 0;
    int map_pi = -1;
    for (Walk<SG> w(&bp, sc.split, t_begin, t_end); w.valid(); w.next(), ++q) {
      int ok = 1;
      if (lane == 0) ok = mm::wait_or_abort(&bars->empty[buf], phase ^ 1u, abort_) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;  // uniform across the warp
      produce_stage<MB, SG>(dyn, bars, (int)buf, w.P(), w.pi, map_pi, w.s, w.n0(), lane);
      if (++buf == (uint32_t)kNS) buf = 0, phase ^= 1u;
    }
    // drain: every issued copy lands before the CTA exits (waited on even
    // after an abort; bounded by the wall-time limit)
    mm::cp_async_wait<0>();
    if (lane == 0) {
      for (uint32_t k = (q > (uint32_t)kNS ? q - kNS : 0); k < q; ++k) mbar_wait(&bars->full[k % kNS], (k / kNS) & 1u);
    }
  }
  __syncthreads();
}

// ------------------------------------------------------------ sequence
// Dependency-ordered sequence of problems (one token): problem p + 1 starts
// only after every CTA has finished problem p, as the layers of a model need
// (q/k/v, then o, then gate/up, then down, layer after layer; the attention,
// norms and activation between them are outside this library).  One
// persistent launch: for each problem every CTA takes its share of the
// second-plane tiles and then of the 256-row tiles' stage units (tiles cut so
// that the problem's units cover the CTAs), adding everything into y2 (fp32
// atomics, zeroed by the prep kernel); a grid-wide barrier (a counter in the
// workspace, bounded by the wall-time limit) ends the problem, after which
// every CTA converts its slice of y2 into y.  The producer warp streams the
// stages without waiting at the barriers (weights do not depend on earlier
// problems).  barrier_extra > 0 makes every barrier wait for CTAs that do not
// exist, so that its bounded wait runs out (the failure-path self-test).
struct SeqWalk {
  const BatchParams *bp;
  int cta, ctas, p, unit, u_end, u, nst, tile, s, s_end;
  __device__ void enter() {
    const Problem &P = bp->prob[p];
    const int G = P.K / kGroup, tiles = (P.N + kRows - 1) / kRows;
    const int64_t share = ((int64_t)tiles * G + ctas - 1) / ctas;
    const int split = share >= G ? 0 : (int)(share < 1 ? 1 : share);
    u = unit_parts(P.K, 8, split);
    nst = nstages(P.K, 8);
    const int64_t U = (int64_t)tiles * u;
    unit = (int)(U * cta / ctas);
    u_end = (int)(U * (cta + 1) / ctas);
    if (unit < u_end) locate();
  }
  __device__ void locate() {
    tile = unit / u;
    const int k = unit - tile * u;
    s = k * nst / u;
    s_end = (k + 1) * nst / u;
  }
  __device__ SeqWalk(const BatchParams *b, int c, int n) : bp(b), cta(c), ctas(n), p(0), unit(0), u_end(0) { enter(); }
  __device__ const Problem &P() const { return bp->prob[p]; }
  __device__ bool has_stage() const { return unit < u_end; }
  __device__ bool unit_end() const { return s + 1 == s_end; }
  __device__ int n0() const { return tile * kRows; }
  __device__ void next_stage() {
    if (++s < s_end) return;
    if (++unit < u_end) locate();
  }
  __device__ bool next_problem() {
    if (++p >= bp->count) return false;
    enter();
    return true;
  }
};

__device__ __forceinline__ int ld_acquire(const int32_t *p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// A decode warp's share of problem P's second-plane tiles (one token): the
// CTA's contiguous share of the index's 16-entry tiles, cut among the WD
// decode warps; runs of tiles of one group go through mm::p2_tiles with the
// group's activation fragment of the per-group layout.
template <int WD>
__device__ __forceinline__ void second_plane_share(const Problem &P, int cta, int ctas, int warp, int lane,
                                                   uint32_t tag) {
  const int G = P.K / kGroup, c = lane & 3;
  const int T2 = __ldg(P.p2idx + G) >> 4;  // tiles (group starts are multiples of 16 entries)
  const int lo = (int)((int64_t)T2 * cta / ctas), hi = (int)((int64_t)T2 * (cta + 1) / ctas);
  const int wlo = lo + (hi - lo) * warp / WD, whi = lo + (hi - lo) * (warp + 1) / WD;
  for (int t = wlo; t < whi;) {
    // the tile's group: the last g with colptr[g] <= 16 t
    int g = 0;
    for (int step = 1 << (31 - __clz(G)); step >= 1; step >>= 1)
      if (g + step < G && __ldg(P.p2idx + g + step) <= 16 * t) g += step;
    const int64_t e0 = __ldg(P.p2idx + g);
    const int n = min(whi, __ldg(P.p2idx + g + 1) >> 4) - t;
    if (n <= 0) break;  // malformed index: stop rather than loop
    const unsigned char *Bg = P.wsB + (int64_t)g * mm::kBTok + c * mm::kBLane;
    uint32_t b[20];
#pragma unroll
    for (int cp = 0; cp < mm::kCP; ++cp) {
      const uint4 v = __ldg(reinterpret_cast<const uint4 *>(Bg + cp * 4 * mm::kBLane));
      b[4 * cp] = v.x, b[4 * cp + 1] = v.y, b[4 * cp + 2] = v.z, b[4 * cp + 3] = v.w;
    }
    const float2 Cv = __ldg(reinterpret_cast<const float2 *>(P.wsCS + (int64_t)g * (mm::kCSGroup / 4)));
    mm::p2_tiles<true, false>(P, 1, g % mm::kStageG, e0, t - (int)(e0 >> 4), n, b, b, Cv, Cv, lane, tag);
    t += n;
  }
}

// The CTA's share of problem P's second-plane records (the tiles that
// second_plane_share gives it) into L2, one bulk prefetch: they are weights,
// so they can be fetched while the problem before P still runs.
__device__ __forceinline__ void prefetch_second_plane(const Problem &P, int cta, int ctas) {
  const int G = P.K / kGroup;
  const int T2 = __ldg(P.p2idx + G) >> 4;
  const int lo = (int)((int64_t)T2 * cta / ctas), hi = (int)((int64_t)T2 * (cta + 1) / ctas);
  if (hi <= lo) return;
  const unsigned char *slots = reinterpret_cast<const unsigned char *>(P.p2idx) + mm::c_slot_off(P.K);
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(slots + (int64_t)lo * 512),
               "r"((uint32_t)(hi - lo) * 512u)
               : "memory");
}

template <bool F32>
__global__ void __launch_bounds__((kWD1 + 1) * 32, 1)
    gemv_seq_kernel(const __grid_constant__ BatchParams bp, int32_t barrier_extra) {
  constexpr int SG = 8, MB = 1, WD = kWD1, TL = kTL1;
  using C = Cfg<SG>;
  constexpr int kNS = C::kNS;
  extern __shared__ __align__(1024) unsigned char dyn[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (smem_u32(dyn) != kDynShared) {
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  Bars *bars = reinterpret_cast<Bars *>(dyn + C::kOffBars);
  volatile int32_t *abort_ = &bars->abort_;
  setup_cta<SG, WD>(dyn, tid, (WD + 1) * 32);
  __syncthreads();
  grid_dep_wait();  // the prep kernel's operands, maps, zeroed y2 and counter
  int32_t *counter = reinterpret_cast<int32_t *>(static_cast<unsigned char *>(bp.prob[0].map()) + 448);

  if (warp < WD) {
    // ============================================================ decode
    const int g = lane >> 2, c = lane & 3;
    const uint32_t tag = kLutShared | ((uint32_t)lane << 2);
    const int wb = 52 * c, rA = 16 * TL * warp + g;
    const bool realB = (g >> 1) == c;
    float y[TL][2][MB];
#pragma unroll
    for (int t = 0; t < TL; ++t) y[t][0][0] = y[t][1][0] = 0.f;
    uint32_t bz[kBSets][4] = {};
    uint32_t buf = 0, phase = 0;
    SeqWalk w(&bp, blockIdx.x, gridDim.x);
    for (bool more = true; more; more = w.next_problem()) {
      const Problem &P = w.P();
      if (warp == 0 && lane == 0 && w.p + 1 < bp.count && bp.prob[w.p + 1].nnz > 0)
        prefetch_second_plane(bp.prob[w.p + 1], blockIdx.x, gridDim.x);
      if (P.nnz > 0) second_plane_share<WD>(P, blockIdx.x, gridDim.x, warp, lane, tag);
      bool ok = true;
      for (; w.has_stage(); w.next_stage()) {
        ok = __all_sync(0xffffffffu, mm::wait_or_abort(&bars->full[buf], phase, abort_));
        if (!ok) break;
        decode_stage<MB, SG, TL>(dyn, (int)buf, w.s, rA, wb, c, g, realB, tag, bz, y);
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->empty[buf]);
        if (w.unit_end()) {
          quad_sum<MB, TL>(y);
#pragma unroll
          for (int t = 0; t < TL; ++t)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int n = w.n0() + rA + 16 * t + 8 * h;
              if (((2 * t + h) & 3) == c && n < P.N) atomicAdd(P.y2() + n, y[t][h][0]);
              y[t][h][0] = 0.f;
            }
        }
        if (++buf == (uint32_t)kNS) buf = 0, phase ^= 1u;
      }
      // the problem's barrier: every CTA's additions into y2 are done
      named_bar(1, WD * 32);
      if (warp == 0 && lane == 0 && ok && !*abort_) {
        __threadfence();
        atomicAdd(counter, 1);
        const int target = (w.p + 1) * ((int)gridDim.x + barrier_extra);
        const uint64_t t0 = global_ns();
        while (ld_acquire(counter) < target) {
          if (*abort_) break;
          if (global_ns() - t0 > kWaitLimitNs) {
            atomicOr(&g_tq_device_status, kStatusTimeout);
            *abort_ = 1;
            break;
          }
          __nanosleep(32);  // 1.603 ms per Qwen3-8B step against 1.610 with 128 ns (spinning: 1.611)
        }
        __threadfence();
      }
      // stop together: the flag may be raised (by the producer) while
      // the warps read it, so they decide by one reduction over the barrier
      if (named_bar_any(1, WD * 32, *abort_ != 0)) break;
      // this CTA's slice of the problem's output
      const int r0 = (int)((int64_t)P.N * blockIdx.x / gridDim.x), r1 = (int)((int64_t)P.N * (blockIdx.x + 1) / gridDim.x);
      for (int n = r0 + warp * 32 + lane; n < r1; n += WD * 32) {
        const float v = __ldcg(P.y2() + n);
        if (F32)
          static_cast<float *>(P.y)[n] = v;
        else
          static_cast<__half *>(P.y)[n] = __float2half_rn(v);
      }
    }
  } else if (warp == WD) {
    // ========================================================== producer
    uint32_t buf = 0, phase = 0, q = 0;
    int map_pi = -1;
    SeqWalk w(&bp, blockIdx.x, gridDim.x);
    bool ok = true;
    for (bool more = true; more && ok; more = w.next_problem()) {
      for (; w.has_stage(); w.next_stage(), ++q) {
        int r = 1;
        if (lane == 0) r = mm::wait_or_abort(&bars->empty[buf], phase ^ 1u, abort_) ? 1 : 0;
        if (!__shfl_sync(0xffffffffu, r, 0)) {
          ok = false;
          break;
        }
        produce_stage<MB, SG>(dyn, bars, (int)buf, w.P(), w.p, map_pi, w.s, w.n0(), lane);
        if (++buf == (uint32_t)kNS) buf = 0, phase ^= 1u;
      }
    }
    mm::cp_async_wait<0>();
    if (lane == 0) {
      for (uint32_t k = (q > (uint32_t)kNS ? q - kNS : 0); k < q; ++k) mbar_wait(&bars->full[k % kNS], (k / kNS) & 1u);
    }
  }
  __syncthreads();
}

// ------------------------------------------------- second plane, one token
// The second plane of one token with the group-ordered index, in the first
// plane's one-group-per-lane layout: an m16 tile takes, for each of the 8
// groups of one stage, 16 consecutive entries of that group (group 2c + h
// of the stage in MMA column 2c + h).  Lane (r, c) loads the slots of
// entries r and r + 8 of the stage's groups 2c (record at slot byte 0) and
// 2c + 1 (record at byte 2): the even record's words 0..5, one PRMT of its
// word 6 with the odd record's word 0, then the odd record's words 1..6 are
// the 13 window words of an 8-group stage row, so the decode and the B
// operands (the stage's activation slices, copied per unit into the warp's
// shared-memory slot) are the first plane's.  The accumulator fragment of lane (r, c) then holds the
// dot products of exactly its own four records, each added as s2 (D - C)
// to y2 of the record's row (fp32 atomics; the prep kernel zeroes y2).
// Warps take units (problem, stage, share of the stage's tiles) from a
// counter in the workspace.
// Shared memory per warp: its unit's two activation slices; the first
// kP2rLow warps use the space below the table, the others the space above it.
constexpr int kP2rWarps = 20;
// activation register sets and accumulator chains: two sets free the
// registers for three chains within the 96 a thread may hold with 20 warps
// (0.4995 ms per Qwen3-8B step against 0.5005 with four sets and one chain;
// five chains spill)
constexpr int kP2rBSets = 2;
constexpr int kP2rChains = 3;
constexpr int kP2rTiles = 8;  // most m16 tiles (128 entries) per unit
constexpr int kP2rSlices = 2 * Cfg<8>::kSlice;
constexpr int kP2rLow = kArena1 / kP2rSlices;
constexpr int kP2rDyn = kArena1 + kLutBytes + (kP2rWarps - kP2rLow) * kP2rSlices;
static_assert(kP2rDyn <= kDynBytes && kP2rLow < kP2rWarps, "p2r shared memory");

struct P2rBase {
  int32_t count;
  int32_t tiles;                   // target tiles per unit (1 .. kP2rTiles)
  int32_t base[TQ_MAX_BATCH + 1];  // first unit of problem p (base[count]: all units)
};

// Units per stage of a problem: the expected tiles of a stage over the
// call's target tiles per unit, rounded up, 1 .. 64.
__host__ __device__ inline int p2r_parts(int K, int64_t nnz, int tiles) {
  const int64_t per = (int64_t)nstages(K, 8) * 8 * 16 * tiles;
  const int64_t q = (nnz + per - 1) / per;
  return (int)(q < 1 ? 1 : q > 64 ? 64 : q);
}

__global__ void __launch_bounds__(kP2rWarps * 32, 1)
    gemv_p2r_kernel(const __grid_constant__ P2rBase pb, const __grid_constant__ BatchParams bp, int32_t *counter) {
  extern __shared__ __align__(1024) unsigned char dynr[];
  const int tid = threadIdx.x, lane = tid & 31;
  if (smem_u32(dynr) != kDynShared) {
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  mm::lut_fill_replicated(reinterpret_cast<uint32_t *>(dynr + kArena1), tid, kP2rWarps * 32);
  __syncthreads();
  // the work below reads the prep kernel's output (launched programmatically
  // after it); the first-plane kernel may start its set-up meanwhile
  grid_dep_wait();
  grid_dep_launch_next();
  const int g16 = lane >> 2, c = lane & 3, warp = tid >> 5;
  const uint32_t tag = kLutShared | ((uint32_t)lane << 2);
  const bool realB = (g16 >> 1) == c;
  unsigned char *bw = warp < kP2rLow ? dynr + warp * kP2rSlices
                                     : dynr + kArena1 + kLutBytes + (warp - kP2rLow) * kP2rSlices;
  const int count = pb.count, total = pb.base[count];
  const int top = 1 << (31 - __clz(max(count, 1)));
  uint32_t bz[kP2rBSets][4] = {};  // activation registers (zero-column lanes: zero throughout)
  for (;;) {
    int u = 0;
    if (lane == 0) u = atomicAdd(counter, 1);
    u = __shfl_sync(0xffffffffu, u, 0);
    if (u >= total) break;
    int pi = 0;  // the unit's problem: the last with base <= u
    for (int step = top; step >= 1; step >>= 1)
      if (pi + step < count && pb.base[pi + step] <= u) pi += step;
    const Problem &P = bp.prob[pi];
    const int G = P.K / kGroup, S = p2r_parts(P.K, P.nnz, pb.tiles), local = u - pb.base[pi];
    const int s = local / S, part = local - s * S;
    // the stage's groups' entry ranges (16-entry multiples, clamped into the
    // index): lane q < 8 reads group 8 s + q; the tiles are the longest's
    const int64_t cap = mm::c_capacity(P.K, P.nnz);
    int64_t gb = 0;
    int gn = 0;
    if (lane < 8 && 8 * s + lane < G) {
      const int g = 8 * s + lane;
      gb = min(max((int64_t)__ldg(P.p2idx + g), (int64_t)0), cap) & ~(int64_t)15;
      const int64_t ge = min(max((int64_t)__ldg(P.p2idx + g + 1), gb), cap) & ~(int64_t)15;
      gn = (int)((ge - gb) >> 4);
    }
    int T = gn;
#pragma unroll
    for (int o = 4; o; o >>= 1) T = max(T, __shfl_xor_sync(0xffffffffu, T, o));
    T = __shfl_sync(0xffffffffu, T, 0);
    const int t0 = (int)((int64_t)T * part / S), t1 = (int)((int64_t)T * (part + 1) / S);
    if (t0 >= t1) continue;
    // this lane's two groups (stage columns 2c, 2c + 1)
    const int64_t gbE = __shfl_sync(0xffffffffu, gb, 2 * c), gbO = __shfl_sync(0xffffffffu, gb, 2 * c + 1);
    const int gnE = __shfl_sync(0xffffffffu, gn, 2 * c), gnO = __shfl_sync(0xffffffffu, gn, 2 * c + 1);
    const unsigned char *slots = reinterpret_cast<const unsigned char *>(P.p2idx) + mm::c_slot_off(P.K);
    {
      // the stage's two slices (contiguous in the workspace) into the warp's slot
      const uint4 *src = reinterpret_cast<const uint4 *>(ws_b(P) + (int64_t)s * 2 * slice_bytes(8));
      __syncwarp();  // the previous unit's reads are done
      for (int i = lane; i < 2 * slice_bytes(8) / 16; i += 32) {
        const int sl = i / (slice_bytes(8) / 16), k = i - sl * (slice_bytes(8) / 16);
        reinterpret_cast<uint4 *>(bw + sl * Cfg<8>::kSlice)[k] = __ldg(src + i);
      }
      __syncwarp();
    }
    const unsigned char *bq = bw + (g16 & 1) * Cfg<8>::kSlice + c * 16;
    const float4 cs = __ldg(reinterpret_cast<const float4 *>(ws_cs(P, 1) + s * kCSStage + c * 16));
    float *y2 = P.y2();
    for (int t = t0; t < t1; ++t) {
      // slots of entries r, r + 8 of tile t: words in slot order (0, 4, 1, 5 | 2, 6, 3, 7)
      uint4 sl[2][2][2];  // [h: row r / r + 8][odd][half]
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int o = 0; o < 2; ++o) {
          const int r = 16 * t + g16 + 8 * h;
          const bool ok = r < 16 * (o ? gnO : gnE);
          const uint4 *p = reinterpret_cast<const uint4 *>(slots + ((o ? gbO : gbE) + r) * 32);
          sl[h][o][0] = ok ? __ldcs(p) : make_uint4(0u, 0u, 0u, 0u);
          sl[h][o][1] = ok ? __ldcs(p + 1) : make_uint4(0u, 0u, 0u, 0u);
        }
      // window word i of row h
      auto win = [&](int h, int i) -> uint32_t {
        const uint4 &e0 = sl[h][0][0], &e1 = sl[h][0][1], &o0 = sl[h][1][0], &o1 = sl[h][1][1];
        switch (i) {
          case 0: return e0.x;
          case 1: return e0.z;
          case 2: return e1.x;
          case 3: return e1.z;
          case 4: return e0.y;
          case 5: return e0.w;
          case 6: return mm::prmt(e1.y, o0.x, 0x7610u);
          case 7: return o0.z;
          case 8: return o1.x;
          case 9: return o1.z;
          case 10: return o0.y;
          case 11: return o0.w;
          default: return o1.y;
        }
      };
      float dc[kP2rChains][4];
      dc[0][0] = dc[0][2] = -cs.x;
      dc[0][1] = dc[0][3] = -cs.y;
#pragma unroll
      for (int k = 1; k < kP2rChains; ++k) dc[k][0] = dc[k][1] = dc[k][2] = dc[k][3] = 0.f;
#pragma unroll
      for (int i = 0; i < words(8); ++i) {
        uint32_t a[2][10];
        decode_word(win(0, i), tag, a[0]);
        decode_word(win(1, i), tag, a[1]);
#pragma unroll
        for (int m = 0; m < 5; ++m) {
          const int j = 5 * i + m;
          uint32_t(&r)[4] = bz[(j >> 1) % kP2rBSets];
          if ((j & 1) == 0) ld_b_real(r, bq + (j >> 1) * 64, realB);
          const uint32_t b0 = (j & 1) ? r[2] : r[0], b1 = (j & 1) ? r[3] : r[1];
          mm::mma16816(dc[j % kP2rChains], a[0][2 * m], a[1][2 * m], a[0][2 * m + 1], a[1][2 * m + 1], b0, b1);
        }
      }
      float d[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        d[e] = dc[0][e];
#pragma unroll
        for (int k = 1; k < kP2rChains; ++k) d[e] += dc[k][e];
      }
      // d: (row r: even, odd), (row r + 8: even, odd); s2 beside each record
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int r = 16 * t + g16 + 8 * h;
        const int nE = (int)sl[h][0][1].w, nO = (int)sl[h][1][1].w;
        const float s2E = mm::half_of<true>(sl[h][0][1].y), s2O = mm::half_of<false>(sl[h][1][0].x);
        if (r < 16 * gnE && nE >= 0 && nE < P.N) atomicAdd(&y2[nE], s2E * d[2 * h]);
        if (r < 16 * gnO && nO >= 0 && nO < P.N) atomicAdd(&y2[nO], s2O * d[2 * h + 1]);
      }
    }
  }
}

}  // namespace g4

TQ_STATUS_ACCESSOR(read_status_gemv_g4)

static_assert(sizeof(BatchParams) + sizeof(g4::Sched) <= 32764, "one-group-per-lane kernel parameters");

int64_t g4_workspace_bytes(int M, int N, int K) {
  return g4::pad256(g4::b_bytes(M, K)) + g4::pad256(g4::cs_bytes(M, K)) + g4::pad256(g4::ticket_bytes(N));
}

// Target groups per work unit for an M <= 2 batch: 0 (whole tiles) when the
// largest tile costs no more than a CTA's fair share of the batch, else
// that share, so that no unit holds up the end of the call.
int g4_split_for(const BatchParams &bp, int num_sms) {
  const int ctas = std::min(num_sms, 256);
  int64_t total = 0;
  int gmax = 0;
  for (int i = 0; i < bp.count; ++i) {
    const int G = bp.prob[i].K / kGroup;
    total += (int64_t)((bp.prob[i].N + g4::kRows - 1) / g4::kRows) * G;
    gmax = std::max(gmax, G);
  }
  const int64_t share = (total + ctas - 1) / ctas;
  return share >= gmax ? 0 : (int)std::max<int64_t>(1, share);
}

// The M <= 2 decode kernel over a batch whose prep (activation slots, maps,
// y2, tickets) and second plane have been launched on the same stream.
cudaError_t launch_gemv_g4(const BatchParams &bp, int num_sms, cudaStream_t s) {
  thread_local g4::Sched sc;
  if (!g4::takes(bp) || bp.g4_split < 0) return cudaErrorInvalidValue;
  const int ctas = min(num_sms, 256);
  const int SG = g4::stage_groups(bp.M);
  sc.split = bp.g4_split;
  // contiguous unit ranges of about equal cost (groups per unit)
  int64_t total_cost = 0;
  for (int i = 0; i < bp.count; ++i) total_cost += (int64_t)((bp.prob[i].N + g4::kRows - 1) / g4::kRows) * (bp.prob[i].K / kGroup);
  int c = 0, unit = 0;
  int64_t run2 = 0;  // twice the cost before the current unit
  sc.cta_unit[0] = 0;
  for (int i = 0; i < bp.count; ++i) {
    const int nst = g4::nstages(bp.prob[i].K, SG), G = bp.prob[i].K / kGroup;
    const int u = g4::unit_parts(bp.prob[i].K, SG, sc.split);
    const int tiles_i = (bp.prob[i].N + g4::kRows - 1) / g4::kRows;
    for (int t = 0; t < tiles_i; ++t)
      for (int k = 0; k < u; ++k, ++unit) {
        // the unit's groups: its stages' share of G
        const int64_t s0 = (int64_t)k * nst / u, s1 = (int64_t)(k + 1) * nst / u;
        const int64_t cost = std::min<int64_t>(G, s1 * SG) - s0 * SG;
        const int64_t mid2 = run2 + cost;
        while (c < ctas - 1 && mid2 * ctas >= 2 * total_cost * (int64_t)(c + 1)) sc.cta_unit[++c] = unit;
        run2 += 2 * cost;
      }
  }
  while (c < ctas) sc.cta_unit[++c] = unit;
  using g4::kTL1;
  using g4::kTL2;
  using g4::kWD1;
  using g4::kWD2;
  auto kern = bp.M == 1
                  ? (bp.out_f32 ? g4::gemv_g4_kernel<true, 1, 8, kWD1, kTL1> : g4::gemv_g4_kernel<false, 1, 8, kWD1, kTL1>)
                  : (bp.out_f32 ? g4::gemv_g4_kernel<true, 2, 4, kWD2, kTL2> : g4::gemv_g4_kernel<false, 2, 4, kWD2, kTL2>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, g4::kDynBytes);
  if (e != cudaSuccess) return e;
  // launched programmatically: its CTAs set up (table, barriers) while the
  // second-plane kernel finishes, then wait for it (grid_dep_wait)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ctas);
  cfg.blockDim = dim3(((bp.M == 1 ? kWD1 : kWD2) + 1) * 32);
  cfg.dynamicSmemBytes = g4::kDynBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, bp, sc);
}

// The second plane of one token through gemv_p2r_kernel (every problem
// with a second plane has its index): units numbered problem by problem,
// launched programmatically after the prep kernel, which zeroes y2 and the
// unit counter.
cudaError_t launch_gemv_p2r(const BatchParams &bp, int num_sms, int32_t *counter, cudaStream_t s) {
  thread_local g4::P2rBase pb;
  if (bp.M != 1) return cudaErrorInvalidValue;
  pb.count = bp.count;
  // tiles per unit: about one and a half units per warp of the grid, at
  // most kP2rTiles (measured best for the Qwen3-8B step; small calls get
  // one tile per unit)
  const int ctas = std::min(num_sms, 256);
  int64_t tiles = 0;
  for (int p = 0; p < bp.count; ++p) tiles += (bp.prob[p].nnz + 127) / 128;
  pb.tiles = (int)std::max<int64_t>(1, std::min<int64_t>(g4::kP2rTiles, 2 * tiles / (3LL * ctas * g4::kP2rWarps)));
  pb.base[0] = 0;
  for (int p = 0; p < bp.count; ++p) {
    const Problem &P = bp.prob[p];
    pb.base[p + 1] = pb.base[p] + (P.nnz > 0 ? g4::nstages(P.K, 8) * g4::p2r_parts(P.K, P.nnz, pb.tiles) : 0);
  }
  cudaError_t e = cudaFuncSetAttribute(g4::gemv_p2r_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, g4::kP2rDyn);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ctas);
  cfg.blockDim = dim3(g4::kP2rWarps * 32);
  cfg.dynamicSmemBytes = g4::kP2rDyn;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, g4::gemv_p2r_kernel, pb, bp, counter);
}

// The dependency-ordered sequence kernel (one token), launched
// programmatically after its prep kernel.
cudaError_t launch_gemv_seq(const BatchParams &bp, int num_sms, int barrier_extra, cudaStream_t s) {
  if (bp.M != 1 || bp.count < 1) return cudaErrorInvalidValue;
  const int ctas = std::min(num_sms, 256);
  auto kern = bp.out_f32 ? g4::gemv_seq_kernel<true> : g4::gemv_seq_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, g4::kDynBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(ctas);
  cfg.blockDim = dim3((g4::kWD1 + 1) * 32);
  cfg.dynamicSmemBytes = g4::kDynBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, bp, (int32_t)barrier_extra);
}

}  // namespace tq
