// tq_gemv_tc.cu - decode-path linear (M <= 16 tokens) on the tcgen05 tensor
// cores, straight from the packed bytes.
//
// What is computed (per-group reading of the paper's eq. W-hat, "Model and
// Representation"; packed execution as in "Direct Packed Execution"):
//   y[m][n] = sum_g ( s1[n,g] * P1[n,g,m] + off[n,g] * S[g,m]
//                   + sal[n,g] * s2[j(n,g)] * P2[n,g,m] )
//   P1 = sum_{k in g} T1[n,k] x[m,k],  P2 likewise with T2,  S = sum_{k in g} x[m,k].
// P1 and P2 are fp32 tensor-core accumulations of exact products.
//
// Operand encoding.  A packed byte (digits d0..d4, digit = trit + 1) selects
// one 32-bit word W of a lane-replicated shared-memory table; one PRMT builds
// the table address from the byte.  W itself is the first fp16x2 A register:
//   lo = 4 + d0 + d2/4 + d4/16,  hi = 4 + d1 + d3/4 + d4/16   (exact fp16)
// and two LOP3 extract  16 + d2 | 16 + d3  and  64 + d4 | 64 + d4.
// The activation slots are chosen so that the MMA sees every digit with its
// own activation: y = (x0, x1, x2 - x0/4, x3 - x1/4, x4 - (x0+x1)/16, 0)
// (fp16, rounded once).  Subtracting C = the same MMA for an all-zero-trit
// row (every digit 1) leaves sum_i t_i x_i, exact up to that rounding.
// y, C and S per (group, token) are prepared once per call by
// gemv_prep_kernel into the caller's workspace.
//
// Roles (one persistent CTA per SM over a contiguous, cost-balanced range of
// 128-row tiles; every tile is walked in 8-group stages):
//  * warp 12 (producer): per stage, 1-D bulk copies of the 128 rows' packed
//    bytes (208 B each), the stage's activation slots and C/S into a ring of
//    shared-memory stage slots;
//  * warps 0-3 and 4-7 (decode quads, thread r = row r): even / odd groups;
//    each group's 26 bytes become 80 tensor-memory columns of the MMA's A
//    operand in a 3-slot ring; decoders wait for MMAs only to reuse a slot;
//  * warp 13 (one thread): 10 MMAs (M=128, N=16, K=16) per group into a
//    per-group fp32 accumulator slot; the chunks of two groups are
//    interleaved so that two accumulation chains are in flight (MMAs on one
//    accumulator serialize), and plane-2 batches are issued as they arrive;
//  * warps 8-11 (epilogue quad, thread r = row r): applies s1 / off per
//    group, and runs plane 2: the stage's salient (row, group) pairs are
//    compacted one per thread, decoded into a tensor-memory A slot and
//    multiplied by the stage's B blocks stacked along N (each record reads
//    its own group's columns); s2 * P2 goes to the row's shared-memory
//    accumulator; a stage's plane-2 result is collected one stage later.
//    The epilogue quad writes y.
// Every wait is bounded (tq_sm100.cuh); a timeout raises a CTA-wide abort.
#include "tq_common.cuh"
#include "tq_sm100.cuh"

namespace tq {

#ifdef TQ_TRACE
// debugging aid (trace builds only): clock64 stamps from CTA 0
static __device__ unsigned long long g_trace[4096];
#define TQ_STAMP(idx)                                                        \
  do {                                                                       \
    if (blockIdx.x == 0 && (idx) < 4096) g_trace[(idx)] = clock64();         \
  } while (0)
#else
#define TQ_STAMP(idx) \
  do {                \
  } while (0)
#endif

#ifdef TQ_CHECKS
// debugging aid (check builds only): first failed check id and its value
static __device__ uint32_t g_check[2];
#define TQ_CHK(cond, id, val)                                   \
  ((cond) ? true                                                \
          : (atomicOr(&g_tq_device_status, 8u), atomicCAS(&g_check[0], 0u, (uint32_t)(id)), \
             atomicCAS(&g_check[1], 0u, (uint32_t)(val)), false))
#else
#define TQ_CHK(cond, id, val) true
#endif

namespace tc {

constexpr int kRows = 128;        // tile rows = MMA M
constexpr int kStageG = 8;        // groups per stage
constexpr int kStageBytes = 208;  // plane-1 bytes per row per stage (13 x 16)
constexpr int kACols = 80;        // tensor-memory columns of A per group (160 K slots)
constexpr int kMmaPerGroup = 10;  // K = 16 each
constexpr int kQuad = 128;        // threads per quad
constexpr int kWarpEpi = 8, kWarpProd = 12, kWarpMma = 13;
constexpr int kThreads = 14 * 32;
constexpr int kBHalf = 2560;      // one 8-row x 160-slot activation block
constexpr int kLutBytes = 65536;  // 256 byte values x 256 B (32 lanes x 4 B used)
constexpr uint32_t kDynShared = 1024;  // shared-window offset of dynamic smem
constexpr int kDynBytes = 232448;      // whole opt-in shared memory of a CTA
constexpr int kArena1 = 65536 - (int)kDynShared;          // below the table
constexpr int kArena2 = kDynBytes - kArena1 - kLutBytes;  // above the table
constexpr uint32_t kTmemCols = 512;
constexpr int kRA = 3;  // A slots

template <int MP>
struct Cfg {
  static constexpr int NS = MP == 8 ? 3 : 2;        // stage slots
  static constexpr int RD = MP == 8 ? 8 : 4;        // accumulator slots (16 columns)
  static constexpr int BGroup = (MP / 8) * kBHalf;  // activation block of one group
  // MP = 8: an N=16 MMA of group g reads rows 8..15 from the next block
  // (harmless: those accumulator columns are never read), hence one extra.
  static constexpr int BStage = kStageG * BGroup + (MP == 8 ? kBHalf : 0);
  static constexpr int CSGroup = 2 * MP * 4;  // C[MP], S[MP] floats
  static constexpr int CSStage = kStageG * CSGroup;
  static constexpr int StageBuf = kRows * kStageBytes;
  // tensor-memory columns
  static constexpr uint32_t ColA = 0;
  static constexpr uint32_t ColD = kRA * kACols;
  static constexpr uint32_t ColA2 = ColD + RD * 16;
  static constexpr uint32_t ColD2 = ColA2 + kACols;
  static_assert(ColD2 + 8 * MP <= kTmemCols, "tensor memory overflow");
  // shared memory
  static constexpr int AccBytes = 2 * kRows * MP * 4;  // 2 tile parities x 128 rows x MP
  static constexpr bool AccIn1 = MP == 8;
  static constexpr int oBytes1 = 0;
  static constexpr int oList = oBytes1 + 2 * StageBuf;  // 128 x int2
  static constexpr int oBar = oList + kRows * 8;
  static constexpr int oAcc1 = oBar + 512;
  static constexpr int kArena1Used = oAcc1 + (AccIn1 ? AccBytes : 0);
  static constexpr int oBytes2 = 0;
  static constexpr int oB = oBytes2 + (NS - 2) * StageBuf;
  static constexpr int oCS = oB + NS * BStage;
  static constexpr int oAcc2 = oCS + NS * CSStage;
  static constexpr int kArena2Used = oAcc2 + (AccIn1 ? 0 : AccBytes);
  static_assert(kArena1Used <= kArena1, "arena 1 overflow");
  static_assert(kArena2Used <= kArena2, "arena 2 overflow");
};

struct Bars {
  uint64_t full[3], empty[3];
  uint64_t a_full[kRA], a_free[kRA];
  uint64_t d_full[8], d_free[8];
  uint64_t a2_full, g2_done;
  uint32_t tmem_slot;
  // plane-2 batch handed from the epilogue quad to the MMA thread
  uint32_t p2_rows;   // records in the batch (0: nothing to multiply)
  uint32_t p2_buf;    // stage slot whose activation blocks it uses
  uint32_t p2_last;   // 1 if it is the last batch of its stage
  int32_t wtot[4];
  int32_t abort_;
};

// Schedule: CTA c processes global tiles [cta_tile[c], cta_tile[c+1]).
struct Sched {
  int32_t cta_tile[257];
};

__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, volatile int32_t *abort_) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0) {
      if (*abort_) return false;
      if (global_ns() - t0 > kWaitLimitNs) break;
    }
  }
  atomicOr(&g_tq_device_status, kStatusTimeout);
  *abort_ = 1;
  return false;
}

// Table word of a byte value (see the file comment); invalid bytes map to
// the exponent pattern alone.
__device__ __forceinline__ uint32_t lut_word(int v) {
  uint32_t w = 0x44004400u;
  if (v <= 242) {
    const uint32_t d0 = v % 3, d1 = (v / 3) % 3, d2 = (v / 9) % 3, d3 = (v / 27) % 3, d4 = v / 81;
    w |= (d0 << 8) | (d2 << 6) | (d4 << 4) | (d1 << 24) | (d3 << 22) | (d4 << 20);
  }
  return w;
}

template <int K>
__device__ __forceinline__ void decode_byte(uint32_t word, uint32_t lanebase, uint32_t *out) {
  uint32_t addr, w;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(addr) : "r"(word), "r"(lanebase), "n"(0x7604 | (K << 4)));
  asm("ld.shared.u32 %0, [%1];" : "=r"(w) : "r"(addr) : "memory");
  out[0] = w;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(out[1]) : "r"(w), "n"(0x00C000C0), "n"(0x4C004C00));
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(out[2]) : "r"(w), "n"(0x00300030), "n"(0x54005400));
}

// Decode 26 bytes starting at byte offset O0 of the word window `w`.
template <int O0>
__device__ __forceinline__ void decode_group(const uint32_t *w, uint32_t lanebase, uint32_t *a) {
#pragma unroll
  for (int b = 0; b < 26; ++b) {
    const int o = O0 + b;
    const uint32_t word = w[o >> 2];
    switch (o & 3) {
      case 0: decode_byte<0>(word, lanebase, a + 3 * b); break;
      case 1: decode_byte<1>(word, lanebase, a + 3 * b); break;
      case 2: decode_byte<2>(word, lanebase, a + 3 * b); break;
      default: decode_byte<3>(word, lanebase, a + 3 * b); break;
    }
  }
  a[78] = 0u;
  a[79] = 0u;
}

__device__ __forceinline__ void store_a(uint32_t taddr, const uint32_t *a) {
#pragma unroll
  for (int c = 0; c < kACols; c += 16) tmem_st16(taddr + c, a + c);
}

// Decode group G (0..7) of this row's stage bytes in shared memory: loads the
// 16-byte chunks that cover bytes [26G, 26G + 26).
template <int G>
__device__ __forceinline__ void decode_stage_group(const unsigned char *row, uint32_t lanebase, uint32_t *a) {
  constexpr int c0 = (26 * G) / 16, c1 = (26 * G + 25) / 16;
  uint32_t w[12];
#pragma unroll
  for (int c = c0; c <= c1; ++c) {
    const uint4 v = *reinterpret_cast<const uint4 *>(row + 16 * c);
    w[4 * (c - c0) + 0] = v.x;
    w[4 * (c - c0) + 1] = v.y;
    w[4 * (c - c0) + 2] = v.z;
    w[4 * (c - c0) + 3] = v.w;
  }
  decode_group<26 * G - 16 * c0>(w, lanebase, a);
}

__device__ __forceinline__ void decode_stage_group_rt(int g, const unsigned char *row, uint32_t lanebase,
                                                      uint32_t *a) {
  switch (g) {
    case 0: decode_stage_group<0>(row, lanebase, a); break;
    case 1: decode_stage_group<1>(row, lanebase, a); break;
    case 2: decode_stage_group<2>(row, lanebase, a); break;
    case 3: decode_stage_group<3>(row, lanebase, a); break;
    case 4: decode_stage_group<4>(row, lanebase, a); break;
    case 5: decode_stage_group<5>(row, lanebase, a); break;
    case 6: decode_stage_group<6>(row, lanebase, a); break;
    default: decode_stage_group<7>(row, lanebase, a); break;
  }
}

// Loads the 26-byte plane-2 record j without reading past the end of plane 2
// and returns it as 7 words (bytes 0..25, little-endian).
__device__ __forceinline__ void load_record(const uint8_t *plane2, int64_t j, uint32_t *rw) {
  const int64_t off0 = j * kGroupBytes;
  const int64_t base4 = off0 & ~(int64_t)3;
  const int sh = (int)(off0 - base4);  // 0 or 2
  const uint32_t *src = reinterpret_cast<const uint32_t *>(plane2 + base4);
  uint32_t r8[8];
#pragma unroll
  for (int i = 0; i < 6; ++i) r8[i] = __ldg(src + i);
  r8[6] = sh ? __ldg(src + 6) : (uint32_t)__ldg(reinterpret_cast<const uint16_t *>(src + 6));
  r8[7] = 0u;
#pragma unroll
  for (int i = 0; i < 7; ++i) rw[i] = sh ? __funnelshift_r(r8[i], r8[i + 1], 16) : r8[i];
}

// Iterates (tile, stage) in the CTA's order; every role walks the same list.
struct Walk {
  int tile, t_end, pi, s, nstages, gs;
  const BatchParams *bp;
  __device__ void set_tile() {
    while (pi + 1 < bp->count && bp->prob[pi + 1].tile_begin <= tile) ++pi;
    const int G = bp->prob[pi].K / kGroup;
    nstages = (G + kStageG - 1) / kStageG;
    s = 0;
    gs = min(kStageG, G);
  }
  __device__ Walk(const BatchParams *b, int t0, int t1)
      : tile(t0), t_end(t1), pi(0), s(0), nstages(0), gs(0), bp(b) {
    if (tile < t_end) set_tile();
  }
  __device__ bool valid() const { return tile < t_end; }
  __device__ const Problem &P() const { return bp->prob[pi]; }
  __device__ bool last_stage() const { return s + 1 == nstages; }
  __device__ void next() {
    if (++s < nstages) {
      const int G = bp->prob[pi].K / kGroup;
      gs = min(kStageG, G - s * kStageG);
    } else if (++tile < t_end) {
      set_tile();
    }
  }
};

// ------------------------------------------------------------------ prep
// Activation slots y, C (the all-zero-trit MMA value) and S = sum x for every
// (problem, group, token); rows m in [M, MP) are zero.  Layout per problem:
// B[g][h][kc][r][8 halves] (8-row x 160-slot blocks in the no-swizzle K-major
// core-matrix layout of the MMA's B operand), then CS[g][C[MP], S[MP]].
template <int MP>
__global__ void gemv_prep_kernel(const __grid_constant__ BatchParams bp) {
  const int p = blockIdx.y;
  if (p >= bp.count) return;
  const Problem &P = bp.prob[p];
  const int G = P.K / kGroup;
  const int task = blockIdx.x * blockDim.x + threadIdx.x;
  if (task >= G * MP) return;
  const int g = task / MP, m = task % MP;
  const bool real = m < bp.M;
  unsigned char *Bblk = P.wsB + (int64_t)g * Cfg<MP>::BGroup + (m >> 3) * kBHalf + (m & 7) * 16;
  float C = 0.f, S = 0.f;
  const __half *xr = P.x + (int64_t)(real ? m : 0) * P.K + (int64_t)g * kGroup;
  for (int b = 0; b < 26; ++b) {
    const int ntr = b < 25 ? 5 : 3;
    float x[5];
#pragma unroll
    for (int i = 0; i < 5; ++i) x[i] = (real && i < ntr) ? __half2float(xr[5 * b + i]) : 0.f;
    const float ya = x[0], yb = x[1];
    const float yc = __half2float(__float2half_rn(x[2] - 0.25f * ya));
    const float yd = ntr == 5 ? __half2float(__float2half_rn(x[3] - 0.25f * yb)) : 0.f;
    const float ye = ntr == 5 ? __half2float(__float2half_rn(x[4] - 0.0625f * (ya + yb))) : 0.f;
    C += 5.3125f * (ya + yb) + 17.f * (yc + yd) + 65.f * ye;
    S += x[0] + x[1] + x[2] + x[3] + x[4];
    const float ys[6] = {ya, yb, yc, yd, ye, 0.f};
#pragma unroll
    for (int q = 0; q < 3; ++q) {
      const int slot = 6 * b + 2 * q, kc = slot >> 3, e = slot & 7;
      *reinterpret_cast<__half2 *>(Bblk + kc * 128 + e * 2) = __floats2half2_rn(ys[2 * q], ys[2 * q + 1]);
    }
  }
  // pad slots 156..159 (core matrix 19, elements 4..7)
  *reinterpret_cast<uint2 *>(Bblk + 19 * 128 + 8) = make_uint2(0u, 0u);
  float *cs = P.wsCS + (int64_t)g * 2 * MP;
  cs[m] = C;
  cs[MP + m] = S;
}

// ------------------------------------------------------------------ main
template <int MP, bool F32>
__global__ void __launch_bounds__(kThreads, 1)
    gemv_tc_kernel(const __grid_constant__ BatchParams bp, const __grid_constant__ Sched sc) {
  using C_ = Cfg<MP>;
  extern __shared__ __align__(1024) unsigned char dyn[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int M = bp.M;
  if (smem_u32(dyn) != kDynShared) {
    // the layout assumes the dynamic window starts right after the reserved
    // 1 KiB of shared memory; anything else is reported, not guessed at
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  unsigned char *ar1 = dyn, *lut_p = dyn + kArena1, *ar2 = dyn + kArena1 + kLutBytes;
  const uint32_t lut_s = kDynShared + kArena1;  // 65536
  auto bytes_buf = [&](int b) -> unsigned char * {
    return b < 2 ? ar1 + C_::oBytes1 + b * C_::StageBuf : ar2 + C_::oBytes2;
  };
  int2 *list = reinterpret_cast<int2 *>(ar1 + C_::oList);
  Bars *bars = reinterpret_cast<Bars *>(ar1 + C_::oBar);
  unsigned char *B_p = ar2 + C_::oB;
  float *CS_p = reinterpret_cast<float *>(ar2 + C_::oCS);
  float *acc_s = reinterpret_cast<float *>(C_::AccIn1 ? ar1 + C_::oAcc1 : ar2 + C_::oAcc2);
  volatile int32_t *abort_ = &bars->abort_;

  // ---- one-time set-up
  {
    uint32_t *lut = reinterpret_cast<uint32_t *>(lut_p);
    for (int i = tid; i < 256 * 32; i += kThreads) lut[(i >> 5) * 64 + (i & 31)] = lut_word(i >> 5);
    uint32_t *bz = reinterpret_cast<uint32_t *>(B_p);
    for (int i = tid; i < C_::NS * C_::BStage / 4; i += kThreads) bz[i] = 0u;
    for (int i = tid; i < 2 * kRows * MP; i += kThreads) acc_s[i] = 0.f;
  }
  if (tid == 0) {
    for (int i = 0; i < C_::NS; ++i) {
      mbar_init(&bars->full[i], 1);
      mbar_init(&bars->empty[i], 2 * kQuad + 1);
    }
    for (int i = 0; i < kRA; ++i) {
      mbar_init(&bars->a_full[i], kQuad);
      mbar_init(&bars->a_free[i], 1);
    }
    for (int i = 0; i < C_::RD; ++i) {
      mbar_init(&bars->d_full[i], 1);
      mbar_init(&bars->d_free[i], kQuad);
    }
    mbar_init(&bars->a2_full, kQuad);
    mbar_init(&bars->g2_done, 1);
    bars->abort_ = 0;
    bars->p2_rows = 0;
    bars->p2_buf = 0;
    bars->p2_last = 0;
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(&bars->tmem_slot, kTmemCols);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_slot;
  const int t_begin = sc.cta_tile[blockIdx.x], t_end = sc.cta_tile[blockIdx.x + 1];
  const uint32_t lane_tm = (uint32_t)((warp & 3) * 32) << 16;  // this warp's tensor-memory lanes

  if (warp < kWarpEpi) {
    // ================================================================ decode
    const int qd = warp >> 2;
    const int r = tid & (kQuad - 1);
    const uint32_t lanebase = lut_s | ((uint32_t)lane << 2);
    {
      uint32_t z[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) z[i] = 0u;
      for (int c = qd * 16; c < kRA * kACols; c += 32) tmem_st16(tmem + lane_tm + C_::ColA + c, z);
      tmem_wait_st();
    }
    uint32_t q = 0, G = 0;  // global stage and group counters
    // the abort test is a warp vote: tcgen05.st / wait are warp-collective
    for (Walk w(&bp, t_begin, t_end); w.valid() && !__any_sync(0xffffffffu, *abort_ != 0); w.next(), ++q) {
      const int buf = (int)(q % C_::NS);
      bool have_bytes = false;
      const unsigned char *rowp = bytes_buf(buf) + r * kStageBytes;
#pragma unroll 1
      for (int g = 0; g < w.gs; ++g, ++G) {
        if ((int)(G & 1u) != qd) continue;
        const bool st0 = (tid == 0 && G < 512);
        if (st0) TQ_STAMP((G / 2) * 4 + 0);
        if (!have_bytes) {
          wait_or_abort(&bars->full[buf], (q / C_::NS) & 1u, abort_);
          have_bytes = true;
        }
        const uint32_t slot = G % kRA;
        if (G >= (uint32_t)kRA) wait_or_abort(&bars->a_free[slot], (G / kRA - 1) & 1u, abort_);
        if (st0) TQ_STAMP((G / 2) * 4 + 1);
        uint32_t a[kACols];
        decode_stage_group_rt(g, rowp, lanebase, a);
        if (st0) TQ_STAMP((G / 2) * 4 + 2);
        store_a(tmem + lane_tm + C_::ColA + slot * kACols, a);
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&bars->a_full[slot]);
        if (st0) TQ_STAMP((G / 2) * 4 + 3);
      }
      // this quad is done with the stage's bytes; a quad without a group in a
      // (partial) stage still waits for the stage to land first, so that its
      // arrival counts toward this stage's phase of the slot
      if (!have_bytes) wait_or_abort(&bars->full[buf], (q / C_::NS) & 1u, abort_);
      mbar_arrive(&bars->empty[buf]);
    }
  } else if (warp < kWarpProd) {
    // ============================================================== epilogue
    const int r = tid - kWarpEpi * 32;
    const uint32_t lanebase = lut_s | ((uint32_t)lane << 2);
    const uint32_t a2 = tmem + lane_tm + C_::ColA2;
    {
      uint32_t z[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) z[i] = 0u;
      for (int c = 0; c < kACols; c += 16) tmem_st16(a2 + c, z);
      tmem_wait_st();
    }
    float acc[MP];
#pragma unroll
    for (int m = 0; m < MP; ++m) acc[m] = 0.f;
    uint32_t q = 0, G = 0, bc = 0;
    // the plane-2 batch whose MMA is in flight
    bool pend = false;
    int pend_buf = 0, pend_gs = 0, pend_rows = 0;
    int2 pend_rec = make_int2(-1, 0);
    float pend_s2 = 0.f;
    // the tile whose y is written when its last stage's plane 2 is collected
    bool fin = false, fin_valid = false;
    int fin_par = 0, fin_n = 0, fin_N = 0;
    void *fin_y = nullptr;

    // collects the batch in flight: s2 * P2 of every record into acc_s
    auto collect = [&](bool release_stage) {
      wait_or_abort(&bars->g2_done, bc & 1u, abort_);
      ++bc;
      tc_fence_after();
      if (pend_rows > 0) {
        const int g = pend_rec.x >= 0 ? ((pend_rec.x >> 8) & 0xff) : 0;  // bits 8..15: group
        uint32_t d[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) d[i] = 0u;
        // one column address per warp-collective load: walk the groups
#pragma unroll 1
        for (int gg = 0; gg < pend_gs; ++gg) {
          uint32_t t[16];
          tmem_ld_cols<MP>(tmem + lane_tm + C_::ColD2 + gg * MP, t);
          tmem_wait_ld();
          if (gg == g) {
#pragma unroll
            for (int i = 0; i < MP; ++i) d[i] = t[i];
          }
        }
        if (pend_rec.x >= 0 && TQ_CHK(g < kStageG && pend_buf < C_::NS && (pend_rec.x & 0xff) < kRows, 1, pend_rec.x)) {
          const float *Cg = CS_p + pend_buf * (C_::CSStage / 4) + g * 2 * MP;
          const int par = (pend_rec.x >> 16) & 1;  // bit 16: tile parity
          float *dst = acc_s + (par * kRows + (pend_rec.x & 0xff)) * MP;
#pragma unroll
          for (int m = 0; m < MP; ++m)
            if (m < M) atomicAdd(dst + m, pend_s2 * (__uint_as_float(d[m]) - Cg[m]));
        }
      }
      tc_fence_before();
      named_bar(1, kQuad);  // the batch's contributions are in acc_s; A2 / D2 are free
      pend = false;
      if (release_stage && r == 0) mbar_arrive(&bars->empty[pend_buf]);
      if (release_stage && fin) {
        float *src = acc_s + (fin_par * kRows + r) * MP;
        if (fin_valid) {
#pragma unroll
          for (int m = 0; m < MP; ++m) {
            if (m < M) {
              const float v = src[m];
              if (F32)
                static_cast<float *>(fin_y)[(int64_t)m * fin_N + fin_n] = v;
              else
                static_cast<__half *>(fin_y)[(int64_t)m * fin_N + fin_n] = __float2half_rn(v);
            }
          }
        }
#pragma unroll
        for (int m = 0; m < MP; ++m) src[m] = 0.f;
        fin = false;
      }
    };

    bool eq_abort = false;  // uniform across the quad (decided at a barrier)
    for (Walk w(&bp, t_begin, t_end); w.valid() && !eq_abort; w.next(), ++q) {
      const Problem &P = w.P();
      const int K = P.K, Gk = K / kGroup, W = sal_words_of(K);
      const int n = (w.tile - P.tile_begin) * kRows + r;
      const bool valid = n < P.N;
      const int g0 = w.s * kStageG, gs = w.gs;
      const int buf = (int)(q % C_::NS);
      const int tpar = w.tile & 1;
      // ---- per-row data of the stage
      float s1v[kStageG], offv[kStageG];
#pragma unroll
      for (int g = 0; g < kStageG; ++g) {
        s1v[g] = (valid && g < gs) ? __half2float(P.s1[(int64_t)n * Gk + g0 + g]) : 0.f;
        offv[g] = (valid && g < gs) ? __half2float(P.off[(int64_t)n * Gk + g0 + g]) : 0.f;
      }
      uint32_t bits = 0;
      int j0 = 0;
      if (valid) {
        const uint32_t *srow = P.sal + (int64_t)n * W;
        const uint32_t word = srow[g0 >> 5];
        bits = (word >> (g0 & 31)) & ((1u << gs) - 1u);
        if (bits) {
          int before = 0;
          for (int ww = 0; ww < (g0 >> 5); ++ww) before += __popc(srow[ww]);
          before += __popc(word & ((1u << (g0 & 31)) - 1u));
          j0 = P.rowptr[n] + before;
        }
      }
      const bool se = (r == 0 && q < 128);
      if (se) TQ_STAMP(1024 + q * 8 + 0);
      // ---- plane 1: one accumulator slot per group
      wait_or_abort(&bars->full[buf], (q / C_::NS) & 1u, abort_);
      if (se) TQ_STAMP(1024 + q * 8 + 1);
      const float *cs = CS_p + buf * (C_::CSStage / 4);
#pragma unroll 1
      for (int g = 0; g < gs; ++g, ++G) {
        const uint32_t ds = G % C_::RD;
        wait_or_abort(&bars->d_full[ds], (G / C_::RD) & 1u, abort_);
        tc_fence_after();
        uint32_t d[16];
        tmem_ld_cols<MP>(tmem + lane_tm + C_::ColD + ds * 16, d);
        tmem_wait_ld();
        tc_fence_before();
        mbar_arrive(&bars->d_free[ds]);
        const float *Cg = cs + g * 2 * MP, *Sg = Cg + MP;
        float s1g = 0.f, offg = 0.f;
#pragma unroll
        for (int gg = 0; gg < kStageG; ++gg)
          if (gg == g) {
            s1g = s1v[gg];
            offg = offv[gg];
          }
#pragma unroll
        for (int m = 0; m < MP; ++m) acc[m] = fmaf(s1g, __uint_as_float(d[m]) - Cg[m], fmaf(offg, Sg[m], acc[m]));
      }
      if (se) TQ_STAMP(1024 + q * 8 + 2);
      if (w.last_stage()) {
        // the row's plane-1 part is complete: park it in the tile's slot
        float *dst = acc_s + (tpar * kRows + r) * MP;
#pragma unroll
        for (int m = 0; m < MP; ++m) {
          if (m < M) atomicAdd(dst + m, acc[m]);
          acc[m] = 0.f;
        }
      }
      // ---- plane 2 of the previous stage
      if (pend) collect(true);
      if (se) TQ_STAMP(1024 + q * 8 + 3);
      // ---- plane 2 of this stage: compact the salient (row, group) pairs
      const int c = __popc(bits);
      int incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      if (lane == 31) bars->wtot[warp & 3] = incl;
      named_bar(1, kQuad);
      int wbase = 0, total = 0;
#pragma unroll
      for (int ww = 0; ww < 4; ++ww) {
        const int t = bars->wtot[ww];
        wbase += ww < (warp & 3) ? t : 0;
        total += t;
      }
      const int my0 = wbase + incl - c;
      const int nb = total > kRows ? (total + kRows - 1) / kRows : 1;
      for (int b = 0; b < nb; ++b) {
        const int b0 = b * kRows;
        // more than 128 pairs in one stage (rare): the earlier batch is
        // collected first, its A / D slots are reused
        if (b > 0) collect(false);
        {
          int o = my0, jj = j0;
          uint32_t bb = bits;
          while (bb) {
            const int g = __ffs(bb) - 1;
            bb &= bb - 1;
            if (o >= b0 && o < b0 + kRows && TQ_CHK(g < gs, 2, g)) list[o - b0] = make_int2(r | (g << 8) | (tpar << 16), jj);
            ++o;
            ++jj;
          }
        }
        const int rows_here = min(total - b0, kRows);
        if (r == 0) {
          bars->p2_rows = (uint32_t)rows_here;
          bars->p2_buf = (uint32_t)buf;
          bars->p2_last = b + 1 == nb ? 1u : 0u;
        }
        named_bar(1, kQuad);
        int2 rec = make_int2(-1, 0);
        float s2v = 0.f;
        uint32_t a[kACols];
        if (r < rows_here && P.nnz > 0 && TQ_CHK(rows_here <= kRows, 3, rows_here)) {
          rec = list[r];
          TQ_CHK(rec.y >= 0 && rec.y < P.nnz, 4, rec.y);
          const int jj = min(max(rec.y, 0), P.nnz - 1);
          s2v = __half2float(P.s2[jj]);
          uint32_t rw[7];
          load_record(P.plane2, jj, rw);
          decode_group<0>(rw, lanebase, a);
        } else {
#pragma unroll
          for (int i = 0; i < kACols; ++i) a[i] = 0u;
        }
        if (se) TQ_STAMP(1024 + q * 8 + 4);
        store_a(a2, a);
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&bars->a2_full);
        if (se) TQ_STAMP(1024 + q * 8 + 5);
        pend = true;
        pend_buf = buf;
        pend_gs = gs;
        pend_rows = rows_here;
        pend_rec = rec;
        pend_s2 = s2v;
      }
      if (w.last_stage()) {
        fin = true;
        fin_valid = valid;
        fin_par = tpar;
        fin_n = n;
        fin_N = P.N;
        fin_y = P.y;
      }
      eq_abort = named_bar_any(1, kQuad, *abort_ != 0);
      if (se) TQ_STAMP(1024 + q * 8 + 6);
    }
    if (pend && !eq_abort) collect(true);
  } else if (warp == kWarpProd) {
    // ============================================================== producer
    uint32_t q = 0;
    for (Walk w(&bp, t_begin, t_end); w.valid(); w.next(), ++q) {
      const Problem &P = w.P();
      const int64_t RB = row_bytes_of(P.K);
      const int n0 = (w.tile - P.tile_begin) * kRows;
      const int rows = min(kRows, P.N - n0);
      const int s = w.s, gs = w.gs;
      const uint32_t rb = (uint32_t)((gs * kGroupBytes + 15) / 16 * 16);
      const uint32_t bb = (uint32_t)(gs * C_::BGroup);
      const uint32_t cb = (uint32_t)(gs * C_::CSGroup);
      const int buf = (int)(q % C_::NS);
      int ok = 1;
      if (lane == 0) ok = wait_or_abort(&bars->empty[buf], ((q / C_::NS) & 1u) ^ 1u, abort_) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;  // uniform across the warp
      if (lane == 0) {
        mbar_arrive_expect_tx(&bars->full[buf], rb * (uint32_t)rows + bb + cb);
        bulk_g2s(B_p + buf * C_::BStage, P.wsB + (int64_t)s * kStageG * C_::BGroup, bb, &bars->full[buf]);
        bulk_g2s(reinterpret_cast<unsigned char *>(CS_p) + buf * C_::CSStage,
                 reinterpret_cast<const unsigned char *>(P.wsCS) + (int64_t)s * kStageG * C_::CSGroup, cb,
                 &bars->full[buf]);
      }
      __syncwarp();
      TQ_CHK((int64_t)s * kStageBytes + rb <= RB && rows >= 1 && rows <= kRows, 7, s * 1000 + rows);
      for (int rr = lane; rr < rows; rr += 32)
        bulk_g2s(bytes_buf(buf) + rr * kStageBytes, P.plane1 + (int64_t)(n0 + rr) * RB + (int64_t)s * kStageBytes,
                 rb, &bars->full[buf]);
    }
    // drain: every issued copy lands before the CTA exits (waited on even
    // after an abort; bounded by the wall-time limit)
    if (lane == 0) {
      for (uint32_t k = (q > (uint32_t)C_::NS ? q - C_::NS : 0); k < q; ++k)
        mbar_wait(&bars->full[k % C_::NS], (k / C_::NS) & 1u);
    }
  } else if (warp == kWarpMma && lane == 0) {
    // =================================================================== MMA
    const uint32_t idesc1 = idesc_f16_f32(128, 16);
    const uint32_t idesc2 = idesc_f16_f32(128, 8 * MP);
    uint32_t q = 0, G = 0, bc = 0;
    uint32_t p2_stages_done = 0;
    bool stop = false;
    // issues the next plane-2 batch if the epilogue has handed one over
    auto try_plane2 = [&](bool block) -> bool {
      if (block) {
        if (!wait_or_abort(&bars->a2_full, bc & 1u, abort_)) {
          stop = true;
          return false;
        }
      } else if (!mbar_try_wait(&bars->a2_full, bc & 1u)) {
        return false;
      }
      ++bc;
      tc_fence_after();
      const uint32_t rows = bars->p2_rows, buf = bars->p2_buf, last = bars->p2_last;
      if (rows > 0 && TQ_CHK(buf < (uint32_t)C_::NS && rows <= (uint32_t)kRows, 5, buf * 1000 + rows)) {
        const uint32_t Bst = smem_u32(B_p + buf * C_::BStage);
#pragma unroll
        for (int i = 0; i < kMmaPerGroup; ++i)
          mma_tmemA(tmem + C_::ColD2, tmem + C_::ColA2 + 8 * i, smem_desc(Bst + 2 * i * 128, 128, kBHalf), idesc2,
                    i > 0 ? 1u : 0u);
        mma_commit(&bars->g2_done);
      } else {
        mbar_arrive(&bars->g2_done);
      }
      p2_stages_done += last;
      return true;
    };
    // waits for `bar`, issuing plane-2 batches while it is not ready
    auto wait_serving = [&](uint64_t *bar, uint32_t parity) -> bool {
      const uint64_t t0 = global_ns();
      for (uint32_t i = 0;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        try_plane2(false);
        if ((i & 63u) == 63u) {
          if (*abort_) return false;
          if (global_ns() - t0 > kWaitLimitNs) {
            atomicOr(&g_tq_device_status, kStatusTimeout);
            *abort_ = 1;
            return false;
          }
        }
      }
    };
    for (Walk w(&bp, t_begin, t_end); w.valid() && !stop; w.next(), ++q) {
      const int buf = (int)(q % C_::NS);
      const uint32_t Bst = smem_u32(B_p + buf * C_::BStage);
      // plane 1: groups in pairs, chunks interleaved (two accumulation chains)
      for (int g = 0; g < w.gs && !stop; g += 2) {
        const int ng = min(2, w.gs - g);
        for (int k = 0; k < ng && !stop; ++k) {
          const uint32_t Gk = G + k;
          if (!wait_serving(&bars->a_full[Gk % kRA], (Gk / kRA) & 1u)) stop = true;
          if (!stop && Gk >= (uint32_t)C_::RD && !wait_serving(&bars->d_free[Gk % C_::RD], (Gk / C_::RD - 1) & 1u))
            stop = true;
        }
        if (stop) break;
        if (G / 2 < 512) TQ_STAMP(2048 + (G / 2) * 2);
        tc_fence_after();
        if (!TQ_CHK(g + ng <= kStageG && buf < C_::NS, 6, g * 100 + ng)) {
          stop = true;
          break;
        }
#pragma unroll 1
        for (int i = 0; i < kMmaPerGroup; ++i) {
          for (int k = 0; k < ng; ++k) {
            const uint32_t Gk = G + k;
            const uint32_t bg = Bst + (g + k) * C_::BGroup;
            mma_tmemA(tmem + C_::ColD + (Gk % C_::RD) * 16, tmem + C_::ColA + (Gk % kRA) * kACols + 8 * i,
                      smem_desc(bg + 2 * i * 128, 128, kBHalf), idesc1, i > 0 ? 1u : 0u);
          }
        }
        for (int k = 0; k < ng; ++k) {
          const uint32_t Gk = G + k;
          mma_commit(&bars->a_free[Gk % kRA]);
          mma_commit(&bars->d_full[Gk % C_::RD]);
        }
        if (G / 2 < 512) TQ_STAMP(2048 + (G / 2) * 2 + 1);
        G += ng;
      }
    }
    // the remaining plane-2 batches: one stage's last batch per stage
    while (!stop && p2_stages_done < q) try_plane2(true);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace tc

// -------------------------------------------------------------- launcher
static int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

int tc_rows_per_tile() { return tc::kRows; }

// Workspace bytes of one problem (activation slots + C/S) for M tokens.
size_t tc_workspace_bytes(int M, int K) {
  const int MP = M <= 8 ? 8 : 16;
  const size_t G = (size_t)(K / kGroup);
  return G * ((size_t)(MP / 8) * tc::kBHalf + (size_t)2 * MP * 4);
}

size_t tc_workspace_b_bytes(int M, int K) {
  const int MP = M <= 8 ? 8 : 16;
  return (size_t)(K / kGroup) * (size_t)(MP / 8) * tc::kBHalf;
}

TQ_STATUS_ACCESSOR(read_status_gemv_tc)

#ifdef TQ_TRACE
extern "C" __attribute__((visibility("default"))) int tq_debug_trace(unsigned long long *out, int n) {
  return (int)cudaMemcpyFromSymbol(out, g_trace, sizeof(unsigned long long) * (n < 4096 ? n : 4096));
}
#endif

#ifdef TQ_CHECKS
extern "C" __attribute__((visibility("default"))) int tq_debug_checks(uint32_t *out) {
  return (int)cudaMemcpyFromSymbol(out, g_check, sizeof(uint32_t) * 2);
}
#endif

template <int MP, bool F32>
static cudaError_t launch_tc(const BatchParams &bp, cudaStream_t s) {
  static tc::Sched sc;
  const int ctas = min(num_sms(), 256);
  int64_t total_cost = 0;
  for (int i = 0; i < bp.count; ++i) {
    const int tiles_i = (bp.prob[i].N + tc::kRows - 1) / tc::kRows;
    total_cost += (int64_t)tiles_i * (bp.prob[i].K / kGroup);
  }
  // contiguous tile ranges: a tile goes to the CTA whose equal share of the
  // total cost contains the tile's midpoint
  int c = 0, tile = 0;
  int64_t run = 0;
  sc.cta_tile[0] = 0;
  for (int i = 0; i < bp.count; ++i) {
    const int tiles_i = (bp.prob[i].N + tc::kRows - 1) / tc::kRows;
    const int64_t cost = bp.prob[i].K / kGroup;
    for (int t = 0; t < tiles_i; ++t, ++tile) {
      const int64_t mid2 = 2 * run + cost;
      while (c < ctas - 1 && mid2 * ctas >= 2 * total_cost * (int64_t)(c + 1)) sc.cta_tile[++c] = tile;
      run += cost;
    }
  }
  while (c < ctas) sc.cta_tile[++c] = tile;
  // activation slots for every problem, then the decode kernel
  int gmax = 0;
  for (int i = 0; i < bp.count; ++i) gmax = max(gmax, bp.prob[i].K / kGroup);
  dim3 pgrid((gmax * MP + 127) / 128, bp.count);
  tc::gemv_prep_kernel<MP><<<pgrid, 128, 0, s>>>(bp);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(tc::gemv_tc_kernel<MP, F32>, cudaFuncAttributeMaxDynamicSharedMemorySize, tc::kDynBytes);
  if (e != cudaSuccess) return e;
  tc::gemv_tc_kernel<MP, F32><<<ctas, tc::kThreads, tc::kDynBytes, s>>>(bp, sc);
  return cudaGetLastError();
}

cudaError_t launch_gemv_tc(const BatchParams &bp, cudaStream_t s) {
  if (bp.M <= 8) return bp.out_f32 ? launch_tc<8, true>(bp, s) : launch_tc<8, false>(bp, s);
  return bp.out_f32 ? launch_tc<16, true>(bp, s) : launch_tc<16, false>(bp, s);
}

}  // namespace tq
