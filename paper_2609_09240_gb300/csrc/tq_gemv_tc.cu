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
// Schedule (one persistent CTA per SM, a contiguous cost-balanced range of
// 128-row tiles): every 8-group stage of a tile is handled by one of two
// decode quads (warps 0-3, 4-7; stages alternate), thread r = row r.  Warp 8
// streams each stage's packed rows (1-D bulk copies, 208 B per row), its
// activation slots and C/S into a shared-memory slot ring; warp 9 issues the
// MMAs (lane 0 for quad 0, lane 1 for quad 1): 10 MMAs (M=128, N=16, K=16)
// per group, A from tensor memory, B from shared memory, one fp32 column
// block per group.  After a stage the quad reads the block back once and
// applies s1 / off.  Plane 2: the stage's salient (row, group) pairs are
// compacted one per thread, decoded into the quad's A slot, multiplied by the
// stage's B blocks stacked along N (each record reads its own group's
// columns), scaled by s2 and added into the row accumulator in shared
// memory.  The last quad to finish a tile's row writes y.
// Every wait is bounded (tq_sm100.cuh); a timeout raises a CTA-wide abort.
#include "tq_common.cuh"
#include "tq_sm100.cuh"

namespace tq {

namespace tc {

constexpr int kRows = 128;        // tile rows = MMA M
constexpr int kStageG = 8;        // groups per stage
constexpr int kStageBytes = 208;  // plane-1 bytes per row per stage (13 x 16)
constexpr int kACols = 80;        // tensor-memory columns of A per group (160 K slots)
constexpr int kMmaPerGroup = 10;  // K = 16 each
constexpr int kQuad = 128;        // threads per decode quad
constexpr int kThreads = 320;     // 2 quads + producer warp + MMA warp
constexpr int kBHalf = 2560;      // one 8-row x 160-slot activation block
constexpr int kLutBytes = 65536;  // 256 byte values x 256 B (32 lanes x 4 B used)
constexpr uint32_t kDynShared = 1024;  // shared-window offset of dynamic smem
constexpr int kDynBytes = 232448;      // whole opt-in shared memory of a CTA
constexpr int kArena1 = 65536 - (int)kDynShared;          // below the table
constexpr int kArena2 = kDynBytes - kArena1 - kLutBytes;  // above the table
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kQuadTmem = 256;  // tensor-memory columns per quad

template <int MP>
struct Cfg {
  static constexpr int NS = MP == 8 ? 3 : 2;        // stage slots
  static constexpr int DEPTH = MP == 8 ? 2 : 1;     // A slots per quad
  static constexpr int BGroup = (MP / 8) * kBHalf;  // activation block of one group
  // MP = 8: group g's N=16 MMA reads rows 8..15 from group g+1's block (its
  // columns 8..15 are overwritten by group g+1 later), so one extra block.
  static constexpr int BStage = kStageG * BGroup + (MP == 8 ? kBHalf : 0);
  static constexpr int CSGroup = 2 * MP * 4;  // C[MP], S[MP] floats
  static constexpr int CSStage = kStageG * CSGroup;
  static constexpr int DStep = MP == 8 ? 8 : 16;    // accumulator columns per group
  static constexpr uint32_t ColD = DEPTH * kACols;  // accumulator block offset in a quad
  static constexpr int StageBuf = kRows * kStageBytes;
  // arena 1 (below the table): two byte buffers, record lists, barriers and,
  // for MP = 8, the shared row accumulators
  static constexpr int AccBytes = 2 * kRows * MP * 4;  // 2 tile parities x 128 rows x MP
  static constexpr bool AccIn1 = MP == 8;
  static constexpr int oBytes1 = 0;
  static constexpr int oList = oBytes1 + 2 * StageBuf;  // 2 quads x 128 x int2
  static constexpr int oBar = oList + 2 * kRows * 8;
  static constexpr int oAcc1 = oBar + 512;
  static constexpr int kArena1Used = oAcc1 + (AccIn1 ? AccBytes : 0);
  // arena 2 (above the table): third byte buffer, B, C/S, counters (and acc)
  static constexpr int oBytes2 = 0;
  static constexpr int oB = oBytes2 + (NS - 2) * StageBuf;
  static constexpr int oCS = oB + NS * BStage;
  static constexpr int oCnt = oCS + NS * CSStage;  // 2 tile parities x 128 int
  static constexpr int oAcc2 = oCnt + 2 * kRows * 4;
  static constexpr int kArena2Used = oAcc2 + (AccIn1 ? 0 : AccBytes);
  static_assert(kArena1Used <= kArena1, "arena 1 overflow");
  static_assert(kArena2Used <= kArena2, "arena 2 overflow");
};

struct Bars {
  uint64_t full[3], empty[3];
  uint64_t a1_full[2][2], mma_done[2][2], d1_done[2], a2_full[2], mma2_done[2];
  uint32_t tmem_slot;
  uint32_t nrec[2];
  int32_t wtot[2][4];
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
  // stage byte buffers: two below the table, the third (MP = 8) above it
  auto bytes_buf = [&](int b) -> unsigned char * {
    return b < 2 ? ar1 + C_::oBytes1 + b * C_::StageBuf : ar2 + C_::oBytes2;
  };
  int2 *lists = reinterpret_cast<int2 *>(ar1 + C_::oList);
  int32_t *cnt = reinterpret_cast<int32_t *>(ar2 + C_::oCnt);
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
    for (int i = tid; i < 2 * kRows; i += kThreads) cnt[i] = 0;
  }
  if (tid == 0) {
    for (int i = 0; i < C_::NS; ++i) {
      mbar_init(&bars->full[i], 1);
      mbar_init(&bars->empty[i], kQuad);
    }
    for (int q = 0; q < 2; ++q) {
      for (int i = 0; i < 2; ++i) {
        mbar_init(&bars->a1_full[q][i], kQuad);
        mbar_init(&bars->mma_done[q][i], 1);
      }
      mbar_init(&bars->d1_done[q], 1);
      mbar_init(&bars->a2_full[q], kQuad);
      mbar_init(&bars->mma2_done[q], 1);
      bars->nrec[q] = 0;
    }
    bars->abort_ = 0;
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(&bars->tmem_slot, kTmemCols);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_slot;
  const int t_begin = sc.cta_tile[blockIdx.x], t_end = sc.cta_tile[blockIdx.x + 1];

  if (warp < 8) {
    // =============================================================== decode
    const int qd = warp >> 2;           // quad
    const int r = tid & (kQuad - 1);    // row within the tile
    const uint32_t lane_tm = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t qt = tmem + lane_tm + qd * kQuadTmem;  // this quad's tensor-memory base
    const uint32_t lanebase = lut_s | ((uint32_t)lane << 2);
    const uint32_t barid = 1 + qd;
    int2 *list = lists + qd * kRows;
    {
      uint32_t z[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) z[i] = 0u;
      for (int c = 0; c < C_::DEPTH * kACols; c += 16) tmem_st16(qt + c, z);
      tmem_wait_st();
    }
    float acc[MP];
#pragma unroll
    for (int m = 0; m < MP; ++m) acc[m] = 0.f;
    uint32_t q = 0, gcount = 0, own = 0, bcount = 0;  // global stage, own groups, own stages, plane-2 batches
    bool dec_abort = false;
    int pi = 0;
    for (int tile = t_begin; tile < t_end && !dec_abort; ++tile) {
      while (pi + 1 < bp.count && bp.prob[pi + 1].tile_begin <= tile) ++pi;
      const Problem &P = bp.prob[pi];
      const int K = P.K, G = K / kGroup, W = sal_words_of(K);
      const int n0 = (tile - P.tile_begin) * kRows;
      const int n = n0 + r;
      const bool valid = n < P.N;
      const int nstages = (G + kStageG - 1) / kStageG;
      const int tpar = tile & 1;
      for (int s = 0; s < nstages && !dec_abort; ++s, ++q) {
        if ((int)(q & 1u) != qd) continue;
        const int gs = min(kStageG, G - s * kStageG);
        const int g0 = s * kStageG;
        const int buf = (int)(q % C_::NS);
        // ---- per-row data of the stage, loaded early
        float s1v[kStageG], offv[kStageG];
        uint32_t bits = 0;
        int j0 = 0;
#pragma unroll
        for (int g = 0; g < kStageG; ++g) {
          s1v[g] = (valid && g < gs) ? __half2float(P.s1[(int64_t)n * G + g0 + g]) : 0.f;
          offv[g] = (valid && g < gs) ? __half2float(P.off[(int64_t)n * G + g0 + g]) : 0.f;
        }
        if (valid) {
          const uint32_t *srow = P.sal + (int64_t)n * W;
          const uint32_t word = srow[g0 >> 5];
          bits = (word >> (g0 & 31)) & ((1u << gs) - 1u);
          if (bits) {
            int before = 0;
            for (int w = 0; w < (g0 >> 5); ++w) before += __popc(srow[w]);
            before += __popc(word & ((1u << (g0 & 31)) - 1u));
            j0 = P.rowptr[n] + before;
          }
        }
        // ---- plane 1
        wait_or_abort(&bars->full[buf], (q / C_::NS) & 1u, abort_);
        const unsigned char *rowp = bytes_buf(buf) + r * kStageBytes;
#pragma unroll 1
        for (int g = 0; g < gs; ++g, ++gcount) {
          const uint32_t slot = gcount % C_::DEPTH;
          const uint32_t use = gcount / C_::DEPTH;
          if (use > 0) wait_or_abort(&bars->mma_done[qd][slot], (use - 1) & 1u, abort_);
          uint32_t a[kACols];
          decode_stage_group_rt(g, rowp, lanebase, a);
          store_a(qt + slot * kACols, a);
          tmem_wait_st();
          tc_fence_before();
          mbar_arrive(&bars->a1_full[qd][slot]);
        }
        // ---- compact this stage's plane-2 records (one per thread)
        const int c = __popc(bits);
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += v;
        }
        if (lane == 31) bars->wtot[qd][warp & 3] = incl;
        named_bar(barid, kQuad);
        int wbase = 0, total = 0;
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int t = bars->wtot[qd][w];
          wbase += w < (warp & 3) ? t : 0;
          total += t;
        }
        const int my0 = wbase + incl - c;
        // ---- epilogue of plane 1 (one accumulator column block per group)
        wait_or_abort(&bars->d1_done[qd], own & 1u, abort_);
        tc_fence_after();
        const float *cs = CS_p + buf * (C_::CSStage / 4);
#pragma unroll 1
        for (int g = 0; g < gs; ++g) {
          uint32_t d[16];
          tmem_ld_cols<MP>(qt + C_::ColD + g * C_::DStep, d);
          tmem_wait_ld();
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
        // ---- plane 2 of the stage, in batches of 128 records
        for (int b0 = 0;; b0 += kRows) {
          named_bar(barid, kQuad);  // earlier readers of the list are done
          {
            int o = my0, jj = j0;
            uint32_t bb = bits;
            while (bb) {
              const int g = __ffs(bb) - 1;
              bb &= bb - 1;
              if (o >= b0 && o < b0 + kRows) list[o - b0] = make_int2(r | (g << 8), jj);
              ++o;
              ++jj;
            }
          }
          if (r == 0) bars->nrec[qd] = (uint32_t)total;
          named_bar(barid, kQuad);
          const int rows_here = min(total - b0, kRows);
          int2 rec = make_int2(-1, 0);
          uint32_t a[kACols];
          if (r < rows_here && P.nnz > 0) {
            rec = list[r];
            const int64_t jj = min(max((int64_t)rec.y, (int64_t)0), (int64_t)P.nnz - 1);
            const int64_t off0 = jj * kGroupBytes;
            const int64_t base4 = off0 & ~(int64_t)3;
            const int sh = (int)(off0 - base4);  // 0 or 2
            const uint32_t *src = reinterpret_cast<const uint32_t *>(P.plane2 + base4);
            uint32_t r8[8];
#pragma unroll
            for (int i = 0; i < 6; ++i) r8[i] = __ldg(src + i);
            // the record's last bytes without reading past the end of plane 2
            r8[6] = sh ? __ldg(src + 6) : (uint32_t)__ldg(reinterpret_cast<const uint16_t *>(src + 6));
            r8[7] = 0u;
            uint32_t rw[7];
#pragma unroll
            for (int i = 0; i < 7; ++i) rw[i] = sh ? __funnelshift_r(r8[i], r8[i + 1], 16) : r8[i];
            decode_group<0>(rw, lanebase, a);
          } else {
#pragma unroll
            for (int i = 0; i < kACols; ++i) a[i] = 0u;
          }
          store_a(qt, a);  // A slot 0 is free: every plane-1 MMA of the stage is done
          tmem_wait_st();
          tc_fence_before();
          mbar_arrive(&bars->a2_full[qd]);
          wait_or_abort(&bars->mma2_done[qd], bcount & 1u, abort_);
          ++bcount;
          tc_fence_after();
          if (rows_here > 0) {
            const int g = rec.x >= 0 ? (rec.x >> 8) : 0;
            uint32_t d[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) d[i] = 0u;
            // one column address per warp-collective load: walk the groups
#pragma unroll 1
            for (int gg = 0; gg < gs; ++gg) {
              uint32_t t[16];
              tmem_ld_cols<MP>(qt + C_::ColD + gg * MP, t);
              tmem_wait_ld();
              if (gg == g) {
#pragma unroll
                for (int i = 0; i < MP; ++i) d[i] = t[i];
              }
            }
            if (rec.x >= 0) {
              const float s2 = __half2float(P.s2[min(max(rec.y, 0), P.nnz - 1)]);
              const float *Cg = cs + g * 2 * MP;
              float *dst = acc_s + (tpar * kRows + (rec.x & 0xff)) * MP;
#pragma unroll
              for (int m = 0; m < MP; ++m)
                if (m < M) atomicAdd(dst + m, s2 * (__uint_as_float(d[m]) - Cg[m]));
            }
          }
          if (b0 + kRows >= total) break;
        }
        named_bar(barid, kQuad);  // the stage's plane-2 atomics are complete
        mbar_arrive(&bars->empty[buf]);
        ++own;
        // ---- this quad's last stage of the tile: hand the row over
        if (s + 2 >= nstages) {
          const int quads = nstages >= 2 ? 2 : 1;
          float *dst = acc_s + (tpar * kRows + r) * MP;
#pragma unroll
          for (int m = 0; m < MP; ++m)
            if (m < M) atomicAdd(dst + m, acc[m]);
          __threadfence_block();
          const int prev = atomicAdd(cnt + tpar * kRows + r, 1);
          if (prev == quads - 1) {
            __threadfence_block();
            if (valid) {
#pragma unroll
              for (int m = 0; m < MP; ++m) {
                if (m < M) {
                  const float v = atomicAdd(dst + m, 0.f);
                  if (F32)
                    static_cast<float *>(P.y)[(int64_t)m * P.N + n] = v;
                  else
                    static_cast<__half *>(P.y)[(int64_t)m * P.N + n] = __float2half_rn(v);
                }
              }
            }
#pragma unroll
            for (int m = 0; m < MP; ++m) dst[m] = 0.f;
            cnt[tpar * kRows + r] = 0;
          }
#pragma unroll
          for (int m = 0; m < MP; ++m) acc[m] = 0.f;
        }
        dec_abort = named_bar_any(barid, kQuad, *abort_ != 0);
      }
    }
  } else if (warp == 8) {
    // ============================================================ producer
    uint32_t q = 0;
    int pi = 0;
    bool stop = false;
    for (int tile = t_begin; tile < t_end && !stop; ++tile) {
      while (pi + 1 < bp.count && bp.prob[pi + 1].tile_begin <= tile) ++pi;
      const Problem &P = bp.prob[pi];
      const int K = P.K, G = K / kGroup;
      const int64_t RB = row_bytes_of(K);
      const int n0 = (tile - P.tile_begin) * kRows;
      const int rows = min(kRows, P.N - n0);
      const int nstages = (G + kStageG - 1) / kStageG;
      for (int s = 0; s < nstages; ++s, ++q) {
        const int gs = min(kStageG, G - s * kStageG);
        const uint32_t rb = (uint32_t)((gs * kGroupBytes + 15) / 16 * 16);
        const uint32_t bb = (uint32_t)(gs * C_::BGroup);
        const uint32_t cb = (uint32_t)(gs * C_::CSGroup);
        const int buf = (int)(q % C_::NS);
        if (!wait_or_abort(&bars->empty[buf], ((q / C_::NS) & 1u) ^ 1u, abort_)) {
          stop = true;
          break;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(&bars->full[buf], rb * (uint32_t)rows + bb + cb);
          bulk_g2s(B_p + buf * C_::BStage, P.wsB + (int64_t)s * kStageG * C_::BGroup, bb, &bars->full[buf]);
          bulk_g2s(reinterpret_cast<unsigned char *>(CS_p) + buf * C_::CSStage,
                   reinterpret_cast<const unsigned char *>(P.wsCS) + (int64_t)s * kStageG * C_::CSGroup, cb,
                   &bars->full[buf]);
        }
        __syncwarp();
        for (int rr = lane; rr < rows; rr += 32)
          bulk_g2s(bytes_buf(buf) + rr * kStageBytes,
                   P.plane1 + (int64_t)(n0 + rr) * RB + (int64_t)s * kStageBytes, rb, &bars->full[buf]);
      }
    }
    // drain: every issued copy lands before the CTA exits (waited on even
    // after an abort; bounded by the wall-time limit)
    if (lane == 0) {
      for (uint32_t k = (q > (uint32_t)C_::NS ? q - C_::NS : 0); k < q; ++k)
        mbar_wait(&bars->full[k % C_::NS], (k / C_::NS) & 1u);
    }
  } else if (lane < 2) {
    // ================================================================= MMA
    const int qd = lane;  // lane 0 serves quad 0, lane 1 quad 1
    const uint32_t qt = tmem + qd * kQuadTmem;
    const uint32_t idesc1 = idesc_f16_f32(128, 16);
    const uint32_t idesc2 = idesc_f16_f32(128, 8 * MP);
    uint32_t q = 0, gcount = 0, bcount = 0;
    int pi = 0;
    bool stop = false;
    for (int tile = t_begin; tile < t_end && !stop; ++tile) {
      while (pi + 1 < bp.count && bp.prob[pi + 1].tile_begin <= tile) ++pi;
      const Problem &P = bp.prob[pi];
      const int G = P.K / kGroup;
      const int nstages = (G + kStageG - 1) / kStageG;
      for (int s = 0; s < nstages && !stop; ++s, ++q) {
        if ((int)(q & 1u) != qd) continue;
        const int gs = min(kStageG, G - s * kStageG);
        const int buf = (int)(q % C_::NS);
        const uint32_t Bst = smem_u32(B_p + buf * C_::BStage);
        for (int g = 0; g < gs; ++g, ++gcount) {
          const uint32_t slot = gcount % C_::DEPTH;
          if (!wait_or_abort(&bars->a1_full[qd][slot], (gcount / C_::DEPTH) & 1u, abort_)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t bg = Bst + g * C_::BGroup;
#pragma unroll
          for (int i = 0; i < kMmaPerGroup; ++i)
            mma_tmemA(qt + C_::ColD + g * C_::DStep, qt + slot * kACols + 8 * i,
                      smem_desc(bg + 2 * i * 128, 128, kBHalf), idesc1, i > 0 ? 1u : 0u);
          mma_commit(&bars->mma_done[qd][slot]);
        }
        if (stop) break;
        mma_commit(&bars->d1_done[qd]);
        // plane-2 batches of the stage (at least one, possibly empty)
        uint32_t nb = 1;
        for (uint32_t b = 0; b < nb; ++b) {
          if (!wait_or_abort(&bars->a2_full[qd], bcount & 1u, abort_)) {
            stop = true;
            break;
          }
          ++bcount;
          tc_fence_after();
          const uint32_t total = bars->nrec[qd];
          nb = total > (uint32_t)kRows ? (total + kRows - 1) / kRows : 1u;
          if (total > b * (uint32_t)kRows) {
#pragma unroll
            for (int i = 0; i < kMmaPerGroup; ++i)
              mma_tmemA(qt + C_::ColD, qt + 8 * i, smem_desc(Bst + 2 * i * 128, 128, kBHalf), idesc2,
                        i > 0 ? 1u : 0u);
            mma_commit(&bars->mma2_done[qd]);
          } else {
            mbar_arrive(&bars->mma2_done[qd]);
          }
        }
      }
    }
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
