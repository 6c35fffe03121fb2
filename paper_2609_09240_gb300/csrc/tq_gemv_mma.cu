// tq_gemv_mma.cu - decode-path linear for M <= 16 tokens: packed bytes are
// streamed from HBM into shared memory by bulk copies, decoded in registers
// and contracted on the tensor cores with warp-level m16n8k16 MMAs (fp16
// operands, fp32 accumulators).
//
// What is computed (per-group reading of the paper's eq. W-hat, "Model and
// Representation"; packed execution as in "Direct Packed Execution"):
//   y[m][n] = sum_g ( s1[n,g] * P1[n,g,m] + off[n,g] * S[g,m]
//                   + sal[n,g] * s2[j(n,g)] * P2[n,g,m] )
//   P1 = sum_{k in g} T1[n,k] x[m,k],  P2 likewise with T2,  S = sum_{k in g} x[m,k].
//
// Operand encoding (five MMA slots per packed byte, the minimum: the five
// digits d0..d4 of a byte, digit = trit + 1, are five independent linear
// functions of the byte value v = sum_i d_i 3^i).  A lane-replicated table
// maps v to the fp16x2 word
//   W  = (4 + d0 + d2/4, 4 + d1 + d3/4)
// and one LOP3 gives W' = (16 + d2, 16 + d3).  The fifth slot is the byte
// value itself, 4 + v/256: one PRMT puts two bytes of a packed word under
// the exponent byte 0x44.  With z_i = x_i - 3^i x4 / 81 the activation slots
//   y_a = z0, y_b = z1, y_c = z2 - z0/4, y_d = z3 - z1/4, y_e = 256 x4 / 81
// make the MMA return  const + sum_i d_i x_i  (exact up to the rounding of
// the slots to fp16); subtracting C, the same MMA for all digits 1 (all
// trits 0), leaves sum_i t_i x_i.  Slots, C and S per (group, token) come
// from gemv_mma_prep_kernel into the caller's workspace.
//
// Fragment layout.  In an m16n8k16 MMA, lane (g, c) (g = lane / 4,
// c = lane % 4) holds A's k-pairs c and c + 4 of rows g and g + 8; B's
// column g is token g (with more than 8 tokens a second MMA on the same A
// takes tokens 8 + g, and C/S come in one block per 8-token tile).  Lane c
// of a row decodes the two words of the group's window (the aligned words
// covering its 26 bytes) whose index is c mod 4, loaded straight from the
// stage row in shared memory (the 32 lanes hit 32 different banks): 8 bytes,
// whose 20 A words (W, W' of each byte, then 4 V words) feed the group's 10
// MMAs, chunk j taking words 2j and 2j + 1.  Window bytes outside the group
// get zero activations, so every lane runs the same code.  The prep kernel
// writes B (the activation slots) in exactly this order for each of the 8
// positions a group can take in its stage.
//
// Kernels (one step = three launches):
//  * gemv_mma_prep_kernel: B fragments, C and S per (problem, group, token);
//  * the second plane, s2 * P2 per row into the workspace (y2, fp32):
//    gemv_mma_p2v3_kernel (persistent over row spans: a counting sort of the
//    span's records by group, then m16n8k16 MMAs over 16 records of one group
//    at a time); gemv_mma_p2_kernel, one CTA per 128-row tile, when a row has
//    more salience words than the former's staging holds;
//  * gemv_mma_kernel (one persistent CTA per SM over a cost-balanced range
//    of 128-row tiles, 8-group stages): warp 8 fills a ring of shared-memory
//    slots, per stage the tile's 208 bytes of 128 rows (one 2-D tensor copy
//    through the problem's tensor map, which the prep kernel writes into
//    the workspace), the B fragments and C/S (bulk copies) and s1 / off
//    (16-byte asynchronous copies); warps 0..7 each own 16 rows of the tile,
//    decode and multiply, apply s1 / off per group, and at the tile's end
//    add y2 and write y.
// Every wait is bounded (tq_sm100.cuh); a timeout raises a CTA-wide abort.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <type_traits>

#include "tq_common.cuh"
#include "tq_decode_ops.cuh"
#include "tq_p2_tile.cuh"
#include "tq_sm100.cuh"

namespace tq {
namespace mm {

constexpr int kRows = 128;        // tile rows (8 m16 tiles)
constexpr int kWarpsP1 = 8, kWarpProd = 8;
constexpr int kThreads = 9 * 32;
constexpr int kBytesSlot = kRows * kStageBytes;           // 26624
constexpr int kSOSlot = 2 * kRows * 16;                   // s1 then off, 16 B per row

constexpr int kBarOff = 2 * kBytesSlot;                   // barriers in arena 1
static_assert(kBarOff + 512 <= kArena1, "arena 1 overflow");

__host__ __device__ constexpr int num_slots(int MB) { return MB <= 2 ? 4 : MB <= 8 ? 3 : 2; }
__host__ __device__ constexpr int b_stage_bytes(int MB) { return kStageG * kBTok * MB; }
// C/S bytes per group: C[8], S[8] of tokens 0..7, then (more than 8 tokens)
// the same for tokens 8..15
__host__ __device__ constexpr int cs_group_bytes(int MB) { return MB > 8 ? 2 * kCSGroup : kCSGroup; }

// Stage-slot layout for MB tokens: plane-1 slots 0, 1 in arena 1, the rest
// in arena 2 followed by the B, s1/off and C/S slots.
struct Layout {
  int NS, BStage, CSStage;
  int oBytes2, oB, oSO, oCS, used2;
  __host__ __device__ explicit Layout(int MB) {
    NS = num_slots(MB);
    BStage = b_stage_bytes(MB);
    CSStage = kStageG * cs_group_bytes(MB);
    oBytes2 = 0;
    oB = oBytes2 + (NS - 2) * kBytesSlot;
    oSO = oB + NS * BStage;
    oCS = oSO + NS * kSOSlot;
    used2 = oCS + NS * CSStage;
  }
};

struct Bars {
  uint64_t full[4], empty[4];
  int32_t abort_;
};

// Schedule: CTA c processes global tiles [cta_tile[c], cta_tile[c+1]).
struct Sched {
  int32_t cta_tile[257];
};



// The same from a compact (not replicated) 256-word table at `lut`.
__device__ __forceinline__ void decode_words_compact(uint32_t w0, uint32_t w1, const uint32_t *lut, uint32_t *a) {
  uint32_t v[8];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    v[k] = (w0 >> (8 * k)) & 0xffu;
    v[4 + k] = (w1 >> (8 * k)) & 0xffu;
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t w = lut[v[i]];
    a[2 * i] = w;
    a[2 * i + 1] = w_prime(w);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) a[16 + i] = 0x44004400u | v[2 * i] | (v[2 * i + 1] << 16);
}


// Iterates (tile, stage) in the CTA's order.
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

// Tensor-map templates, one per distinct (tensor kind, row length, row
// count) in a batch, encoded on the host; idx[p] / idx_so[p] pick problem
// p's.  The prep kernel only puts in the problem's address: a template
// encoded for the same sizes then equals the host encoding byte for byte.
constexpr int kMaxMapTemplates = 10;
constexpr uint8_t kNoMap = 255;
// The prep kernel reads the indices by its problem and the templates only at
// constant offsets (a loop over the template slots): indexed or
// address-taken reads of a parameter block this far into the parameter
// space have returned wrong data.
struct MapTemplates {
  uint8_t idx[TQ_MAX_BATCH];     // plane 1's template
  uint8_t idx_so[TQ_MAX_BATCH];  // s1's and off's template, or kNoMap (then asynchronous copies)
  uint4 t[kMaxMapTemplates][8];  // the encoded templates (128 bytes each)
};
static_assert(sizeof(CUtensorMap) == 8 * sizeof(uint4), "tensor map size");
// Workspace slot of a problem's tensor maps: plane 1, s1, off, then the
// indexed second-plane kernel's unit counter.
constexpr int kMapSlotBytes = 512;
constexpr int kMapS1 = 128, kMapOff = 256, kCounterOff = 384;
// problem 0's slot also holds the sequence kernel's problem barrier counter
constexpr int kSeqCounterOff = 448;
static_assert(kSeqCounterOff + 4 <= kMapSlotBytes, "map slot");

// ------------------------------------------------------------------ prep
constexpr int kPrepTasks = 16;  // (group, token) tasks per 128-thread prep block

__global__ void gemv_mma_prep_kernel(const __grid_constant__ BatchParams bp, const __grid_constant__ MapTemplates mt,
                                     int32_t *unit_counter) {
  const int p = blockIdx.y;
  if (p >= bp.count) return;
  const Problem &P = bp.prob[p];
  // the next kernel (second plane or main) may start its own set-up now
  grid_dep_launch_next();
  // launched programmatically: the stream's previous kernel (often the
  // last call's decode kernel, whose workspace this may be) has finished
  // and its writes are visible past this point
  grid_dep_wait();
  const bool g4_shared = g4::takes(bp) && bp.g4_split > 0;  // split tiles add their partial sums into y2
  // (the sequence kernel, g4_split < 0, adds every partial sum into y2)
  if (P.nnz > 0 || g4_shared || bp.g4_split < 0) {
    // y2 starts at zero (the indexed second-plane kernel adds into it)
    float *y2 = P.y2();
    const int64_t n = (int64_t)P.N * bp.M;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
      y2[i] = 0.f;
  }
  if (bp.g4_split < 0 && p == 0 && blockIdx.x == 0 && threadIdx.x == 0) {
    // the sequence kernel's problem barrier counter starts at zero
    *reinterpret_cast<int32_t *>(static_cast<unsigned char *>(P.map()) + kSeqCounterOff) = 0;
  }
  if (g4_shared) {
    // the arrival counters of split tiles start at zero
    const int MBx = bp.M;
    int32_t *tk = reinterpret_cast<int32_t *>(P.wsB + P.map_off + kMapSlotBytes + g4::pad256(g4::b_bytes(MBx, P.K)) +
                                              g4::pad256(g4::cs_bytes(MBx, P.K)));
    const int64_t n = g4::ticket_bytes(P.N) / 4;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
      tk[i] = 0;
  }
  if (p == 0 && blockIdx.x == 0 && threadIdx.x == 0 && unit_counter) *unit_counter = 0;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    // plane 1 as a 2-D byte tensor (row_bytes x N) for the main kernel's
    // stage copies: the template of its sizes with this problem's address
    auto build = [&](unsigned char *m, int t, const void *addr) {
      uint4 *dst = reinterpret_cast<uint4 *>(m);
#pragma unroll
      for (int k = 0; k < kMaxMapTemplates; ++k)
        if (k == t) {
#pragma unroll
          for (int i = 0; i < 8; ++i) dst[i] = mt.t[k][i];
        }
      asm volatile("tensormap.replace.tile.global_address.global.b1024.b64 [%0], %1;" ::"l"(m), "l"(addr) : "memory");
    };
    unsigned char *m = static_cast<unsigned char *>(P.map());
    build(m, mt.idx[p], P.plane1);
    if (mt.idx_so[p] != kNoMap) {
      // s1 and off as 2-D fp16 tensors (G x N), for the stage copies of their 8 groups
      build(m + kMapS1, mt.idx_so[p], P.s1);
      build(m + kMapOff, mt.idx_so[p], P.off);
    }
    asm volatile("fence.proxy.tensormap::generic.release.gpu;" ::: "memory");
  }
  const int MB = bp.M;
  const int G = P.K / kGroup;
  // eight threads per (group, token) task: thread `sub` forms the slots of
  // group bytes 4 sub .. 4 sub + 3 (bytes past 25 are none), the task's
  // threads exchange them through shared memory and each writes a share of
  // the task's outputs; C and S are summed over the eight.
  __shared__ __half sv[kPrepTasks][26][5];
  const int tib = threadIdx.x >> 3, sub = threadIdx.x & 7;
  const int task = blockIdx.x * kPrepTasks + tib;
  // with M <= 2 the one-group-per-lane kernel runs; its operands cover whole
  // stages of SG groups (groups past G get zero activations and C/S)
  const int SG = g4::stage_groups(MB);
  const bool g4ops = g4::takes(bp);
  const int Gx = g4ops ? SG * g4::nstages(P.K, SG) : G;
  const bool live = task < Gx * MB;
  const int g = live ? task / MB : 0, m = live ? task % MB : 0;
  const bool real = live && g < G;
  float C = 0.f, S = 0.f;
  if (real) {
    const __half *xr = P.x + (int64_t)m * P.K + (int64_t)g * kGroup;
    // this thread's activations: trits 20 sub .. min(20 sub + 19, 127)
    // (group rows are 16-byte aligned, so the 40-byte runs are 8-byte
    // aligned)
    const int nb = sub < 6 ? 4 : sub == 6 ? 2 : 0;
    uint2 xv[5];
#pragma unroll
    for (int i = 0; i < 5; ++i)
      xv[i] = (4 * i < kGroup - 20 * sub) ? __ldg(reinterpret_cast<const uint2 *>(xr + 20 * sub) + i) : make_uint2(0u, 0u);
    auto xg = [&](int j) -> float {  // activation 20 sub + j (0 past the group)
      const uint2 &v = xv[j >> 2];
      const uint32_t w = (j & 2) ? v.y : v.x;
      return __half2float(__ushort_as_half((unsigned short)((j & 1) ? (w >> 16) : (w & 0xffffu))));
    };
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (q >= nb) break;
      const int b = 4 * sub + q;
      const int ntr = b < 25 ? 5 : 3;
      float x[5];
#pragma unroll
      for (int i = 0; i < 5; ++i) x[i] = i < ntr ? xg(5 * q + i) : 0.f;
      const float z0 = x[0] - x[4] * (1.f / 81.f), z1 = x[1] - x[4] * (3.f / 81.f);
      const float z2 = x[2] - x[4] * (9.f / 81.f), z3 = x[3] - x[4] * (27.f / 81.f);
      const __half ha = __float2half_rn(z0), hb = __float2half_rn(z1);
      const float fa = __half2float(ha), fb = __half2float(hb);
      const __half hc = __float2half_rn(z2 - 0.25f * fa), hd = __float2half_rn(z3 - 0.25f * fb);
      const __half he = __float2half_rn(x[4] * (256.f / 81.f));
      sv[tib][b][0] = ha, sv[tib][b][1] = hb, sv[tib][b][2] = hc, sv[tib][b][3] = hd, sv[tib][b][4] = he;
      // all digits 1: slots 4 + 1 + 1/4, 16 + 1, 4 + 121/256
      C += 5.25f * (fa + fb) + 17.f * (__half2float(hc) + __half2float(hd)) + (4.f + 121.f / 256.f) * __half2float(he);
      S += x[0] + x[1] + x[2] + x[3] + x[4];
    }
  }
#pragma unroll
  for (int o = 1; o < 8; o <<= 1) {
    C += __shfl_xor_sync(0xffffffffu, C, o);
    S += __shfl_xor_sync(0xffffffffu, S, o);
  }
  __syncwarp();
  if (!live) return;
  const __half z = __float2half_rn(0.f);
  // slot k (0..4) of group byte b, zero outside the group
  auto slot = [&](int b, int k) -> __half { return (b >= 0 && b < 26) ? sv[tib][b][k] : z; };
  auto pk = [](__half lo, __half hi) -> uint32_t {
    __half2 v = __halves2half2(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
  };
  // the group's lane position and slice: 4-group stages, group g % 4 and
  // token m; 8-group stages, lane (g % 8) / 2 and the lane's group g % 2
  const int gs = g / SG, gp = g % SG;
  const int g4c = SG == 8 ? gp >> 1 : gp, g4sl = SG == 8 ? gp & 1 : m;
  if (g4ops) {
    unsigned char *g4b = P.wsB + P.map_off + kMapSlotBytes;
    float *g4cs = reinterpret_cast<float *>(g4b + g4::pad256(g4::b_bytes(MB, P.K)));
    unsigned char *g4dst = g4b + (int64_t)(gs * 2 + g4sl) * g4::slice_bytes(SG) + g4c * 16;
    // activation slots for the one-group-per-lane kernel: MMA j = 5 i + r
    // of the lane's window words takes W, W' of window byte 4 i + r (r < 4)
    // or the fifth-slot words of window bytes 4 i .. 4 i + 3 (r = 4);
    // window byte beta is group byte beta - offs (offs = 26 for the second
    // group of a lane in an 8-group stage, 2 for the odd groups of a
    // 4-group stage)
    const int offs = SG == 8 ? (g4sl ? 26 : 0) : (g & 1 ? 2 : 0);
    const int nj = 5 * g4::words(SG);
    for (int jp = sub; jp < g4::pairs(SG); jp += 8) {
      uint32_t w[4];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int j = 2 * jp + h, i = j / 5, r5 = j % 5;
        uint32_t b0 = 0u, b1 = 0u;
        if (real && j < nj) {
          if (r5 < 4) {
            const int b = 4 * i + r5 - offs;
            if (b >= 0 && b < 26) {
              b0 = pk(sv[tib][b][0], sv[tib][b][1]);
              b1 = pk(sv[tib][b][2], sv[tib][b][3]);
            }
          } else {
            b0 = pk(slot(4 * i - offs, 4), slot(4 * i + 1 - offs, 4));
            b1 = pk(slot(4 * i + 2 - offs, 4), slot(4 * i + 3 - offs, 4));
          }
        }
        w[2 * h] = b0;
        w[2 * h + 1] = b1;
      }
      *reinterpret_cast<uint4 *>(g4dst + jp * 64) = make_uint4(w[0], w[1], w[2], w[3]);
    }
    if (sub == 0) {
      float *g4q = g4cs + (gs * 4 + g4c) * 4;  // (C_a, C_b, S_a, S_b) of the lane position
      g4q[g4sl] = C;
      g4q[2 + g4sl] = S;
    }
  }
  if (!real || bp.g4_only) return;
  // the general decode kernels' per-group layout: lane position c's two
  // window words give W, W' of their bytes (words 0..15) and the four
  // fifth-slot words (16..19), as chunk pairs of 16 bytes
  const int GL = g % kStageG;  // the group's index in its stage fixes its window
  unsigned char *Bg = P.wsB + (int64_t)g * kBTok * MB;
  for (int it = sub; it < 4 * kCP; it += 8) {
    const int c = it / kCP, cp = it % kCP;
    // group byte of byte k of lane c's word i (0: first, 1: second), or -1
    auto byte_of = [&](int i, int k) -> int {
      const int b = 4 * (first_word(GL, c) + 4 * i) + k - 26 * GL;
      return (b >= 0 && b < 26) ? b : -1;
    };
    uint32_t w[4];
    if (cp < 4) {
      // words 4 cp .. 4 cp + 3: W, W' of bytes k = 2 cp and 2 cp + 1 of the words (i = cp / 2)
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int bi = 2 * cp + e, b = byte_of(bi >> 2, bi & 3);
        w[2 * e] = b >= 0 ? pk(sv[tib][b][0], sv[tib][b][1]) : 0u;
        w[2 * e + 1] = b >= 0 ? pk(sv[tib][b][2], sv[tib][b][3]) : 0u;
      }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int b0 = byte_of(i >> 1, 2 * (i & 1)), b1 = byte_of(i >> 1, 2 * (i & 1) + 1);
        w[i] = pk(b0 >= 0 ? sv[tib][b0][4] : z, b1 >= 0 ? sv[tib][b1][4] : z);
      }
    }
    *reinterpret_cast<uint4 *>(Bg + ((m * kCP + cp) * 4 + c) * kBLane) = make_uint4(w[0], w[1], w[2], w[3]);
  }
  if (sub == 0) {
    // C, S of token m in its 8-token tile's block; unused tokens' entries zero
    float *cs = P.wsCS + (int64_t)g * (cs_group_bytes(MB) / 4);
    cs[(m >> 3) * 16 + (m & 7)] = C;
    cs[(m >> 3) * 16 + 8 + (m & 7)] = S;
    if (m == 0)
      for (int q = MB; q < (MB > 8 ? 16 : 8); ++q) cs[(q >> 3) * 16 + (q & 7)] = cs[(q >> 3) * 16 + 8 + (q & 7)] = 0.f;
  }
}

// ------------------------------------------------------------ plane 2
// One CTA (4 warps) per 128-row tile of one problem.  For each 32-group
// salience word, thread t = row t compacts the tile's salient pairs into
// per-group row lists; then the records (the 28 aligned bytes around each)
// and their s2 are staged in shared memory with asynchronous copies, one
// round of at most kRecCap records at a time, and each warp multiplies
// 16-record items of one group like the first plane (the activation
// fragments of the next item are loaded while the current one computes).
// s2 * P2 per row accumulates in shared memory and goes to the workspace
// (y2, fp32) at the end.
constexpr int kP2Threads = 128;
constexpr int kRecCap = 512;
constexpr int kMaxItems = kRecCap / 16 + 32;

__device__ __forceinline__ void cp_async4(void *dst, const void *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}

__device__ __forceinline__ void load_b_frag(const Problem &P, int g, int MB, int gq, int c, uint32_t *b, float2 &Cv) {
  const unsigned char *Bg = P.wsB + (int64_t)g * kBTok * MB;
#pragma unroll
  for (int cp = 0; cp < kCP; ++cp) {
    uint4 q = make_uint4(0u, 0u, 0u, 0u);
    if (gq < MB) q = __ldg(reinterpret_cast<const uint4 *>(Bg + ((gq * kCP + cp) * 4 + c) * kBLane));
    b[4 * cp] = q.x;
    b[4 * cp + 1] = q.y;
    b[4 * cp + 2] = q.z;
    b[4 * cp + 3] = q.w;
  }
  Cv = __ldg(reinterpret_cast<const float2 *>(P.wsCS + (int64_t)g * (kCSGroup / 4) + 2 * c));
}

__global__ void __launch_bounds__(kP2Threads) gemv_mma_p2_kernel(const __grid_constant__ BatchParams bp) {
  const int p = blockIdx.y;
  if (p >= bp.count) return;
  const Problem &P = bp.prob[p];
  const int n0 = blockIdx.x * kRows;
  if (n0 >= P.N) return;
  const int MB = bp.M;
  __shared__ uint32_t lut[256];
  __shared__ uint8_t rowl[32][kRows];  // row of each salient pair, per group
  __shared__ int jbase[kRows];         // record index of the row's first pair in this word
  __shared__ uint32_t bitsv[kRows];    // the row's salience bits of this word
  __shared__ int cnt[4][32];
  __shared__ int eoff[33];             // per-group offsets in the flat (group-major) pair order
  __shared__ int itm[kMaxItems];       // item: group << 16 | first flat pair
  __shared__ int nitm;
  __shared__ __align__(16) uint32_t rec[kRecCap][8];  // 28 record bytes + the record's word offset
  __shared__ float s2s[kRecCap];
  __shared__ float acc[kRows][8];
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  for (int i = t; i < 256; i += kP2Threads) lut[i] = lut_word(i);
  for (int i = t; i < kRows * 8; i += kP2Threads) (&acc[0][0])[i] = 0.f;
  const int n = n0 + t;
  const bool valid = n < P.N;
  const int G = P.K / kGroup, W = sal_words_of(P.K);
  int j = (valid && P.nnz > 0) ? P.rowptr[n] : 0;
  const uint32_t lt = (1u << lane) - 1u;
  const int gq = lane >> 2, c = lane & 3;
  __syncthreads();
  for (int w = 0; w < W && P.nnz > 0; ++w) {
    const int gbase = 32 * w, gw = min(32, G - gbase);
    uint32_t bits = valid ? P.sal[(int64_t)n * W + w] : 0u;
    if (gw < 32) bits &= (1u << gw) - 1u;
    jbase[t] = j;
    bitsv[t] = bits;
    for (int gl = 0; gl < 32; ++gl) {
      const uint32_t m = __ballot_sync(0xffffffffu, (bits >> gl) & 1u);
      if (lane == 0) cnt[warp][gl] = __popc(m);
    }
    __syncthreads();
    if (t < 32) {
      int s = 0;
      for (int ww = 0; ww < 4; ++ww) {
        const int v = cnt[ww][t];
        cnt[ww][t] = s;  // becomes the warp's base within the group
        s += v;
      }
      // exclusive scan of the group totals across the warp
      int incl = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      eoff[t] = incl - s;
      if (t == 31) eoff[32] = incl;
    }
    __syncthreads();
    for (int gl = 0; gl < 32; ++gl) {
      const uint32_t m = __ballot_sync(0xffffffffu, (bits >> gl) & 1u);
      if ((bits >> gl) & 1u) rowl[gl][cnt[warp][gl] + __popc(m & lt)] = (uint8_t)t;
    }
    j += __popc(bits);
    __syncthreads();
    const int E = eoff[32];
    for (int r0 = 0; r0 < E; r0 += kRecCap) {
      const int r1 = min(E, r0 + kRecCap);
      // ---- stage the round's records and s2
      for (int e = r0 + t; e < r1; e += kP2Threads) {
        int gl = 0;
#pragma unroll
        for (int step = 16; step >= 1; step >>= 1)
          if (gl + step < 32 && eoff[gl + step] <= e) gl += step;
        const int row = rowl[gl][e - eoff[gl]];
        const int64_t jj = min(max((int64_t)jbase[row] + __popc(bitsv[row] & ((1u << gl) - 1u)), (int64_t)0),
                               (int64_t)P.nnz - 1);
        const uint8_t *A = P.plane2 + jj * kGroupBytes;
        const int sh = (int)(jj & 1) * 2;  // plane 2 is 16-byte aligned: the record starts 0 or 2 bytes into a word
        const uint32_t *src = reinterpret_cast<const uint32_t *>(A - sh);
        uint32_t *dst = rec[e - r0];
#pragma unroll
        for (int i = 0; i < 6; ++i) cp_async4(dst + i, src + i);
        if (sh) {
          cp_async4(dst + 6, src + 6);
        } else {  // bytes 24, 25 only: the word after them may lie past the end of plane 2
          dst[6] = (uint32_t)__ldg(reinterpret_cast<const uint16_t *>(src + 6));
        }
        dst[7] = (uint32_t)sh;
        s2s[e - r0] = __half2float(P.s2[jj]);
      }
      asm volatile("cp.async.wait_all;" ::: "memory");
      if (t == 0) {
        int k = 0;
        for (int gl = 0; gl < gw; ++gl) {
          const int a = max(eoff[gl], r0), b = min(eoff[gl + 1], r1);
          for (int e = a; e < b; e += 16) itm[k++] = (gl << 16) | e;
        }
        nitm = k;
      }
      __syncthreads();
      // ---- items
      const int ni = nitm;
      uint32_t b[20], bn[20];
      float2 Cv = make_float2(0.f, 0.f), Cn = Cv;
      if (warp < ni) load_b_frag(P, gbase + (itm[warp] >> 16), MB, gq, c, b, Cv);
      for (int k = warp; k < ni; k += 4) {
        if (k + 4 < ni) load_b_frag(P, gbase + (itm[k + 4] >> 16), MB, gq, c, bn, Cn);
        const int gl = itm[k] >> 16, e0 = itm[k] & 0xffff;
        const int seg_end = min(eoff[gl + 1], r1);
        const int g = gbase + gl, GL = g % kStageG;
        const int o = (GL & 1) * 2;
        const int jw1 = ((c - win_start(GL)) % 4 + 4) % 4;
        uint32_t aL[20], aH[20];
        int rows[2] = {-1, -1};
        float s2v[2] = {0.f, 0.f};
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int e = e0 + gq + 8 * h;
          uint32_t win[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) win[i] = 0u;
          if (e < seg_end) {
            rows[h] = rowl[gl][e - eoff[gl]];
            s2v[h] = s2s[e - r0];
            const uint4 q0 = *reinterpret_cast<const uint4 *>(rec[e - r0]);
            const uint4 q1 = *reinterpret_cast<const uint4 *>(rec[e - r0] + 4);
            const uint32_t wv[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, 0u};
            const int sh = (int)q1.w;
            // place the record o = 26 GL % 4 bytes into its window
            if (sh == o) {
#pragma unroll
              for (int i = 0; i < 7; ++i) win[i] = wv[i];
            } else if (o == 2) {
#pragma unroll
              for (int i = 0; i < 7; ++i) win[i] = __funnelshift_l(i ? wv[i - 1] : 0u, wv[i], 16);
            } else {
#pragma unroll
              for (int i = 0; i < 7; ++i) win[i] = __funnelshift_r(wv[i], wv[i + 1], 16);
            }
          }
          uint32_t w0 = win[0], w1 = win[4];
#pragma unroll
          for (int i = 1; i < 4; ++i)
            if (jw1 == i) {
              w0 = win[i];
              w1 = win[i + 4];
            }
          decode_words_compact(w0, w1, lut, h ? aH : aL);
        }
        float d[4];
        group_mma(aL, aH, b, d);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          if (rows[h] < 0) continue;
          const float cc[2] = {Cv.x, Cv.y};
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            const int m = 2 * c + i;
            if (m < MB) atomicAdd(&acc[rows[h]][m], s2v[h] * (d[2 * h + i] - cc[i]));
          }
        }
#pragma unroll
        for (int i = 0; i < 20; ++i) b[i] = bn[i];
        Cv = Cn;
      }
      __syncthreads();  // the round's buffers are free again
    }
  }
  __syncthreads();
  if (valid) {
    float *y2 = P.y2() + (int64_t)n * MB;
    for (int m = 0; m < MB; ++m) y2[m] = acc[t][m];
  }
}

// Second plane, tensor-core version (1..8 tokens).  Persistent over the
// main kernel's tile ranges, in spans of 1..4 consecutive tiles of one
// problem (as many as keep the span's expected records within the record
// buffer).  For each span the CTA stages the rows' rowptr and salience words
// and the span's contiguous range of plane-2 records and s2 in shared
// memory, one span ahead (asynchronous copies; each span's metadata carries
// the next span's record bounds, so the next records can be requested at
// once; a span whose records exceed the buffer is done in several record
// ranges).  Warp w takes groups g = w, w + 16, ...: per 128 rows a ballot
// gives the rows whose bit g is set, compacted into a per-warp list with
// their records' places; 16 list entries form one m16 tile whose rows are
// records, decoded with the same encoding as the first plane and multiplied
// by group g's B fragment.  s2 * (D - C) per record accumulates per row in
// shared memory and goes to the workspace (y2) at the span's end.
constexpr int kQThreads = 512, kQWarps = 16;
constexpr int kQMaxSpanTiles = 4, kQMaxSpanRows = kQMaxSpanTiles * kRows;
constexpr int kQRecBuf = 47104;                                   // record bytes per buffer
constexpr int kQRecCap = (kQRecBuf - 16) / kGroupBytes;           // records per range
constexpr int kQRecPerThread = (kQRecCap + kQThreads - 1) / kQThreads;
constexpr int kQMaxW = 10;                                        // salience words per row
constexpr int kQMaxG = kQMaxW * 32;
constexpr int kQS2Buf = ((2 * kQRecCap + 8 + 15) / 16) * 16;      // s2 bytes per buffer
constexpr int kQMetaSal = 2304;                                   // salience words per span
struct QMeta {
  int32_t rp[kQMaxSpanRows + 4];  // rowptr of the span's rows (rows + 1 used)
  int32_t next[4];                // record bounds of the next span
  uint32_t sal[kQMetaSal];        // salience words, [row][W]
};
constexpr int kQMetaOff = 0;                                          // QMeta[2]
constexpr int kQListOff = kQMetaOff + 2 * (int)sizeof(QMeta);         // records by group: entry, s2
constexpr int kQCntOff = kQListOff + kQRecCap * 8;                    // per group: count, first entry
constexpr int kQAccOff = kQCntOff + 2 * kQMaxG * 4;                   // float [span row][8]
constexpr int kQS2Off = kQAccOff + kQMaxSpanRows * 8 * 4;             // s2 buffers
constexpr int kQEndA = kQS2Off + 2 * kQS2Buf;
static_assert(kQEndA <= kArena1, "plane-2 arrays overflow the region below the table");
constexpr int kQRecOff = kArena1 + kLutBytes;                         // record buffers, above the table
constexpr int kQRecStride = kQRecBuf + 64;
constexpr int kQDynBytes = kQRecOff + 2 * kQRecStride;
static_assert(kQDynBytes <= kDynBytes, "plane-2 shared memory");
static_assert(kQMetaSal >= kRows * kQMaxW, "one tile's salience words fit a span");

__device__ __forceinline__ void cp_async16_zfill(void *dst, const void *src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async4_zfill(void *dst, const void *src, int src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}

// Tiles per span of a problem: the expected records of a span (the mean
// per row, nnz / N) stay below 85 % of the buffer, the salience words fit.
__device__ __forceinline__ int q_span_tiles(const Problem &P) {
  const int W = sal_words_of(P.K);
  const int by_meta = kQMetaSal / (kRows * W);
  const int64_t per_tile = ((int64_t)kRows * P.nnz + P.N - 1) / P.N;
  const int by_rec = (int)min((int64_t)kQMaxSpanTiles, (int64_t)(kQRecCap * 85 / 100) / max(per_tile, (int64_t)1));
  return max(1, min(by_meta, by_rec));
}

// The span starting at the first tile at or after `tile` (below t_end) of
// a problem with a second plane; q is the problem to start the search from.
struct QSpan {
  int tile, ntiles, q, n0, rows;
  bool valid;
};
__device__ __forceinline__ QSpan q_span(const BatchParams &bp, int tile, int q, int t_end) {
  QSpan S{0, 0, 0, 0, 0, false};
  while (tile < t_end) {
    while (q + 1 < bp.count && bp.prob[q + 1].tile_begin <= tile) ++q;
    const Problem &P = bp.prob[q];
    const int p_end = P.tile_begin + (P.N + kRows - 1) / kRows;
    if (P.nnz > 0) {
      S.tile = tile, S.q = q;
      S.ntiles = min(q_span_tiles(P), min(p_end, t_end) - tile);
      S.n0 = (tile - P.tile_begin) * kRows;
      S.rows = min(S.ntiles * kRows, P.N - S.n0);
      S.valid = true;
      return S;
    }
    tile = p_end;  // skip the problem
  }
  return S;
}

// A record range: records [lo, hi) of plane 2 (of the span's [r0, end)),
// staged from the 16-byte boundary at or below byte 26 lo (delta bytes
// earlier); s2 from the 4-byte boundary at or below s2 + lo (ds bytes earlier).
struct QRange {
  int64_t lo, hi, end;
  int delta, ds;
};
__device__ __forceinline__ QRange q_range(const Problem &P, int32_t first, int32_t last, int64_t lo) {
  QRange R;
  const int64_t nnz = P.nnz;
  const int64_t r0 = min(max((int64_t)first, (int64_t)0), nnz);
  R.end = min(max((int64_t)last, r0), nnz);
  R.lo = lo < 0 ? r0 : lo;
  R.hi = min(R.end, R.lo + kQRecCap);
  R.delta = (int)((R.lo * kGroupBytes) & 15);
  R.ds = (int)(((uintptr_t)(P.s2 + R.lo)) & 3u);
  return R;
}

// The span's rowptr and salience words, and the next span's record bounds.
__device__ __forceinline__ void q_issue_meta(const BatchParams &bp, const QSpan &S, const QSpan &Sn, QMeta *M) {
  const Problem &P = bp.prob[S.q];
  const int W = sal_words_of(P.K);
  for (int i = threadIdx.x; i <= S.rows; i += kQThreads) cp_async4(&M->rp[i], P.rowptr + S.n0 + i);
  for (int i = threadIdx.x; i < S.rows * W; i += kQThreads) cp_async4(&M->sal[i], P.sal + (int64_t)S.n0 * W + i);
  if (Sn.valid && threadIdx.x < 2) {
    const Problem &Pn = bp.prob[Sn.q];
    cp_async4(&M->next[threadIdx.x], Pn.rowptr + Sn.n0 + (threadIdx.x ? Sn.rows : 0));
  }
}

__device__ __forceinline__ void q_issue_records(const Problem &P, const QRange &R, unsigned char *rec,
                                                unsigned char *s2b) {
  const int64_t a0 = R.lo * kGroupBytes - R.delta, end = R.hi * kGroupBytes, lim = P.nnz * kGroupBytes;
  const int nch = (int)((end - a0 + 15) / 16);
  for (int k = threadIdx.x; k < nch; k += kQThreads) {
    const int64_t off = a0 + 16 * (int64_t)k;
    cp_async16_zfill(rec + 16 * k, P.plane2 + off, (int)min((int64_t)16, lim - off));
  }
  const unsigned char *b0 = reinterpret_cast<const unsigned char *>(P.s2 + R.lo) - R.ds;
  const unsigned char *bend = reinterpret_cast<const unsigned char *>(P.s2 + R.hi);
  const unsigned char *blim = reinterpret_cast<const unsigned char *>(P.s2 + P.nnz);
  const int nw = (int)((bend - b0 + 3) / 4);
  for (int k = threadIdx.x; k < nw; k += kQThreads)
    cp_async4_zfill(s2b + 4 * k, b0 + 4 * k, (int)min((ptrdiff_t)4, blim - (b0 + 4 * k)));
}

template <bool ONE>
__global__ void __launch_bounds__(kQThreads, 1)
    gemv_mma_p2v3_kernel(const __grid_constant__ BatchParams bp, const __grid_constant__ Sched sc) {
  extern __shared__ __align__(1024) unsigned char dynq[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (smem_u32(dynq) != kDynShared) {
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  const int t_end = sc.cta_tile[blockIdx.x + 1];
  QSpan S = q_span(bp, sc.cta_tile[blockIdx.x], 0, t_end);
  if (!S.valid) return;
  QMeta *meta = reinterpret_cast<QMeta *>(dynq + kQMetaOff);
  uint32_t *list = reinterpret_cast<uint32_t *>(dynq + kQListOff);
  float *lists2 = reinterpret_cast<float *>(list + kQRecCap);
  int *gcnt = reinterpret_cast<int *>(dynq + kQCntOff);
  int *goff = gcnt + kQMaxG;
  float *acc = reinterpret_cast<float *>(dynq + kQAccOff);
  unsigned char *s2buf = dynq + kQS2Off;
  unsigned char *recbuf = dynq + kQRecOff;
  {
    uint32_t *lut = reinterpret_cast<uint32_t *>(dynq + kArena1);
    lut_fill_replicated(lut, tid, kQThreads);
    for (int i = tid; i < kQMaxSpanRows * 8; i += kQThreads) acc[i] = 0.f;
    for (int i = tid; i < kQMaxG; i += kQThreads) gcnt[i] = 0;
  }
  const int MB = ONE ? 1 : bp.M;
  const int g16 = lane >> 2, c = lane & 3;
  const uint32_t tag = kLutShared | ((uint32_t)lane << 2);

  // prologue: the first span's metadata (with the next span's record bounds), then its records
  QSpan S1 = q_span(bp, S.tile + S.ntiles, S.q, t_end);
  q_issue_meta(bp, S, S1, &meta[0]);
  cp_async_commit();
  cp_async_wait<0>();
  __syncthreads();
  q_issue_records(bp.prob[S.q], q_range(bp.prob[S.q], meta[0].rp[0], meta[0].rp[S.rows], -1), recbuf, s2buf);
  cp_async_commit();

  for (int k = 0; S.valid; ++k) {
    const int cur = k & 1, nxt = cur ^ 1;
    QMeta &M = meta[cur];
    cp_async_wait<0>();
    __syncthreads();  // this span's records and metadata are in; the previous span is done
    // request the next span's records (bounds from this span's metadata) and
    // its metadata (with the record bounds of the one after)
    QSpan S2{0, 0, 0, 0, 0, false};
    if (S1.valid) {
      S2 = q_span(bp, S1.tile + S1.ntiles, S1.q, t_end);
      q_issue_records(bp.prob[S1.q], q_range(bp.prob[S1.q], M.next[0], M.next[1], -1), recbuf + nxt * kQRecStride,
                      s2buf + nxt * kQS2Buf);
      q_issue_meta(bp, S1, S2, &meta[nxt]);
      cp_async_commit();
    }
    const Problem &P = bp.prob[S.q];
    const int G = P.K / kGroup, W = sal_words_of(P.K), rows = S.rows;
    unsigned char *rec = recbuf + cur * kQRecStride;
    unsigned char *s2b = s2buf + cur * kQS2Buf;
    const int rp0 = M.rp[0];
    QRange R = q_range(P, M.rp[0], M.rp[rows], -1);
    for (;;) {
      const int n_rel = (int)(R.hi - R.lo);
      // records of the range by group (counting sort): a record's row is the
      // last r with rp[r] <= j, its group the rank-th set bit of that row
      int rj[kQRecPerThread], gj[kQRecPerThread], pj[kQRecPerThread];
#pragma unroll
      for (int u = 0; u < kQRecPerThread; ++u) {
        const int jr = tid + u * kQThreads;
        gj[u] = -1;
        if (jr < n_rel) {
          const int j = (int)(R.lo - rp0) + jr;  // relative to the span's first record
          int r = 0;
#pragma unroll
          for (int step = kQMaxSpanRows / 2; step >= 1; step >>= 1)
            if (r + step < rows && M.rp[r + step] - rp0 <= j) r += step;
          int rank = j - (M.rp[r] - rp0), g = -1;
          for (int w = 0; w < W; ++w) {
            const uint32_t word = M.sal[r * W + w];
            const int cnt = __popc(word);
            if (rank < cnt) {
              g = 32 * w + (int)__fns(word, 0u, rank + 1);
              break;
            }
            rank -= cnt;
          }
          if (g >= 0 && g < G) {
            rj[u] = r;
            gj[u] = g;
            pj[u] = atomicAdd(&gcnt[g], 1);
          }
        }
      }
      __syncthreads();
      if (warp == 0) {
        // exclusive scan of the group counts (each lane a run of groups)
        const int per = (G + 31) / 32, g0 = lane * per;
        int run = 0;
        for (int i = 0; i < per; ++i)
          if (g0 + i < G) run += gcnt[g0 + i];
        int incl = run;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += v;
        }
        int base = incl - run;
        for (int i = 0; i < per; ++i)
          if (g0 + i < G) {
            goff[g0 + i] = base;
            base += gcnt[g0 + i];
          }
      }
      __syncthreads();
      // entry = span row | (4 + byte offset of the record's window in the buffer) << 9
#pragma unroll
      for (int u = 0; u < kQRecPerThread; ++u) {
        if (gj[u] < 0) continue;
        const int jr = tid + u * kQThreads, g = gj[u], GL = g % kStageG;
        const int pos = goff[g] + pj[u];
        list[pos] = (uint32_t)rj[u] | ((uint32_t)(R.delta + kGroupBytes * jr - 2 * (GL & 1) + 4) << 9);
        lists2[pos] = __half2float(*reinterpret_cast<const __half *>(s2b + R.ds + 2 * jr));
      }
      __syncthreads();
      for (int g = warp; g < G; g += kQWarps) {
        const int count = gcnt[g];
        if (count == 0) continue;
        const uint32_t *lg = list + goff[g];
        const float *sg = lists2 + goff[g];
        const int GL = g % kStageG;
        // the group's B fragment (lanes of absent tokens repeat the last token) and C
        const unsigned char *Bg = P.wsB + (int64_t)g * kBTok * MB + min(g16, MB - 1) * kBTok + c * kBLane;
        uint32_t b[20];
#pragma unroll
        for (int cp = 0; cp < kCP; ++cp) {
          const uint4 v = __ldg(reinterpret_cast<const uint4 *>(Bg + cp * 4 * kBLane));
          b[4 * cp] = v.x, b[4 * cp + 1] = v.y, b[4 * cp + 2] = v.z, b[4 * cp + 3] = v.w;
        }
        const float2 Cv = __ldg(reinterpret_cast<const float2 *>(P.wsCS + (int64_t)g * (kCSGroup / 4) + 2 * c));
        // lane c's window words: win_start + jw and + 4 (the record starts o bytes in)
        const int jw = (c - win_start(GL)) & 3;
        for (int e0 = 0; e0 < count; e0 += 16) {
          uint32_t aL[20], aH[20];
          int rowv[2];
          float s2v[2];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int s = e0 + g16 + 8 * h;
            const uint32_t e = s < count ? lg[s] : 4u << 9;
            rowv[h] = s < count ? (int)(e & 511u) : -1;
            s2v[h] = sg[s < count ? s : 0];
            const uint32_t a = (e >> 9) + 4 * jw, sh = (a & 3u) * 8u;
            const uint32_t *wp = reinterpret_cast<const uint32_t *>(rec - 4 + (a & ~3u));
            decode_words(__funnelshift_r(wp[0], wp[1], sh), __funnelshift_r(wp[4], wp[5], sh), tag, h ? aH : aL);
          }
          float d[4];
          group_mma(aL, aH, b, d);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            if (rowv[h] < 0) continue;
            if (ONE) {
              if (c == 0) atomicAdd(&acc[rowv[h] * 8], s2v[h] * (d[2 * h] - Cv.x));
            } else {
#pragma unroll
              for (int i = 0; i < 2; ++i) {
                const int m = 2 * c + i;
                if (m < MB) atomicAdd(&acc[rowv[h] * 8 + m], s2v[h] * (d[2 * h + i] - (i ? Cv.y : Cv.x)));
              }
            }
          }
        }
      }
      __syncthreads();
      for (int i = tid; i < G; i += kQThreads) gcnt[i] = 0;
      if (R.hi >= R.end) break;
      // a further record range of this span (the buffer holds kQRecCap records)
      __syncthreads();
      R = q_range(P, M.rp[0], M.rp[rows], R.hi);
      q_issue_records(P, R, rec, s2b);
      cp_async_commit();
      cp_async_wait<0>();
      __syncthreads();
    }
    __syncthreads();
    for (int i = tid; i < rows * MB; i += kQThreads) {
      const int r = ONE ? i : i / MB, m = ONE ? 0 : i - r * MB;
      P.y2()[(int64_t)(S.n0 + r) * MB + m] = acc[r * 8 + m];
      acc[r * 8 + m] = 0.f;
    }
    S = S1;
    S1 = S2;
  }
  cp_async_wait<0>();
}

// Second plane with the group-ordered index (1..8 tokens).  Persistent
// warps take units from a counter in the workspace: a unit is one of the
// c_parts contiguous shares of one group's 16-entry tiles, numbered problem
// by problem (CBase: the first unit of each problem).  For its unit a warp
// loads group g's B fragment and C once and runs the tiles as m16 tiles:
// lane (r, c) loads slot words 2 jw, 2 jw + 1 of entries r and r + 8 (its
// two window words, one 8-byte load per entry; a quad's loads cover the
// slot), decodes them with the lane-replicated table and, after the MMAs,
// takes the entries' rows and s2 from the quad's lanes that hold them;
// s2 (D - C) per entry is added to y2 of the entry's row with a global
// atomic (the prep kernel zeroes y2).
// threads per CTA: 1024 (64 registers) for up to 8 tokens, 768 for the
// second token tile's extra fragment registers
__host__ __device__ constexpr int c_threads(bool two) { return two ? 768 : 1024; }
constexpr int kCDynBytes2 = kArena1 + kLutBytes;  // the table of codes at its fixed address
constexpr int kCUnitTiles = 32;                   // target tiles per unit

// The kernel's first parameter, so that the loop's indexed reads of it stay
// at the low offsets of the parameter space.
struct CBase {
  int32_t count;                   // problems
  int32_t base[TQ_MAX_BATCH + 1];  // first unit of problem p (base[count]: all units)
};

// Units per group: the mean tiles per group over kCUnitTiles, rounded up, 1 .. 32.
__host__ __device__ __forceinline__ int c_parts(int K, int64_t nnz) {
  const int64_t per = (int64_t)(K / kGroup) * 16 * kCUnitTiles;
  const int64_t q = (nnz + per - 1) / per;
  return (int)(q < 1 ? 1 : q > 32 ? 32 : q);
}

template <bool ONE, bool TWO>
__global__ void __launch_bounds__(c_threads(TWO), 1)
    gemv_mma_p2c_kernel(const __grid_constant__ CBase cb, const __grid_constant__ BatchParams bp, int32_t *counter) {
  extern __shared__ __align__(1024) unsigned char dync[];
  const int tid = threadIdx.x, lane = tid & 31;
  if (smem_u32(dync) != kDynShared) {
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  {
    uint32_t *lut = reinterpret_cast<uint32_t *>(dync + kArena1);
    lut_fill_replicated(lut, tid, c_threads(TWO));
  }
  __syncthreads();
  // the work below reads the prep kernel's output (launched programmatically
  // after it); the main kernel may start its set-up meanwhile
  grid_dep_wait();
  grid_dep_launch_next();
  const int MB = ONE ? 1 : bp.M, g16 = lane >> 2, c = lane & 3, quad = lane & ~3;
  const uint32_t tag = kLutShared | ((uint32_t)lane << 2);
  const int count = cb.count, total = cb.base[count];
  for (;;) {
    int u = 0;
    if (lane == 0) u = atomicAdd(counter, 1);
    u = __shfl_sync(0xffffffffu, u, 0);
    if (u >= total) break;
    int i = 0;  // the unit's problem: the last i with base[i] <= u
    for (int step = 128; step >= 1; step >>= 1)
      if (i + step < count && cb.base[i + step] <= u) i += step;
    const Problem &P = bp.prob[i];
    const int S = c_parts(P.K, P.nnz), local = u - cb.base[i];
    const int g = local / S, part = local - g * S, GL = g % kStageG;
    // the group's entries, clamped into the index (whole tiles)
    const int64_t cap = c_capacity(P.K, P.nnz);
    const int64_t e0 = min(max((int64_t)__ldg(P.p2idx + g), (int64_t)0), cap) & ~(int64_t)15;
    const int64_t e1 = min(max((int64_t)__ldg(P.p2idx + g + 1), e0), cap) & ~(int64_t)15;
    const uint32_t nt = (uint32_t)((e1 - e0) >> 4);  // below 2^27: nt * 32 fits 32 bits
    const int t0 = (int)(nt * (uint32_t)part / (uint32_t)S);
    const int n = (int)(nt * (uint32_t)(part + 1) / (uint32_t)S) - t0;
    if (n <= 0) continue;
    // the group's B fragment (lanes of absent tokens repeat the last token) and C
    const unsigned char *Bg = P.wsB + (int64_t)g * kBTok * MB + min(g16, MB - 1) * kBTok + c * kBLane;
    uint32_t b[20], b2[20];  // tokens g16 and (more than 8 tokens) 8 + g16 as MMA columns
#pragma unroll
    for (int cp = 0; cp < kCP; ++cp) {
      const uint4 v = __ldg(reinterpret_cast<const uint4 *>(Bg + cp * 4 * kBLane));
      b[4 * cp] = v.x, b[4 * cp + 1] = v.y, b[4 * cp + 2] = v.z, b[4 * cp + 3] = v.w;
    }
    const float *csg = P.wsCS + (int64_t)g * (cs_group_bytes(MB) / 4);
    const float2 Cv = __ldg(reinterpret_cast<const float2 *>(csg + (ONE ? 0 : 2 * c)));
    float2 Cv2 = make_float2(0.f, 0.f);
    if (TWO) {
      const unsigned char *Bg2 = P.wsB + (int64_t)g * kBTok * MB + min(8 + g16, MB - 1) * kBTok + c * kBLane;
#pragma unroll
      for (int cp = 0; cp < kCP; ++cp) {
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(Bg2 + cp * 4 * kBLane));
        b2[4 * cp] = v.x, b2[4 * cp + 1] = v.y, b2[4 * cp + 2] = v.z, b2[4 * cp + 3] = v.w;
      }
      Cv2 = __ldg(reinterpret_cast<const float2 *>(csg + 16 + 2 * c));
    }
    p2_tiles<ONE, TWO>(P, MB, GL, e0, t0, n, b, b2, Cv, Cv2, lane, tag);
  }
}

// ------------------------------------------------------------------ main
template <bool F32, bool ONE, bool TWO>
__global__ void __launch_bounds__(kThreads, 1)
    gemv_mma_kernel(const __grid_constant__ BatchParams bp, const __grid_constant__ Sched sc) {
  extern __shared__ __align__(1024) unsigned char dyn[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int M = ONE ? 1 : bp.M, MB = M;
  if (smem_u32(dyn) != kDynShared) {
    // the table address trick needs the dynamic window right after the
    // reserved 1 KiB of shared memory; anything else is reported
    if (tid == 0) atomicOr(&g_tq_device_status, 2u);
    return;
  }
  const Layout L(MB);
  const int NS = L.NS;
  unsigned char *ar1 = dyn, *ar2 = dyn + kArena1 + kLutBytes;
  auto bytes_buf = [&](int b) -> unsigned char * {
    return b < 2 ? ar1 + b * kBytesSlot : ar2 + L.oBytes2 + (b - 2) * kBytesSlot;
  };
  Bars *bars = reinterpret_cast<Bars *>(ar1 + kBarOff);
  volatile int32_t *abort_ = &bars->abort_;

  // ---- one-time set-up: the lane-replicated table, barriers
  {
    uint32_t *lut = reinterpret_cast<uint32_t *>(dyn + kArena1);
    lut_fill_replicated(lut, tid, kThreads);
  }
  if (tid == 0) {
    for (int i = 0; i < NS; ++i) {
      mbar_init(&bars->full[i], 1 + 32);  // the producer's expect-tx arrival + its lanes' s1/off arrivals
      mbar_init(&bars->empty[i], kWarpsP1);
    }
    bars->abort_ = 0;
    mbar_fence_init();
  }
  __syncthreads();
  const int t_begin = sc.cta_tile[blockIdx.x], t_end = sc.cta_tile[blockIdx.x + 1];

  if (warp < kWarpsP1) {
    // ============================================================ decode
    // Warp mt owns the 16 rows of m16 tile mt and every group of a stage.
    {
      const int mt = warp;
      const int g = lane >> 2, c = lane & 3;
      const int R0 = mt * 16 + g, R1 = R0 + 8;
      const uint32_t tag = kLutShared | ((uint32_t)lane << 2);
      uint32_t b[20], b2[20];  // tokens g, and (more than 8 tokens) 8 + g, as MMA columns
      float y[4] = {0.f, 0.f, 0.f, 0.f};  // (R0, 2c), (R0, 2c+1), (R1, 2c), (R1, 2c+1)
      float y2t[4] = {0.f, 0.f, 0.f, 0.f};  // the same for tokens 8 + 2c, 8 + 2c + 1
      constexpr int CSF = (TWO ? 2 : 1) * kCSGroup / 4;  // C/S floats per group
      uint32_t buf = 0, phase = 0;
      for (Walk w(&bp, t_begin, t_end); w.valid(); w.next()) {
        // the stage's rows, s1 / off, B and C / S are in slot buf
        const bool ok = __all_sync(0xffffffffu, wait_or_abort(&bars->full[buf], phase, abort_));
        if (!ok) break;
        const unsigned char *Bst = ar2 + L.oB + buf * L.BStage;
        // this lane's B words (lanes of absent tokens load the last token's:
        // their output columns are never written)
        const unsigned char *Bl = Bst + min(g, MB - 1) * kBTok + c * kBLane;
        const unsigned char *Bl2 = Bst + min(8 + g, MB - 1) * kBTok + c * kBLane;
        const float *CSst = reinterpret_cast<const float *>(ar2 + L.oCS + buf * L.CSStage);
        const unsigned char *SO = ar2 + L.oSO + buf * kSOSlot;
        const uint4 s1a = *reinterpret_cast<const uint4 *>(SO + R0 * 16);
        const uint4 s1b = *reinterpret_cast<const uint4 *>(SO + R1 * 16);
        const uint4 ofa = *reinterpret_cast<const uint4 *>(SO + kRows * 16 + R0 * 16);
        const uint4 ofb = *reinterpret_cast<const uint4 *>(SO + kRows * 16 + R1 * 16);
        const uint32_t s1w[2][4] = {{s1a.x, s1a.y, s1a.z, s1a.w}, {s1b.x, s1b.y, s1b.z, s1b.w}};
        const uint32_t ofw[2][4] = {{ofa.x, ofa.y, ofa.z, ofa.w}, {ofb.x, ofb.y, ofb.z, ofb.w}};
        const int gs = w.gs;
        // s1 / off / C / S of group GL applied to its accumulators d
        auto epilogue = [&](auto glc, const float *d, const float *d2) {
          constexpr int GL = decltype(glc)::value;
          if (ONE) {
            // one token: only column 0 (lanes c = 0) is ever written
            const float Cx = CSst[GL * CSF + 2 * c], Sx = CSst[GL * CSF + 8 + 2 * c];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const float s1 = half_of<(GL & 1) != 0>(s1w[h][GL >> 1]);
              const float of = half_of<(GL & 1) != 0>(ofw[h][GL >> 1]);
              y[2 * h] = fmaf(s1, d[2 * h] - Cx, fmaf(of, Sx, y[2 * h]));
            }
            return;
          }
          const float2 Cv = *reinterpret_cast<const float2 *>(CSst + GL * CSF + 2 * c);
          const float2 Sv = *reinterpret_cast<const float2 *>(CSst + GL * CSF + 8 + 2 * c);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const float s1 = half_of<(GL & 1) != 0>(s1w[h][GL >> 1]);
            const float of = half_of<(GL & 1) != 0>(ofw[h][GL >> 1]);
            y[2 * h] = fmaf(s1, d[2 * h] - Cv.x, fmaf(of, Sv.x, y[2 * h]));
            y[2 * h + 1] = fmaf(s1, d[2 * h + 1] - Cv.y, fmaf(of, Sv.y, y[2 * h + 1]));
          }
          if (TWO) {
            // tokens 8 + 2c, 8 + 2c + 1: the second C/S block
            const float2 Cw = *reinterpret_cast<const float2 *>(CSst + GL * CSF + 16 + 2 * c);
            const float2 Sw = *reinterpret_cast<const float2 *>(CSst + GL * CSF + 24 + 2 * c);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const float s1 = half_of<(GL & 1) != 0>(s1w[h][GL >> 1]);
              const float of = half_of<(GL & 1) != 0>(ofw[h][GL >> 1]);
              y2t[2 * h] = fmaf(s1, d2[2 * h] - Cw.x, fmaf(of, Sw.x, y2t[2 * h]));
              y2t[2 * h + 1] = fmaf(s1, d2[2 * h + 1] - Cw.y, fmaf(of, Sw.y, y2t[2 * h + 1]));
            }
          }
        };
        // Software pipeline over the stage's groups: the MMAs of group GL run
        // while group GL + 1 is decoded; GL's epilogue comes after that.
        float dp[4] = {0.f, 0.f, 0.f, 0.f}, dp2[4] = {0.f, 0.f, 0.f, 0.f};
        // lane (g, c)'s window words of a group at shift k = win_start % 4:
        // stage-row words win_start + ((c - k) & 3) (+ 4) of rows R0, R1
        const unsigned char *rowp = bytes_buf(buf) + R0 * kStageBytes;
        const unsigned char *wb[4] = {rowp + 4 * (c & 3), rowp + 4 * ((c - 1) & 3), rowp + 4 * ((c - 2) & 3),
                                      rowp + 4 * ((c - 3) & 3)};
        auto group = [&](auto glc, auto fullc) {
          constexpr int GL = decltype(glc)::value;
          constexpr bool FULL = decltype(fullc)::value;
          if (FULL || GL < gs) {
            constexpr int ws = win_start(GL);
            const unsigned char *src = wb[ws % 4] + 4 * ws;
            const uint32_t x00 = *reinterpret_cast<const uint32_t *>(src);
            const uint32_t x01 = *reinterpret_cast<const uint32_t *>(src + 16);
            const uint32_t x10 = *reinterpret_cast<const uint32_t *>(src + 8 * kStageBytes);
            const uint32_t x11 = *reinterpret_cast<const uint32_t *>(src + 8 * kStageBytes + 16);
            uint32_t aL[20], aH[20];
            decode_words(x00, x01, tag, aL);
            decode_words(x10, x11, tag, aH);
            {
              const uint4 *bq = reinterpret_cast<const uint4 *>(Bl + GL * kBTok * MB);
#pragma unroll
              for (int cp = 0; cp < kCP; ++cp) {
                const uint4 v = bq[cp * 4];
                b[4 * cp] = v.x, b[4 * cp + 1] = v.y, b[4 * cp + 2] = v.z, b[4 * cp + 3] = v.w;
              }
              if (TWO) {
                const uint4 *bq2 = reinterpret_cast<const uint4 *>(Bl2 + GL * kBTok * MB);
#pragma unroll
                for (int cp = 0; cp < kCP; ++cp) {
                  const uint4 v = bq2[cp * 4];
                  b2[4 * cp] = v.x, b2[4 * cp + 1] = v.y, b2[4 * cp + 2] = v.z, b2[4 * cp + 3] = v.w;
                }
              }
            }
            float d[4], d2[4] = {0.f, 0.f, 0.f, 0.f};
            // one token tile: two chains; two tiles: one chain each (the
            // tiles' MMAs are independent already, and the registers short)
            if (TWO) {
              group_mma(aL, aH, b, d);
              group_mma(aL, aH, b2, d2);
            } else {
              group_mma2(aL, aH, b, d);
            }
            if constexpr (GL >= 1) epilogue(std::integral_constant<int, GL - 1>{}, dp, dp2);
#pragma unroll
            for (int i = 0; i < 4; ++i) dp[i] = d[i], dp2[i] = d2[i];
          }
        };
        auto stage = [&](auto fullc) {
          group(std::integral_constant<int, 0>{}, fullc);
          group(std::integral_constant<int, 1>{}, fullc);
          group(std::integral_constant<int, 2>{}, fullc);
          group(std::integral_constant<int, 3>{}, fullc);
          group(std::integral_constant<int, 4>{}, fullc);
          group(std::integral_constant<int, 5>{}, fullc);
          group(std::integral_constant<int, 6>{}, fullc);
          group(std::integral_constant<int, 7>{}, fullc);
        };
        if (gs == kStageG) {
          // a full stage: straight-line code
          stage(std::true_type{});
          epilogue(std::integral_constant<int, kStageG - 1>{}, dp, dp2);
        } else {
          stage(std::false_type{});
          // the epilogue of the stage's last group
          auto last = [&](auto glc) {
            constexpr int GL = decltype(glc)::value;
            if (GL < gs && GL + 1 >= gs) epilogue(glc, dp, dp2);
          };
          last(std::integral_constant<int, 0>{});
          last(std::integral_constant<int, 1>{});
          last(std::integral_constant<int, 2>{});
          last(std::integral_constant<int, 3>{});
          last(std::integral_constant<int, 4>{});
          last(std::integral_constant<int, 5>{});
          last(std::integral_constant<int, 6>{});
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->empty[buf]);
        if (w.last_stage()) {
          // add the second plane and write y
          {
            const Problem &P = w.P();
            const int nb = (w.tile - P.tile_begin) * kRows;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int n = nb + (h ? R1 : R0);
              if (n < P.N) {
#pragma unroll
                for (int t2 = 0; t2 < (TWO ? 2 : 1); ++t2)
#pragma unroll
                  for (int i = 0; i < 2; ++i) {
                    const int m = 8 * t2 + 2 * c + i;
                    if (m < M) {
                      float v = t2 ? y2t[2 * h + i] : y[2 * h + i];
                      if (P.nnz > 0) v += P.y2()[(int64_t)n * MB + m];
                      if (F32)
                        static_cast<float *>(P.y)[(int64_t)m * P.N + n] = v;
                      else
                        static_cast<__half *>(P.y)[(int64_t)m * P.N + n] = __float2half_rn(v);
                    }
                  }
              }
            }
          }
#pragma unroll
          for (int i = 0; i < 4; ++i) y[i] = 0.f, y2t[i] = 0.f;
        }
        if (++buf == (uint32_t)NS) buf = 0, phase ^= 1u;
      }
    }
  } else if (warp == kWarpProd) {
    // ========================================================== producer
    // Per stage: the tile's plane-1 bytes (one 2-D tensor copy), B and C / S
    // (bulk copies), counted in bytes on full[buf]; s1 / off (16-byte
    // asynchronous copies spread over the lanes), each lane arriving on
    // full[buf] once its copies landed.
    uint32_t buf = 0, phase = 0, q = 0;
    int map_pi = -1;
    for (Walk w(&bp, t_begin, t_end); w.valid(); w.next(), ++q) {
      const Problem &P = w.P();
      const int gs = w.gs, g0 = w.s * kStageG;
      const int n0 = (w.tile - P.tile_begin) * kRows, rows = min(kRows, P.N - n0);
      const uint32_t bb = (uint32_t)(gs * kBTok * MB);
      const uint32_t cb = (uint32_t)(gs * cs_group_bytes(MB));
      int ok = 1;
      if (lane == 0) ok = wait_or_abort(&bars->empty[buf], phase ^ 1u, abort_) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, ok, 0)) break;  // uniform across the warp
      uint64_t *full = &bars->full[buf];
      // s1 / off go by tensor copies when their rows are whole 16-byte units
      // (the prep kernel then built their maps), else by asynchronous copies
      const int G = P.K / kGroup;
      const bool so_map = (G % 8 == 0) && ((((uintptr_t)P.s1) | ((uintptr_t)P.off)) & 15u) == 0;
      unsigned char *so = ar2 + L.oSO + buf * kSOSlot;
      const unsigned char *maps = static_cast<const unsigned char *>(P.map());
      if (lane == 0) {
        if (w.pi != map_pi) {
          // the problem's tensor maps, written by the prep kernel
          asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps) : "memory");
          if (so_map) {
            asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps + kMapS1) : "memory");
            asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(maps + kMapOff) : "memory");
          }
          map_pi = w.pi;
        }
        mbar_arrive_expect_tx(full, bb + cb + (uint32_t)kBytesSlot + (so_map ? (uint32_t)kSOSlot : 0u));
        bulk_g2s(ar2 + L.oB + buf * L.BStage, P.wsB + (int64_t)g0 * kBTok * MB, bb, full);
        bulk_g2s(ar2 + L.oCS + buf * L.CSStage, reinterpret_cast<const unsigned char *>(P.wsCS) + (int64_t)g0 * cs_group_bytes(MB),
                 cb, full);
        // the stage's 208 bytes of the tile's 128 rows (rows past N and bytes
        // past the row's end arrive as zeros)
        asm volatile(
            "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                smem_u32(bytes_buf((int)buf))),
            "l"(maps), "r"(w.s * kStageBytes), "r"(n0), "r"(smem_u32(full))
            : "memory");
        if (so_map) {
          // the stage's 8 groups of s1 and of off for the 128 rows (16 bytes a row)
          asm volatile(
              "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                  smem_u32(so)),
              "l"(maps + kMapS1), "r"(g0), "r"(n0), "r"(smem_u32(full))
              : "memory");
          asm volatile(
              "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
                  smem_u32(so + kRows * 16)),
              "l"(maps + kMapOff), "r"(g0), "r"(n0), "r"(smem_u32(full))
              : "memory");
        }
      }
      __syncwarp();
      if (so_map) {
        mbar_arrive(full);  // the lanes' arrivals (the barrier counts 1 + 32)
      } else {
        {
          for (int r = lane; r < rows; r += 32) {
            const int64_t o = (int64_t)(n0 + r) * G + g0;
            __half *d1 = reinterpret_cast<__half *>(so + r * 16);
            __half *d2 = reinterpret_cast<__half *>(so + kRows * 16 + r * 16);
            for (int gg = 0; gg < kStageG; ++gg) {
              d1[gg] = gg < gs ? P.s1[o + gg] : __float2half_rn(0.f);
              d2[gg] = gg < gs ? P.off[o + gg] : __float2half_rn(0.f);
            }
          }
          mbar_arrive(full);
        }
      }
      if (++buf == (uint32_t)NS) buf = 0, phase ^= 1u;
    }
    cp_async_wait<0>();  // nothing of this warp in flight at exit
    // drain: every issued copy lands before the CTA exits (waited on even
    // after an abort; bounded by the wall-time limit)
    if (lane == 0) {
      for (uint32_t k = (q > (uint32_t)NS ? q - NS : 0); k < q; ++k) mbar_wait(&bars->full[k % NS], (k / NS) & 1u);
    }
  }
  __syncthreads();
}

}  // namespace mm

// -------------------------------------------------------------- launcher
cudaError_t launch_gemv_g4(const BatchParams &bp, int num_sms, cudaStream_t s);
cudaError_t launch_gemv_p2r(const BatchParams &bp, int num_sms, int32_t *counter, cudaStream_t s);
int g4_split_for(const BatchParams &bp, int num_sms);
cudaError_t launch_gemv_seq(const BatchParams &bp, int num_sms, int barrier_extra, cudaStream_t s);

static int num_sms_mm() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

int mma_rows_per_tile() { return mm::kRows; }

// Workspace bytes of one problem for M <= 16 tokens: B fragments, C/S, y2.
void mma_workspace_parts(int M, int N, int K, size_t *b, size_t *cs, size_t *y2) {
  const size_t G = (size_t)(K / kGroup);
  *b = G * (size_t)mm::kBTok * (size_t)M;
  *cs = G * (size_t)mm::cs_group_bytes(M);
  *y2 = (size_t)N * (size_t)M * 4;
}

TQ_STATUS_ACCESSOR(read_status_gemv_mma)

// Template tensor maps, encoded once per (kind, row length, rows) and cached:
// kind 0 = plane 1 as a 2-D byte tensor of rows of `len` bytes (box 208 x 128
// bytes); kind 1 = s1 / off as a 2-D fp16 tensor of rows of `len` halves (box
// 8 x 128); kinds 2, 3 and 4 for the one-group-per-lane kernel of M <= 2:
// plane 1 in boxes of 112 x 256 bytes (4-group stages, two tokens) or
// 208 x 256 (8-group stages, one token), s1 / off in boxes of 8 x 256 halves.
// No swizzle, zero fill.
// The prep kernel puts in each problem's address.
static bool map_template(int kind, int64_t len, const void *addr, int N, CUtensorMap *out) {
  // the driver's encoder, looked up through the runtime (no link-time
  // dependence on the driver library)
  static PFN_cuTensorMapEncodeTiled_v12000 encode = [] {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      fn = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }();
  if (!encode) return false;
  static std::mutex mu;
  static int64_t keys[64];
  static CUtensorMap maps[64];
  static int n = 0;
  const int64_t key = ((int64_t)N << 32) | (len << 3) | kind;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < n; ++i)
    if (keys[i] == key) {
      *out = maps[i];
      return true;
    }
  CUtensorMap m;
  const bool halves = (kind & 1) != 0;
  const int esz = halves ? 2 : 1;
  cuuint64_t dims[2] = {(cuuint64_t)len, (cuuint64_t)N};
  cuuint64_t strides[1] = {(cuuint64_t)(len * esz)};
  const cuuint32_t box_rows = kind >= 2 ? (cuuint32_t)g4::kRows : (cuuint32_t)mm::kRows;
  const cuuint32_t box_x = halves ? 8u : (kind == 0 || kind == 4) ? (cuuint32_t)mm::kStageBytes : 112u;
  cuuint32_t box[2] = {box_x, box_rows};
  cuuint32_t estr[2] = {1, 1};
  if (encode(&m, halves ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(addr),
             dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return false;
  if (n < 64) keys[n] = key, maps[n] = m, ++n;
  *out = m;
  return true;
}

// s1 / off of a problem go by tensor copies (rows of whole 16-byte units)
static bool scales_by_map(const Problem &P) {
  return (P.K / kGroup) % 8 == 0 && (((uintptr_t)P.s1 | (uintptr_t)P.off) & 15u) == 0;
}

static_assert(sizeof(BatchParams) + sizeof(mm::MapTemplates) + 8 <= 32764, "prep kernel parameters");
static_assert(sizeof(mm::CBase) + sizeof(BatchParams) + 8 <= 32764, "indexed second-plane kernel parameters");
static_assert(sizeof(BatchParams) + sizeof(mm::Sched) <= 32764, "main kernel parameters");

// Distinct tensor-map templates of a batch's problems (up to `cap` + 1 are
// counted): (row length, rows) of plane 1, and (groups, rows) of scales by map.
static int distinct_row_lengths(const BatchParams &bp, int first, int last, int cap) {
  int64_t seen[mm::kMaxMapTemplates + 2] = {};
  int n = 0;
  auto add = [&](int64_t key) {
    int k = 0;
    while (k < n && seen[k] != key) ++k;
    if (k == n) seen[n++] = key;
  };
  for (int i = first; i < last && n <= cap; ++i) {
    const int64_t rows = (int64_t)bp.prob[i].N << 32;
    add(rows | (row_bytes_of(bp.prob[i].K) << 1));
    if (scales_by_map(bp.prob[i])) add(rows | ((int64_t)(bp.prob[i].K / kGroup) << 1) | 1);
  }
  return n;
}

// The tensor-map templates of a batch (one per distinct kind and size) and
// each problem's template indices.  g4path: the one-group-per-lane layouts
// (kinds 2/4 and 3) instead of the general kernel's (0 and 1).
static cudaError_t build_templates(const BatchParams &bp, bool g4path, mm::MapTemplates &mt) {
  int64_t keys[mm::kMaxMapTemplates] = {};
  int nt = 0;
  auto slot = [&](int kind, int64_t len, const void *addr, int N) -> int {
    const int64_t key = ((int64_t)N << 32) | (len << 3) | kind;
    int k = 0;
    while (k < nt && keys[k] != key) ++k;
    if (k == nt) {
      if (nt == mm::kMaxMapTemplates) return -1;  // launch_mm splits such batches
      CUtensorMap enc;
      if (!map_template(kind, len, addr, N, &enc)) return -2;
      std::memcpy(&mt.t[nt][0], &enc, sizeof(enc));
      keys[nt++] = key;
    }
    return k;
  };
  for (int i = 0; i < bp.count; ++i) {
    const Problem &P = bp.prob[i];
    const int k1 = slot(g4path ? (bp.M == 1 ? 4 : 2) : 0, row_bytes_of(P.K), P.plane1, P.N);
    if (k1 < 0) return k1 == -1 ? cudaErrorNotSupported : cudaErrorInvalidValue;
    mt.idx[i] = (uint8_t)k1;
    mt.idx_so[i] = mm::kNoMap;
    if (scales_by_map(P)) {
      const int k2 = slot(g4path ? 3 : 1, P.K / kGroup, P.s1, P.N);
      if (k2 < 0) return k2 == -1 ? cudaErrorNotSupported : cudaErrorInvalidValue;
      mt.idx_so[i] = (uint8_t)k2;
    }
  }
  return cudaSuccess;
}

// The prep kernel, launched programmatically after the stream's previous
// kernel (it waits for that kernel before touching memory), so that its
// launch overlaps the previous kernel's tail.
static cudaError_t launch_prep(const BatchParams &bp, const mm::MapTemplates &mt, int32_t *counter, int gtasks,
                               cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((gtasks + mm::kPrepTasks - 1) / mm::kPrepTasks, bp.count);
  cfg.blockDim = dim3(128);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, mm::gemv_mma_prep_kernel, bp, mt, counter);
}

template <bool F32>
static cudaError_t launch_mm_one(const BatchParams &bp, cudaStream_t s);

// A batch with more distinct row lengths than tensor-map templates runs as
// consecutive sub-batches (in order, same stream).
template <bool F32>
static cudaError_t launch_mm(const BatchParams &bp, cudaStream_t s) {
  if (distinct_row_lengths(bp, 0, bp.count, mm::kMaxMapTemplates) <= mm::kMaxMapTemplates) return launch_mm_one<F32>(bp, s);
  thread_local BatchParams sub;
  int i = 0;
  while (i < bp.count) {
    int j = i + 1;
    while (j < bp.count && distinct_row_lengths(bp, i, j + 1, mm::kMaxMapTemplates) <= mm::kMaxMapTemplates) ++j;
    sub.count = j - i;
    sub.M = bp.M;
    sub.out_f32 = bp.out_f32;
    int tiles = 0;
    for (int k = 0; k < sub.count; ++k) {
      sub.prob[k] = bp.prob[i + k];
      sub.prob[k].tile_begin = tiles;
      tiles += (sub.prob[k].N + mm::kRows - 1) / mm::kRows;
    }
    sub.total_tiles = tiles;
    const cudaError_t e = launch_mm_one<F32>(sub, s);
    if (e != cudaSuccess) return e;
    i = j;
  }
  return cudaSuccess;
}

template <bool F32>
static cudaError_t launch_mm_one(const BatchParams &bp_in, cudaStream_t s) {
  // the batch with the M <= 2 kernel's tile split filled in
  thread_local BatchParams bp;
  bp = bp_in;
  bp.g4_split = g4::takes(bp) ? g4_split_for(bp, num_sms_mm()) : 1;
  thread_local mm::Sched sc;
  if (bp.M < 1 || bp.M > 16 || mm::Layout(bp.M).used2 > mm::kArena2) return cudaErrorInvalidValue;
  const int ctas = min(num_sms_mm(), 256);
  int64_t total_cost = 0;
  for (int i = 0; i < bp.count; ++i) {
    const int tiles_i = (bp.prob[i].N + mm::kRows - 1) / mm::kRows;
    total_cost += (int64_t)tiles_i * (bp.prob[i].K / kGroup);
  }
  int c = 0, tile = 0;
  int64_t run = 0;
  sc.cta_tile[0] = 0;
  for (int i = 0; i < bp.count; ++i) {
    const int tiles_i = (bp.prob[i].N + mm::kRows - 1) / mm::kRows;
    const int64_t cost = bp.prob[i].K / kGroup;
    for (int t = 0; t < tiles_i; ++t, ++tile) {
      const int64_t mid2 = 2 * run + cost;
      while (c < ctas - 1 && mid2 * ctas >= 2 * total_cost * (int64_t)(c + 1)) sc.cta_tile[++c] = tile;
      run += cost;
    }
  }
  while (c < ctas) sc.cta_tile[++c] = tile;
  int gmax = 0, tmax = 0;
  bool any2 = false;
  for (int i = 0; i < bp.count; ++i) {
    gmax = max(gmax, bp.prob[i].K / kGroup);
    tmax = max(tmax, (bp.prob[i].N + mm::kRows - 1) / mm::kRows);
    any2 = any2 || bp.prob[i].nnz > 0;
  }
  // one or two tokens: the one-group-per-lane kernel (tq_gemv_g4.cu)
  const bool g4path = g4::takes(bp);
  thread_local mm::MapTemplates mt;
  if (cudaError_t e = build_templates(bp, g4path, mt)) return e;
  // second plane: the indexed kernel when every weight with a second plane
  // has its index, else the span kernel (or, for rows of more than
  // kQMaxW salience words, the per-tile one)
  bool all_idx = true;
  for (int i = 0; i < bp.count; ++i)
    if (bp.prob[i].nnz > 0 && !bp.prob[i].p2idx)
      all_idx = false;
  int32_t *counter = nullptr;
  thread_local mm::CBase cb;
  if (any2 && all_idx) {
    cb.count = bp.count;
    cb.base[0] = 0;
    for (int p = 0; p < bp.count; ++p) {
      const Problem &P = bp.prob[p];
      cb.base[p + 1] = cb.base[p] + (P.nnz > 0 ? P.K / kGroup * mm::c_parts(P.K, P.nnz) : 0);
    }
    counter = reinterpret_cast<int32_t *>(static_cast<unsigned char *>(bp.prob[0].map()) + mm::kCounterOff);
  }
  const int sg = g4::stage_groups(bp.M);
  const int gtasks = (g4path ? sg * ((gmax + sg - 1) / sg) : gmax) * bp.M;
  // the general layout is read by the general decode kernels and by the
  // second-plane kernels other than the one-token indexed one
  bp.g4_only = g4path && (!any2 || (all_idx && bp.M == 1)) ? 1 : 0;
  cudaError_t e = launch_prep(bp, mt, counter, gtasks, s);
  if (e != cudaSuccess) return e;
  // more than 8 tokens in one pass needs every second plane indexed (the
  // other plane-2 kernels take 8 tokens at most)
  if (bp.M > 8 && any2 && !all_idx) return cudaErrorInvalidValue;
  if (any2 && all_idx && g4path && bp.M == 1) {
    // one token: the second plane in the first plane's layout (tq_gemv_g4.cu)
    e = launch_gemv_p2r(bp, num_sms_mm(), counter, s);
    if (e != cudaSuccess) return e;
  } else if (any2 && all_idx) {
    auto kern = bp.M == 1 ? mm::gemv_mma_p2c_kernel<true, false>
                          : (bp.M > 8 ? mm::gemv_mma_p2c_kernel<false, true> : mm::gemv_mma_p2c_kernel<false, false>);
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, mm::kCDynBytes2);
    if (e != cudaSuccess) return e;
    // launched programmatically after the prep kernel (it sets up its table,
    // then waits for the prep kernel's output)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(ctas);
    cfg.blockDim = dim3(mm::c_threads(bp.M > 8));
    cfg.dynamicSmemBytes = mm::kCDynBytes2;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, cb, bp, counter);
    if (e != cudaSuccess) return e;
  } else if (any2 && gmax <= mm::kQMaxG) {
    auto kern = bp.M == 1 ? mm::gemv_mma_p2v3_kernel<true> : mm::gemv_mma_p2v3_kernel<false>;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, mm::kQDynBytes);
    if (e != cudaSuccess) return e;
    kern<<<ctas, mm::kQThreads, mm::kQDynBytes, s>>>(bp, sc);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  } else if (any2) {
    mm::gemv_mma_p2_kernel<<<dim3(tmax, bp.count), mm::kP2Threads, 0, s>>>(bp);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (g4path) return launch_gemv_g4(bp, num_sms_mm(), s);
  auto main_kern = bp.M == 1 ? mm::gemv_mma_kernel<F32, true, false>
                             : (bp.M > 8 ? mm::gemv_mma_kernel<F32, false, true> : mm::gemv_mma_kernel<F32, false, false>);
  e = cudaFuncSetAttribute(main_kern, cudaFuncAttributeMaxDynamicSharedMemorySize, mm::kDynBytes);
  if (e != cudaSuccess) return e;
  main_kern<<<ctas, mm::kThreads, mm::kDynBytes, s>>>(bp, sc);
  return cudaGetLastError();
}

// The dependency-ordered sequence (one token): prep (operands of every
// problem, maps, zeroed y2 and barrier counter), then the persistent
// sequence kernel (tq_gemv_g4.cu).  Every problem with a second plane must
// carry its index.  A sequence's problems must fit one set of tensor-map
// templates (cudaErrorNotSupported otherwise).
cudaError_t launch_gemv_sequence(const BatchParams &bp_in, int barrier_extra, cudaStream_t s) {
  if (bp_in.M != 1) return cudaErrorInvalidValue;
  thread_local BatchParams bp;
  bp = bp_in;
  bp.g4_split = -1;  // sequence mode: y2 and the barrier counter zeroed by prep
  int gmax = 0;
  for (int i = 0; i < bp.count; ++i) {
    gmax = max(gmax, bp.prob[i].K / kGroup);
    if (bp.prob[i].nnz > 0 && !bp.prob[i].p2idx) return cudaErrorInvalidValue;
  }
  thread_local mm::MapTemplates mt;
  if (cudaError_t e = build_templates(bp, true, mt)) return e;
  const int gtasks = g4::stage_groups(1) * ((gmax + g4::stage_groups(1) - 1) / g4::stage_groups(1));
  const cudaError_t e = launch_prep(bp, mt, nullptr, gtasks, s);
  if (e != cudaSuccess) return e;
  return launch_gemv_seq(bp, num_sms_mm(), barrier_extra, s);
}

cudaError_t launch_gemv_mma(const BatchParams &bp, cudaStream_t s) {
  return bp.out_f32 ? launch_mm<true>(bp, s) : launch_mm<false>(bp, s);
}

}  // namespace tq
