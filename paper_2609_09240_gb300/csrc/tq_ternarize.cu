// tq_ternarize.cu - E2M-ATQ ternarization of fp16 weights straight into the
// packed format (paper "Conversion Pipeline", subsection "E2M-ATQ"; the
// representation of "Model and Representation", eq. for W-hat, read per
// (row, group of 128) block).
//
// Per block w (128 fp16 weights of one row and group):
//   mu = mean(w), c = w - mu, Delta0 = 0.75 mean|c|, T0 = sign(c) where
//   |c| > Delta0, alpha0 = least-squares scale of c on T0; residual
//   r = c - alpha0 T0 with energy E = sum r^2.  The projection's nnz blocks
//   of largest E (ties: lower block id) are salient: their residual gets a
//   second support T1 by the same threshold rule and its least-squares
//   scale alpha1.  Then `sweeps` alternating refinements of mu, alpha0,
//   alpha1 with the supports fixed.  Stored: offset = fp16(mu), scale1 =
//   fp16(alpha0), scale2 = fp16(alpha1), plane 1 = T0, plane 2 = T1.
//
// The supports, thresholds and the salience are integer decisions taken from
// floats, so their arithmetic is fixed: IEEE float32 with explicit
// round-to-nearest operations (never contracted into fused multiply-adds),
// every sum over a block in index order 0..127 from +0, means as sums times
// 1/128.  One thread owns one block, which makes index order its natural
// order.  The refinement decides nothing and runs on per-block moments (see
// plane2_blocks); its fp16 outputs agree with in-order passes to one ulp.
//
// Kernels, in launch order:
//   tern_stats_kernel   per block: mu, Delta0, alpha0 and E (key = E's bits)
//   tern_hist_kernel    4 passes of an 8-bit radix select of the nnz-th
//                       largest key; the last CTA of a pass to finish picks
//                       the digit (no CTA waits for another)
//   tern_count_kernel   keys equal to the selected key, per chunk of
//                       salience words
//   tern_mark_kernel    salience words: keys above the selected key, and the
//                       first `need` equal keys in block-id order
//   rowptr (tq_codec.cu), then
//   tern_planes_kernel  per block: supports, second plane, refinement, and
//                       the packed bytes and fp16 parameters (salient blocks
//                       by record, in CTAs of their own).
#include "tq_common.cuh"

namespace tq {

cudaError_t launch_rowptr(int N, int K, const uint32_t *sal, int32_t *rowptr, uint32_t *status,
                          cudaStream_t s);

namespace tz {

constexpr int kBlockThreads = 128;  // per-block kernels: one thread per (row, group)
constexpr int kSelThreads = 1024;   // histogram kernels
constexpr int kMarkThreads = 128;   // count / mark kernels: one salience word per thread
constexpr float kInvGroup = 0.0078125f;  // 1 / 128, exact
constexpr float kThresh = 0.75f;         // E2M-ATQ threshold factor

// Radix-select state after each pass: bits of the selected key fixed so far,
// and how many keys with that prefix are still to take.
struct SelState {
  uint32_t prefix[5];
  uint32_t pad_;
  int64_t need[5];
};

struct SelWork {
  uint32_t hist[4][256];
  uint32_t done[4];  // CTAs finished per pass
  uint32_t pad_[4];
  SelState st;
};

// A block's 128 fp16 weights, staged in shared memory by the thread that
// owns the block: its word j (weights 2j, 2j+1) at word j * kBlockThreads +
// thread, so that a warp's loads of one word hit 32 consecutive banks.
// Every pass re-reads the block with volatile loads, which the compiler can
// neither merge nor hoist, so a thread's registers hold only the supports'
// bit masks and scalars (kept in registers, a block's 128 floats plus the
// per-element support decisions exceed the register file).
struct Blk {
  uint32_t base;  // shared address of the thread's word 0
  __device__ __forceinline__ float2 pair(int j) const {
    uint32_t w;
    asm volatile("ld.volatile.shared.u32 %0, [%1];" : "=r"(w) : "r"(base + 4u * (uint32_t)(j * kBlockThreads)));
    return __half22float2(*reinterpret_cast<const __half2 *>(&w));
  }
  // fn(q, bit, x) for the weights in index order: weight 32 q + bit is x;
  // done(q) after each 32 weights (one mask word).
  template <class Fn, class Done>
  __device__ __forceinline__ void each(Fn fn, Done done) const {
#pragma unroll 1
    for (int q = 0; q < 4; ++q) {
#pragma unroll 4
      for (int jj = 0; jj < 16; ++jj) {
        const float2 v = pair(16 * q + jj);
        fn(q, 2 * jj, v.x);
        fn(q, 2 * jj + 1, v.y);
      }
      done(q);
    }
  }
  template <class Fn>
  __device__ __forceinline__ void each(Fn fn) const {
    each(fn, [](int) {});
  }
};

__device__ __forceinline__ Blk stage_block(const uint16_t *W, int64_t b, uint32_t *sx) {
  const uint4 *src = reinterpret_cast<const uint4 *>(W + b * kGroup);
  const uint32_t col = (uint32_t)__cvta_generic_to_shared(sx + threadIdx.x);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint4 v = __ldg(src + j);
    const uint32_t a = col + 4u * (uint32_t)(4 * j * kBlockThreads);
    asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(a), "r"(v.x));
    asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(a + 4u * kBlockThreads), "r"(v.y));
    asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(a + 8u * kBlockThreads), "r"(v.z));
    asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(a + 12u * kBlockThreads), "r"(v.w));
  }
  return Blk{col};
}

__device__ __forceinline__ uint32_t pick4(const uint32_t (&m)[4], int q) {
  return q == 0 ? m[0] : q == 1 ? m[1] : q == 2 ? m[2] : m[3];
}
__device__ __forceinline__ void put4(uint32_t (&m)[4], int q, uint32_t v) {
  m[0] = q == 0 ? v : m[0];
  m[1] = q == 1 ? v : m[1];
  m[2] = q == 2 ? v : m[2];
  m[3] = q == 3 ? v : m[3];
}
// a * t for the trit t of bit `bit` of mask words (nz: t != 0, ng: t < 0):
// +a, -a (the sign bit flipped) or +0.
__device__ __forceinline__ float times_bit(float a, uint32_t nz, uint32_t ng, int bit) {
  const uint32_t keep = 0u - ((nz >> bit) & 1u);
  const uint32_t sign = (ng << (31 - bit)) & 0x80000000u;
  return __uint_as_float((__float_as_uint(a) ^ sign) & keep);
}

__device__ __forceinline__ int popc4(const uint32_t (&m)[4]) {
  return __popc(m[0]) + __popc(m[1]) + __popc(m[2]) + __popc(m[3]);
}

// Support of v (v(x) per weight) at threshold d (E2M-ATQ, eq. for T0): +1
// above d, -1 below -d; on(x, t) sees each weight with its trit.  Returns
// the support's size.
template <class V, class On>
__device__ __forceinline__ int support(const Blk &B, V v, float d, uint32_t (&nz)[4], uint32_t (&ng)[4], On on) {
  uint32_t mz = 0u, mg = 0u;
  B.each(
      [&](int q, int bit, float x) {
        const float c = v(q, bit, x);
        const int t = c > d ? 1 : (c < -d ? -1 : 0);
        if (t) mz |= 1u << bit;
        if (t < 0) mg |= 1u << bit;
        on(x, t);
      },
      [&](int q) {
        put4(nz, q, mz);
        put4(ng, q, mg);
        mz = 0u, mg = 0u;
      });
  return popc4(nz);
}

// First plane of a block: mu, Delta0, T0, alpha0 (least squares with mu fixed).
struct First {
  float mu, d0, a0;
  int n0;
  uint32_t nz[4], ng[4];
};

__device__ __forceinline__ void first_plane(const Blk &B, First &f, bool *bad) {
  float s = 0.f;
  bool nf = false;
  B.each([&](int, int, float x) {
    s = __fadd_rn(s, x);
    nf |= !isfinite(x);
  });
  *bad = nf;
  const float mu = __fmul_rn(s, kInvGroup);
  float a = 0.f;
  B.each([&](int, int, float x) { a = __fadd_rn(a, fabsf(__fsub_rn(x, mu))); });
  const float d0 = __fmul_rn(kThresh, __fmul_rn(a, kInvGroup));
  f.n0 = support(B, [&](int, int, float x) { return __fsub_rn(x, mu); }, d0, f.nz, f.ng, [](float, int) {});
  float p = 0.f;
  B.each([&](int q, int bit, float x) {
    p = __fadd_rn(p, times_bit(__fsub_rn(x, mu), pick4(f.nz, q), pick4(f.ng, q), bit));
  });
  f.mu = mu, f.d0 = d0;
  f.a0 = f.n0 > 0 ? __fdiv_rn(p, (float)f.n0) : 0.f;
}

// ------------------------------------------------------------ statistics
__global__ void __launch_bounds__(kBlockThreads) tern_stats_kernel(int64_t NB, const uint16_t *W, float4 *stats,
                                                                   uint32_t *keys, uint32_t *status) {
  __shared__ uint32_t sx[64 * kBlockThreads];
  for (int64_t b = (int64_t)blockIdx.x * kBlockThreads + threadIdx.x; b < NB;
       b += (int64_t)gridDim.x * kBlockThreads) {
    const Blk B = stage_block(W, b, sx);
    First f;
    bool bad;
    first_plane(B, f, &bad);
    if (bad) atomicOr(status, TQ_DATA_BAD_WEIGHT);
    float e = 0.f;
    B.each([&](int q, int bit, float x) {
      const float r = __fsub_rn(__fsub_rn(x, f.mu), times_bit(f.a0, pick4(f.nz, q), pick4(f.ng, q), bit));
      e = __fadd_rn(e, __fmul_rn(r, r));
    });
    stats[b] = make_float4(f.mu, f.d0, f.a0, 0.f);
    keys[b] = __float_as_uint(e);
  }
}

// --------------------------------------------------------------- select
// Warp 0 of the last CTA of a pass: the digit d (255 down to 0) at which the
// counts of hist, added from the top, reach need; returns need minus the
// counts above d.
__device__ void pick_digit(const uint32_t *hist, int64_t need, int &digit, int64_t &need_out) {
  const int lane = threadIdx.x & 31;
  uint32_t c[8];
  int64_t loc = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    c[j] = __ldcg(hist + 255 - 8 * lane - j);
    loc += c[j];
  }
  int64_t incl = loc;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  const int64_t excl = incl - loc;
  const unsigned owner = __ballot_sync(0xffffffffu, excl < need && need <= incl);
  // need <= the count of keys with the current prefix, so exactly one lane owns it
  const int src = owner ? __ffs(owner) - 1 : 0;
  int d = 0;
  int64_t rem = 1;
  if (lane == src) {
    int64_t cum = excl;
    bool found = false;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (found) continue;
      if (cum + c[j] >= need) {
        d = 255 - 8 * lane - j;
        rem = need - cum;
        found = true;
      } else {
        cum += c[j];
      }
    }
  }
  digit = __shfl_sync(0xffffffffu, d, src);
  need_out = __shfl_sync(0xffffffffu, rem, src);
}

__global__ void __launch_bounds__(kSelThreads) tern_hist_kernel(int pass, int64_t NB, int64_t nnz,
                                                                const uint32_t *keys, SelWork *sw) {
  __shared__ uint32_t hs[256];
  __shared__ bool last;
  const int tid = threadIdx.x;
  if (tid < 256) hs[tid] = 0u;
  const uint32_t prefix = pass ? sw->st.prefix[pass] : 0u;
  const int64_t need = pass ? sw->st.need[pass] : nnz;
  const int shift = 24 - 8 * pass;
  // keys whose bits above `shift + 8` match the prefix (all keys in pass 0)
  const uint32_t hi_mask = pass ? (0xffffffffu << (shift + 8)) : 0u;
  __syncthreads();
  for (int64_t b = (int64_t)blockIdx.x * kSelThreads + tid; b < NB; b += (int64_t)gridDim.x * kSelThreads) {
    const uint32_t k = keys[b];
    if ((k & hi_mask) == prefix) atomicAdd(&hs[(k >> shift) & 255u], 1u);
  }
  __syncthreads();
  if (tid < 256 && hs[tid]) atomicAdd(&sw->hist[pass][tid], hs[tid]);
  __threadfence();
  __syncthreads();
  if (tid == 0) last = atomicAdd(&sw->done[pass], 1u) == gridDim.x - 1;
  __syncthreads();
  if (last && tid < 32) {
    __threadfence();
    int d;
    int64_t rem;
    pick_digit(sw->hist[pass], need, d, rem);
    if (tid == 0) {
      sw->st.prefix[pass + 1] = prefix | ((uint32_t)d << shift);
      sw->st.need[pass + 1] = rem;
    }
  }
}

// Masks of the 32 salience words w0 .. w0 + 31 (word w: row w / SW, word
// w % SW) against the selected key T, built by one warp: per word, lane l
// reads the key of group 32 (w % SW) + l (one coalesced load) and two
// ballots give the valid groups above T and equal to T; lane k keeps word
// w0 + k's masks.
__device__ __forceinline__ void warp_word_masks(const uint32_t *keys, int G, int SW, int NW, int w0, uint32_t T,
                                                uint32_t &gt, uint32_t &eq) {
  const int lane = threadIdx.x & 31;
  gt = 0u, eq = 0u;
  uint32_t v[32];
  bool ok[32];
  // all 32 loads first (in flight together), then the ballots
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    const int w = w0 + k, n = w / SW, j = w - n * SW;
    ok[k] = w < NW && lane < G - 32 * j;
    v[k] = ok[k] ? keys[(int64_t)n * G + 32 * j + lane] : 0u;
  }
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    const uint32_t bg = __ballot_sync(0xffffffffu, ok[k] && v[k] > T);
    const uint32_t be = __ballot_sync(0xffffffffu, ok[k] && v[k] == T);
    if (lane == k) gt = bg, eq = be;
  }
}

__device__ __forceinline__ int block_sum(int v, int *red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  int t = 0;
  for (int i = 0; i < kMarkThreads / 32; ++i) t += red[i];
  return t;
}

// Keys equal to the selected key, per chunk of kMarkThreads salience words.
__global__ void __launch_bounds__(kMarkThreads) tern_count_kernel(int NW, int G, int SW, const uint32_t *keys,
                                                                  const SelWork *sw, uint32_t *chunk_eq) {
  __shared__ int red[kMarkThreads / 32];
  const int w0 = (int)blockIdx.x * kMarkThreads + (threadIdx.x & ~31);
  uint32_t gt, eq;
  warp_word_masks(keys, G, SW, NW, w0, sw->st.prefix[4], gt, eq);
  const int t = block_sum(__popc(eq), red);
  if (threadIdx.x == 0) chunk_eq[blockIdx.x] = (uint32_t)t;
}

// Salience words of a chunk: groups above the selected key, and equal ones
// while fewer than `need` equal keys precede them in block-id order.
__global__ void __launch_bounds__(kMarkThreads) tern_mark_kernel(int NW, int G, int SW, const uint32_t *keys,
                                                                 const SelWork *sw, const uint32_t *chunk_eq,
                                                                 uint32_t *sal) {
  __shared__ int red[kMarkThreads / 32];
  __shared__ int wpre[kMarkThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const uint32_t T = sw->st.prefix[4];
  const int64_t need = sw->st.need[4];
  // equal keys in earlier chunks
  int before = 0;
  for (int c = tid; c < (int)blockIdx.x; c += kMarkThreads) before += (int)chunk_eq[c];
  const int64_t base = block_sum(before, red);
  const int w0 = (int)blockIdx.x * kMarkThreads + (tid & ~31);
  uint32_t gt, eq;
  warp_word_masks(keys, G, SW, NW, w0, T, gt, eq);
  // exclusive scan of the equal counts over the chunk's words (block-id order)
  const int cnt = __popc(eq);
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) wpre[wid] = incl;
  __syncthreads();
  int wbase = 0;
  for (int i = 0; i < wid; ++i) wbase += wpre[i];
  int64_t rank = base + wbase + incl - cnt;  // equal keys before this word
  uint32_t take = 0u;
  for (uint32_t m = eq; m && rank < need; m &= m - 1u, ++rank) take |= m & (~m + 1u);
  const int w = w0 + lane;
  if (w < NW) sal[w] = gt | take;
}

// ----------------------------------------------------------------- pack
// 26 packed bytes of a block's trits (five per byte, digit = trit + 1, first
// trit least significant; tail byte: trits 125..127 and two pad digits 1)
// stored as 13 two-byte words at dst (2-byte aligned).
__device__ __forceinline__ void store_group(const uint32_t (&nz)[4], const uint32_t (&ng)[4], uint8_t *dst) {
  uint16_t *d16 = reinterpret_cast<uint16_t *>(dst);
  uint32_t prev = 0;
#pragma unroll
  for (int j = 0; j < kGroupBytes; ++j) {
    uint32_t v = 0, p3 = 1;
#pragma unroll
    for (int q = 0; q < 5; ++q) {
      const int i = 5 * j + q;
      const uint32_t bit = 1u << (i & 31);
      const uint32_t dgt = i >= kGroup ? 1u : (nz[i >> 5] & bit) ? ((ng[i >> 5] & bit) ? 0u : 2u) : 1u;
      v += dgt * p3;
      p3 *= 3u;
    }
    if (j & 1)
      d16[j >> 1] = (uint16_t)(prev | (v << 8));
    else
      prev = v;
  }
}

// Blocks without a second plane (the CTAs from p2_ctas on of
// tern_planes_kernel): the first support from the statistics, then `sweeps`
// refinements of mu and alpha0 (alpha1 = 0) on the block's moments (see
// plane2_blocks).
// Salient blocks are skipped here; plane2_blocks writes them.  Also
// zeroes each row's pad bytes.
__device__ __forceinline__ void plane1_blocks(int cta, int ctas, uint32_t *sx, int N, int K, int sweeps,
                                              const uint16_t *W, const float4 *stats, const uint32_t *sal,
                                              uint8_t *plane1, __half *s1, __half *off) {
  const int G = K / kGroup, SW = sal_words_of(K);
  const int64_t NB = (int64_t)N * G, RB = row_bytes_of(K);
  for (int64_t b = (int64_t)cta * kBlockThreads + threadIdx.x; b < NB; b += (int64_t)ctas * kBlockThreads) {
    const int64_t n = b / G;
    const int g = (int)(b - n * G);
    uint8_t *row = plane1 + n * RB;
    if (g == G - 1)
      for (int64_t i = (int64_t)kGroupBytes * G; i < RB; ++i) row[i] = 0;
    if ((sal[n * SW + (g >> 5)] >> (g & 31)) & 1u) continue;
    const Blk B = stage_block(W, b, sx);
    const float4 st = stats[b];
    float mu = st.x, a0 = st.z;
    uint32_t nz0[4] = {0u, 0u, 0u, 0u}, ng0[4] = {0u, 0u, 0u, 0u};
    float mw = 0.f, mw0 = 0.f;  // sum w, sum w T0
    const int n0 = support(B, [&](int, int, float x) { return __fsub_rn(x, mu); }, st.y, nz0, ng0,
                           [&](float x, int t) { mw += x, mw0 += t > 0 ? x : (t < 0 ? -x : 0.f); });
    const int z0 = n0 - 2 * popc4(ng0);  // sum T0
    for (int sw = 0; sw < sweeps; ++sw) {
      mu = (mw - a0 * z0) * kInvGroup;
      a0 = n0 > 0 ? (mw0 - mu * z0) / n0 : 0.f;
    }
    off[b] = __float2half_rn(mu);
    s1[b] = __float2half_rn(a0);
    store_group(nz0, ng0, row + (int64_t)kGroupBytes * g);
  }
}

// Salient blocks (the first p2_ctas CTAs of tern_planes_kernel, scheduled
// first because they take longest), one thread per plane-2 record j < nnz:
// the record's row
// (the last n with rowptr[n] <= j) and group (the (j - rowptr[n])-th set
// salience bit of the row), then both supports, the refinement of mu,
// alpha0 and alpha1, and both planes' bytes and parameters.
//
// The refinement decides nothing (the supports are fixed), so it runs on
// the block's moments: with n0 = |T0|, n1 = |T1|, s0 = sum T0, s1 = sum T1,
// s01 = sum T0 T1 and the sums w, w T0, w T1, a sweep is
//   mu = (sum w - alpha0 s0 - alpha1 s1) / 128,
//   alpha0 = (sum w T0 - mu s0 - alpha1 s01) / n0,
//   alpha1 = (sum w T1 - mu s1 - alpha0 s01) / n1,
// the exact coordinate updates of the least-squares fit, without a pass
// over the weights.  Supports and thresholds keep the in-order sums.
__device__ __forceinline__ void plane2_blocks(int cta, int ctas, uint32_t *sx, int N, int K, int sweeps,
                                              int64_t nnz, const uint16_t *W, const float4 *stats,
                                              const uint32_t *sal, const int32_t *rowptr, uint8_t *plane1,
                                              uint8_t *plane2, __half *s1, __half *off, __half *s2,
                                              uint32_t *status) {
  const int G = K / kGroup, SW = sal_words_of(K);
  const int64_t RB = row_bytes_of(K);
  for (int64_t j = (int64_t)cta * kBlockThreads + threadIdx.x; j < nnz; j += (int64_t)ctas * kBlockThreads) {
    int lo = 0, hi = N;  // rowptr[lo] <= j < rowptr[hi] for a consistent rowptr
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (rowptr[mid] <= j) lo = mid; else hi = mid;
    }
    const int n = lo;
    int rank = (int)(j - rowptr[n]), g = -1;
    for (int w = 0; w < SW && g < 0; ++w) {
      uint32_t m = sal[(int64_t)n * SW + w];
      if (G - 32 * w < 32) m &= (1u << (G - 32 * w)) - 1u;
      const int c = __popc(m);
      if (rank < c) {
        for (int k = 0; k < rank; ++k) m &= m - 1u;
        g = 32 * w + __ffs(m) - 1;
      } else {
        rank -= c;
      }
    }
    if (g < 0 || rank < 0) {
      atomicOr(status, TQ_DATA_BAD_ROWPTR);  // rowptr disagrees with the salience map
      continue;
    }
    const int64_t b = (int64_t)n * G + g;
    const Blk B = stage_block(W, b, sx);
    const float4 st = stats[b];
    float mu = st.x, a0 = st.z, a1 = 0.f;
    uint32_t nz0[4] = {0u, 0u, 0u, 0u}, ng0[4] = {0u, 0u, 0u, 0u};
    uint32_t nz1[4] = {0u, 0u, 0u, 0u}, ng1[4] = {0u, 0u, 0u, 0u};
    float mw = 0.f, mw0 = 0.f, mw1 = 0.f;  // sum w, sum w T0, sum w T1
    const int n0 = support(B, [&](int, int, float x) { return __fsub_rn(x, mu); }, st.y, nz0, ng0,
                           [&](float x, int t) { mw += x, mw0 += t > 0 ? x : (t < 0 ? -x : 0.f); });
    auto t0a = [&](float a, int q, int bit) { return times_bit(a, pick4(nz0, q), pick4(ng0, q), bit); };
    // second support on the residual r = c - alpha0 T0, same threshold rule
    auto resid = [&](int q, int bit, float x) { return __fsub_rn(__fsub_rn(x, mu), t0a(a0, q, bit)); };
    float bsum = 0.f;
    B.each([&](int q, int bit, float x) { bsum = __fadd_rn(bsum, fabsf(resid(q, bit, x))); });
    const float d1 = __fmul_rn(kThresh, __fmul_rn(bsum, kInvGroup));
    const int n1 = support(B, resid, d1, nz1, ng1,
                           [&](float x, int t) { mw1 += t > 0 ? x : (t < 0 ? -x : 0.f); });
    const int z0 = n0 - 2 * popc4(ng0), z1 = n1 - 2 * popc4(ng1);  // sum T0, sum T1
    int z01 = 0;  // sum T0 T1: +1 where both are nonzero with equal signs, -1 with opposite signs
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint32_t both = nz0[k] & nz1[k], opp = ng0[k] ^ ng1[k];
      z01 += __popc(both & ~opp) - __popc(both & opp);
    }
    // alpha1 = sum r T1 / n1 with r = w - mu - alpha0 T0
    a1 = n1 > 0 ? (mw1 - mu * z1 - a0 * z01) / n1 : 0.f;
    for (int sw = 0; sw < sweeps; ++sw) {
      mu = (mw - a0 * z0 - a1 * z1) * kInvGroup;
      a0 = n0 > 0 ? (mw0 - mu * z0 - a1 * z01) / n0 : 0.f;
      if (n1 > 0) a1 = (mw1 - mu * z1 - a0 * z01) / n1;
    }
    off[b] = __float2half_rn(mu);
    s1[b] = __float2half_rn(a0);
    store_group(nz0, ng0, plane1 + (int64_t)n * RB + (int64_t)kGroupBytes * g);
    store_group(nz1, ng1, plane2 + j * kGroupBytes);
    s2[j] = __float2half_rn(a1);
  }
}

// Both kinds of blocks in one launch: CTAs below p2_ctas take the salient
// records, the rest the other blocks, so the two run side by side.
__global__ void __launch_bounds__(kBlockThreads) tern_planes_kernel(int N, int K, int sweeps, int64_t nnz, int p2_ctas,
                                                                   const uint16_t *W, const float4 *stats,
                                                                   const uint32_t *sal, const int32_t *rowptr,
                                                                   uint8_t *plane1, uint8_t *plane2, __half *s1,
                                                                   __half *off, __half *s2, uint32_t *status) {
  __shared__ uint32_t sx[64 * kBlockThreads];
  if ((int)blockIdx.x < p2_ctas)
    plane2_blocks(blockIdx.x, p2_ctas, sx, N, K, sweeps, nnz, W, stats, sal, rowptr, plane1, plane2, s1, off, s2,
                  status);
  else
    plane1_blocks(blockIdx.x - p2_ctas, gridDim.x - p2_ctas, sx, N, K, sweeps, W, stats, sal, plane1, s1, off);
}

int grid_blocks(int64_t NB) {
  int64_t g = (NB + kBlockThreads - 1) / kBlockThreads;
  return (int)(g < 1 ? 1 : g > 152 * 16 ? 152 * 16 : g);
}

}  // namespace tz

size_t ternarize_ws_bytes(int N, int K) {
  const int64_t NB = (int64_t)N * (K / kGroup);
  const int64_t NW = (int64_t)N * sal_words_of(K);
  const int64_t chunks = (NW + tz::kMarkThreads - 1) / tz::kMarkThreads;
  auto pad = [](int64_t b) { return (b + 255) / 256 * 256; };
  return (size_t)(pad(NB * 16) + pad(NB * 4) + pad(sizeof(tz::SelWork)) + pad(chunks * 4));
}

cudaError_t launch_ternarize(int N, int K, const uint16_t *W, int64_t nnz, int sweeps, uint8_t *plane1,
                             uint32_t *sal, int32_t *rowptr, uint8_t *plane2, uint16_t *scale1, uint16_t *offset,
                             uint16_t *scale2, unsigned char *ws, uint32_t *status, cudaStream_t s) {
  using namespace tz;
  const int G = K / kGroup, SW = sal_words_of(K);
  const int64_t NB = (int64_t)N * G, NW = (int64_t)N * SW;
  const int64_t chunks = (NW + kMarkThreads - 1) / kMarkThreads;
  auto pad = [](int64_t b) { return (b + 255) / 256 * 256; };
  float4 *stats = reinterpret_cast<float4 *>(ws);
  uint32_t *keys = reinterpret_cast<uint32_t *>(ws + pad(NB * 16));
  SelWork *sw = reinterpret_cast<SelWork *>(ws + pad(NB * 16) + pad(NB * 4));
  uint32_t *chunk_eq = reinterpret_cast<uint32_t *>(ws + pad(NB * 16) + pad(NB * 4) + pad(sizeof(SelWork)));
  tern_stats_kernel<<<grid_blocks(NB), kBlockThreads, 0, s>>>(NB, W, stats, keys, status);
  if (nnz > 0) {
    cudaError_t e = cudaMemsetAsync(sw, 0, sizeof(SelWork), s);
    if (e != cudaSuccess) return e;
    int hg = (int)((NB + kSelThreads - 1) / kSelThreads);
    if (hg > 152 * 2) hg = 152 * 2;
    for (int p = 0; p < 4; ++p) tern_hist_kernel<<<hg, kSelThreads, 0, s>>>(p, NB, nnz, keys, sw);
    tern_count_kernel<<<(unsigned)chunks, kMarkThreads, 0, s>>>((int)NW, G, SW, keys, sw, chunk_eq);
    tern_mark_kernel<<<(unsigned)chunks, kMarkThreads, 0, s>>>((int)NW, G, SW, keys, sw, chunk_eq, sal);
  } else {
    cudaError_t e = cudaMemsetAsync(sal, 0, (size_t)NW * 4, s);
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  e = launch_rowptr(N, K, sal, rowptr, status, s);
  if (e != cudaSuccess) return e;
  __half *h1 = reinterpret_cast<__half *>(scale1), *ho = reinterpret_cast<__half *>(offset);
  const int p2 = nnz > 0 ? grid_blocks(nnz) : 0;
  tern_planes_kernel<<<p2 + grid_blocks(NB), kBlockThreads, 0, s>>>(N, K, sweeps, nnz, p2, W, stats, sal, rowptr,
                                                                    plane1, plane2, h1, ho,
                                                                    reinterpret_cast<__half *>(scale2), status);
  return cudaGetLastError();
}

}  // namespace tq
