// tq_ew.cu - the linear layer of the element-wise four-mask representation
// (paper "Model and Representation": four disjoint salience masks with
// orders [2, 2, 1, 1], W-hat = (mu + alpha0 T0 + alpha1 T1) (.) M, one mu /
// alpha0 per row and mask, alpha1 for the two order-2 masks).
//
// With mask 3 the largest (86.5 % of a recorded projection), the layer is
//   y[m][n] = mu3 S[m] + alpha0_3 P0[m][n]
//           + sum over the elements k of the row's other masks q of
//             x[m][k] ((mu_q - mu3) + (alpha0_q - alpha0_3) T0[n,k] + alpha1_q T1[n,k]),
// S = sum_k x, P0 = sum_k T0 x.  The first line is the group format's
// linear over plane 1 with s1 = alpha0_3 and off = mu3 in every group and no
// second plane: the library's decode or prefill path runs it, through
// per-call views of s1 / off in the workspace (views_kernel), into an fp32
// buffer.  correct_kernel then adds the second line and writes y.
#include <algorithm>

#include "tq_common.cuh"

namespace tq {
namespace ew {

constexpr int kWarps = 8;  // warps per block of correct_kernel

// One problem of a batched call, as the views kernel sees it ...
struct ViewProb {
  const __half *mu, *a0;  // [N][4]
  __half *s1v, *offv;     // views [N][G]
  uint32_t *salv;         // [N][sal_words] (zero)
  int32_t *rpv;           // [N+1] (zero)
  int32_t N, K;
};
// ... and as correct_kernel sees it: its weight, x, the fp32 plane-1
// result and y; S warps per row and the kernel's blocks for it.
struct Prob {
  const uint32_t *mask;     // [N][K/16]
  const uint8_t *plane1;    // [N][row_bytes]
  const int32_t *p2rowptr;  // [N+1]
  const uint8_t *plane2;
  const __half *mu, *a0, *a1;  // [N][4], [N][4], [N][2]
  const __half *x;             // [M][K]
  const float *ydense;         // [M][N]
  void *y;                     // [M][N], fp16 or fp32
  int32_t N, K, S, blocks;
};
template <typename T>
struct Batch {
  int32_t count;
  T prob[TQ_MAX_BATCH];
};
static_assert(sizeof(Batch<Prob>) <= 32764 && sizeof(Batch<ViewProb>) <= 32764, "launch parameters");

// Block row blockIdx.y = problem; thread per (row, group): s1 view = alpha0
// of mask 3, off view = mu of mask 3; the views' salience words and rowptr
// are zero (no second plane).
__global__ void views_kernel(const __grid_constant__ Batch<ViewProb> bt) {
  const ViewProb &P = bt.prob[blockIdx.y];
  const int N = P.N, G = P.K / kGroup, W = sal_words_of(P.K);
  const int64_t total = (int64_t)N * G;
  const int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x, step = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = i0; i < total; i += step) {
    const int64_t n = i / G;
    P.s1v[i] = P.a0[n * 4 + 3];
    P.offv[i] = P.mu[n * 4 + 3];
  }
  for (int64_t i = i0; i < (int64_t)N * W; i += step) P.salv[i] = 0u;
  for (int64_t i = i0; i <= N; i += step) P.rpv[i] = 0;
}

// The five base-3 digits of a byte (values above 242 read as 242), two bits
// each, first digit in bits 0..1.
__device__ __forceinline__ uint32_t digit_code(int v) {
  v = v > 242 ? 242 : v;
  uint32_t c = 0;
#pragma unroll
  for (int i = 0; i < 5; ++i) {
    c |= (uint32_t)(v % 3) << (2 * i);
    v /= 3;
  }
  return c;
}

__device__ __forceinline__ float ldx(const __half *p) {
  return __half2float(__ushort_as_half(__ldg(reinterpret_cast<const unsigned short *>(p))));
}

// Four 2-bit fields (bits 0..15 hold eight) spread to 4-bit spacing: field
// j of x at bits 2j..2j+1 -> bits 4j..4j+1.
__device__ __forceinline__ uint32_t spread2(uint32_t x) {
  x &= 0xffffu;
  x = (x | (x << 8)) & 0x00ff00ffu;
  x = (x | (x << 4)) & 0x0f0f0f0fu;
  x = (x | (x << 2)) & 0x33333333u;
  return x;
}

// Adds the elements of masks 0..2 to the dense fp32 result of tokens
// [m0, m0 + mt) (mt <= MT) and writes y.  S warps share a row, warp s taking
// a contiguous range of the row's 512-element chunks.
//
// Per chunk a lane owns one mask word (16 elements) and its 16 activations
// per token.  The chunk's plane-1 bytes (four groups of 26) are read as
// 32-bit words by the first lanes and each lane takes the four bytes
// holding its 16 trits by two shuffles and a funnel shift; a shared table
// turns each byte into five two-bit digits, so the word's T0 digits line up
// with its mask fields.  Each element's mask q and digit d0 form a 4-bit
// code (q << 2 | d0); two neighbouring elements' codes form a byte, and the
// row's 256-entry pair table gives both elements' weights
// (mu_q - mu_3) + (alpha0_q - alpha0_3) (d0 - 1) in one 8-byte load (mask-3
// codes give 0), so the sixteen elements cost eight loads and no branch.
// The order-2 elements (masks 0, 1; 3.6 % of a recorded projection) add
// alpha1_q T1 x in a loop over their bits: the T1 trit is plane 2's trit at
// the element's rank among the row's order-2 elements, the warp's exclusive
// scan of the words' order-2 counts plus the count of the row's earlier
// warps (a first pass over the mask words gives each warp its count).
template <bool F32, int MT>
__global__ void __launch_bounds__(32 * kWarps) correct_kernel(const __grid_constant__ Batch<Prob> bt, int m0, int mt) {
  const Prob &w = bt.prob[blockIdx.y];
  if ((int)blockIdx.x >= w.blocks) return;
  const int N = w.N, K = w.K, S = w.S;
  __shared__ uint32_t dig[256];
  __shared__ float2 ptab[kWarps][256];
  __shared__ int cnt[kWarps];
  __shared__ float part[kWarps][MT];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < 256; i += blockDim.x) dig[i] = digit_code(i);
  const int r_in = warp / S, seg = warp - r_in * S;
  const int n = blockIdx.x * (kWarps / S) + r_in;
  const bool live = n < N;
  const int WK = K / 16, C = (WK + 31) / 32, G = K / kGroup;
  const int c_lo = (int)((int64_t)seg * C / S), c_hi = (int)((int64_t)(seg + 1) * C / S);
  const int64_t nr = live ? n : 0;
  const uint32_t *mrow = w.mask + nr * WK;
  {
    // code q << 2 | d0 -> weight (zero for mask 3 and the unused d0 = 3)
    float v = 0.f;
    const int q = lane >> 2, d0 = lane & 3;
    if (live && lane < 12 && d0 < 3) {
      const float mu3 = __half2float(w.mu[nr * 4 + 3]), a03 = __half2float(w.a0[nr * 4 + 3]);
      v = (__half2float(w.mu[nr * 4 + q]) - mu3) + (__half2float(w.a0[nr * 4 + q]) - a03) * (float)(d0 - 1);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e = lane + 32 * i;
      const float wa = __shfl_sync(0xffffffffu, v, e & 15), wb = __shfl_sync(0xffffffffu, v, e >> 4);
      ptab[warp][e] = make_float2(wa, wb);
    }
  }
  int mine = 0;
  if (live)
    for (int c = c_lo; c < c_hi; ++c) {
      const int wi = c * 32 + lane;
      if (wi < WK) mine += __popc(~__ldg(mrow + wi) & 0xaaaaaaaau);
    }
#pragma unroll
  for (int o = 16; o; o >>= 1) mine += __shfl_xor_sync(0xffffffffu, mine, o);
  if (lane == 0) cnt[warp] = mine;
  __syncthreads();
  float acc[MT];
#pragma unroll
  for (int t = 0; t < MT; ++t) acc[t] = 0.f;
  if (live) {
    int base = 0;  // order-2 elements of the row before this warp's chunk
    for (int s = 0; s < seg; ++s) base += cnt[r_in * S + s];
    const uint8_t *p1 = w.plane1 + nr * row_bytes_of(K);
    const uint8_t *p2 = w.plane2 + w.p2rowptr[nr];
    const __half *xm = w.x + (int64_t)m0 * K;
    const int e0 = 16 * (lane & 7), s2 = 2 * (e0 % 5);
    const int B = (lane >> 3) * kGroupBytes + e0 / 5;  // first plane-1 byte of the lane's word in its chunk
    const float2 *pt = ptab[warp];
    const float a1_0 = __half2float(w.a1[nr * 2]), a1_1 = __half2float(w.a1[nr * 2 + 1]);
    for (int c = c_lo; c < c_hi; ++c) {
      const int wi = c * 32 + lane;
      const bool in = wi < WK;
      const uint32_t mw = in ? __ldg(mrow + wi) : 0xffffffffu;  // absent words read as all mask 3
      const int nw = (min(4, G - 4 * c) * kGroupBytes + 3) / 4;
      const uint32_t pw = lane < nw ? __ldg(reinterpret_cast<const uint32_t *>(p1 + (int64_t)c * 4 * kGroupBytes) + lane) : 0u;
      const uint32_t lo = __shfl_sync(0xffffffffu, pw, B >> 2), hi = __shfl_sync(0xffffffffu, pw, (B >> 2) + 1);
      uint4 xv[MT][2];
#pragma unroll
      for (int t = 0; t < MT; ++t) {
        const uint4 *xp = reinterpret_cast<const uint4 *>(xm + (int64_t)t * K + wi * 16);
        const bool ok = in && t < mt;
        xv[t][0] = ok ? __ldg(xp) : make_uint4(0u, 0u, 0u, 0u);
        xv[t][1] = ok ? __ldg(xp + 1) : make_uint4(0u, 0u, 0u, 0u);
      }
      const uint32_t o2 = ~mw & 0xaaaaaaaau;  // high bit of each order-2 field (mask 0, 1)
      const int c2 = __popc(o2);
      int incl = c2;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      const uint32_t rank0 = (uint32_t)(base + incl - c2);
      base += __shfl_sync(0xffffffffu, incl, 31);
      const uint32_t v = __funnelshift_r(lo, hi, 8 * (B & 3));
      const uint64_t code = (uint64_t)dig[v & 255u] | (uint64_t)dig[(v >> 8) & 255u] << 10 |
                            (uint64_t)dig[(v >> 16) & 255u] << 20 | (uint64_t)dig[v >> 24] << 30;
      const uint32_t T = (uint32_t)(code >> s2);  // T0 digit of field j in bits 2j..2j+1
      const uint32_t nib[2] = {spread2(mw) << 2 | spread2(T), spread2(mw >> 16) << 2 | spread2(T >> 16)};
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float2 wp = pt[(nib[k >> 2] >> (8 * (k & 3))) & 255u];
#pragma unroll
        for (int t = 0; t < MT; ++t) {
          const uint4 &q4 = xv[t][k >> 2];
          const uint32_t hw = (k & 3) == 0 ? q4.x : (k & 3) == 1 ? q4.y : (k & 3) == 2 ? q4.z : q4.w;
          const float2 xf = __half22float2(*reinterpret_cast<const __half2 *>(&hw));
          acc[t] = fmaf(wp.x, xf.x, fmaf(wp.y, xf.y, acc[t]));
        }
      }
      for (uint32_t bits = o2; bits; bits &= bits - 1) {
        const int jb = __ffs(bits) - 1;  // 2 j + 1
        const uint32_t r = rank0 + __popc(o2 & ((1u << jb) - 1u));
        const uint32_t rb = r / 5u;
        const int t1 = (int)((dig[__ldg(p2 + rb)] >> (2u * (r - 5u * rb))) & 3u) - 1;
        if (t1 == 0) continue;
        const float a1 = ((mw >> (jb - 1)) & 1u) ? a1_1 : a1_0;
        const float wc = t1 > 0 ? a1 : -a1;
        const __half *xk = xm + wi * 16 + (jb >> 1);
#pragma unroll
        for (int t = 0; t < MT; ++t)
          if (t < mt) acc[t] = fmaf(wc, ldx(xk + (int64_t)t * K), acc[t]);
      }
    }
  }
#pragma unroll
  for (int t = 0; t < MT; ++t) {
    float v = acc[t];
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == t) part[warp][t] = v;
  }
  __syncthreads();
  if (live && seg == 0 && lane < mt) {
    float v = 0.f;
    for (int s = 0; s < S; ++s) v += part[r_in * S + s][lane];
    const int64_t i = (int64_t)(m0 + lane) * N + n;
    v += w.ydense[i];
    if (F32)
      static_cast<float *>(w.y)[i] = v;
    else
      static_cast<__half *>(w.y)[i] = __float2half_rn(v);
  }
}

// Warps per row: the largest power of two up to 8 that leaves each warp at
// least three chunks, raised (up to one chunk per warp) while the grid holds
// fewer than four blocks per SM.
int warps_per_row(int N, int K, int num_sms) {
  const int C = (K / 16 + 31) / 32;
  int S = 1;
  while (S < kWarps && C / (2 * S) >= 3) S *= 2;
  while (S < kWarps && 2 * S <= C && (int64_t)N * S / kWarps < 4LL * num_sms) S *= 2;
  return S;
}

template <bool F32, int MT>
cudaError_t launch_correct(int M, const Batch<Prob> &bt, int max_blocks, cudaStream_t s) {
  for (int m0 = 0; m0 < M; m0 += MT) {
    correct_kernel<F32, MT><<<dim3(max_blocks, bt.count), 32 * kWarps, 0, s>>>(bt, m0, std::min(MT, M - m0));
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace ew

// The views of every problem (one launch).
cudaError_t launch_ew_views(const EwCall *calls, int count, cudaStream_t s) {
  thread_local ew::Batch<ew::ViewProb> bt;  // large: kept off the stack
  bt.count = count;
  int64_t most = 1;
  for (int i = 0; i < count; ++i) {
    const EwCall &c = calls[i];
    ew::ViewProb &P = bt.prob[i];
    P.mu = reinterpret_cast<const __half *>(c.w->mu);
    P.a0 = reinterpret_cast<const __half *>(c.w->alpha0);
    P.s1v = reinterpret_cast<__half *>(c.s1v);
    P.offv = reinterpret_cast<__half *>(c.offv);
    P.salv = c.salv;
    P.rpv = c.rpv;
    P.N = c.w->N;
    P.K = c.w->K;
    most = std::max<int64_t>(most, (int64_t)P.N * (P.K / kGroup));
  }
  const int blocks = (int)std::min<int64_t>((most + 255) / 256, 1024);
  ew::views_kernel<<<dim3(blocks, count), 256, 0, s>>>(bt);
  return cudaGetLastError();
}

// Masks 0..2 of every problem added to its plane-1 result, y written (one
// launch per pass of up to 8 tokens).
cudaError_t launch_ew_correct(int M, const EwCall *calls, int count, bool f32, cudaStream_t s) {
  thread_local ew::Batch<ew::Prob> bt;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  bt.count = count;
  int most = 1;
  for (int i = 0; i < count; ++i) {
    const EwCall &c = calls[i];
    ew::Prob &P = bt.prob[i];
    P.mask = c.w->mask;
    P.plane1 = c.w->plane1;
    P.p2rowptr = c.w->p2rowptr;
    P.plane2 = c.w->plane2;
    P.mu = reinterpret_cast<const __half *>(c.w->mu);
    P.a0 = reinterpret_cast<const __half *>(c.w->alpha0);
    P.a1 = reinterpret_cast<const __half *>(c.w->alpha1);
    P.x = reinterpret_cast<const __half *>(c.x);
    P.ydense = c.ydense;
    P.y = c.y;
    P.N = c.w->N;
    P.K = c.w->K;
    P.S = ew::warps_per_row(P.N, P.K, sms);
    const int rows = ew::kWarps / P.S;
    P.blocks = (P.N + rows - 1) / rows;
    most = std::max(most, P.blocks);
  }
  if (M == 1) return f32 ? ew::launch_correct<true, 1>(M, bt, most, s) : ew::launch_correct<false, 1>(M, bt, most, s);
  if (M == 2) return f32 ? ew::launch_correct<true, 2>(M, bt, most, s) : ew::launch_correct<false, 2>(M, bt, most, s);
  if (M <= 4) return f32 ? ew::launch_correct<true, 4>(M, bt, most, s) : ew::launch_correct<false, 4>(M, bt, most, s);
  return f32 ? ew::launch_correct<true, 8>(M, bt, most, s) : ew::launch_correct<false, 8>(M, bt, most, s);
}

}  // namespace tq
