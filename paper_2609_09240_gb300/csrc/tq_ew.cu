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

constexpr int kRowWarps = 4;
constexpr int kTok = 8;  // tokens per pass of correct_kernel

// Thread per (row, group): s1 view = alpha0 of mask 3, off view = mu of mask
// 3; the views' salience words and rowptr are zero (no second plane).
__global__ void views_kernel(int N, int K, const __half *mu, const __half *a0, __half *s1v, __half *offv,
                             uint32_t *salv, int32_t *rpv) {
  const int G = K / kGroup, W = sal_words_of(K);
  const int64_t total = (int64_t)N * G;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t n = i / G;
    s1v[i] = a0[n * 4 + 3];
    offv[i] = mu[n * 4 + 3];
  }
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < (int64_t)N * W;
       i += (int64_t)gridDim.x * blockDim.x)
    salv[i] = 0u;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i <= N; i += (int64_t)gridDim.x * blockDim.x)
    rpv[i] = 0;
}

struct View {
  const uint32_t *mask;    // [N][K/16]
  const uint8_t *plane1;   // [N][row_bytes]
  const int32_t *p2rowptr;  // [N+1]
  const uint8_t *plane2;
  const __half *mu, *a0, *a1;  // [N][4], [N][4], [N][2]
};

__device__ __forceinline__ int digit_of(int v, int i) {
  // digit i of a base-3 byte (v <= 242)
  const int p = i == 0 ? 1 : i == 1 ? 3 : i == 2 ? 9 : i == 3 ? 27 : 81;
  return (v / p) % 3;
}

// Warp per row, tokens [m0, m0 + mt) of this pass (mt <= kTok): adds the
// elements of masks 0..2 to the dense fp32 result and writes y.  A lane
// takes one mask word (16 elements) of each 32-word chunk; the warp's
// exclusive scan of the words' order-2 counts gives each word the rank of
// its first order-2 element in the row (plane 2 is in rank order).
template <bool F32>
__global__ void __launch_bounds__(32 * kRowWarps) correct_kernel(int M, int N, int K, View w, const __half *x,
                                                                 const float *ydense, void *y, int m0, int mt) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
  if (n >= N) return;
  const int WK = K / 16;
  const int64_t RB = row_bytes_of(K);
  const uint32_t *mrow = w.mask + (int64_t)n * WK;
  const uint8_t *p1 = w.plane1 + (int64_t)n * RB;
  const uint8_t *p2 = w.plane2 + w.p2rowptr[n];
  float mu[4], a0[4], a1[2];
#pragma unroll
  for (int q = 0; q < 4; ++q) mu[q] = __half2float(w.mu[(int64_t)n * 4 + q]), a0[q] = __half2float(w.a0[(int64_t)n * 4 + q]);
  a1[0] = __half2float(w.a1[(int64_t)n * 2]);
  a1[1] = __half2float(w.a1[(int64_t)n * 2 + 1]);
  float corr[kTok];
#pragma unroll
  for (int t = 0; t < kTok; ++t) corr[t] = 0.f;
  int base = 0;  // order-2 elements of the row before this chunk
  for (int w0 = 0; w0 < WK; w0 += 32) {
    const int wi = w0 + lane;
    const uint32_t mw = wi < WK ? mrow[wi] : 0xffffffffu;  // absent words read as all mask 3
    const uint32_t o2 = ~mw & 0xaaaaaaaau;                  // high bit of each order-2 field (mask 0, 1)
    const uint32_t non3 = ~(mw & (mw >> 1)) & 0x55555555u;  // low bit of each field that is not mask 3
    const int c2 = __popc(o2);
    int incl = c2;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    const int rank0 = base + incl - c2;
    base += __shfl_sync(0xffffffffu, incl, 31);
    for (uint32_t bits = non3; bits; bits &= bits - 1) {
      const int j = (__ffs(bits) - 1) >> 1;  // field index in the word
      const int k = wi * 16 + j;
      const int q = (mw >> (2 * j)) & 3;
      const int kg = k & (kGroup - 1);
      const int t0 = digit_of(p1[(k / kGroup) * kGroupBytes + kg / 5], kg % 5) - 1;
      float wc = (mu[q] - mu[3]) + (a0[q] - a0[3]) * (float)t0;
      if (q <= 1) {
        const int r = rank0 + __popc(o2 & ((1u << (2 * j)) - 1u));
        const int t1 = digit_of(p2[r / 5], r % 5) - 1;
        wc += a1[q] * (float)t1;
      }
#pragma unroll
      for (int t = 0; t < kTok; ++t)
        if (t < mt) corr[t] = fmaf(wc, __half2float(x[(int64_t)(m0 + t) * K + k]), corr[t]);
    }
  }
#pragma unroll
  for (int t = 0; t < kTok; ++t) {
    if (t >= mt) break;
    float v = corr[t];
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == t) {
      const int64_t i = (int64_t)(m0 + t) * N + n;
      v += ydense[i];
      if (F32)
        static_cast<float *>(y)[i] = v;
      else
        static_cast<__half *>(y)[i] = __float2half_rn(v);
    }
  }
}

}  // namespace ew

cudaError_t launch_ew_views(int N, int K, const uint16_t *mu, const uint16_t *a0, uint16_t *s1v, uint16_t *offv,
                            uint32_t *salv, int32_t *rpv, cudaStream_t s) {
  const int64_t total = (int64_t)N * (K / kGroup);
  const int blocks = (int)std::min<int64_t>((total + 255) / 256 + 1, 4096);
  ew::views_kernel<<<blocks, 256, 0, s>>>(N, K, reinterpret_cast<const __half *>(mu), reinterpret_cast<const __half *>(a0),
                                          reinterpret_cast<__half *>(s1v), reinterpret_cast<__half *>(offv), salv, rpv);
  return cudaGetLastError();
}

cudaError_t launch_ew_correct(int M, int N, int K, const tq_ew_weight *w, const uint16_t *x, const float *ydense,
                              void *y, bool f32, cudaStream_t s) {
  ew::View v{w->mask, w->plane1, w->p2rowptr, w->plane2, reinterpret_cast<const __half *>(w->mu),
             reinterpret_cast<const __half *>(w->alpha0), reinterpret_cast<const __half *>(w->alpha1)};
  const int blocks = (N + ew::kRowWarps - 1) / ew::kRowWarps;
  for (int m0 = 0; m0 < M; m0 += ew::kTok) {
    const int mt = std::min(ew::kTok, M - m0);
    if (f32)
      ew::correct_kernel<true><<<blocks, 32 * ew::kRowWarps, 0, s>>>(M, N, K, v, reinterpret_cast<const __half *>(x), ydense,
                                                                     y, m0, mt);
    else
      ew::correct_kernel<false><<<blocks, 32 * ew::kRowWarps, 0, s>>>(M, N, K, v, reinterpret_cast<const __half *>(x), ydense,
                                                                      y, m0, mt);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace tq
