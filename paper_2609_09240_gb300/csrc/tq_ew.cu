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
  const int32_t *idx_off;      // correction index (or null): offsets [N nb + 1]
  const uint16_t *idx;         //   and entries
  const __half *x;             // [M][K]
  const float *ydense;         // [M][N]
  void *y;                     // [M][N], fp16 or fp32
  int32_t N, K, S, blocks;     // blocks = 0: the problem is the other kernel's
  int32_t row_begin;           // first row of the problem among the index kernel's rows
};
template <typename T>
struct Batch {
  int32_t count;
  T prob[TQ_MAX_BATCH];
};
static_assert(sizeof(Batch<Prob>) <= 32764 && sizeof(Batch<ViewProb>) <= 32764, "launch parameters");

// Block row blockIdx.y = problem: s1 view = alpha0 of mask 3, off view =
// mu of mask 3 in every group of the row (eight groups per 16-byte store
// when a row's views are whole 16-byte units); the views' salience words
// and rowptr are zero (no second plane).
__global__ void views_kernel(const __grid_constant__ Batch<ViewProb> bt) {
  const ViewProb &P = bt.prob[blockIdx.y];
  const int N = P.N, G = P.K / kGroup, W = sal_words_of(P.K);
  const int i0 = blockIdx.x * blockDim.x + threadIdx.x, step = gridDim.x * blockDim.x;
  const __half *mu = P.mu, *a0 = P.a0;
  if (G % 8 == 0) {
    const int G8 = G / 8;
    uint4 *s1 = reinterpret_cast<uint4 *>(P.s1v), *of = reinterpret_cast<uint4 *>(P.offv);
    for (int i = i0; i < N * G8; i += step) {
      const int n = i / G8;
      const uint32_t a = __half_as_ushort(a0[n * 4 + 3]) * 0x10001u, m = __half_as_ushort(mu[n * 4 + 3]) * 0x10001u;
      s1[i] = make_uint4(a, a, a, a);
      of[i] = make_uint4(m, m, m, m);
    }
  } else {
    for (int i = i0; i < N * G; i += step) {
      const int n = i / G;
      P.s1v[i] = a0[n * 4 + 3];
      P.offv[i] = mu[n * 4 + 3];
    }
  }
  for (int i = i0; i < N * W; i += step) P.salv[i] = 0u;
  for (int i = i0; i <= N; i += step) P.rpv[i] = 0;
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

constexpr int kIdxBlock = 2048, kIdxShift = 11;  // the correction index's blocks and code position
constexpr uint32_t kIdxNone = 31u << kIdxShift;  // a code that weighs nothing (pads a step)

// The same correction from the correction index: warp per row, the warps
// striding over the rows of every indexed problem of the call; the lanes
// take a block's entries two at a time per step.  An entry names its element
// k (within its block) and code = 9 q + 3 d0 + d1 (digits d = trit + 1),
// whose weight (mu_q - mu_3) + (alpha0_q - alpha0_3) T0 + alpha1_q T1 is read
// from the row's 27-entry table.  Only the entries and x are read: no mask
// plane, plane-1 or plane-2 bytes.
template <bool F32, int MT>
__global__ void __launch_bounds__(32 * kWarps) correct_idx_kernel(const __grid_constant__ Batch<Prob> bt,
                                                                  int total_rows, int m0, int mt) {
  __shared__ float tab[kWarps][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int top = 1 << (31 - __clz(max(bt.count, 1)));
  for (int r = blockIdx.x * kWarps + warp; r < total_rows; r += gridDim.x * kWarps) {
    // the problem of row r: the last with row_begin <= r (problems without
    // an index have no rows: their row_begin equals the next one's)
    int p = 0;
    for (int step = top; step >= 1; step >>= 1)
      if (p + step < bt.count && bt.prob[p + step].row_begin <= r) p += step;
    const Prob &w = bt.prob[p];
    const int n = r - w.row_begin, N = w.N, K = w.K;
    {
      // codes 27..31 (none in a valid index but the step padding) weigh nothing
      const int q = lane / 9, d0 = (lane / 3) % 3, d1 = lane % 3;
      float v = 0.f;
      if (lane < 27) {
        const __half *mu = w.mu + (int64_t)n * 4, *a0 = w.a0 + (int64_t)n * 4;
        v = (__half2float(mu[q]) - __half2float(mu[3])) + (__half2float(a0[q]) - __half2float(a0[3])) * (float)(d0 - 1);
        if (q < 2) v += __half2float(w.a1[(int64_t)n * 2 + q]) * (float)(d1 - 1);
      }
      tab[warp][lane] = v;
    }
    __syncwarp();
    const float *tw = tab[warp];
    const uint16_t *idx = w.idx;
    const unsigned short *xm = reinterpret_cast<const unsigned short *>(w.x) + (int64_t)m0 * K;
    const int nb = (K + kIdxBlock - 1) / kIdxBlock;
    const int32_t *offr = w.idx_off + (int64_t)n * nb;
    float acc[MT];
#pragma unroll
    for (int t = 0; t < MT; ++t) acc[t] = 0.f;
    int e = __ldg(offr);
    for (int b = 0; b < nb; ++b) {
      const int e1 = __ldg(offr + b + 1);
      const int kb = b * kIdxBlock, kmax = K - 1 - kb;
      for (int e0 = e + lane; e0 < e1; e0 += 64) {
        const uint32_t v0 = __ldg(idx + e0);
        const uint32_t v1 = e0 + 32 < e1 ? __ldg(idx + e0 + 32) : kIdxNone;
        const int k0 = kb + min((int)(v0 & (kIdxBlock - 1)), kmax), k1 = kb + min((int)(v1 & (kIdxBlock - 1)), kmax);
        const float w0 = tw[v0 >> kIdxShift], w1 = tw[v1 >> kIdxShift];
#pragma unroll
        for (int t = 0; t < MT; ++t)
          if (t < mt) {
            const float x0 = __half2float(__ushort_as_half(__ldg(xm + t * K + k0)));
            const float x1 = __half2float(__ushort_as_half(__ldg(xm + t * K + k1)));
            acc[t] = fmaf(w0, x0, fmaf(w1, x1, acc[t]));
          }
      }
      e = e1;
    }
#pragma unroll
    for (int t = 0; t < MT; ++t) {
      float v = acc[t];
#pragma unroll
      for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == t && t < mt) {
        const int64_t i = (int64_t)(m0 + t) * N + n;
        v += w.ydense[i];
        if (F32)
          static_cast<float *>(w.y)[i] = v;
        else
          static_cast<__half *>(w.y)[i] = __float2half_rn(v);
      }
    }
    __syncwarp();  // the table is rewritten for the next row
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

// indexed: grid blocks striding over `rows` rows; else grid x count.
template <bool F32, int MT>
cudaError_t launch_correct(int M, const Batch<Prob> &bt, int grid, int rows, bool indexed, cudaStream_t s) {
  for (int m0 = 0; m0 < M; m0 += MT) {
    if (indexed)
      correct_idx_kernel<F32, MT><<<grid, 32 * kWarps, 0, s>>>(bt, rows, m0, std::min(MT, M - m0));
    else
      correct_kernel<F32, MT><<<dim3(grid, bt.count), 32 * kWarps, 0, s>>>(bt, m0, std::min(MT, M - m0));
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

template <bool F32>
cudaError_t launch_correct_mt(int M, const Batch<Prob> &bt, int grid, int rows, bool indexed, cudaStream_t s) {
  if (M == 1) return launch_correct<F32, 1>(M, bt, grid, rows, indexed, s);
  if (M == 2) return launch_correct<F32, 2>(M, bt, grid, rows, indexed, s);
  if (M <= 4) return launch_correct<F32, 4>(M, bt, grid, rows, indexed, s);
  return launch_correct<F32, 8>(M, bt, grid, rows, indexed, s);
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

// Masks 0..2 of every problem added to its plane-1 result, y written: the
// problems with a correction index through correct_idx_kernel, the others
// through correct_kernel (one launch of each kind present per pass of up
// to 8 tokens).
cudaError_t launch_ew_correct(int M, const EwCall *calls, int count, bool f32, cudaStream_t s) {
  thread_local ew::Batch<ew::Prob> bt;
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  bt.count = count;
  for (int pass = 0; pass < 2; ++pass) {
    const bool indexed = pass == 1;
    int most = 0, total = 0;
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
      P.idx_off = c.w->idx_off;
      P.idx = c.w->idx;
      P.x = reinterpret_cast<const __half *>(c.x);
      P.ydense = c.ydense;
      P.y = c.y;
      P.N = c.w->N;
      P.K = c.w->K;
      const bool mine = (c.w->idx_off && c.w->idx) == indexed;
      P.S = ew::warps_per_row(P.N, P.K, sms);
      const int rows = ew::kWarps / P.S;
      P.blocks = mine && !indexed ? (P.N + rows - 1) / rows : 0;
      P.row_begin = total;
      if (mine && indexed) total += P.N;
      most = std::max(most, P.blocks);
    }
    if (indexed ? total == 0 : most == 0) continue;
    const int grid = indexed ? std::min((total + ew::kWarps - 1) / ew::kWarps, 8 * sms) : most;
    const cudaError_t e = f32 ? ew::launch_correct_mt<true>(M, bt, grid, total, indexed, s)
                              : ew::launch_correct_mt<false>(M, bt, grid, total, indexed, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace tq
