// tq_codec.cu - pack / unpack / salience row-prefix kernels.
//
// The lattice-aware serialization of the paper ("Packing: From Quantization
// to Serialization") stores the discrete supports (trit codes) and their
// parameters instead of fp16 values.  Byte layout (library definition, the
// paper prints none): five trits per byte as a base-3 numeral, digit =
// trit + 1, first trit least significant; a 128-trit group is 26 bytes
// (25 full bytes, then a tail byte with trits 125..127 and pad digits 1);
// plane-1 rows are padded with 0x00 to a multiple of 16 bytes.  Plane 2
// holds only salient groups in (row, group) order.
//
// Every kernel validates what it reads and ORs TQ_DATA_* bits into the
// caller's status word; no kernel traps, and every plane-2 index is checked
// against rowptr[N] before it is used.
#include "tq_common.cuh"

namespace tq {

__device__ __forceinline__ int sal_bit(const uint32_t *sal, int W, int n, int g) {
  return (int)((sal[(int64_t)n * W + (g >> 5)] >> (g & 31)) & 1u);
}

// Number of salient groups of row n before group g.
__device__ __forceinline__ int sal_rank(const uint32_t *sal, int W, int n, int g) {
  const uint32_t *row = sal + (int64_t)n * W;
  int r = 0;
  for (int w = 0; w < (g >> 5); ++w) r += __popc(row[w]);
  uint32_t part = row[g >> 5] & ((1u << (g & 31)) - 1u);
  return r + __popc(part);
}

// Set bits of row n at valid group positions, and whether pad bits are set.
__device__ __forceinline__ int row_popc(const uint32_t *sal, int W, int G, int n, bool *pad_bad) {
  const uint32_t *row = sal + (int64_t)n * W;
  int r = 0;
  for (int w = 0; w < W; ++w) {
    uint32_t v = row[w];
    int valid = G - 32 * w;  // valid bits in this word
    if (valid < 32) {
      uint32_t mask = valid > 0 ? ((1u << valid) - 1u) : 0u;
      if (v & ~mask) *pad_bad = true;
      v &= mask;
    }
    r += __popc(v);
  }
  return r;
}

// ---------------------------------------------------------------- rowptr
// One block: each thread sums a contiguous run of rows, then a block scan.
__global__ void __launch_bounds__(1024) rowptr_kernel(int N, int K, const uint32_t *sal,
                                                      int32_t *rowptr, uint32_t *status) {
  const int G = K / kGroup, W = sal_words_of(K);
  const int per = (N + blockDim.x - 1) / blockDim.x;
  const int r0 = threadIdx.x * per;
  const int r1 = min(N, r0 + per);
  bool pad_bad = false;
  int local = 0;
  for (int n = r0; n < r1; ++n) local += row_popc(sal, W, G, n, &pad_bad);
  // inclusive warp scan, then scan of warp totals
  __shared__ int warp_tot[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  int incl = local;
  for (int o = 1; o < 32; o <<= 1) {
    int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) warp_tot[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    int nw = blockDim.x >> 5;
    int v = lane < nw ? warp_tot[lane] : 0;
    for (int o = 1; o < 32; o <<= 1) {
      int u = __shfl_up_sync(0xffffffffu, v, o);
      if (lane >= o) v += u;
    }
    if (lane < nw) warp_tot[lane] = v;  // inclusive over warps
  }
  __syncthreads();
  int base = (wid > 0 ? warp_tot[wid - 1] : 0) + incl - local;
  for (int n = r0; n < r1; ++n) {
    rowptr[n] = base;
    bool dummy = false;
    base += row_popc(sal, W, G, n, &dummy);
  }
  if (threadIdx.x == blockDim.x - 1) rowptr[N] = warp_tot[(blockDim.x >> 5) - 1];
  if (pad_bad) atomicOr(status, TQ_DATA_BAD_PAD);
}

// Thread per row: rowptr[0] == 0 and rowptr[n+1] - rowptr[n] == popcount.
__global__ void check_rowptr_kernel(int N, int K, const uint32_t *sal, const int32_t *rowptr,
                                    uint32_t *status) {
  const int G = K / kGroup, W = sal_words_of(K);
  int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= N) return;
  bool pad_bad = false;
  int c = row_popc(sal, W, G, n, &pad_bad);
  uint32_t st = 0;
  if (pad_bad) st |= TQ_DATA_BAD_PAD;
  if (rowptr[n + 1] - rowptr[n] != c) st |= TQ_DATA_BAD_ROWPTR;
  if (n == 0 && rowptr[0] != 0) st |= TQ_DATA_BAD_ROWPTR;
  if (st) atomicOr(status, st);
}

// ------------------------------------------------------------------- pack
__device__ __forceinline__ uint8_t encode_codes(const int8_t *t, int ntr, uint32_t *st) {
  int v = 0, p = 1;
  for (int i = 0; i < 5; ++i) {
    int d = 1;  // pad digit (trit 0)
    if (i < ntr) {
      int c = t[i];
      if (c < -1 || c > 1) {
        *st |= TQ_DATA_BAD_CODE;
        c = c < -1 ? -1 : 1;
      }
      d = c + 1;
    }
    v += d * p;
    p *= 3;
  }
  return (uint8_t)v;
}

// Thread per plane-1 byte (n, b): blocks stride over rows, threads over a
// row's bytes.
__global__ void pack_kernel(int N, int K, const int8_t *T1, const int8_t *T2, const uint32_t *sal,
                            const int32_t *rowptr, uint8_t *plane1, uint8_t *plane2,
                            uint32_t *status) {
  const int G = K / kGroup, W = sal_words_of(K);
  const int RB = (int)row_bytes_of(K);
  const int32_t nnz = rowptr[N];
  for (int n = blockIdx.x; n < N; n += gridDim.x)
  for (int b = threadIdx.x; b < RB; b += blockDim.x) {
    const int64_t idx = (int64_t)n * RB + b;
    uint32_t st = 0;
    if (b >= G * kGroupBytes) {
      plane1[idx] = 0;
      continue;
    }
    const int g = b / kGroupBytes, pos = b - g * kGroupBytes;
    const int ntr = pos < kFullBytes ? 5 : kTailTrits;
    const int64_t k0 = (int64_t)n * K + (int64_t)g * kGroup + 5 * pos;
    plane1[idx] = encode_codes(T1 + k0, ntr, &st);
    const int s = sal_bit(sal, W, n, g);
    if (T2) {
      if (s) {
        int64_t j = (int64_t)rowptr[n] + sal_rank(sal, W, n, g);
        if (j >= 0 && j < nnz)
          plane2[j * kGroupBytes + pos] = encode_codes(T2 + k0, ntr, &st);
        else
          st |= TQ_DATA_BAD_ROWPTR;
      } else {
        for (int i = 0; i < ntr; ++i)
          if (T2[k0 + i] != 0) st |= TQ_DATA_T2_OUTSIDE;
      }
    } else if (s) {
      st |= TQ_DATA_T2_OUTSIDE;
    }
    if (st) atomicOr(status, st);
  }
}

// ----------------------------------------------------------------- unpack
__device__ __forceinline__ void decode_to(uint8_t v, int ntr, int8_t *t, uint32_t *st) {
  if (v > 242) {
    *st |= TQ_DATA_BAD_BYTE;
    for (int i = 0; i < ntr; ++i) t[i] = 0;
    return;
  }
  int q = v;
  for (int i = 0; i < 5; ++i) {
    int d = q % 3;
    q /= 3;
    if (i < ntr)
      t[i] = (int8_t)(d - 1);
    else if (d != 1)
      *st |= TQ_DATA_BAD_PAD;
  }
}

// Thread per plane-1 byte (n, b): blocks stride over rows, threads over a
// row's bytes.
__global__ void unpack_kernel(int N, int K, const uint8_t *plane1, const uint8_t *plane2,
                              const uint32_t *sal, const int32_t *rowptr, int8_t *T1, int8_t *T2,
                              uint32_t *status) {
  const int G = K / kGroup, W = sal_words_of(K);
  const int RB = (int)row_bytes_of(K);
  const int32_t nnz = rowptr[N];
  for (int n = blockIdx.x; n < N; n += gridDim.x)
  for (int b = threadIdx.x; b < RB; b += blockDim.x) {
    const int64_t idx = (int64_t)n * RB + b;
    uint32_t st = 0;
    const uint8_t v = plane1[idx];
    if (b >= G * kGroupBytes) {
      if (v != 0) atomicOr(status, TQ_DATA_BAD_PAD);
      continue;
    }
    const int g = b / kGroupBytes, pos = b - g * kGroupBytes;
    const int ntr = pos < kFullBytes ? 5 : kTailTrits;
    const int64_t k0 = (int64_t)n * K + (int64_t)g * kGroup + 5 * pos;
    decode_to(v, ntr, T1 + k0, &st);
    if (T2) {
      if (sal_bit(sal, W, n, g)) {
        int64_t j = (int64_t)rowptr[n] + sal_rank(sal, W, n, g);
        if (plane2 && j >= 0 && j < nnz) {
          decode_to(plane2[j * kGroupBytes + pos], ntr, T2 + k0, &st);
        } else {
          st |= TQ_DATA_BAD_ROWPTR;
          for (int i = 0; i < ntr; ++i) T2[k0 + i] = 0;
        }
      } else {
        for (int i = 0; i < ntr; ++i) T2[k0 + i] = 0;
      }
    }
    if (st) atomicOr(status, st);
  }
}

// ------------------------------------------------ row-staged pack / unpack
// The same byte layout and status bits as pack_kernel / unpack_kernel, with
// one CTA per row at a time.  The row's codes move between global and
// shared memory in 16-byte units (coalesced), and the per-byte encode or
// decode works on shared memory; the salience rank of each group is formed
// once per row.  Taken when the code arrays are 16-byte aligned and a row's
// codes fit in shared memory.
constexpr int kPackThreads = 128;    // pack: up to 16 CTAs (rows in flight) per SM
constexpr int kUnpackThreads = 256;
constexpr int kRowMaxK = 49152;  // 2 x 48 KiB of codes per row

// The byte of the five codes row[k0 .. k0 + 4] (a full byte): two 32-bit
// shared-memory loads and a funnel shift give the codes, their digits
// (code + 1) come bytewise without carries between bytes, and one dp4a
// forms sum d_i 3^i.  A code outside {-1, 0, 1} goes through encode_codes,
// which clamps it and flags the status.
__device__ __forceinline__ uint8_t encode5(const int8_t *row, int k0, uint32_t *st) {
  const uint32_t *w = reinterpret_cast<const uint32_t *>(row) + (k0 >> 2);
  const uint32_t sh = 8u * (uint32_t)(k0 & 3);
  const uint32_t lo = w[0], hi = w[1];
  const uint32_t c4 = __funnelshift_r(lo, hi, sh), c5 = (hi >> sh) & 0xFFu;
  const uint32_t d4 = ((c4 & 0x7F7F7F7Fu) + 0x01010101u) ^ (c4 & 0x80808080u);
  const uint32_t d5 = ((c5 & 0x7Fu) + 1u) ^ (c5 & 0x80u);
  if ((((d4 | d5) & 0xFCFCFCFCu) | (d4 & (d4 >> 1) & 0x01010101u) | (d5 & (d5 >> 1) & 1u)) != 0)
    return encode_codes(row + k0, 5, st);
  return (uint8_t)__dp4a(d4, 0x1B090301u, 81u * d5);
}

__host__ __device__ inline int rows_smem_bytes(int K) { return 2 * K + 4 * (K / kGroup); }

// rk[g]: rank of group g among row n's salient groups, -1 if not salient.
__device__ __forceinline__ void row_ranks(const uint32_t *sal, int W, int G, int n, int32_t *rk) {
  for (int g = threadIdx.x; g < G; g += blockDim.x) rk[g] = sal_bit(sal, W, n, g) ? sal_rank(sal, W, n, g) : -1;
}

__global__ void __launch_bounds__(kPackThreads) pack_rows_kernel(int N, int K, const int8_t *T1, const int8_t *T2,
                                                               const uint32_t *sal, const int32_t *rowptr,
                                                               uint8_t *plane1, uint8_t *plane2, uint32_t *status) {
  extern __shared__ __align__(16) unsigned char smr[];
  const int G = K / kGroup, W = sal_words_of(K);
  const int RB = (int)row_bytes_of(K);
  const int32_t nnz = rowptr[N];
  int8_t *t1 = reinterpret_cast<int8_t *>(smr), *t2 = t1 + K;
  int32_t *rk = reinterpret_cast<int32_t *>(smr + 2 * K);
  uint32_t st = 0;
  for (int n = blockIdx.x; n < N; n += gridDim.x) {
    __syncthreads();  // the previous row's shared-memory reads are done
    row_ranks(sal, W, G, n, rk);
    const int4 *s1 = reinterpret_cast<const int4 *>(T1 + (int64_t)n * K);
    for (int i = threadIdx.x; i < K / 16; i += blockDim.x) reinterpret_cast<int4 *>(t1)[i] = __ldcs(s1 + i);
    if (T2) {
      const int4 *s2 = reinterpret_cast<const int4 *>(T2 + (int64_t)n * K);
      for (int i = threadIdx.x; i < K / 16; i += blockDim.x) {
        const int4 v = __ldcs(s2 + i);
        reinterpret_cast<int4 *>(t2)[i] = v;
        // second-plane codes outside the salient groups must be zero
        if ((v.x | v.y | v.z | v.w) != 0 && !sal_bit(sal, W, n, (16 * i) / kGroup)) st |= TQ_DATA_T2_OUTSIDE;
      }
    }
    __syncthreads();
    const int64_t p1 = (int64_t)n * RB;
    const int32_t rp = rowptr[n];
    for (int b = threadIdx.x; b < RB; b += blockDim.x) {
      if (b >= G * kGroupBytes) {
        plane1[p1 + b] = 0;
        continue;
      }
      const int g = b / kGroupBytes, pos = b - g * kGroupBytes;
      const int ntr = pos < kFullBytes ? 5 : kTailTrits;
      const int k0 = g * kGroup + 5 * pos;
      plane1[p1 + b] = ntr == 5 ? encode5(t1, k0, &st) : encode_codes(t1 + k0, ntr, &st);
      const int r = rk[g];
      if (r >= 0) {
        if (T2) {
          const int64_t j = (int64_t)rp + r;
          if (j >= 0 && j < nnz)
            plane2[j * kGroupBytes + pos] = ntr == 5 ? encode5(t2, k0, &st) : encode_codes(t2 + k0, ntr, &st);
          else
            st |= TQ_DATA_BAD_ROWPTR;
        } else {
          st |= TQ_DATA_T2_OUTSIDE;
        }
      }
    }
  }
  if (st) atomicOr(status, st);
}

__global__ void __launch_bounds__(kUnpackThreads) unpack_rows_kernel(int N, int K, const uint8_t *plane1,
                                                                 const uint8_t *plane2, const uint32_t *sal,
                                                                 const int32_t *rowptr, int8_t *T1, int8_t *T2,
                                                                 uint32_t *status) {
  extern __shared__ __align__(16) unsigned char smr[];
  const int G = K / kGroup, W = sal_words_of(K);
  const int RB = (int)row_bytes_of(K);
  const int32_t nnz = rowptr[N];
  int8_t *t1 = reinterpret_cast<int8_t *>(smr), *t2 = t1 + K;
  int32_t *rk = reinterpret_cast<int32_t *>(smr + 2 * K);
  uint32_t st = 0;
  for (int n = blockIdx.x; n < N; n += gridDim.x) {
    __syncthreads();  // the previous row's stores have read shared memory
    row_ranks(sal, W, G, n, rk);
    // second-plane codes are zero outside the salient groups: the row starts
    // zeroed by 16-byte stores, and only salient groups are decoded into it
    if (T2)
      for (int i = threadIdx.x; i < K / 16; i += blockDim.x) reinterpret_cast<int4 *>(t2)[i] = make_int4(0, 0, 0, 0);
    __syncthreads();
    const int64_t p1 = (int64_t)n * RB;
    const int32_t rp = rowptr[n];
    for (int b = threadIdx.x; b < RB; b += blockDim.x) {
      const uint8_t v = __ldcs(plane1 + p1 + b);
      if (b >= G * kGroupBytes) {
        if (v != 0) st |= TQ_DATA_BAD_PAD;
        continue;
      }
      const int g = b / kGroupBytes, pos = b - g * kGroupBytes;
      const int ntr = pos < kFullBytes ? 5 : kTailTrits;
      const int k0 = g * kGroup + 5 * pos;
      decode_to(v, ntr, t1 + k0, &st);
      if (T2) {
        const int r = rk[g];
        const int64_t j = (int64_t)rp + r;
        if (r >= 0 && plane2 && j >= 0 && j < nnz)
          decode_to(plane2[j * kGroupBytes + pos], ntr, t2 + k0, &st);
        else if (r >= 0)
          st |= TQ_DATA_BAD_ROWPTR;
      }
    }
    __syncthreads();
    int4 *d1 = reinterpret_cast<int4 *>(T1 + (int64_t)n * K);
    for (int i = threadIdx.x; i < K / 16; i += blockDim.x) __stcs(d1 + i, reinterpret_cast<const int4 *>(t1)[i]);
    if (T2) {
      int4 *d2 = reinterpret_cast<int4 *>(T2 + (int64_t)n * K);
      for (int i = threadIdx.x; i < K / 16; i += blockDim.x) __stcs(d2 + i, reinterpret_cast<const int4 *>(t2)[i]);
    }
  }
  if (st) atomicOr(status, st);
}

// ------------------------------------------------------ second-plane index
// One block per group g walks the rows in chunks of blockDim.x, in order;
// a block-wide count (and, for the fill, an exclusive scan of the row bits)
// gives each salient row its place in group g's list.  Group lists start at
// multiples of 16; the entries after a group's last pair, up to the next
// start, are empty.
constexpr int kIdxThreads = 256;

__host__ __device__ __forceinline__ int64_t p2index_capacity(int K, int64_t nnz) {
  return (nnz + 15 * (int64_t)(K / kGroup) + 15) & ~(int64_t)15;
}
__host__ __device__ __forceinline__ int64_t p2index_slot_off(int K) {
  return ((int64_t)(K / kGroup + 1) * 4 + 127) & ~(int64_t)127;
}

// Rows are taken in chunks of kIdxChunk: block (g, c) handles group g's
// rows [kIdxChunk c, kIdxChunk (c + 1)).
constexpr int kIdxChunk = 1024;

// Salient rows of group g in rows [r0, r1) (the block's threads together;
// every thread gets the total).
__device__ __forceinline__ int p2index_block_count(const uint32_t *sal, int W, int g, int r0, int r1, int *red) {
  int c = 0;
  for (int n = r0 + (int)threadIdx.x; n < r1; n += kIdxThreads) c += sal_bit(sal, W, n, g);
  for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = c;
  __syncthreads();
  int t = 0;
  for (int w = 0; w < kIdxThreads / 32; ++w) t += red[w];
  __syncthreads();
  return t;
}

// colptr[g + 1] += salient rows of group g in the block's chunk (colptr
// zeroed by p2index_zero_kernel).
__global__ void __launch_bounds__(kIdxThreads) p2index_count_kernel(int N, int K, const uint32_t *sal,
                                                                     int32_t *colptr) {
  __shared__ int red[kIdxThreads / 32];
  const int g = blockIdx.x, c = blockIdx.y, W = sal_words_of(K);
  const int r0 = c * kIdxChunk, r1 = min(N, r0 + kIdxChunk);
  const int t = p2index_block_count(sal, W, g, r0, r1, red);
  if (threadIdx.x == 0 && t) atomicAdd(colptr + g + 1, t);
}

__global__ void p2index_zero_kernel(int G, int32_t *colptr) {
  for (int i = threadIdx.x; i <= G; i += blockDim.x) colptr[i] = 0;
}

// colptr[g+1] = colptr[g] + count rounded up to 16, at most the capacity
// (which the counts of a consistent salience map never reach).
__global__ void p2index_scan_kernel(int G, int64_t cap, int32_t *colptr) {
  if (threadIdx.x != 0) return;
  colptr[0] = 0;
  int64_t run = 0;
  for (int g = 0; g < G; ++g) {
    run = min(run + (((int64_t)colptr[g + 1] + 15) & ~(int64_t)15), cap);
    colptr[g + 1] = (int32_t)run;
  }
}

// One slot: 8 words in the order of logical words 0, 4, 1, 5, 2, 6, 3, 7.
__device__ __forceinline__ void p2index_store_slot(uint8_t *slot, const uint32_t *L) {
  uint4 *d = reinterpret_cast<uint4 *>(slot);
  d[0] = make_uint4(L[0], L[4], L[1], L[5]);
  d[1] = make_uint4(L[2], L[6], L[3], L[7]);
}

__device__ __forceinline__ void p2index_empty_slot(uint8_t *slot) {
  const uint32_t L[8] = {0, 0, 0, 0, 0, 0, 0, 0xffffffffu};
  p2index_store_slot(slot, L);
}

// Entry e of group g: the record j of row n (plane 2 and s2 are 2-byte
// aligned at a record, so the record is read as 13 halves).
__device__ __forceinline__ void p2index_fill_slot(uint8_t *slot, int g, int n, int64_t j, int64_t nnz,
                                                  const uint8_t *plane2, const uint16_t *scale2) {
  if (j < 0 || j >= nnz) {
    p2index_empty_slot(slot);
    return;
  }
  uint32_t L[8] = {0, 0, 0, 0, 0, 0, 0, (uint32_t)n};
  const int h0 = (g % 8) & 1;  // the record starts at logical half h0 (byte o = 2 h0)
  const uint16_t *rec = reinterpret_cast<const uint16_t *>(plane2 + j * kGroupBytes);
#pragma unroll
  for (int i = 0; i < kGroupBytes / 2; ++i) {
    const int h = h0 + i;
    L[h >> 1] |= (uint32_t)rec[i] << (16 * (h & 1));
  }
  const int hs = h0 ? 0 : kGroupBytes / 2;  // s2 in the free half next to the record
  L[hs >> 1] |= (uint32_t)scale2[j] << (16 * (hs & 1));
  p2index_store_slot(slot, L);
}

// Block (g, c) fills the entries of group g's salient rows of chunk c
// (their place: colptr[g] plus the salient rows of the group's earlier
// chunks, counted by the block itself); the group's last chunk empties the
// slots after its last entry.  Block (G, 0) empties the slots from
// colptr[G] to the capacity.
__global__ void __launch_bounds__(kIdxThreads) p2index_fill_kernel(int N, int K, const uint32_t *sal,
                                                                    const int32_t *rowptr, int64_t nnz,
                                                                    const uint8_t *plane2, const uint16_t *scale2,
                                                                    int32_t *index) {
  __shared__ int warp_base[kIdxThreads / 32 + 1];
  __shared__ int red[kIdxThreads / 32];
  const int G = K / kGroup, g = blockIdx.x, c = blockIdx.y, W = sal_words_of(K);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint8_t *slots = reinterpret_cast<uint8_t *>(index) + p2index_slot_off(K);
  if (g == G) {
    if (c != 0) return;
    const int64_t cap = p2index_capacity(K, nnz);
    for (int64_t e = index[G] + threadIdx.x; e < cap; e += kIdxThreads) p2index_empty_slot(slots + 32 * e);
    return;
  }
  const int r0 = c * kIdxChunk, r1 = min(N, r0 + kIdxChunk);
  if (r0 >= N) return;
  const int64_t lim = index[g + 1];
  int64_t base = index[g] + p2index_block_count(sal, W, g, 0, r0, red);
  for (int n0 = r0; n0 < r1; n0 += kIdxThreads) {
    const int n = n0 + threadIdx.x;
    const bool bit = n < r1 && sal_bit(sal, W, n, g);
    const uint32_t m = __ballot_sync(0xffffffffu, bit);
    if (lane == 0) warp_base[warp] = __popc(m);
    __syncthreads();
    if (threadIdx.x == 0) {
      int run = 0;
      for (int w = 0; w < kIdxThreads / 32; ++w) {
        const int cnt = warp_base[w];
        warp_base[w] = run;
        run += cnt;
      }
      warp_base[kIdxThreads / 32] = run;
    }
    __syncthreads();
    if (bit) {
      const int64_t pos = base + warp_base[warp] + __popc(m & ((1u << lane) - 1u));
      if (pos < lim) {  // within the group's entries (the capacity cuts an inconsistent map short)
        const int64_t j = (int64_t)rowptr[n] + sal_rank(sal, W, n, g);
        p2index_fill_slot(slots + 32 * pos, g, n, j, nnz, plane2, scale2);
      }
    }
    base += warp_base[kIdxThreads / 32];
    __syncthreads();
  }
  if (r1 == N)
    for (int64_t e = base + threadIdx.x; e < lim; e += kIdxThreads) p2index_empty_slot(slots + 32 * e);
}

// ------------------------------------------------------------- launchers
static int grid_for(int64_t work, int block) {
  int64_t g = (work + block - 1) / block;
  if (g > 152 * 32) g = 152 * 32;
  return (int)(g < 1 ? 1 : g);
}

cudaError_t launch_rowptr(int N, int K, const uint32_t *sal, int32_t *rowptr, uint32_t *status,
                          cudaStream_t s) {
  rowptr_kernel<<<1, 1024, 0, s>>>(N, K, sal, rowptr, status);
  return cudaGetLastError();
}

cudaError_t launch_check_rowptr(int N, int K, const uint32_t *sal, const int32_t *rowptr,
                                uint32_t *status, cudaStream_t s) {
  check_rowptr_kernel<<<(N + 255) / 256, 256, 0, s>>>(N, K, sal, rowptr, status);
  return cudaGetLastError();
}

cudaError_t launch_pack(int N, int K, const int8_t *T1, const int8_t *T2, const uint32_t *sal,
                        const int32_t *rowptr, uint8_t *plane1, uint8_t *plane2, uint32_t *status,
                        cudaStream_t s) {
  if (K <= kRowMaxK && ((((uintptr_t)T1) | ((uintptr_t)T2)) & 15u) == 0) {
    const int sm = rows_smem_bytes(K);
    if (sm > 48 * 1024) {
      const cudaError_t e = cudaFuncSetAttribute(pack_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
      if (e != cudaSuccess) return e;
    }
    pack_rows_kernel<<<std::min(N, 152 * 16), kPackThreads, sm, s>>>(N, K, T1, T2, sal, rowptr, plane1, plane2,
                                                                    status);
    return cudaGetLastError();
  }
  pack_kernel<<<std::min(N, 152 * 16), 256, 0, s>>>(N, K, T1, T2, sal, rowptr, plane1, plane2, status);
  return cudaGetLastError();
}

cudaError_t launch_unpack(int N, int K, const uint8_t *plane1, const uint8_t *plane2,
                          const uint32_t *sal, const int32_t *rowptr, int8_t *T1, int8_t *T2,
                          uint32_t *status, cudaStream_t s) {
  if (K <= kRowMaxK && ((((uintptr_t)T1) | ((uintptr_t)T2)) & 15u) == 0) {
    const int sm = rows_smem_bytes(K);
    if (sm > 48 * 1024) {
      const cudaError_t e = cudaFuncSetAttribute(unpack_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
      if (e != cudaSuccess) return e;
    }
    unpack_rows_kernel<<<std::min(N, 152 * 8), kUnpackThreads, sm, s>>>(N, K, plane1, plane2, sal, rowptr, T1, T2,
                                                                      status);
    return cudaGetLastError();
  }
  unpack_kernel<<<std::min(N, 152 * 16), 256, 0, s>>>(N, K, plane1, plane2, sal, rowptr, T1, T2,
                                                     status);
  return cudaGetLastError();
}

cudaError_t launch_plane2_index(int N, int K, const uint32_t *sal, const int32_t *rowptr, int64_t nnz,
                                const uint8_t *plane2, const uint16_t *scale2, int32_t *index, cudaStream_t s) {
  const int G = K / kGroup, C = (N + kIdxChunk - 1) / kIdxChunk;
  p2index_zero_kernel<<<1, 256, 0, s>>>(G, index);
  p2index_count_kernel<<<dim3(G, C), kIdxThreads, 0, s>>>(N, K, sal, index);
  p2index_scan_kernel<<<1, 32, 0, s>>>(G, p2index_capacity(K, nnz), index);
  p2index_fill_kernel<<<dim3(G + 1, C), kIdxThreads, 0, s>>>(N, K, sal, rowptr, nnz, plane2, scale2, index);
  return cudaGetLastError();
}

// ------------------------------------------ element-wise four-mask format
// The paper's representation with four disjoint masks of orders [2, 2, 1, 1]
// ("Model and Representation"), stored as: a 2-bit mask-id plane (element k
// of row n in bits 2 (k mod 16) of word [n][k / 16]); T0 of every element in
// plane 1's group layout (the codec above); per row, the T1 trits of its
// order-2 elements (masks 0 and 1) in increasing k, five per byte, the last
// byte padded with digit 1, row n's bytes from byte rowptr[n].
constexpr int kEwRowWarps = 4;  // rows (warps) per block of the per-row kernels

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Warp per row: plane-2 bytes of the row (ceil(order-2 elements / 5)) into
// rowptr[n + 1]; mask ids above 3 set BAD_CODE.
__global__ void __launch_bounds__(32 * kEwRowWarps) ew_count_kernel(int N, int K, const uint8_t *mask,
                                                                   int32_t *rowptr, uint32_t *status) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kEwRowWarps + (threadIdx.x >> 5);
  if (n >= N) return;
  const uint8_t *row = mask + (int64_t)n * K;
  int c = 0;
  uint32_t st = 0;
  for (int k = lane; k < K; k += 32) {
    const uint8_t m = row[k];
    c += m <= 1;
    if (m > 3) st |= TQ_DATA_BAD_CODE;
  }
  for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) {
    rowptr[n + 1] = (c + 4) / 5;
    if (n == 0) rowptr[0] = 0;
    if (st) atomicOr(status, st);
  }
}

// One block: rowptr[1..N] (bytes per row) into offsets, in place.
__global__ void __launch_bounds__(1024) ew_scan_kernel(int N, int32_t *rowptr) {
  __shared__ int32_t part[1024];
  const int t = threadIdx.x;
  const int r0 = (int)((int64_t)N * t / 1024), r1 = (int)((int64_t)N * (t + 1) / 1024);
  int32_t sum = 0;
  for (int n = r0; n < r1; ++n) sum += rowptr[n + 1];
  part[t] = sum;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {
    const int32_t v = t >= o ? part[t - o] : 0;
    __syncthreads();
    part[t] += v;
    __syncthreads();
  }
  int32_t run = part[t] - sum;  // exclusive prefix of this thread's rows
  for (int n = r0; n < r1; ++n) {
    run += rowptr[n + 1];
    rowptr[n + 1] = run;
  }
}

// Thread per mask word.
__global__ void ew_mask_pack_kernel(int N, int K, const uint8_t *mask, uint32_t *plane, uint32_t *status) {
  const int64_t total = (int64_t)N * (K / 16);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const uint8_t *src = mask + i * 16;
    uint32_t w = 0, st = 0;
    for (int j = 0; j < 16; ++j) {
      uint32_t m = src[j];
      if (m > 3) st |= TQ_DATA_BAD_CODE, m = 3;
      w |= m << (2 * j);
    }
    plane[i] = w;
    if (st) atomicOr(status, st);
  }
}

// Thread per plane-1 byte: T0 of every element (the group layout).
__global__ void ew_plane1_pack_kernel(int N, int K, const int8_t *T0, uint8_t *plane1, uint32_t *status) {
  const int G = K / kGroup;
  const int64_t RB = row_bytes_of(K), total = (int64_t)N * RB;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int n = (int)(idx / RB), b = (int)(idx - (int64_t)n * RB);
    if (b >= G * kGroupBytes) {
      plane1[idx] = 0;
      continue;
    }
    uint32_t st = 0;
    const int g = b / kGroupBytes, pos = b - g * kGroupBytes;
    plane1[idx] = encode_codes(T0 + (int64_t)n * K + (int64_t)g * kGroup + 5 * pos, pos < kFullBytes ? 5 : kTailTrits, &st);
    if (st) atomicOr(status, st);
  }
}

// Warp per row: the row's order-2 T1 trits in order, five per byte.  Each
// 32-element chunk ranks its order-2 elements by ballot; their digits join
// the (fewer than 5) left over from earlier chunks in a per-warp ring, whole
// bytes are written, the rest carried on.
__global__ void __launch_bounds__(32 * kEwRowWarps) ew_plane2_pack_kernel(int N, int K, const int8_t *T1,
                                                                         const uint8_t *mask, const int32_t *rowptr,
                                                                         uint8_t *plane2, uint32_t *status) {
  __shared__ uint8_t dig[kEwRowWarps][40];
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  const int n = blockIdx.x * kEwRowWarps + wi;
  if (n >= N) return;
  uint8_t *d = dig[wi];
  const int8_t *t1 = T1 + (int64_t)n * K;
  const uint8_t *mk = mask + (int64_t)n * K;
  const int64_t b0 = rowptr[n], nb = (int64_t)rowptr[n + 1] - rowptr[n];
  int pend = 0;   // digits carried into this chunk
  int64_t out = 0;  // bytes written
  uint32_t st = 0;
  for (int k0 = 0; k0 < K; k0 += 32) {
    const int k = k0 + lane;
    const bool in = k < K;
    const bool o2 = in && mk[k] <= 1;
    int c = in ? t1[k] : 0;
    if (c < -1 || c > 1) st |= TQ_DATA_BAD_CODE, c = c < -1 ? -1 : 1;
    if (in && !o2 && c != 0) st |= TQ_DATA_T2_OUTSIDE;
    const uint32_t bal = __ballot_sync(0xffffffffu, o2);
    if (o2) d[pend + __popc(bal & lanemask_lt())] = (uint8_t)(c + 1);
    __syncwarp();
    const int tot = pend + __popc(bal), full = tot / 5, rem = tot - 5 * full;
    if (lane < full) {
      const uint8_t *q = d + 5 * lane;
      const int v = q[0] + 3 * q[1] + 9 * q[2] + 27 * q[3] + 81 * q[4];
      if (out + lane < nb) plane2[b0 + out + lane] = (uint8_t)v;
    }
    const uint8_t carry = lane < rem ? d[5 * full + lane] : 0;
    __syncwarp();
    if (lane < rem) d[lane] = carry;
    __syncwarp();
    out += full;
    pend = rem;
  }
  if (pend > 0 && lane == 0) {
    int v = 0, p = 1;
    for (int i = 0; i < 5; ++i, p *= 3) v += (i < pend ? d[i] : 1) * p;
    if (out < nb) plane2[b0 + out] = (uint8_t)v;
    ++out;
  }
  if (lane == 0 && out != nb) st |= TQ_DATA_BAD_ROWPTR;
  if (st) atomicOr(status, st);
}

// Thread per mask word: mask ids back.
__global__ void ew_mask_unpack_kernel(int N, int K, const uint32_t *plane, uint8_t *mask) {
  const int64_t total = (int64_t)N * (K / 16);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t w = plane[i];
    for (int j = 0; j < 16; ++j) mask[i * 16 + j] = (uint8_t)((w >> (2 * j)) & 3u);
  }
}

// Thread per plane-1 byte: T0 back (pad bytes must be 0).
__global__ void ew_plane1_unpack_kernel(int N, int K, const uint8_t *plane1, int8_t *T0, uint32_t *status) {
  const int G = K / kGroup;
  const int64_t RB = row_bytes_of(K), total = (int64_t)N * RB;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int n = (int)(idx / RB), b = (int)(idx - (int64_t)n * RB);
    const uint8_t v = plane1[idx];
    if (b >= G * kGroupBytes) {
      if (v != 0) atomicOr(status, TQ_DATA_BAD_PAD);
      continue;
    }
    uint32_t st = 0;
    const int g = b / kGroupBytes, pos = b - g * kGroupBytes;
    decode_to(v, pos < kFullBytes ? 5 : kTailTrits, T0 + (int64_t)n * K + (int64_t)g * kGroup + 5 * pos, &st);
    if (st) atomicOr(status, st);
  }
}

// Warp per row: T1 back from plane 2 (zeros on order-1 elements); bytes
// above 242 and pad digits other than 1 in the row's last byte are flagged.
__global__ void __launch_bounds__(32 * kEwRowWarps) ew_plane2_unpack_kernel(int N, int K, const uint32_t *plane,
                                                                           const int32_t *rowptr,
                                                                           const uint8_t *plane2, int8_t *T1,
                                                                           uint32_t *status) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kEwRowWarps + (threadIdx.x >> 5);
  if (n >= N) return;
  const int64_t b0 = rowptr[n], nb = (int64_t)rowptr[n + 1] - rowptr[n];
  const uint32_t *mw = plane + (int64_t)n * (K / 16);
  int base = 0;
  uint32_t st = 0;
  for (int k0 = 0; k0 < K; k0 += 32) {
    const int k = k0 + lane;
    const bool in = k < K;
    const bool o2 = in && ((mw[k >> 4] >> (2 * (k & 15))) & 3u) <= 1;
    const uint32_t bal = __ballot_sync(0xffffffffu, o2);
    int8_t t = 0;
    if (o2) {
      const int r = base + __popc(bal & lanemask_lt());
      if (r / 5 < nb) {
        int v = plane2[b0 + r / 5];
        if (v > 242) st |= TQ_DATA_BAD_BYTE, v = 0;
        for (int i = 0; i < r % 5; ++i) v /= 3;
        t = (int8_t)(v % 3 - 1);
      } else {
        st |= TQ_DATA_BAD_ROWPTR;
      }
    }
    if (in) T1[(int64_t)n * K + k] = t;
    base += __popc(bal);
  }
  if (lane == 0) {
    if ((base + 4) / 5 != nb) st |= TQ_DATA_BAD_ROWPTR;
    if (base % 5 && nb > 0 && (base + 4) / 5 == nb) {
      int v = plane2[b0 + nb - 1];
      if (v <= 242) {
        for (int i = 0; i < 5; ++i, v /= 3)
          if (i >= base % 5 && v % 3 != 1) st |= TQ_DATA_BAD_PAD;
      }
    }
  }
  if (st) atomicOr(status, st);
}

// ----------------------------------------------- element-wise correction index
// Entries of masks 0..2 per row and 2048-element block (uint16
// (k mod 2048) | code << 11, code = 9 q + 3 (T0 + 1) + (T1 + 1)), with int32
// offsets[n nb + b] (nb = ceil(K / 2048)).
constexpr int kIdxBlock = 2048, kIdxShift = 11;

// Warp per row: the count of each block's mask-0..2 elements into
// off[n nb + b + 1] (off[0] = 0); ew_scan_kernel turns them into offsets.
__global__ void __launch_bounds__(32 * kEwRowWarps) ew_index_count_kernel(int N, int K, const uint32_t *plane,
                                                                          int32_t *off) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kEwRowWarps + (threadIdx.x >> 5);
  if (n >= N) return;
  const int WK = K / 16, nb = (K + kIdxBlock - 1) / kIdxBlock;
  const uint32_t *mw = plane + (int64_t)n * WK;
  for (int b = 0; b < nb; ++b) {
    int c = 0;
    for (int wi = b * (kIdxBlock / 16) + lane; wi < min(WK, (b + 1) * (kIdxBlock / 16)); wi += 32) {
      const uint32_t m = mw[wi];
      c += __popc(~(m & (m >> 1)) & 0x55555555u);
    }
    for (int o = 16; o; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if (lane == 0) off[(int64_t)n * nb + b + 1] = c;
  }
  if (n == 0 && lane == 0) off[0] = 0;
}

__device__ __forceinline__ int base3_digit(int v, int i) {
  for (int j = 0; j < i; ++j) v /= 3;
  return v % 3;
}

// Warp per row, 32 elements per step (lane = element): each mask-0..2
// element's entry at its rank in the row; T0 from plane 1, T1 from plane 2
// at the element's rank among the row's order-2 elements.  A row whose
// offsets or plane-2 rowptr do not match its mask plane is skipped and
// reported (TQ_DATA_BAD_ROWPTR), so nothing is written outside its range.
__global__ void __launch_bounds__(32 * kEwRowWarps) ew_index_fill_kernel(int N, int K, const uint32_t *plane,
                                                                         const uint8_t *plane1,
                                                                         const int32_t *rowptr,
                                                                         const uint8_t *plane2, const int32_t *off,
                                                                         uint16_t *idx, uint32_t *status) {
  const int lane = threadIdx.x & 31;
  const int n = blockIdx.x * kEwRowWarps + (threadIdx.x >> 5);
  if (n >= N) return;
  const int WK = K / 16, nb = (K + kIdxBlock - 1) / kIdxBlock;
  const uint32_t *mw = plane + (int64_t)n * WK;
  const int64_t e0 = off[(int64_t)n * nb];
  int c3 = 0, c2 = 0;
  for (int wi = lane; wi < WK; wi += 32) {
    const uint32_t m = mw[wi];
    c3 += __popc(~(m & (m >> 1)) & 0x55555555u);
    c2 += __popc(~m & 0xaaaaaaaau);
  }
  for (int o = 16; o; o >>= 1) {
    c3 += __shfl_xor_sync(0xffffffffu, c3, o);
    c2 += __shfl_xor_sync(0xffffffffu, c2, o);
  }
  const int64_t b2 = rowptr[n], nb2 = (int64_t)rowptr[n + 1] - rowptr[n];
  if ((int64_t)off[(int64_t)n * nb + nb] - e0 != c3 || (c2 + 4) / 5 != nb2) {
    if (lane == 0) atomicOr(status, TQ_DATA_BAD_ROWPTR);
    return;
  }
  const uint8_t *p1 = plane1 + (int64_t)n * row_bytes_of(K);
  uint32_t st = 0;
  int run = 0, r2 = 0;
  for (int k0 = 0; k0 < K; k0 += 32) {
    if (k0 % kIdxBlock == 0 && run != (int)(off[(int64_t)n * nb + k0 / kIdxBlock] - e0)) {
      st |= TQ_DATA_BAD_ROWPTR;  // per-block offsets that do not match the mask plane
      break;
    }
    const int k = k0 + lane;
    const uint32_t q = k < K ? (mw[k >> 4] >> (2 * (k & 15))) & 3u : 3u;
    const uint32_t bal3 = __ballot_sync(0xffffffffu, q != 3u), bal2 = __ballot_sync(0xffffffffu, q <= 1u);
    if (q != 3u) {
      const int kg = k % kGroup;
      int v = p1[(int64_t)(k / kGroup) * kGroupBytes + kg / 5];
      if (v > 242) st |= TQ_DATA_BAD_BYTE, v = 242;
      const int d0 = base3_digit(v, kg % 5);
      int d1 = 1;
      if (q <= 1u) {
        const int r = r2 + __popc(bal2 & lanemask_lt());
        int u = plane2[b2 + r / 5];
        if (u > 242) st |= TQ_DATA_BAD_BYTE, u = 242;
        d1 = base3_digit(u, r % 5);
      }
      const uint32_t code = 9u * q + 3u * (uint32_t)d0 + (uint32_t)d1;
      idx[e0 + run + __popc(bal3 & lanemask_lt())] = (uint16_t)((uint32_t)(k % kIdxBlock) | (code << kIdxShift));
    }
    run += __popc(bal3);
    r2 += __popc(bal2);
  }
  for (int o = 16; o; o >>= 1) st |= __shfl_xor_sync(0xffffffffu, st, o);
  if (lane == 0 && st) atomicOr(status, st);
}

cudaError_t launch_ew_index_offsets(int N, int K, const uint32_t *mplane, int32_t *off, cudaStream_t s) {
  const int nb = (K + kIdxBlock - 1) / kIdxBlock;
  ew_index_count_kernel<<<(N + kEwRowWarps - 1) / kEwRowWarps, 32 * kEwRowWarps, 0, s>>>(N, K, mplane, off);
  ew_scan_kernel<<<1, 1024, 0, s>>>(N * nb, off);
  return cudaGetLastError();
}

cudaError_t launch_ew_index_fill(int N, int K, const uint32_t *mplane, const uint8_t *plane1, const int32_t *rowptr,
                                 const uint8_t *plane2, const int32_t *off, uint16_t *idx, uint32_t *status,
                                 cudaStream_t s) {
  ew_index_fill_kernel<<<(N + kEwRowWarps - 1) / kEwRowWarps, 32 * kEwRowWarps, 0, s>>>(N, K, mplane, plane1, rowptr,
                                                                                       plane2, off, idx, status);
  return cudaGetLastError();
}

cudaError_t launch_ew_rowptr(int N, int K, const uint8_t *mask, int32_t *rowptr, uint32_t *status, cudaStream_t s) {
  ew_count_kernel<<<(N + kEwRowWarps - 1) / kEwRowWarps, 32 * kEwRowWarps, 0, s>>>(N, K, mask, rowptr, status);
  ew_scan_kernel<<<1, 1024, 0, s>>>(N, rowptr);
  return cudaGetLastError();
}

cudaError_t launch_ew_pack(int N, int K, const int8_t *T0, const int8_t *T1, const uint8_t *mask,
                           const int32_t *rowptr, uint32_t *mplane, uint8_t *plane1, uint8_t *plane2,
                           uint32_t *status, cudaStream_t s) {
  ew_mask_pack_kernel<<<grid_for((int64_t)N * (K / 16), 256), 256, 0, s>>>(N, K, mask, mplane, status);
  ew_plane1_pack_kernel<<<grid_for((int64_t)N * row_bytes_of(K), 256), 256, 0, s>>>(N, K, T0, plane1, status);
  ew_plane2_pack_kernel<<<(N + kEwRowWarps - 1) / kEwRowWarps, 32 * kEwRowWarps, 0, s>>>(N, K, T1, mask, rowptr,
                                                                                        plane2, status);
  return cudaGetLastError();
}

cudaError_t launch_ew_unpack(int N, int K, const uint32_t *mplane, const uint8_t *plane1, const int32_t *rowptr,
                             const uint8_t *plane2, int8_t *T0, int8_t *T1, uint8_t *mask, uint32_t *status,
                             cudaStream_t s) {
  ew_mask_unpack_kernel<<<grid_for((int64_t)N * (K / 16), 256), 256, 0, s>>>(N, K, mplane, mask);
  ew_plane1_unpack_kernel<<<grid_for((int64_t)N * row_bytes_of(K), 256), 256, 0, s>>>(N, K, plane1, T0, status);
  ew_plane2_unpack_kernel<<<(N + kEwRowWarps - 1) / kEwRowWarps, 32 * kEwRowWarps, 0, s>>>(N, K, mplane, rowptr,
                                                                                          plane2, T1, status);
  return cudaGetLastError();
}

}  // namespace tq
