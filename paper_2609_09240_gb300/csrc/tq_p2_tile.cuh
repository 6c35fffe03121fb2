// tq_p2_tile.cuh - the decode path's per-group operand layout (the general
// decode kernels' stages of 8 groups, each group's window in its stage row)
// and the second-plane tile routine shared by the second-plane kernel and
// the dependency-ordered sequence kernel: 16-entry tiles of one group of the
// group-ordered second-plane index, decoded into m16n8k16 MMAs against the
// group's activation fragment, s2 (D - C) per entry added to y2 of its row.
#pragma once

#include "tq_decode_ops.cuh"

namespace tq {
namespace mm {

constexpr int kStageG = 8;        // groups per stage
constexpr int kStageBytes = 208;  // plane-1 bytes per row per stage (13 x 16)
constexpr int kChunks = 10;       // k16 chunks per group (160 K slots)
constexpr int kCP = 5;            // chunk pairs
constexpr int kBLane = 16;        // B bytes per (chunk pair, token, lane position)
constexpr int kBTok = kCP * 4 * kBLane;  // 320 B of B per group and token
constexpr int kCSGroup = 64;             // C[8], S[8] floats per group and 8-token tile

// Window of a group: the aligned words of the stage row that cover its 26
// bytes, words wstart .. wstart + 6 with wstart = 26 GL / 4 (GL = the
// group's index in its stage); the group starts o = 26 GL % 4 bytes into
// the first.  Lane c of a row owns the window words whose stage-row index
// is c mod 4 (two words: the first at or after wstart, and the one four
// words later; bytes outside the group get zero activations).
__host__ __device__ constexpr int win_start(int GL) { return (26 * GL) / 4; }
// Stage-row word index of lane c's first window word.
__host__ __device__ constexpr int first_word(int GL, int c) {
  return win_start(GL) + ((c - win_start(GL)) % 4 + 4) % 4;
}

// The 20 A words of one row and group from the lane's two window words
// (lane-replicated table; `tag` = table base | lane * 4, so that one PRMT
// yields the entry's address): W, W' of bytes 0..3 of the first word, then
// of the second, then the four V words, each made by one PRMT of a word's
// byte pair with the fifth slot's exponent byte 0x44.
__device__ __forceinline__ void decode_words(uint32_t w0, uint32_t w1, uint32_t tag, uint32_t *a) {
  uint32_t r[8];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    r[k] = prmt(w0, tag, 0x7604u | (k << 4));
    r[4 + k] = prmt(w1, tag, 0x7604u | (k << 4));
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t w = lut_load(r[i]);
    a[2 * i] = w;
    a[2 * i + 1] = w_prime(w);
  }
  const uint32_t e44 = 0x44444444u;
  a[16] = prmt(w0, e44, 0x4140u);
  a[17] = prmt(w0, e44, 0x4342u);
  a[18] = prmt(w1, e44, 0x4140u);
  a[19] = prmt(w1, e44, 0x4342u);
}

// The MMAs of one group: rows g (aL) and g + 8 (aH), B words of this lane
// (b[2j], b[2j+1] for chunk j), one accumulation chain (measured faster than
// two or four chains summed at the end: the adds cost more than the latency).
__device__ __forceinline__ void group_mma(const uint32_t *aL, const uint32_t *aH, const uint32_t *b, float *d) {
  mma16816_z(d, aL[0], aH[0], aL[1], aH[1], b[0], b[1]);
#pragma unroll
  for (int j = 1; j < kChunks; ++j) mma16816(d, aL[2 * j], aH[2 * j], aL[2 * j + 1], aH[2 * j + 1], b[2 * j], b[2 * j + 1]);
}
// As group_mma, in two accumulator chains (even and odd chunks), so that an
// MMA waits for the result of the one two places earlier only (for kernels
// with the registers to spare).
__device__ __forceinline__ void group_mma2(const uint32_t *aL, const uint32_t *aH, const uint32_t *b, float *d) {
  float e[4];
  mma16816_z(d, aL[0], aH[0], aL[1], aH[1], b[0], b[1]);
  mma16816_z(e, aL[2], aH[2], aL[3], aH[3], b[2], b[3]);
#pragma unroll
  for (int j = 2; j < kChunks; ++j)
    mma16816((j & 1) ? e : d, aL[2 * j], aH[2 * j], aL[2 * j + 1], aH[2 * j + 1], b[2 * j], b[2 * j + 1]);
#pragma unroll
  for (int i = 0; i < 4; ++i) d[i] += e[i];
}

// The group-ordered second-plane index (tq_plane2_index): colptr [G + 1]
// padded to 128 bytes, then 32-byte slots of at most c_capacity entries.
__device__ __forceinline__ int64_t c_capacity(int K, int64_t nnz) {
  return (nnz + 15 * (int64_t)(K / kGroup) + 15) & ~(int64_t)15;
}
__device__ __forceinline__ int64_t c_slot_off(int K) { return ((int64_t)(K / kGroup + 1) * 4 + 127) & ~(int64_t)127; }

constexpr int kCDepth = 2;  // tiles in flight per warp (in registers)

// n consecutive 16-entry tiles of group g's entries (from entry e0 + 16 t0),
// as m16 tiles of one warp: lane (r, c) loads slot words 2 jw, 2 jw + 1 of
// entries r and r + 8 (its two window words, one 8-byte load per entry; a
// quad's loads cover the slot), decodes them with the lane-replicated table
// (tag = table base | lane * 4) and, after the MMAs with the group's B words
// b (b2: tokens 8..15) and corrections Cv (Cv2), takes the entries' rows
// and s2 from the quad's lanes that hold them and adds s2 (D - C) to y2.
template <bool ONE, bool TWO>
__device__ __forceinline__ void p2_tiles(const Problem &P, int MB, int GL, int64_t e0, int t0, int n,
                                         const uint32_t *b, const uint32_t *b2, float2 Cv, float2 Cv2, int lane,
                                         uint32_t tag) {
  const int g16 = lane >> 2, c = lane & 3, quad = lane & ~3;
    // lane c's window words jw and jw + 4 are slot words 2 jw, 2 jw + 1; the row is the second
    // word of the lane with jw = 3, s2 a half of the first word of jw = 0 (record at byte 2)
    // or of the second word of jw = 2 (record at byte 0)
    const int ws = win_start(GL), jw = (c - ws) & 3, odd = GL & 1;
    const int c_row = quad + ((3 + ws) & 3), c_s2 = quad + (((odd ? 0 : 2) + ws) & 3);
    const unsigned char *src = reinterpret_cast<const unsigned char *>(P.p2idx) + c_slot_off(P.K) +
                               (e0 + 16 * (int64_t)t0 + g16) * 32 + jw * 8;
    float *y2 = P.y2();
    uint2 pre[kCDepth][2];
#pragma unroll
    for (int k = 0; k < kCDepth; ++k) {
      pre[k][0] = pre[k][1] = make_uint2(0u, 0u);
      if (k < n) {
        pre[k][0] = __ldg(reinterpret_cast<const uint2 *>(src + k * 512));
        pre[k][1] = __ldg(reinterpret_cast<const uint2 *>(src + k * 512 + 256));
      }
    }
    for (int t = 0; t < n; t += kCDepth) {
#pragma unroll
      for (int k = 0; k < kCDepth; ++k) {
        if (t + k < n) {
          const uint2 r0 = pre[k][0], r1 = pre[k][1];
          if (t + k + kCDepth < n) {
            const unsigned char *p = src + (int64_t)(t + k + kCDepth) * 512;
            pre[k][0] = __ldg(reinterpret_cast<const uint2 *>(p));
            pre[k][1] = __ldg(reinterpret_cast<const uint2 *>(p + 256));
          }
          uint32_t aL[20], aH[20];
          decode_words(r0.x, r0.y, tag, aL);
          decode_words(r1.x, r1.y, tag, aH);
          float d[4], d2[4] = {0.f, 0.f, 0.f, 0.f};
          group_mma(aL, aH, b, d);
          if (TWO) group_mma(aL, aH, b2, d2);
          const uint32_t sw0 = __shfl_sync(0xffffffffu, odd ? r0.x : r0.y, c_s2);
          const uint32_t sw1 = __shfl_sync(0xffffffffu, odd ? r1.x : r1.y, c_s2);
          const float s2v0 = odd ? half_of<false>(sw0) : half_of<true>(sw0);
          const float s2v1 = odd ? half_of<false>(sw1) : half_of<true>(sw1);
          if (ONE) {
            // every column of D is token 0: the lane holding the rows adds
            if (lane == c_row) {
              const int n0 = (int)r0.y, n1 = (int)r1.y;
              if (n0 >= 0 && n0 < P.N) atomicAdd(&y2[n0], s2v0 * (d[0] - Cv.x));
              if (n1 >= 0 && n1 < P.N) atomicAdd(&y2[n1], s2v1 * (d[2] - Cv.x));
            }
          } else {
            const int rows[2] = {__shfl_sync(0xffffffffu, (int)r0.y, c_row),
                                 __shfl_sync(0xffffffffu, (int)r1.y, c_row)};
            const float s2v[2] = {s2v0, s2v1};
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int nr = rows[h];
              if (nr < 0 || nr >= P.N) continue;
#pragma unroll
              for (int ii = 0; ii < 2; ++ii) {
                const int m = 2 * c + ii;
                if (m < MB) atomicAdd(&y2[(int64_t)nr * MB + m], s2v[h] * (d[2 * h + ii] - (ii ? Cv.y : Cv.x)));
                if (TWO && 8 + m < MB)
                  atomicAdd(&y2[(int64_t)nr * MB + 8 + m], s2v[h] * (d2[2 * h + ii] - (ii ? Cv2.y : Cv2.x)));
              }
            }
          }
        }
      }
    }
}

}  // namespace mm
}  // namespace tq
