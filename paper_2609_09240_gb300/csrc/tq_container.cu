// tq_container.cu - the packed-weight container (host code) and the
// dequantizing kernel used by provenance checks.
//
// The paper's serialization lesson ("Packing: From Quantization to
// Serialization"): persist the discrete supports and their parameters, not
// a floating reconstruction; and its provenance safeguards ("Provenance
// safeguards"): zero missing or unexpected keys, measurable weight changes,
// no malformed packed tensors.  The container stores each projection's seven
// packed fields under a name, with a hash per field and an optional
// fingerprint of the fp16 source weights; reading an entry re-checks the
// hashes (and that the fields' alignment padding is zero), the shapes, rowptr
// against the salience map and every packed byte.
//
// Layout (little-endian; offsets from the start of the buffer):
//   0   char     magic[8] = "TQPACK01"
//   8   uint32   version (1)          12  uint32 count
//   16  uint64   table offset (64)    24  uint64 data offset
//   32  uint64   total bytes          40  uint64 FNV-1a 64 of the table
//   48  uint64   FNV-1a 64 of bytes 0..47                  56  uint64 0
//   64  count entries of 384 bytes:
//         char name[128] (NUL-terminated, 1..127 bytes, unique)
//         int32 N, K, group (128), flags (0); int64 nnz; uint64 source_hash
//         7 x {uint64 offset, uint64 bytes, uint64 FNV-1a 64} for plane1,
//         salience, rowptr, plane2, scale1, offset, scale2; zero to 384
//   data: the fields, each at a 16-byte aligned offset.
#include <string.h>

#include "tq_common.cuh"

namespace tq {
namespace ct {

constexpr char kMagic[8] = {'T', 'Q', 'P', 'A', 'C', 'K', '0', '1'};
constexpr uint32_t kVersion = 1;
constexpr size_t kHeader = 64, kEntry = 384, kName = 128, kFields = 7;

// FNV-1a, 64-bit (Fowler, Noll, Vo): offset basis 14695981039346656037,
// prime 1099511628211, one byte at a time.
uint64_t fnv1a(const void *p, size_t n, uint64_t h = 14695981039346656037ull) {
  const unsigned char *b = static_cast<const unsigned char *>(p);
  for (size_t i = 0; i < n; ++i) h = (h ^ b[i]) * 1099511628211ull;
  return h;
}

struct Field {
  uint64_t off, bytes, hash;
};
struct Entry {
  char name[kName];
  int32_t N, K, group, flags;
  int64_t nnz;
  uint64_t source_hash;
  Field f[kFields];
  unsigned char pad_[kEntry - kName - 32 - kFields * sizeof(Field)];
};
static_assert(sizeof(Entry) == kEntry, "entry size");
struct Header {
  char magic[8];
  uint32_t version, count;
  uint64_t table_off, data_off, total, table_hash, header_hash, zero;
};
static_assert(sizeof(Header) == kHeader, "header size");

uint64_t up16(uint64_t b) { return (b + 15) / 16 * 16; }

bool shape_ok(int64_t N, int64_t K, int64_t nnz) {
  return N >= 1 && N <= INT32_MAX && K >= kGroup && K % kGroup == 0 && K <= (1 << 20) && nnz >= 0 &&
         nnz <= N * (K / kGroup);
}

// Field sizes of a projection, in the order of the table.
void field_sizes(int64_t N, int64_t K, int64_t nnz, uint64_t out[kFields]) {
  const int64_t G = K / kGroup;
  out[0] = (uint64_t)(N * row_bytes_of((int)K));
  out[1] = (uint64_t)(N * sal_words_of((int)K) * 4);
  out[2] = (uint64_t)((N + 1) * 4);
  out[3] = (uint64_t)(nnz * kGroupBytes);
  out[4] = (uint64_t)(N * G * 2);
  out[5] = (uint64_t)(N * G * 2);
  out[6] = (uint64_t)(nnz * 2);
}

const void *field_ptr(const tq_host_weight &w, int i) {
  switch (i) {
    case 0: return w.plane1;
    case 1: return w.salience;
    case 2: return w.rowptr;
    case 3: return w.plane2;
    case 4: return w.scale1;
    case 5: return w.offset;
    default: return w.scale2;
  }
}

bool name_ok(const char *s) {
  if (!s) return false;
  const size_t n = strnlen(s, kName);
  return n >= 1 && n < kName;
}

// Packed bytes of one 26-byte group: every byte a base-3 numeral (<= 242),
// the tail byte's two pad digits 1 (byte / 27 == 4).
bool group_ok(const uint8_t *g) {
  for (int i = 0; i < kGroupBytes; ++i)
    if (g[i] > 242) return false;
  return g[kGroupBytes - 1] / 27 == 4;
}

// Structure and content of an entry whose fields lie inside the buffer.
tq_status check_content(const Entry &e, const unsigned char *base) {
  const int64_t N = e.N, K = e.K, G = K / kGroup, SW = sal_words_of((int)K), RB = row_bytes_of((int)K);
  const uint8_t *p1 = base + e.f[0].off;
  const uint32_t *sal = reinterpret_cast<const uint32_t *>(base + e.f[1].off);
  const int32_t *rp = reinterpret_cast<const int32_t *>(base + e.f[2].off);
  const uint8_t *p2 = base + e.f[3].off;
  if (rp[0] != 0) return TQ_ERR_SALIENCE;
  for (int64_t n = 0; n < N; ++n) {
    int64_t c = 0;
    for (int64_t w = 0; w < SW; ++w) {
      uint32_t v = sal[n * SW + w];
      const int64_t valid = G - 32 * w;
      if (valid < 32 && (v >> valid)) return TQ_ERR_SALIENCE;  // bits past the last group
      c += __builtin_popcount(v);
    }
    if ((int64_t)rp[n + 1] - rp[n] != c) return TQ_ERR_SALIENCE;
  }
  if (rp[N] != e.nnz) return TQ_ERR_SALIENCE;
  for (int64_t n = 0; n < N; ++n) {
    const uint8_t *row = p1 + n * RB;
    for (int64_t g = 0; g < G; ++g)
      if (!group_ok(row + g * kGroupBytes)) return TQ_ERR_BYTE;
    for (int64_t i = G * kGroupBytes; i < RB; ++i)
      if (row[i]) return TQ_ERR_BYTE;
  }
  for (int64_t j = 0; j < e.nnz; ++j)
    if (!group_ok(p2 + j * kGroupBytes)) return TQ_ERR_BYTE;
  return TQ_OK;
}

// Header and table of a buffer; on success *hdr and the table pointer.
tq_status open_buf(const void *buf, size_t bytes, Header *hdr, const Entry **table) {
  if (!buf || !hdr || !table) return TQ_ERR_NULL;
  if (bytes < kHeader) return TQ_ERR_FORMAT;
  memcpy(hdr, buf, kHeader);
  if (memcmp(hdr->magic, kMagic, 8) || hdr->version != kVersion) return TQ_ERR_FORMAT;
  if (fnv1a(buf, 48) != hdr->header_hash) return TQ_ERR_FORMAT;
  if (hdr->total != bytes || hdr->table_off != kHeader) return TQ_ERR_FORMAT;
  if (hdr->count > (bytes - kHeader) / kEntry) return TQ_ERR_FORMAT;
  const uint64_t tbytes = (uint64_t)hdr->count * kEntry;
  if (hdr->data_off < kHeader + tbytes || hdr->data_off > bytes) return TQ_ERR_FORMAT;
  const unsigned char *b = static_cast<const unsigned char *>(buf);
  if (fnv1a(b + kHeader, tbytes) != hdr->table_hash) return TQ_ERR_FORMAT;
  *table = reinterpret_cast<const Entry *>(b + kHeader);
  if ((uintptr_t)*table % alignof(Entry)) return TQ_ERR_ALIGN;
  return TQ_OK;
}

}  // namespace ct

// ------------------------------------------------------------ dequantize
// W-hat[n][k] = fp16((s1 * t1 + off) + s2 * t2) in float32 (paper "Model and
// Representation", eq. for W-hat, per group): one thread per (row, group),
// 128 outputs as 16 16-byte stores.  status may be null (the prefill path's
// trusted weights): nothing is then reported.
__global__ void __launch_bounds__(128) dequantize_kernel(int N, int K, const uint8_t *plane1, const uint32_t *sal,
                                                         const int32_t *rowptr, const uint8_t *plane2, int64_t nnz,
                                                         const __half *s1, const __half *off, const __half *s2,
                                                         __half *out, uint32_t *status) {
  const int G = K / kGroup, SW = sal_words_of(K);
  const int64_t NB = (int64_t)N * G, RB = row_bytes_of(K);
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < NB; b += (int64_t)gridDim.x * blockDim.x) {
    const int64_t n = b / G;
    const int g = (int)(b - n * G);
    const uint32_t *srow = sal + n * SW;
    int64_t rec = -1;
    if ((srow[g >> 5] >> (g & 31)) & 1u) {
      int rank = 0;
      for (int j = 0; j < (g >> 5); ++j) rank += __popc(srow[j]);
      rank += __popc(srow[g >> 5] & ((1u << (g & 31)) - 1u));
      rec = (int64_t)rowptr[n] + rank;
      if (rec < 0 || rec >= nnz) {
        if (status) atomicOr(status, TQ_DATA_BAD_ROWPTR);
        rec = -1;
      }
    }
    const float a1 = __half2float(s1[b]), o = __half2float(off[b]), a2 = rec >= 0 ? __half2float(s2[rec]) : 0.f;
    const uint8_t *g1 = plane1 + n * RB + (int64_t)kGroupBytes * g;
    const uint8_t *g2 = rec >= 0 ? plane2 + rec * kGroupBytes : nullptr;
    uint4 *dst = reinterpret_cast<uint4 *>(out + b * kGroup);
    // unrolled: every byte index and power of 3 below is a constant
#pragma unroll
    for (int c = 0; c < kGroup / 8; ++c) {
      uint32_t wd[4];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const int k = 8 * c + e, j = k / 5, q = k - 5 * (k / 5);
        const uint32_t p3 = q == 0 ? 1u : q == 1 ? 3u : q == 2 ? 9u : q == 3 ? 27u : 81u;
        const uint32_t v1 = g1[j], v2 = g2 ? g2[j] : 121u;  // 121: five digits 1 (zero trits)
        if (status && (v1 > 242 || v2 > 242)) atomicOr(status, TQ_DATA_BAD_BYTE);
        const int t1 = (int)((v1 / p3) % 3u) - 1, t2 = (int)((v2 / p3) % 3u) - 1;
        float w = __fadd_rn(t1 > 0 ? a1 : (t1 < 0 ? -a1 : 0.f), o);
        w = __fadd_rn(w, t2 > 0 ? a2 : (t2 < 0 ? -a2 : 0.f));
        const uint32_t h = __half_as_ushort(__float2half_rn(w));
        if (e & 1)
          wd[e >> 1] |= h << 16;
        else
          wd[e >> 1] = h;
      }
      dst[c] = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    }
  }
}

cudaError_t launch_dequantize(int N, int K, const tq_weight *w, uint16_t *out, uint32_t *status, cudaStream_t s) {
  const int64_t NB = (int64_t)N * (K / kGroup);
  int64_t grid = (NB + 127) / 128;
  if (grid > 152 * 16) grid = 152 * 16;
  dequantize_kernel<<<(int)grid, 128, 0, s>>>(N, K, w->plane1, w->salience, w->rowptr, w->plane2, w->nnz,
                                              reinterpret_cast<const __half *>(w->scale1),
                                              reinterpret_cast<const __half *>(w->offset),
                                              reinterpret_cast<const __half *>(w->scale2),
                                              reinterpret_cast<__half *>(out), status);
  return cudaGetLastError();
}

}  // namespace tq

using namespace tq;
using namespace tq::ct;

extern "C" {

uint64_t tq_fnv1a64(const void *data, size_t bytes) { return data || !bytes ? fnv1a(data, bytes) : 0; }

size_t tq_container_bytes(int32_t count, const tq_host_weight *w) {
  if (count < 0 || (count > 0 && !w)) return 0;
  uint64_t total = kHeader + (uint64_t)count * kEntry;
  for (int i = 0; i < count; ++i) {
    if (!shape_ok(w[i].N, w[i].K, w[i].nnz)) return 0;
    uint64_t sz[kFields];
    field_sizes(w[i].N, w[i].K, w[i].nnz, sz);
    for (size_t f = 0; f < kFields; ++f) total += up16(sz[f]);
  }
  return (size_t)total;
}

tq_status tq_container_write(int32_t count, const tq_host_weight *w, void *buf, size_t bytes) {
  if (count < 0 || !buf || (count > 0 && !w)) return TQ_ERR_NULL;
  const size_t need = tq_container_bytes(count, w);
  if (need == 0) return TQ_ERR_SHAPE;
  if (bytes < need) return TQ_ERR_SHAPE;
  if ((uintptr_t)buf % 16) return TQ_ERR_ALIGN;
  for (int i = 0; i < count; ++i) {
    if (!name_ok(w[i].name)) return TQ_ERR_KEY;
    for (int j = 0; j < i; ++j)
      if (!strncmp(w[i].name, w[j].name, kName)) return TQ_ERR_KEY;  // duplicate
    uint64_t sz[kFields];
    field_sizes(w[i].N, w[i].K, w[i].nnz, sz);
    for (size_t f = 0; f < kFields; ++f)
      if (sz[f] && !field_ptr(w[i], (int)f)) return TQ_ERR_NULL;
  }
  unsigned char *b = static_cast<unsigned char *>(buf);
  memset(b, 0, need);
  Entry *table = reinterpret_cast<Entry *>(b + kHeader);
  uint64_t at = kHeader + (uint64_t)count * kEntry;
  const uint64_t data_off = at;
  for (int i = 0; i < count; ++i) {
    Entry &e = table[i];
    strncpy(e.name, w[i].name, kName - 1);
    e.N = w[i].N, e.K = w[i].K, e.group = kGroup, e.flags = 0;
    e.nnz = w[i].nnz;
    e.source_hash = w[i].source_hash;
    uint64_t sz[kFields];
    field_sizes(w[i].N, w[i].K, w[i].nnz, sz);
    for (size_t f = 0; f < kFields; ++f) {
      e.f[f].off = at;
      e.f[f].bytes = sz[f];
      if (sz[f]) memcpy(b + at, field_ptr(w[i], (int)f), sz[f]);
      e.f[f].hash = fnv1a(b + at, sz[f]);
      at += up16(sz[f]);
    }
  }
  Header h;
  memcpy(h.magic, kMagic, 8);
  h.version = kVersion;
  h.count = (uint32_t)count;
  h.table_off = kHeader;
  h.data_off = data_off;
  h.total = need;
  h.table_hash = fnv1a(table, (size_t)count * kEntry);
  h.zero = 0;
  memcpy(b, &h, 48);
  h.header_hash = fnv1a(b, 48);
  memcpy(b, &h, kHeader);
  return TQ_OK;
}

tq_status tq_container_count(const void *buf, size_t bytes, int32_t *count) {
  Header h;
  const Entry *t;
  if (!count) return TQ_ERR_NULL;
  if (tq_status s = open_buf(buf, bytes, &h, &t)) return s;
  *count = (int32_t)h.count;
  return TQ_OK;
}

tq_status tq_container_find(const void *buf, size_t bytes, const char *name, int32_t *index) {
  Header h;
  const Entry *t;
  if (!name || !index) return TQ_ERR_NULL;
  if (tq_status s = open_buf(buf, bytes, &h, &t)) return s;
  for (uint32_t i = 0; i < h.count; ++i)
    if (!strncmp(t[i].name, name, kName)) {
      *index = (int32_t)i;
      return TQ_OK;
    }
  return TQ_ERR_KEY;
}

tq_status tq_container_entry(const void *buf, size_t bytes, int32_t index, tq_host_weight *out) {
  Header h;
  const Entry *t;
  if (!out) return TQ_ERR_NULL;
  if (tq_status s = open_buf(buf, bytes, &h, &t)) return s;
  if (index < 0 || (uint32_t)index >= h.count) return TQ_ERR_KEY;
  const Entry &e = t[index];
  if (strnlen(e.name, kName) == 0 || strnlen(e.name, kName) == kName) return TQ_ERR_FORMAT;
  if (e.group != kGroup || e.flags != 0 || !shape_ok(e.N, e.K, e.nnz)) return TQ_ERR_FORMAT;
  uint64_t sz[kFields];
  field_sizes(e.N, e.K, e.nnz, sz);
  const unsigned char *b = static_cast<const unsigned char *>(buf);
  for (size_t f = 0; f < kFields; ++f) {
    if (e.f[f].bytes != sz[f] || e.f[f].off % 16 || e.f[f].off < h.data_off || e.f[f].off > bytes ||
        sz[f] > bytes - e.f[f].off)
      return TQ_ERR_FORMAT;
    if (fnv1a(b + e.f[f].off, sz[f]) != e.f[f].hash) return TQ_ERR_FORMAT;
    // the field's alignment padding (up to 15 bytes) is zero, so that no
    // byte of the data region escapes a check
    const uint64_t end = e.f[f].off + sz[f], pend = up16(end) < bytes ? up16(end) : bytes;
    for (uint64_t i = end; i < pend; ++i)
      if (b[i]) return TQ_ERR_FORMAT;
  }
  if (tq_status s = check_content(e, b)) return s;
  out->name = e.name;
  out->N = e.N, out->K = e.K, out->nnz = e.nnz;
  out->source_hash = e.source_hash;
  out->plane1 = b + e.f[0].off;
  out->salience = reinterpret_cast<const uint32_t *>(b + e.f[1].off);
  out->rowptr = reinterpret_cast<const int32_t *>(b + e.f[2].off);
  out->plane2 = e.nnz ? b + e.f[3].off : nullptr;
  out->scale1 = reinterpret_cast<const uint16_t *>(b + e.f[4].off);
  out->offset = reinterpret_cast<const uint16_t *>(b + e.f[5].off);
  out->scale2 = e.nnz ? reinterpret_cast<const uint16_t *>(b + e.f[6].off) : nullptr;
  return TQ_OK;
}

tq_status tq_container_check_keys(const void *buf, size_t bytes, int32_t n_expected, const char *const *expected,
                                  int32_t *missing, int32_t *unexpected) {
  Header h;
  const Entry *t;
  if (!missing || !unexpected || (n_expected > 0 && !expected) || n_expected < 0) return TQ_ERR_NULL;
  if (tq_status s = open_buf(buf, bytes, &h, &t)) return s;
  int32_t miss = 0, extra = 0;
  for (int32_t i = 0; i < n_expected; ++i) {
    bool found = false;
    for (uint32_t j = 0; j < h.count && !found; ++j) found = expected[i] && !strncmp(t[j].name, expected[i], kName);
    miss += !found;
  }
  for (uint32_t j = 0; j < h.count; ++j) {
    bool found = false;
    for (int32_t i = 0; i < n_expected && !found; ++i) found = expected[i] && !strncmp(t[j].name, expected[i], kName);
    extra += !found;
  }
  *missing = miss, *unexpected = extra;
  return miss || extra ? TQ_ERR_KEY : TQ_OK;
}

}  // extern "C"
