/*
 * tq.h - C ABI of the packed ternary (W1.58A16) linear layer.
 *
 * What is computed (paper: "Model and Representation", eq. for W-hat):
 * every targeted projection W (N rows = outputs, K columns = inputs) is a
 * ternary reconstruction offset + alpha0*T0 + alpha1*T1, the second plane
 * only on salience-selected parts.  This library uses the per-group reading:
 * with g = floor(k / 128),
 *
 *     W[n][k] = s1[n][g] * T1[n][k] + off[n][g] + sal[n][g] * s2[n][g] * T2[n][k]
 *
 * T1, T2 in {-1, 0, +1}; s1, off, s2 fp16; sal a 1-bit salience map.
 * Activations x and outputs y stay fp16 (weight-only A16, paper
 * "Model and Representation").  The layer computes y[m][n] = sum_k x[m][k] W[n][k]
 * with fp32 accumulation, directly from the packed bytes (paper
 * "Direct Packed Execution").
 *
 * Packed ("lattice-aware") format (paper "Packing: From Quantization to
 * Serialization"; the byte layout itself is not printed there, this is the
 * library's definition):
 *   - one byte holds five trits as a base-3 numeral, digit d = t + 1, first
 *     trit least significant: byte = sum_{i<5} d_i * 3^i  (0..242; 243..255
 *     are invalid).  3^5 = 243 <= 256 gives 1.6 bits per trit against the
 *     log2(3) = 1.585-bit bound of the paper's eq. b_T.
 *   - a 128-trit group is 26 bytes: bytes 0..24 hold trits 5j..5j+4, byte 25
 *     holds trits 125..127 in digits 0..2 and pad digits 3,4 = 1 (t = 0).
 *   - plane 1 rows are TQ_GROUP_BYTES * G bytes padded with 0x00 to a
 *     multiple of 16 (tq_row_bytes).
 *   - plane 2 stores only the salient groups, 26 bytes each, in (n, g) order;
 *     rowptr[n] is the number of salient groups in rows 0..n-1.
 *
 * Conventions (all entry points):
 *   - every pointer argument except the tq_weight / tq_problem structs
 *     themselves refers to DEVICE memory owned by the caller;
 *   - every call is asynchronous on `stream` (a cudaStream_t passed as void*,
 *     NULL = legacy default stream); the library never allocates device
 *     memory, never synchronizes and never throws across the ABI;
 *   - argument errors (null pointers, shapes, alignment) are returned
 *     synchronously and nothing is launched;
 *   - data errors found by the codec kernels are OR-ed into the caller's
 *     device word *d_status (TQ_DATA_* bits); the caller zeroes it before the
 *     call and reads it after synchronizing;
 *   - TQ_ERR_CUDA means a launch failed (cudaGetLastError after launch).
 */
#ifndef TQ_H_
#define TQ_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define TQ_API __attribute__((visibility("default")))
#else
#define TQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define TQ_GROUP 128        /* trits per group along K                       */
#define TQ_GROUP_BYTES 26   /* bytes per packed 128-trit group                */
#define TQ_TRITS_PER_BYTE 5 /* 3^5 = 243 <= 256                               */
#define TQ_MAX_SKINNY_M 16  /* M <= this runs the decode (GEMV / skinny) path,
                               larger M the prefill tile path               */

typedef enum {
  TQ_OK = 0,
  TQ_ERR_NULL = -1,     /* a required pointer is NULL                     */
  TQ_ERR_SHAPE = -2,    /* M, N or K out of range, K % 128 != 0, group != 128 */
  TQ_ERR_ALIGN = -3,    /* a pointer is not 16-byte aligned               */
  TQ_ERR_CODE = -4,     /* reserved: invalid trit code (reported in d_status) */
  TQ_ERR_BYTE = -5,     /* reserved: invalid packed byte (d_status)       */
  TQ_ERR_SALIENCE = -6, /* descriptor nnz / salience inconsistent          */
  TQ_ERR_CUDA = -7,     /* a CUDA launch or query failed                  */
  TQ_ERR_TIMEOUT = -8,  /* a bounded device wait ran out                  */
  TQ_ERR_SCRATCH = -9,  /* tq_linear_static: the call needs more scratch than
                           TQ_STATIC_SCRATCH_BYTES                         */
  TQ_ERR_FORMAT = -10,  /* container: bad magic, version, size or hash     */
  TQ_ERR_KEY = -11      /* container: missing, unexpected, duplicate or
                           malformed name                                   */
} tq_status;

/* Bits OR-ed into *d_status by the codec kernels. */
#define TQ_DATA_BAD_CODE 1u     /* a trit code not in {-1, 0, +1}                */
#define TQ_DATA_T2_OUTSIDE 2u   /* T2 != 0 in a group whose salience bit is 0    */
#define TQ_DATA_BAD_BYTE 4u     /* a packed byte > 242                           */
#define TQ_DATA_BAD_PAD 8u      /* a nonzero pad digit (tail byte) or pad byte   */
#define TQ_DATA_BAD_ROWPTR 16u  /* rowptr disagrees with the salience map        */
#define TQ_DATA_BAD_WEIGHT 32u  /* tq_ternarize: an input weight is inf or NaN    */

/* A packed projection.  All pointers: device memory owned by the caller. */
typedef struct {
  int32_t N, K;             /* rows (outputs), columns (inputs); K % 128 == 0  */
  int32_t group;            /* must be TQ_GROUP                                */
  const uint8_t *plane1;    /* [N][tq_row_bytes(K)], 16-byte aligned           */
  const uint32_t *salience; /* [N][tq_sal_words(K)], bit g%32 of word g/32     */
  const int32_t *rowptr;    /* [N+1], exclusive prefix count of salient groups */
  const uint8_t *plane2;    /* [nnz][26], 16-byte aligned; NULL when nnz == 0  */
  const uint16_t *scale1;   /* fp16 bits [N][G]                                */
  const uint16_t *offset;   /* fp16 bits [N][G]                                */
  const uint16_t *scale2;   /* fp16 bits [nnz]; may be NULL when nnz == 0      */
  int64_t nnz;              /* number of salient groups = rowptr[N]            */
  const int32_t *p2index;   /* optional: tq_plane2_index of this weight, or
                               NULL (the decode path then groups the second
                               plane itself on every call)                     */
} tq_weight;

/* Bytes of one packed plane-1 row: roundup(26 * K / 128, 16).  0 if K is not
 * a positive multiple of 128. */
TQ_API size_t tq_row_bytes(int32_t K);
/* 32-bit words of one salience row: ceil((K / 128) / 32). */
TQ_API size_t tq_sal_words(int32_t K);

/* rowptr[n] = number of set salience bits in rows 0..n-1, for n = 0..N
 * (so rowptr[N] = nnz).  sal: [N][tq_sal_words(K)].  Bits at g >= K/128 in
 * the last word of a row must be 0, else TQ_DATA_BAD_PAD is OR-ed into
 * *d_status and those bits are not counted. */
TQ_API tq_status tq_salience_rowptr(int32_t N, int32_t K, const uint32_t *sal, int32_t *rowptr,
                             uint32_t *d_status, void *stream);

/* Second-plane index (no counterpart in the paper; a layout aid for the
 * decode path, M <= 8): plane 2 re-laid out group by group.  The salient
 * (row, group) pairs of each group g, in increasing row order, padded with
 * empty entries to a multiple of 16, each entry a 32-byte slot that holds
 * the pair's plane-2 record, its s2 and its row.  It depends on the weight
 * alone, so it is built once; with it tq_linear runs the second plane one
 * group at a time, 16 entries per tensor-core tile, and reads this copy
 * instead of plane 2 and s2.
 * Layout, with C = tq_plane2_index_capacity(K, nnz) (a multiple of 16):
 *   int32 colptr[G + 1] at byte 0: group g's entries are colptr[g] ..
 *     colptr[g+1] - 1, multiples of 16 (colptr[G] <= C);
 *   slot[C][32] at byte tq_plane2_index_slot_offset(K) (128-byte aligned).
 * A slot's 32 bytes, in logical order L[0..31], o = 2 * ((g % 8) & 1),
 * the decode kernels' window alignment of group g):
 *   L[o .. o+25]  the pair's 26-byte plane-2 record,
 *   L[o ? 0 : 26] the pair's s2 (fp16, two bytes),
 *   L[28 .. 31]   the row n (int32; -1 for an empty entry, whose other bytes
 *                 are zero),
 * stored as 4-byte words in the order of logical words 0, 4, 1, 5, 2, 6, 3,
 * 7 (so logical words i and i + 4, which one lane decodes, are adjacent).
 * Entries from colptr[G] to C are empty too.
 *   index: device, tq_plane2_index_bytes(N, K, nnz) bytes, 16-byte aligned.
 *   sal, rowptr, plane2, scale2 as for tq_linear (rowptr[N] == nnz; bits at
 *   g >= K/128 are ignored; a pair whose record index falls outside
 *   [0, nnz) becomes an empty entry).  Asynchronous on stream. */
TQ_API size_t tq_plane2_index_capacity(int32_t K, int64_t nnz);
TQ_API size_t tq_plane2_index_slot_offset(int32_t K);
TQ_API size_t tq_plane2_index_bytes(int32_t N, int32_t K, int64_t nnz);
TQ_API tq_status tq_plane2_index(int32_t N, int32_t K, const uint32_t *sal, const int32_t *rowptr, int64_t nnz,
                                 const uint8_t *plane2, const uint16_t *scale2, int32_t *index, void *stream);

/* Pack int8 trit codes into the lattice format (paper "Packing").
 *   T1: int8 [N][K] in {-1,0,+1};  T2: int8 [N][K], nonzero only where the
 *   group is salient (NULL means "no second plane": sal must then be all 0);
 *   sal: [N][tq_sal_words(K)];  rowptr: [N+1] as from tq_salience_rowptr;
 *   plane1: out [N][tq_row_bytes(K)] (pad bytes written as 0);
 *   plane2: out [rowptr[N]][26] (NULL iff T2 is NULL).
 * Invalid codes set TQ_DATA_BAD_CODE (the digit is clamped into the byte),
 * T2 != 0 outside salience sets TQ_DATA_T2_OUTSIDE, a rowptr that disagrees
 * with sal sets TQ_DATA_BAD_ROWPTR. */
TQ_API tq_status tq_pack(int32_t N, int32_t K, const int8_t *T1, const int8_t *T2, const uint32_t *sal,
                  const int32_t *rowptr, uint8_t *plane1, uint8_t *plane2, uint32_t *d_status,
                  void *stream);

/* Inverse of tq_pack: T1 [N][K] and (unless NULL) T2 [N][K] int8, T2 = 0 in
 * non-salient groups.  Validates every byte: > 242 -> TQ_DATA_BAD_BYTE (the
 * trits are written as 0), tail pad digit != 1 or row pad byte != 0 ->
 * TQ_DATA_BAD_PAD, rowptr disagreeing with sal -> TQ_DATA_BAD_ROWPTR. */
TQ_API tq_status tq_unpack(int32_t N, int32_t K, const uint8_t *plane1, const uint8_t *plane2,
                    const uint32_t *sal, const int32_t *rowptr, int8_t *T1, int8_t *T2,
                    uint32_t *d_status, void *stream);

/* E2M-ATQ ternarization (paper "Conversion Pipeline", subsection "E2M-ATQ")
 * of a dense fp16 projection straight into the packed format above.
 * Per block of one row and one group of 128 columns, with w its weights:
 *   mu = mean(w), c = w - mu, Delta0 = 0.75 * mean(|c|),
 *   T0 = +1 where c > Delta0, -1 where c < -Delta0, else 0,
 *   alpha0 = sum(c * T0) / sum(T0^2) (0 for an empty support),
 *   residual r = c - alpha0 * T0, energy E = sum(r^2).
 * The nnz blocks of largest E (ties: lower block id n * G + g) are salient:
 * their residual gets a second support T1 by the same rule (threshold
 * 0.75 * mean(|r|)) and alpha1 = sum(r * T1) / sum(T1^2).  Then `sweeps`
 * alternating refinements with the supports fixed: mu = mean(w - alpha0 T0
 * - alpha1 T1), alpha0 = least squares of w - mu - alpha1 T1 on T0, alpha1 =
 * least squares of w - mu - alpha0 T0 on T1.  Outputs: plane1 = T0, plane2
 * = T1 of the salient blocks, offset = fp16(mu), scale1 = fp16(alpha0),
 * scale2 = fp16(alpha1) (round to nearest even), sal and rowptr; together a
 * complete tq_weight with nnz salient groups.
 * Arithmetic of every decision (supports, thresholds, salience): IEEE
 * float32, no fused multiply-add, every sum over a block in index order
 * from +0, means as the sum times 1/128; so the planes and the salience set
 * are reproducible bit for bit by any implementation that does the same.
 * The refinement runs the same coordinate updates on each block's moments
 * (sum w, sum w T0, sum w T1 and the trit counts): its fp16 outputs are
 * within one ulp of sweeps computed as passes over the weights.
 *   W: fp16 [N][K], 16-byte aligned;  nnz: 0 <= nnz <= N * K / 128;
 *   sweeps: 0 .. 64;
 *   plane1: out [N][tq_row_bytes(K)], 16-byte aligned (pad bytes written 0);
 *   sal: out [N][tq_sal_words(K)];  rowptr: out [N + 1];
 *   plane2: out [nnz][26], 16-byte aligned;  scale2: out fp16 [nnz]
 *     (both may be NULL iff nnz == 0);
 *   scale1, offset: out fp16 [N][K / 128];
 *   workspace: tq_ternarize_workspace_bytes(N, K) bytes, 16-byte aligned
 *     (nothing in it needs to start at zero);
 *   d_status: TQ_DATA_BAD_WEIGHT for an inf or NaN weight (the outputs are
 *     then unspecified but written in bounds).
 * Asynchronous on stream: at most nine kernel launches and one memset. */
TQ_API size_t tq_ternarize_workspace_bytes(int32_t N, int32_t K);
TQ_API tq_status tq_ternarize(int32_t N, int32_t K, const uint16_t *W, int64_t nnz, int32_t sweeps,
                              uint8_t *plane1, uint32_t *sal, int32_t *rowptr, uint8_t *plane2,
                              uint16_t *scale1, uint16_t *offset, uint16_t *scale2, void *workspace,
                              size_t workspace_bytes, uint32_t *d_status, void *stream);

/* W-hat of a packed weight as dense fp16 [N][K] (16-byte aligned):
 * fp16((s1 * t1 + off) + s2 * t2), the sums in float32, rounded to nearest
 * even (paper "Model and Representation", eq. for W-hat, per group).  For
 * provenance checks against the source weights and for export.  Invalid
 * bytes set TQ_DATA_BAD_BYTE, a record index outside [0, nnz)
 * TQ_DATA_BAD_ROWPTR (that group's second plane is then left out).
 * Asynchronous on stream. */
TQ_API tq_status tq_dequantize(int32_t N, int32_t K, const tq_weight *w, uint16_t *out, uint32_t *d_status,
                               void *stream);

/* ---- Packed-weight container (HOST memory; no device access, synchronous).
 * Serialization of packed projections under names (paper "Packing: From
 * Quantization to Serialization": the discrete supports and their
 * parameters are what is stored), with the checks of its "Provenance
 * safeguards": every key present and no unexpected one, every field's hash,
 * the shapes, rowptr against the salience map and every packed byte
 * (base-3 numerals <= 242, tail pad digits 1, row pad bytes 0).
 * Layout: a 64-byte header ("TQPACK01", version, count, offsets, total
 * size, FNV-1a 64 hashes of the table and of the header), a 384-byte table
 * entry per projection (name, N, K, group, nnz, the source fingerprint, and
 * offset / size / FNV-1a 64 of each field), then the fields at 16-byte
 * aligned offsets in the order plane1, salience, rowptr, plane2, scale1,
 * offset, scale2, each in the tq_weight layout. */
typedef struct {
  const char *name;          /* 1..127 bytes, NUL-terminated, unique        */
  int32_t N, K;
  int64_t nnz;
  const uint8_t *plane1;     /* the tq_weight fields, in HOST memory        */
  const uint32_t *salience;
  const int32_t *rowptr;
  const uint8_t *plane2;     /* NULL allowed when nnz == 0                  */
  const uint16_t *scale1;
  const uint16_t *offset;
  const uint16_t *scale2;    /* NULL allowed when nnz == 0                  */
  uint64_t source_hash;      /* e.g. tq_fnv1a64 of the source fp16 weights; 0 = none */
} tq_host_weight;

/* FNV-1a 64 (Fowler-Noll-Vo) of a host byte range. */
TQ_API uint64_t tq_fnv1a64(const void *data, size_t bytes);
/* Bytes of a container holding these projections; 0 for an invalid shape. */
TQ_API size_t tq_container_bytes(int32_t count, const tq_host_weight *w);
/* Writes the container into buf (16-byte aligned, >= tq_container_bytes).
 * Fields are copied; hashes computed.  TQ_ERR_KEY: a bad or duplicate name. */
TQ_API tq_status tq_container_write(int32_t count, const tq_host_weight *w, void *buf, size_t bytes);
/* Number of entries, after checking the header and table hashes.
 * `bytes` must be the container's exact size. */
TQ_API tq_status tq_container_count(const void *buf, size_t bytes, int32_t *count);
/* Index of the entry named `name` (TQ_ERR_KEY if absent). */
TQ_API tq_status tq_container_find(const void *buf, size_t bytes, const char *name, int32_t *index);
/* Entry `index`, fully checked (hashes TQ_ERR_FORMAT, rowptr / salience
 * TQ_ERR_SALIENCE, packed bytes TQ_ERR_BYTE); on success *out points into
 * buf (name included).  buf must be 8-byte aligned. */
TQ_API tq_status tq_container_entry(const void *buf, size_t bytes, int32_t index, tq_host_weight *out);
/* Keys: *missing = expected names absent from the container, *unexpected =
 * entries whose name is not expected; TQ_ERR_KEY unless both are 0. */
TQ_API tq_status tq_container_check_keys(const void *buf, size_t bytes, int32_t n_expected,
                                         const char *const *expected, int32_t *missing, int32_t *unexpected);

/* Device workspace of the decode path (M <= TQ_MAX_SKINNY_M): the
 * activations of every call are first rearranged into the tensor-core
 * operand order of the packed weights (with the per-group correction terms),
 * and the second plane's fp32 partial sums of every row are staged there
 * before the first plane is streamed, next to the 128-byte descriptors
 * through which the first plane, s1 and off are copied into shared memory
 * (written by the same call).  A call with 8 < M <= 16 runs tokens 0..7 and
 * then the rest over the same workspace, sized for 8 tokens.  The caller provides this
 * scratch memory (the library never allocates).  Bytes needed for one
 * projection of N rows, K inputs and M tokens; a call with M > 16 (the
 * prefill tile path) uses none and the function returns 256 for it; 0 if M,
 * N or K is invalid. */
TQ_API size_t tq_workspace_bytes(int32_t M, int32_t N, int32_t K);

/* y = x W^T for one packed projection (paper "Direct Packed Execution").
 *   x: fp16 [M][K] row-major, 16-byte aligned; y: fp16 [M][N] (rounded to
 *   nearest even from the fp32 accumulator).  M >= 1.  M <= 16 runs the
 *   decode path straight from the packed bytes; M > 16 runs the prefill
 *   path, which dequantizes each 256-row (or 128-row) x 128-column weight
 *   tile to fp16 (w = s1 t1 + off + s2 t2, rounded once) and multiplies it
 *   by 256-token activation tiles on the tensor cores.
 *   workspace: device scratch of at least tq_workspace_bytes(M, N, K) bytes,
 *   256-byte aligned; its contents are overwritten; calls that share a
 *   workspace must not overlap in time.
 * The packed bytes are trusted (produced by tq_pack): no per-byte
 * validation on this path.
 * Host threads: the linear entry points (tq_linear, tq_linear_f32out,
 * tq_linear_batched, tq_linear_static) keep their launch parameters per
 * host thread, so several threads may call them at once (each with its own
 * workspace; tq_linear_static's one scratch array is the exception). */
TQ_API tq_status tq_linear(int32_t M, int32_t N, int32_t K, const tq_weight *w, const uint16_t *x,
                           uint16_t *y, void *workspace, size_t workspace_bytes, void *stream);

/* As tq_linear but y is fp32 [M][N] (the accumulator before rounding). */
TQ_API tq_status tq_linear_f32out(int32_t M, int32_t N, int32_t K, const tq_weight *w,
                                  const uint16_t *x, float *y, void *workspace, size_t workspace_bytes,
                                  void *stream);

/* Many independent projections in one launch (one decode step of a model:
 * every targeted projection of every layer; or one layer's projections at
 * a prefill's M).  Each problem has its own weight, input and output; all
 * share M.  `problems` is a HOST array read during the call (validated,
 * then passed to the kernel by value in its launch parameters, at most
 * TQ_MAX_BATCH entries).  M <= TQ_MAX_SKINNY_M runs the decode path, M >
 * TQ_MAX_SKINNY_M the prefill tile path with every problem's output tiles
 * in one launch per 16 problems (the longest K first), which fills the
 * SMs' waves better than one launch per projection; it needs no workspace
 * (tq_batched_workspace_bytes returns 256). */
#define TQ_MAX_BATCH 256
typedef struct {
  tq_weight w;
  const uint16_t *x; /* fp16 [M][w.K] */
  uint16_t *y;       /* fp16 [M][w.N] */
} tq_problem;

/* Workspace bytes of a batched call (sum over problems, 256-byte padded). */
TQ_API size_t tq_batched_workspace_bytes(int32_t M, int32_t count, const tq_problem *problems);

TQ_API tq_status tq_linear_batched(int32_t M, int32_t count, const tq_problem *problems, void *workspace,
                                   size_t workspace_bytes, void *stream);

/* Dependency-ordered sequence (paper "Direct Packed Execution": the packed
 * runtime runs one token's layers in order).  Like tq_linear_batched, but
 * problem i + 1 starts only once problem i has completed on every SM, as
 * the layers of a model need: e.g. per layer q/k/v (rows concatenated into
 * one weight), o, gate/up (concatenated), down.  The attention, norms and
 * activation between them are outside this library: every problem's x is
 * an input of the call.  One persistent launch after the activation prep;
 * between problems a grid-wide barrier whose wait is bounded by the wall-
 * time limit (a wait that runs out sets the timeout bit of the device
 * status word, see tq_get_device_status, and the kernel returns).  The
 * fp32 sums of each problem's rows are added in a varying order, so
 * results may differ in the last bits from run to run.
 *   M must be 1 (TQ_ERR_SHAPE otherwise); count <= TQ_MAX_BATCH; every
 *   weight with a second plane must carry its index (p2index, else
 *   TQ_ERR_NULL); the workspace is sized by tq_batched_workspace_bytes;
 *   a sequence's problems may have at most five distinct (N, K) shapes
 *   (TQ_ERR_CUDA otherwise). */
TQ_API tq_status tq_linear_sequence(int32_t M, int32_t count, const tq_problem *problems, void *workspace,
                                    size_t workspace_bytes, void *stream);

/* Failure-path self-test of tq_linear_sequence (no fault involved): runs
 * its kernel on the given problems with every problem barrier expecting one
 * more participant than exists, so that the first barrier's bounded wait
 * runs out after the wall-time limit (about 2 s); the device status word
 * then has its timeout bit set and the launch ends normally.  Arguments as
 * tq_linear_sequence with M = 1. */
TQ_API tq_status tq_sequence_selftest(int32_t count, const tq_problem *problems, void *workspace,
                                      size_t workspace_bytes, void *stream);

/* ---------------------------------------------------------------------
 * Element-wise four-mask representation (paper "Model and Representation":
 * four disjoint salience masks, num_mask = 4, orders = [2, 2, 1, 1], and
 * W-hat = (mu + alpha0 T0 + alpha1 T1) (.) M).  Every element (n, k) has a
 * mask id m in 0..3; its weight is
 *   mu[n][m] + alpha0[n][m] T0[n][k] + alpha1[n][m] T1[n][k],
 * with alpha1 and T1 only for the order-2 masks 0 and 1 (T1 = 0 on the
 * elements of masks 2 and 3).  The paper gives no storage layout; this
 * library's:
 *   mask: uint32 [N][K/16], element k's id in bits 2 (k mod 16) and
 *         2 (k mod 16) + 1 of word k / 16;
 *   plane1: T0 of every element in tq_weight's plane-1 layout;
 *   plane2: per row, the T1 trits of the row's order-2 elements in increasing
 *         k, five per byte (base 3 as plane 1, the row's last byte padded
 *         with digit 1), row n's bytes from byte p2rowptr[n];
 *   mu, alpha0: fp16 [N][4]; alpha1: fp16 [N][2].
 * All device memory owned by the caller; K a multiple of 128. */
typedef struct {
  int32_t N, K;
  const uint32_t *mask;
  const uint8_t *plane1;    /* 16-byte aligned */
  const int32_t *p2rowptr;  /* [N + 1] */
  const uint8_t *plane2;    /* [p2rowptr[N]] bytes; may be NULL when that is 0 */
  const uint16_t *mu;
  const uint16_t *alpha0;
  const uint16_t *alpha1;
  /* Optional correction index (tq_ew_index_offsets / tq_ew_index_fill), or
   * both NULL: with it the linear reads the index instead of the mask plane
   * and planes for the elements of masks 0..2. */
  const int32_t *idx_off;
  const uint16_t *idx;
} tq_ew_weight;

/* p2rowptr[N + 1] from the mask ids (uint8 [N][K], 0..3): bytes per row =
 * ceil(order-2 elements / 5), prefix-summed.  Ids above 3 set
 * TQ_DATA_BAD_CODE in *d_status.  The caller reads p2rowptr[N] to size
 * plane 2. */
TQ_API tq_status tq_ew_rowptr(int32_t N, int32_t K, const uint8_t *mask_ids, int32_t *p2rowptr, uint32_t *d_status,
                              void *stream);
/* int8 T0, T1 [N][K] and mask ids -> mask plane, plane 1, plane 2 (with
 * p2rowptr from tq_ew_rowptr).  Data errors in *d_status: TQ_DATA_BAD_CODE
 * (a code outside {-1, 0, 1} or an id above 3), TQ_DATA_T2_OUTSIDE (T1
 * nonzero on an order-1 element), TQ_DATA_BAD_ROWPTR (p2rowptr does not
 * match the mask ids). */
TQ_API tq_status tq_ew_pack(int32_t N, int32_t K, const int8_t *T0, const int8_t *T1, const uint8_t *mask_ids,
                            const int32_t *p2rowptr, uint32_t *mask, uint8_t *plane1, uint8_t *plane2,
                            uint32_t *d_status, void *stream);
/* The inverse: T0, T1 (int8 [N][K]) and mask ids (uint8 [N][K]); bytes
 * above 242, pad digits other than 1 and pad bytes other than 0 are
 * reported as in tq_unpack. */
TQ_API tq_status tq_ew_unpack(int32_t N, int32_t K, const uint32_t *mask, const uint8_t *plane1,
                              const int32_t *p2rowptr, const uint8_t *plane2, int8_t *T0, int8_t *T1,
                              uint8_t *mask_ids, uint32_t *d_status, void *stream);
/* Correction index (this library's, no counterpart in the paper; derived
 * from a packed weight once, like tq_plane2_index for the group format):
 * for every row n and block b of 2048 elements along K, the elements of
 * masks 0..2 in increasing k as uint16 entries
 *   (k mod 2048) | code << 11,  code = 9 q + 3 (T0 + 1) + (T1 + 1),
 * from entry idx_off[n nb + b] on (nb = ceil(K / 2048); idx_off[N nb] =
 * all entries, 2 bytes each).  tq_ew_index_offsets writes idx_off
 * (int32 [N nb + 1]) from the mask plane; the caller reads idx_off[N nb] to
 * size the entries; tq_ew_index_fill writes them from the weight's mask
 * plane, plane 1, p2rowptr and plane 2 (w's index fields are ignored).
 * Rows whose offsets or p2rowptr do not match the mask plane are skipped
 * and reported as TQ_DATA_BAD_ROWPTR, bytes above 242 as TQ_DATA_BAD_BYTE
 * (in *d_status).  N K must stay below 2^31. */
TQ_API tq_status tq_ew_index_offsets(int32_t N, int32_t K, const uint32_t *mask, int32_t *idx_off, void *stream);
TQ_API tq_status tq_ew_index_fill(int32_t N, int32_t K, const tq_ew_weight *w, const int32_t *idx_off, uint16_t *idx,
                                  uint32_t *d_status, void *stream);
/* Workspace of tq_ew_linear (per-call views of alpha0 / mu of mask 3 for
 * the plane-1 pass, its fp32 result and the decode path's workspace). */
TQ_API size_t tq_ew_workspace_bytes(int32_t M, int32_t N, int32_t K);
/* y = x W-hat^T for the element-wise form, x fp16 [M][K] (16-byte aligned),
 * y fp16 [M][N] (tq_ew_linear_f32out: fp32).  Plane 1 with mask 3's
 * parameters runs through tq_linear's kernels; a second kernel adds, per
 * row, the elements of masks 0..2 and writes y.  The fp32 sums are added in
 * a fixed order. */
TQ_API tq_status tq_ew_linear(int32_t M, int32_t N, int32_t K, const tq_ew_weight *w, const uint16_t *x, uint16_t *y,
                              void *workspace, size_t workspace_bytes, void *stream);
TQ_API tq_status tq_ew_linear_f32out(int32_t M, int32_t N, int32_t K, const tq_ew_weight *w, const uint16_t *x,
                                     float *y, void *workspace, size_t workspace_bytes, void *stream);

/* Many independent element-wise projections sharing M (<= TQ_MAX_SKINNY_M)
 * in three launches plus the decode path's (one decode step's projections
 * of a layer, say): the views of every problem in one launch, every
 * problem's plane-1 pass in one tq_linear_batched-style call, the
 * corrections of every problem in one launch per 8 tokens.  `problems` is a
 * HOST array read during the call (at most TQ_MAX_BATCH entries); y is fp16
 * [M][w.N].  Per-problem results equal tq_ew_linear's up to the order of
 * fp32 additions in split tiles. */
typedef struct {
  tq_ew_weight w;
  const uint16_t *x; /* fp16 [M][w.K], 16-byte aligned */
  uint16_t *y;       /* fp16 [M][w.N] */
} tq_ew_problem;
/* Workspace bytes of a batched element-wise call (0 for invalid arguments). */
TQ_API size_t tq_ew_batched_workspace_bytes(int32_t M, int32_t count, const tq_ew_problem *problems);
TQ_API tq_status tq_ew_linear_batched(int32_t M, int32_t count, const tq_ew_problem *problems, void *workspace,
                                      size_t workspace_bytes, void *stream);

/* ---------------------------------------------------------------------
 * Allocation-free variant (no counterpart in the paper; an integration aid).
 *
 * tq_linear_static is tq_linear with its workspace taken from a scratch
 * array that the library itself holds in device memory (a file-scope
 * __device__ array of TQ_STATIC_SCRATCH_BYTES, reserved when the module
 * loads), so the caller passes no workspace and nothing is allocated at
 * call time.  It is for callers that cannot allocate or own device memory:
 * code inside a region where allocation is not allowed (a stream being
 * captured, where cudaMalloc / cudaFree would invalidate the capture, or a
 * serving loop that forbids allocator calls and their implicit
 * synchronization), and hosts that have no allocator to hand (plain C
 * callers of the library).
 *
 *   - Limit: the call's need, tq_workspace_bytes(M, N, K), must not exceed
 *     TQ_STATIC_SCRATCH_BYTES (1 MiB: every Qwen3-8B projection up to
 *     M = 16); otherwise TQ_ERR_SCRATCH is returned before anything runs.
 *   - Set-up: the first call on a device looks up the scratch array's device
 *     address once (cudaGetSymbolAddress) and caches it for that device; make
 *     that first call before any stream capture on the device.  A failed
 *     lookup returns TQ_ERR_CUDA.  The cached address belongs to the
 *     device's context at the time of the lookup: after cudaDeviceReset (or
 *     any other teardown of that context) it is stale, and this entry point
 *     must not be called on that device again in the same process.
 *   - Nothing in the scratch has to start at zero: every call writes all of
 *     the scratch it reads before reading it.
 *   - There is ONE scratch array per device: calls on the same device that
 *     may overlap in time (different streams, different host threads without
 *     ordering) race on it and produce wrong results.  Serialize them.
 * Arguments, layouts and other errors as tq_linear.
 */
#define TQ_STATIC_SCRATCH_BYTES ((size_t)1 << 20)
TQ_API tq_status tq_linear_static(int32_t M, int32_t N, int32_t K, const tq_weight *w, const uint16_t *x,
                                  uint16_t *y, void *stream);

/* Device status word of the library's linear kernels, OR of:
 *   1 = a bounded device-side wait ran out (the kernel stopped early and its
 *       outputs are incomplete), 2 = shared-memory placement failed.
 * SYNCHRONOUS (unlike every other entry point): copies the word from the
 * device of the current context; clear != 0 resets it to 0 afterwards. */
TQ_API tq_status tq_get_device_status(uint32_t *status_host, int clear);

/* Self-test of the failure path: one kernel makes a bounded wait on a
 * barrier phase that nothing completes.  After its limit (about 2 s) the
 * wait gives up, sets bit 0 of the device status word (as any wait of the
 * library's kernels would) and the kernel returns, writing 0 to
 * *result (device int32; 1 would mean the phase completed).  The context
 * stays usable.  Asynchronous on stream. */
TQ_API tq_status tq_wait_selftest(int32_t *result, void *stream);

/* Human-readable name of a status code (static string). */
TQ_API const char *tq_status_str(tq_status s);

#ifdef __cplusplus
}
#endif

#endif /* TQ_H_ */
