// tq_api.cu - the C ABI (include/tq.h): argument validation and dispatch.
//
// Nothing here allocates device memory or synchronizes; every launch goes to
// the caller's stream.  Shape / null / alignment errors return before any
// launch.
#include <string.h>

#include "tq_common.cuh"

namespace tq {
cudaError_t launch_rowptr(int N, int K, const uint32_t *sal, int32_t *rowptr, uint32_t *status,
                          cudaStream_t s);
cudaError_t launch_check_rowptr(int N, int K, const uint32_t *sal, const int32_t *rowptr,
                                uint32_t *status, cudaStream_t s);
cudaError_t launch_pack(int N, int K, const int8_t *T1, const int8_t *T2, const uint32_t *sal,
                        const int32_t *rowptr, uint8_t *plane1, uint8_t *plane2, uint32_t *status,
                        cudaStream_t s);
cudaError_t launch_plane2_index(int N, int K, const uint32_t *sal, const int32_t *rowptr, int64_t nnz,
                                const uint8_t *plane2, const uint16_t *scale2, int32_t *index, cudaStream_t s);
cudaError_t launch_unpack(int N, int K, const uint8_t *plane1, const uint8_t *plane2,
                          const uint32_t *sal, const int32_t *rowptr, int8_t *T1, int8_t *T2,
                          uint32_t *status, cudaStream_t s);
cudaError_t launch_gemv_mma(const BatchParams &p, cudaStream_t s);
cudaError_t launch_gemv_sequence(const BatchParams &bp, int barrier_extra, cudaStream_t s);
cudaError_t launch_ew_rowptr(int N, int K, const uint8_t *mask, int32_t *rowptr, uint32_t *status, cudaStream_t s);
cudaError_t launch_ew_pack(int N, int K, const int8_t *T0, const int8_t *T1, const uint8_t *mask,
                           const int32_t *rowptr, uint32_t *mplane, uint8_t *plane1, uint8_t *plane2,
                           uint32_t *status, cudaStream_t s);
cudaError_t launch_ew_unpack(int N, int K, const uint32_t *mplane, const uint8_t *plane1, const int32_t *rowptr,
                             const uint8_t *plane2, int8_t *T0, int8_t *T1, uint8_t *mask, uint32_t *status,
                             cudaStream_t s);
cudaError_t launch_ew_index_offsets(int N, int K, const uint32_t *mplane, int32_t *off, cudaStream_t s);
cudaError_t launch_ew_index_fill(int N, int K, const uint32_t *mplane, const uint8_t *plane1, const int32_t *rowptr,
                                 const uint8_t *plane2, const int32_t *off, uint16_t *idx, uint32_t *status,
                                 cudaStream_t s);
cudaError_t launch_ew_views(const EwCall *calls, int count, cudaStream_t s);
cudaError_t launch_ew_correct(int M, const EwCall *calls, int count, bool f32, cudaStream_t s);
int mma_rows_per_tile();
void mma_workspace_parts(int M, int N, int K, size_t *b, size_t *cs, size_t *y2);
cudaError_t read_status_gemv_mma(uint32_t *out, bool clear);
cudaError_t read_status_gemv_g4(uint32_t *out, bool clear);
int64_t g4_workspace_bytes(int M, int N, int K);
cudaError_t launch_prefill(const Problem &P, int M, bool f32, cudaStream_t s);
cudaError_t launch_prefill_batched(const Problem *probs, int count, int M, bool f32, cudaStream_t s);
size_t ternarize_ws_bytes(int N, int K);
cudaError_t launch_dequantize(int N, int K, const tq_weight *w, uint16_t *out, uint32_t *status, cudaStream_t s);
cudaError_t launch_ternarize(int N, int K, const uint16_t *W, int64_t nnz, int sweeps, uint8_t *plane1,
                             uint32_t *sal, int32_t *rowptr, uint8_t *plane2, uint16_t *scale1, uint16_t *offset,
                             uint16_t *scale2, unsigned char *ws, uint32_t *status, cudaStream_t s);
cudaError_t read_status_prefill(uint32_t *out, bool clear);
cudaError_t read_status_selftest(uint32_t *out, bool clear);
cudaError_t launch_wait_selftest(int32_t *result, cudaStream_t s);
}  // namespace tq

using namespace tq;

namespace {

constexpr int kMaxK = 1 << 20;  // 1 Mi inputs per row: far above any projection here

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }
bool aligned2(const void *p) { return ((uintptr_t)p & 1u) == 0; }

tq_status check_shape(int32_t N, int32_t K) {
  if (N < 1 || K < TQ_GROUP || K % TQ_GROUP != 0 || K > kMaxK) return TQ_ERR_SHAPE;
  return TQ_OK;
}

tq_status from_cuda(cudaError_t e) { return e == cudaSuccess ? TQ_OK : TQ_ERR_CUDA; }

tq_status check_weight(const tq_weight *w, int32_t N, int32_t K) {
  if (!w) return TQ_ERR_NULL;
  if (w->group != TQ_GROUP) return TQ_ERR_SHAPE;
  if (w->N != N || w->K != K) return TQ_ERR_SHAPE;
  if (tq_status s = check_shape(N, K)) return s;
  if (!w->plane1 || !w->salience || !w->rowptr || !w->scale1 || !w->offset) return TQ_ERR_NULL;
  if (w->nnz < 0 || w->nnz > (int64_t)N * (K / TQ_GROUP)) return TQ_ERR_SALIENCE;
  if (w->nnz > 0 && (!w->plane2 || !w->scale2)) return TQ_ERR_NULL;
  if (!aligned16(w->plane1)) return TQ_ERR_ALIGN;
  if (w->plane2 && !aligned16(w->plane2)) return TQ_ERR_ALIGN;
  if (w->p2index && !aligned16(w->p2index)) return TQ_ERR_ALIGN;
  if (!aligned2(w->scale1) || !aligned2(w->offset) ||
      (w->scale2 && !aligned2(w->scale2)) || ((uintptr_t)w->salience & 3u) ||
      ((uintptr_t)w->rowptr & 3u))
    return TQ_ERR_ALIGN;
  return TQ_OK;
}

Problem to_problem(const tq_weight *w, const uint16_t *x, void *y) {
  Problem P;
  memset(&P, 0, sizeof(P));
  P.plane1 = w->plane1;
  P.sal = w->salience;
  P.rowptr = w->rowptr;
  P.plane2 = w->plane2;
  P.p2idx = w->nnz > 0 ? w->p2index : nullptr;
  P.s1 = reinterpret_cast<const __half *>(w->scale1);
  P.off = reinterpret_cast<const __half *>(w->offset);
  P.s2 = reinterpret_cast<const __half *>(w->scale2);
  P.x = reinterpret_cast<const __half *>(x);
  P.y = y;
  P.N = w->N;
  P.K = w->K;
  P.nnz = (int32_t)w->nnz;
  return P;
}

size_t pad256(size_t b) { return (b + 255) / 256 * 256; }

// Workspace bytes of one problem for a pass over M <= 16 tokens.  (A call
// whose more than 8 tokens have to run as two passes of at most 8 places the
// smaller 8-token layout in the same space.)
size_t problem_ws_bytes(int M, int N, int K, bool general = false) {
  size_t b, cs, y2;
  mma_workspace_parts(M, N, K, &b, &cs, &y2);
  // + the tensor maps of plane 1, s1, off; with M <= 2 the operands of the
  // one-group-per-lane kernel follow
  const size_t g4 = M <= 2 && !general ? (size_t)g4_workspace_bytes(M, N, K) : 0;
  return pad256(b) + pad256(cs) + pad256(y2) + 512 + g4;
}

}  // namespace

namespace tq {
// Workspace bytes of a call over M tokens (M > TQ_MAX_SKINNY_M runs the
// prefill tile path, which needs none: 256 bytes keep the argument uniform).
size_t call_ws_bytes(int M, int N, int K) {
  if (M > TQ_MAX_SKINNY_M) return 256;
  return problem_ws_bytes(M, N, K);
}
}  // namespace tq

namespace {

// Places every problem's workspace (TQ_ERR_SHAPE when it is too small).
tq_status place(BatchParams &bp, unsigned char *ws, size_t ws_bytes) {
  const int rows = mma_rows_per_tile();
  int tiles = 0;
  size_t off = 0;
  for (int i = 0; i < bp.count; ++i) {
    Problem &P = bp.prob[i];
    P.tile_begin = tiles;
    tiles += (P.N + rows - 1) / rows;
    const size_t tot = problem_ws_bytes(bp.M, P.N, P.K, bp.general != 0);
    if (off + tot > ws_bytes) return TQ_ERR_SHAPE;
    size_t b, cs, y2;
    mma_workspace_parts(bp.M, P.N, P.K, &b, &cs, &y2);
    P.wsB = ws + off;
    P.wsCS = reinterpret_cast<float *>(ws + off + pad256(b));
    P.y2_off = (int32_t)(pad256(b) + pad256(cs));
    P.map_off = (int32_t)(pad256(b) + pad256(cs) + pad256(y2));
    off += tot;
  }
  bp.total_tiles = tiles;
  return TQ_OK;
}

// Places every problem's workspace and runs the decode path for bp.M <= 16
// tokens in one pass (warp-level MMA kernels).  Returns TQ_ERR_SHAPE when the
// workspace is too small.
tq_status run_pass(BatchParams &bp, unsigned char *ws, size_t ws_bytes, cudaStream_t s) {
  if (tq_status st = place(bp, ws, ws_bytes)) return st;
  return from_cuda(launch_gemv_mma(bp, s));
}

// The decode path for bp.M <= 16 tokens.  One pass, unless more than 8
// tokens meet a second plane without its index (the span kernels take 8
// tokens at most): then tokens 0..7 and 8..M-1 run one after the other over
// the same workspace (x and y are token-major, so each pass reads and writes
// one contiguous block of rows).
tq_status run_batch(BatchParams &bp, unsigned char *ws, size_t ws_bytes, cudaStream_t s) {
  bool indexed = true;
  for (int i = 0; i < bp.count; ++i)
    if (bp.prob[i].nnz > 0 && !bp.prob[i].p2idx) indexed = false;
  if (bp.M <= 8 || indexed) return run_pass(bp, ws, ws_bytes, s);
  thread_local BatchParams hi;  // large: kept off the stack
  hi = bp;
  hi.M = bp.M - 8;
  hi.general = 1;  // the workspace holds the 8-token layout, not the one-group-per-lane operands
  for (int i = 0; i < hi.count; ++i) {
    Problem &P = hi.prob[i];
    P.x += (int64_t)8 * P.K;
    P.y = static_cast<unsigned char *>(P.y) + (int64_t)8 * P.N * (hi.out_f32 ? 4 : 2);
  }
  const int M = bp.M;
  bp.M = 8;
  const tq_status st = run_pass(bp, ws, ws_bytes, s);
  bp.M = M;
  if (st != TQ_OK) return st;
  return run_pass(hi, ws, ws_bytes, s);
}

tq_status linear_impl(int32_t M, int32_t N, int32_t K, const tq_weight *w, const uint16_t *x,
                      void *y, bool f32, void *ws, size_t ws_bytes, cudaStream_t s) {
  if (M < 1) return TQ_ERR_SHAPE;
  if (tq_status st = check_weight(w, N, K)) return st;
  if (!x || !y || !ws) return TQ_ERR_NULL;
  if (!aligned16(x) || ((uintptr_t)ws & 255u)) return TQ_ERR_ALIGN;
  if (f32 ? ((uintptr_t)y & 3u) : !aligned2(y)) return TQ_ERR_ALIGN;
  if (ws_bytes < call_ws_bytes(M, N, K)) return TQ_ERR_SHAPE;
  if (M > TQ_MAX_SKINNY_M) {
    // prefill: dequantized weight tiles x activation tiles on the tensor cores
    const Problem P = to_problem(w, x, y);
    return from_cuda(launch_prefill(P, M, f32, s));
  }
  // large (kept off the stack) and per host thread, so that calls from
  // several threads never share launch parameters
  thread_local BatchParams bp;
  bp.count = 1;
  bp.M = M;
  bp.out_f32 = f32 ? 1 : 0;
  bp.prob[0] = to_problem(w, x, y);
  if (tq_status st = run_batch(bp, static_cast<unsigned char *>(ws), ws_bytes, s)) return st;
  return TQ_OK;
}

}  // namespace

extern "C" {

size_t tq_row_bytes(int32_t K) {
  if (check_shape(1, K) != TQ_OK) return 0;
  return (size_t)row_bytes_of(K);
}

size_t tq_sal_words(int32_t K) {
  if (check_shape(1, K) != TQ_OK) return 0;
  return (size_t)sal_words_of(K);
}

tq_status tq_salience_rowptr(int32_t N, int32_t K, const uint32_t *sal, int32_t *rowptr,
                             uint32_t *d_status, void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if (!sal || !rowptr || !d_status) return TQ_ERR_NULL;
  return from_cuda(launch_rowptr(N, K, sal, rowptr, d_status, (cudaStream_t)stream));
}

tq_status tq_pack(int32_t N, int32_t K, const int8_t *T1, const int8_t *T2, const uint32_t *sal,
                  const int32_t *rowptr, uint8_t *plane1, uint8_t *plane2, uint32_t *d_status,
                  void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if (!T1 || !sal || !rowptr || !plane1 || !d_status) return TQ_ERR_NULL;
  if ((T2 == nullptr) != (plane2 == nullptr)) return TQ_ERR_NULL;
  cudaStream_t s = (cudaStream_t)stream;
  if (tq_status st = from_cuda(launch_check_rowptr(N, K, sal, rowptr, d_status, s))) return st;
  return from_cuda(launch_pack(N, K, T1, T2, sal, rowptr, plane1, plane2, d_status, s));
}

tq_status tq_unpack(int32_t N, int32_t K, const uint8_t *plane1, const uint8_t *plane2,
                    const uint32_t *sal, const int32_t *rowptr, int8_t *T1, int8_t *T2,
                    uint32_t *d_status, void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if (!plane1 || !sal || !rowptr || !T1 || !d_status) return TQ_ERR_NULL;
  cudaStream_t s = (cudaStream_t)stream;
  if (tq_status st = from_cuda(launch_check_rowptr(N, K, sal, rowptr, d_status, s))) return st;
  return from_cuda(launch_unpack(N, K, plane1, plane2, sal, rowptr, T1, T2, d_status, s));
}

size_t tq_plane2_index_capacity(int32_t K, int64_t nnz) {
  if (K < TQ_GROUP || K % TQ_GROUP || nnz < 0) return 0;
  return (((size_t)nnz + 15 * (size_t)(K / TQ_GROUP)) + 15) & ~(size_t)15;
}

size_t tq_plane2_index_slot_offset(int32_t K) {
  if (K < TQ_GROUP || K % TQ_GROUP) return 0;
  return ((size_t)(K / TQ_GROUP + 1) * 4 + 127) & ~(size_t)127;
}

size_t tq_plane2_index_bytes(int32_t N, int32_t K, int64_t nnz) {
  if (check_shape(N, K) != TQ_OK || nnz < 0 || nnz > (int64_t)N * (K / TQ_GROUP)) return 0;
  if (tq_plane2_index_capacity(K, nnz) > (size_t)INT32_MAX) return 0;  // colptr is int32
  return tq_plane2_index_slot_offset(K) + 32 * tq_plane2_index_capacity(K, nnz);
}

tq_status tq_plane2_index(int32_t N, int32_t K, const uint32_t *sal, const int32_t *rowptr, int64_t nnz,
                          const uint8_t *plane2, const uint16_t *scale2, int32_t *index, void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if (!sal || !rowptr || !index) return TQ_ERR_NULL;
  if (nnz > 0 && (!plane2 || !scale2)) return TQ_ERR_NULL;
  if (nnz < 0 || nnz > (int64_t)N * (K / TQ_GROUP)) return TQ_ERR_SALIENCE;
  if (tq_plane2_index_bytes(N, K, nnz) == 0) return TQ_ERR_SHAPE;
  if (((uintptr_t)index & 15u) || (plane2 && !aligned16(plane2)) || (scale2 && !aligned2(scale2))) return TQ_ERR_ALIGN;
  return from_cuda(launch_plane2_index(N, K, sal, rowptr, nnz, plane2, scale2, index, (cudaStream_t)stream));
}

tq_status tq_dequantize(int32_t N, int32_t K, const tq_weight *w, uint16_t *out, uint32_t *d_status,
                        void *stream) {
  if (tq_status st = check_weight(w, N, K)) return st;
  if (!out || !d_status) return TQ_ERR_NULL;
  if (!aligned16(out)) return TQ_ERR_ALIGN;
  return from_cuda(launch_dequantize(N, K, w, out, d_status, (cudaStream_t)stream));
}

size_t tq_ternarize_workspace_bytes(int32_t N, int32_t K) {
  if (check_shape(N, K) != TQ_OK || (int64_t)N * (K / TQ_GROUP) > INT32_MAX) return 0;
  return ternarize_ws_bytes(N, K);
}

tq_status tq_ternarize(int32_t N, int32_t K, const uint16_t *W, int64_t nnz, int32_t sweeps, uint8_t *plane1,
                       uint32_t *sal, int32_t *rowptr, uint8_t *plane2, uint16_t *scale1, uint16_t *offset,
                       uint16_t *scale2, void *workspace, size_t workspace_bytes, uint32_t *d_status,
                       void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  const int64_t NB = (int64_t)N * (K / TQ_GROUP);
  if (NB > INT32_MAX || nnz < 0 || nnz > NB || sweeps < 0 || sweeps > 64) return TQ_ERR_SHAPE;
  if (!W || !plane1 || !sal || !rowptr || !scale1 || !offset || !workspace || !d_status) return TQ_ERR_NULL;
  if (nnz > 0 && (!plane2 || !scale2)) return TQ_ERR_NULL;
  if (workspace_bytes < ternarize_ws_bytes(N, K)) return TQ_ERR_SHAPE;
  if (!aligned16(W) || !aligned16(plane1) || !aligned16(workspace) || (plane2 && !aligned16(plane2)) ||
      !aligned2(scale1) || !aligned2(offset) || (scale2 && !aligned2(scale2)) || ((uintptr_t)sal & 3u) ||
      ((uintptr_t)rowptr & 3u))
    return TQ_ERR_ALIGN;
  return from_cuda(launch_ternarize(N, K, W, nnz, sweeps, plane1, sal, rowptr, plane2, scale1, offset, scale2,
                                    static_cast<unsigned char *>(workspace), d_status, (cudaStream_t)stream));
}

size_t tq_workspace_bytes(int32_t M, int32_t N, int32_t K) {
  if (M < 1 || check_shape(N, K) != TQ_OK) return 0;
  return call_ws_bytes(M, N, K);
}

size_t tq_batched_workspace_bytes(int32_t M, int32_t count, const tq_problem *problems) {
  if (M < 1 || count < 1 || count > TQ_MAX_BATCH || !problems) return 0;
  if (M > TQ_MAX_SKINNY_M) {
    // the prefill tile path needs no workspace (256 bytes keep the argument uniform)
    for (int i = 0; i < count; ++i)
      if (check_shape(problems[i].w.N, problems[i].w.K) != TQ_OK) return 0;
    return 256;
  }
  size_t tot = 0;
  for (int i = 0; i < count; ++i) {
    if (check_shape(problems[i].w.N, problems[i].w.K) != TQ_OK) return 0;
    tot += problem_ws_bytes(M, problems[i].w.N, problems[i].w.K);
  }
  return tot;
}

tq_status tq_linear(int32_t M, int32_t N, int32_t K, const tq_weight *w, const uint16_t *x,
                    uint16_t *y, void *workspace, size_t workspace_bytes, void *stream) {
  return linear_impl(M, N, K, w, x, y, false, workspace, workspace_bytes, (cudaStream_t)stream);
}

tq_status tq_linear_f32out(int32_t M, int32_t N, int32_t K, const tq_weight *w,
                           const uint16_t *x, float *y, void *workspace, size_t workspace_bytes,
                           void *stream) {
  return linear_impl(M, N, K, w, x, y, true, workspace, workspace_bytes, (cudaStream_t)stream);
}

tq_status tq_linear_batched(int32_t M, int32_t count, const tq_problem *problems, void *workspace,
                            size_t workspace_bytes, void *stream) {
  if (M < 1 || count < 1 || count > TQ_MAX_BATCH) return TQ_ERR_SHAPE;
  if (!problems || !workspace) return TQ_ERR_NULL;
  if ((uintptr_t)workspace & 255u) return TQ_ERR_ALIGN;
  if (M > TQ_MAX_SKINNY_M) {
    // prefill: every problem's tiles in one launch (per 16 problems)
    thread_local Problem probs[TQ_MAX_BATCH];
    for (int i = 0; i < count; ++i) {
      const tq_problem &q = problems[i];
      if (tq_status st = check_weight(&q.w, q.w.N, q.w.K)) return st;
      if (!q.x || !q.y) return TQ_ERR_NULL;
      if (!aligned16(q.x) || !aligned2(q.y)) return TQ_ERR_ALIGN;
      probs[i] = to_problem(&q.w, q.x, q.y);
    }
    return from_cuda(launch_prefill_batched(probs, count, M, false, (cudaStream_t)stream));
  }
  thread_local BatchParams bp;  // per host thread, as in linear_impl
  bp.count = count;
  bp.M = M;
  bp.out_f32 = 0;
  for (int i = 0; i < count; ++i) {
    const tq_problem &q = problems[i];
    if (tq_status st = check_weight(&q.w, q.w.N, q.w.K)) return st;
    if (!q.x || !q.y) return TQ_ERR_NULL;
    if (!aligned16(q.x)) return TQ_ERR_ALIGN;
    if (!aligned2(q.y)) return TQ_ERR_ALIGN;
    bp.prob[i] = to_problem(&q.w, q.x, q.y);
  }
  return run_batch(bp, static_cast<unsigned char *>(workspace), workspace_bytes, (cudaStream_t)stream);
}

}  // extern "C"

namespace {
// Validates a host problem array into the per-thread launch parameters.
tq_status fill_batch(BatchParams &bp, int32_t M, int32_t count, const tq_problem *problems) {
  bp.count = count;
  bp.M = M;
  bp.out_f32 = 0;
  for (int i = 0; i < count; ++i) {
    const tq_problem &q = problems[i];
    if (tq_status st = check_weight(&q.w, q.w.N, q.w.K)) return st;
    if (!q.x || !q.y) return TQ_ERR_NULL;
    if (!aligned16(q.x)) return TQ_ERR_ALIGN;
    if (!aligned2(q.y)) return TQ_ERR_ALIGN;
    bp.prob[i] = to_problem(&q.w, q.x, q.y);
  }
  return TQ_OK;
}

tq_status run_sequence(int32_t M, int32_t count, const tq_problem *problems, void *workspace,
                       size_t workspace_bytes, int barrier_extra, cudaStream_t s) {
  if (M != 1 || count < 1 || count > TQ_MAX_BATCH) return TQ_ERR_SHAPE;
  if (!problems || !workspace) return TQ_ERR_NULL;
  if ((uintptr_t)workspace & 255u) return TQ_ERR_ALIGN;
  thread_local BatchParams bp;
  if (tq_status st = fill_batch(bp, M, count, problems)) return st;
  for (int i = 0; i < count; ++i)
    if (problems[i].w.nnz > 0 && !problems[i].w.p2index) return TQ_ERR_NULL;
  if (tq_status st = place(bp, static_cast<unsigned char *>(workspace), workspace_bytes)) return st;
  return from_cuda(launch_gemv_sequence(bp, barrier_extra, s));
}
}  // namespace

extern "C" {

tq_status tq_linear_sequence(int32_t M, int32_t count, const tq_problem *problems, void *workspace,
                             size_t workspace_bytes, void *stream) {
  return run_sequence(M, count, problems, workspace, workspace_bytes, 0, (cudaStream_t)stream);
}

tq_status tq_sequence_selftest(int32_t count, const tq_problem *problems, void *workspace, size_t workspace_bytes,
                               void *stream) {
  return run_sequence(1, count, problems, workspace, workspace_bytes, 1, (cudaStream_t)stream);
}

}  // extern "C"

namespace {
// Per-problem workspace parts of the element-wise linear, each 256-byte
// padded: the s1 and off views [N][G] fp16, the views' zero salience words
// and rowptr, the fp32 result of the plane-1 pass [M][N].  The decode
// path's workspace follows (after every problem's parts in a batched call).
struct EwParts {
  size_t s1v, offv, salv, rpv, yd, total;
};
EwParts ew_parts(int32_t M, int32_t N, int32_t K) {
  EwParts p;
  const size_t G = (size_t)(K / TQ_GROUP), W = (size_t)sal_words_of(K);
  p.s1v = 0;
  p.offv = p.s1v + pad256((size_t)N * G * 2);
  p.salv = p.offv + pad256((size_t)N * G * 2);
  p.rpv = p.salv + pad256((size_t)N * W * 4);
  p.yd = p.rpv + pad256(((size_t)N + 1) * 4);
  p.total = p.yd + pad256((size_t)M * N * 4);
  return p;
}

tq_status check_ew(int32_t M, const tq_ew_weight *w, const uint16_t *x, const void *y, bool f32) {
  if (!w || !x || !y) return TQ_ERR_NULL;
  if (tq_status st = check_shape(w->N, w->K)) return st;
  if (!w->mask || !w->plane1 || !w->p2rowptr || !w->mu || !w->alpha0 || !w->alpha1) return TQ_ERR_NULL;
  if (!aligned16(w->plane1) || !aligned16(x) || ((uintptr_t)w->mask & 3u) || ((uintptr_t)w->p2rowptr & 3u) ||
      !aligned2(w->mu) || !aligned2(w->alpha0) || !aligned2(w->alpha1))
    return TQ_ERR_ALIGN;
  if ((w->idx_off == nullptr) != (w->idx == nullptr)) return TQ_ERR_NULL;  // an index has both parts
  if (w->idx_off && (((uintptr_t)w->idx_off & 3u) || !aligned2(w->idx))) return TQ_ERR_ALIGN;
  if (f32 ? ((uintptr_t)y & 3u) : !aligned2(y)) return TQ_ERR_ALIGN;
  (void)M;
  return TQ_OK;
}

// count problems sharing M: every problem's views and plane-1 result, then
// the plane-1 pass (one batched decode-path call; M > 16, a single problem
// only, the prefill path), then the correction of every problem.
tq_status ew_run(int32_t M, int32_t count, const tq_ew_weight *const *wts, const uint16_t *const *xs, void *const *ys,
                 bool f32, void *ws, size_t ws_bytes, cudaStream_t s) {
  thread_local EwCall calls[TQ_MAX_BATCH];
  unsigned char *b = static_cast<unsigned char *>(ws);
  size_t off = 0;
  for (int i = 0; i < count; ++i) {
    const tq_ew_weight *w = wts[i];
    const EwParts p = ew_parts(M, w->N, w->K);
    if (off + p.total > ws_bytes) return TQ_ERR_SHAPE;
    EwCall &c = calls[i];
    c.w = w;
    c.x = xs[i];
    c.y = ys[i];
    c.s1v = reinterpret_cast<uint16_t *>(b + off + p.s1v);
    c.offv = reinterpret_cast<uint16_t *>(b + off + p.offv);
    c.salv = reinterpret_cast<uint32_t *>(b + off + p.salv);
    c.rpv = reinterpret_cast<int32_t *>(b + off + p.rpv);
    c.ydense = reinterpret_cast<float *>(b + off + p.yd);
    off += p.total;
  }
  if (tq_status st = from_cuda(launch_ew_views(calls, count, s))) return st;
  // plane 1 with mask 3's parameters in every group, no second plane
  auto view_weight = [](const EwCall &c) {
    tq_weight tw;
    memset(&tw, 0, sizeof(tw));
    tw.N = c.w->N;
    tw.K = c.w->K;
    tw.group = TQ_GROUP;
    tw.plane1 = c.w->plane1;
    tw.salience = c.salv;
    tw.rowptr = c.rpv;
    tw.scale1 = c.s1v;
    tw.offset = c.offv;
    tw.nnz = 0;
    return tw;
  };
  if (M > TQ_MAX_SKINNY_M) {
    if (count != 1) return TQ_ERR_SHAPE;
    const tq_weight tw = view_weight(calls[0]);
    if (tq_status st = linear_impl(M, tw.N, tw.K, &tw, calls[0].x, calls[0].ydense, true, b + off, ws_bytes - off, s))
      return st;
  } else {
    thread_local BatchParams bp;
    bp.count = count;
    bp.M = M;
    bp.out_f32 = 1;
    for (int i = 0; i < count; ++i) {
      const tq_weight tw = view_weight(calls[i]);
      bp.prob[i] = to_problem(&tw, calls[i].x, calls[i].ydense);
    }
    if (tq_status st = run_batch(bp, b + off, ws_bytes - off, s)) return st;
  }
  return from_cuda(launch_ew_correct(M, calls, count, f32, s));
}

tq_status ew_linear_impl(int32_t M, int32_t N, int32_t K, const tq_ew_weight *w, const uint16_t *x, void *y,
                         bool f32, void *ws, size_t ws_bytes, cudaStream_t s) {
  if (M < 1) return TQ_ERR_SHAPE;
  if (tq_status st = check_ew(M, w, x, y, f32)) return st;
  if (w->N != N || w->K != K) return TQ_ERR_SHAPE;
  if (!ws) return TQ_ERR_NULL;
  if ((uintptr_t)ws & 255u) return TQ_ERR_ALIGN;
  if (ws_bytes < ew_parts(M, N, K).total + call_ws_bytes(M, N, K)) return TQ_ERR_SHAPE;
  void *yv = y;
  return ew_run(M, 1, &w, &x, &yv, f32, ws, ws_bytes, s);
}
}  // namespace

extern "C" {

tq_status tq_ew_rowptr(int32_t N, int32_t K, const uint8_t *mask_ids, int32_t *p2rowptr, uint32_t *d_status,
                       void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if (!mask_ids || !p2rowptr || !d_status) return TQ_ERR_NULL;
  return from_cuda(launch_ew_rowptr(N, K, mask_ids, p2rowptr, d_status, (cudaStream_t)stream));
}

tq_status tq_ew_pack(int32_t N, int32_t K, const int8_t *T0, const int8_t *T1, const uint8_t *mask_ids,
                     const int32_t *p2rowptr, uint32_t *mask, uint8_t *plane1, uint8_t *plane2, uint32_t *d_status,
                     void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if (!T0 || !T1 || !mask_ids || !p2rowptr || !mask || !plane1 || !d_status) return TQ_ERR_NULL;
  if (((uintptr_t)mask & 3u) || ((uintptr_t)p2rowptr & 3u)) return TQ_ERR_ALIGN;
  return from_cuda(launch_ew_pack(N, K, T0, T1, mask_ids, p2rowptr, mask, plane1, plane2, d_status,
                                  (cudaStream_t)stream));
}

tq_status tq_ew_unpack(int32_t N, int32_t K, const uint32_t *mask, const uint8_t *plane1, const int32_t *p2rowptr,
                       const uint8_t *plane2, int8_t *T0, int8_t *T1, uint8_t *mask_ids, uint32_t *d_status,
                       void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if (!mask || !plane1 || !p2rowptr || !T0 || !T1 || !mask_ids || !d_status) return TQ_ERR_NULL;
  if (((uintptr_t)mask & 3u) || ((uintptr_t)p2rowptr & 3u)) return TQ_ERR_ALIGN;
  return from_cuda(launch_ew_unpack(N, K, mask, plane1, p2rowptr, plane2, T0, T1, mask_ids, d_status,
                                    (cudaStream_t)stream));
}

tq_status tq_ew_index_offsets(int32_t N, int32_t K, const uint32_t *mask, int32_t *idx_off, void *stream) {
  if (tq_status st = check_shape(N, K)) return st;
  if ((int64_t)N * K >= (int64_t)1 << 31) return TQ_ERR_SHAPE;
  if (!mask || !idx_off) return TQ_ERR_NULL;
  if (((uintptr_t)mask & 3u) || ((uintptr_t)idx_off & 3u)) return TQ_ERR_ALIGN;
  return from_cuda(launch_ew_index_offsets(N, K, mask, idx_off, (cudaStream_t)stream));
}

tq_status tq_ew_index_fill(int32_t N, int32_t K, const tq_ew_weight *w, const int32_t *idx_off, uint16_t *idx,
                           uint32_t *d_status, void *stream) {
  if (!w || !idx_off || !idx || !d_status) return TQ_ERR_NULL;
  if (w->N != N || w->K != K) return TQ_ERR_SHAPE;
  if (tq_status st = check_shape(N, K)) return st;
  if ((int64_t)N * K >= (int64_t)1 << 31) return TQ_ERR_SHAPE;
  if (!w->mask || !w->plane1 || !w->p2rowptr) return TQ_ERR_NULL;
  if (((uintptr_t)w->mask & 3u) || ((uintptr_t)w->p2rowptr & 3u) || ((uintptr_t)idx_off & 3u) || !aligned2(idx))
    return TQ_ERR_ALIGN;
  return from_cuda(launch_ew_index_fill(N, K, w->mask, w->plane1, w->p2rowptr, w->plane2, idx_off, idx, d_status,
                                        (cudaStream_t)stream));
}

size_t tq_ew_workspace_bytes(int32_t M, int32_t N, int32_t K) {
  if (M < 1 || check_shape(N, K) != TQ_OK) return 0;
  return ew_parts(M, N, K).total + call_ws_bytes(M, N, K);
}

size_t tq_ew_batched_workspace_bytes(int32_t M, int32_t count, const tq_ew_problem *problems) {
  if (M < 1 || M > TQ_MAX_SKINNY_M || count < 1 || count > TQ_MAX_BATCH || !problems) return 0;
  size_t tot = 0;
  for (int i = 0; i < count; ++i) {
    const tq_ew_weight &w = problems[i].w;
    if (check_shape(w.N, w.K) != TQ_OK) return 0;
    tot += ew_parts(M, w.N, w.K).total + problem_ws_bytes(M, w.N, w.K);
  }
  return tot;
}

tq_status tq_ew_linear_batched(int32_t M, int32_t count, const tq_ew_problem *problems, void *workspace,
                               size_t workspace_bytes, void *stream) {
  if (M < 1 || M > TQ_MAX_SKINNY_M || count < 1 || count > TQ_MAX_BATCH) return TQ_ERR_SHAPE;
  if (!problems || !workspace) return TQ_ERR_NULL;
  if ((uintptr_t)workspace & 255u) return TQ_ERR_ALIGN;
  thread_local const tq_ew_weight *wp[TQ_MAX_BATCH];
  thread_local const uint16_t *xp[TQ_MAX_BATCH];
  thread_local void *yp[TQ_MAX_BATCH];
  for (int i = 0; i < count; ++i) {
    const tq_ew_problem &q = problems[i];
    if (tq_status st = check_ew(M, &q.w, q.x, q.y, false)) return st;
    wp[i] = &q.w;
    xp[i] = q.x;
    yp[i] = q.y;
  }
  if (workspace_bytes < tq_ew_batched_workspace_bytes(M, count, problems)) return TQ_ERR_SHAPE;
  return ew_run(M, count, wp, xp, yp, false, workspace, workspace_bytes, (cudaStream_t)stream);
}

tq_status tq_ew_linear(int32_t M, int32_t N, int32_t K, const tq_ew_weight *w, const uint16_t *x, uint16_t *y,
                       void *workspace, size_t workspace_bytes, void *stream) {
  return ew_linear_impl(M, N, K, w, x, y, false, workspace, workspace_bytes, (cudaStream_t)stream);
}

tq_status tq_ew_linear_f32out(int32_t M, int32_t N, int32_t K, const tq_ew_weight *w, const uint16_t *x, float *y,
                              void *workspace, size_t workspace_bytes, void *stream) {
  return ew_linear_impl(M, N, K, w, x, y, true, workspace, workspace_bytes, (cudaStream_t)stream);
}

tq_status tq_get_device_status(uint32_t *status_host, int clear) {
  if (!status_host) return TQ_ERR_NULL;
  uint32_t b = 0, c = 0, d = 0, e = 0;
  if (read_status_gemv_mma(&b, clear != 0) != cudaSuccess) return TQ_ERR_CUDA;
  if (read_status_gemv_g4(&e, clear != 0) != cudaSuccess) return TQ_ERR_CUDA;
  if (read_status_prefill(&c, clear != 0) != cudaSuccess) return TQ_ERR_CUDA;
  if (read_status_selftest(&d, clear != 0) != cudaSuccess) return TQ_ERR_CUDA;
  *status_host = b | c | d | e;
  return TQ_OK;
}

tq_status tq_wait_selftest(int32_t *result, void *stream) {
  if (!result) return TQ_ERR_NULL;
  if ((uintptr_t)result & 3u) return TQ_ERR_ALIGN;
  return from_cuda(launch_wait_selftest(result, (cudaStream_t)stream));
}

const char *tq_status_str(tq_status s) {
  switch (s) {
    case TQ_OK: return "TQ_OK";
    case TQ_ERR_NULL: return "TQ_ERR_NULL: a required pointer is NULL";
    case TQ_ERR_SHAPE: return "TQ_ERR_SHAPE: M, N or K out of range, or K not a multiple of 128";
    case TQ_ERR_ALIGN: return "TQ_ERR_ALIGN: a pointer is not aligned (plane1, plane2 and x need 16 bytes)";
    case TQ_ERR_CODE: return "TQ_ERR_CODE: invalid trit code";
    case TQ_ERR_BYTE: return "TQ_ERR_BYTE: invalid packed byte";
    case TQ_ERR_SALIENCE: return "TQ_ERR_SALIENCE: nnz inconsistent with the salience map";
    case TQ_ERR_CUDA: return "TQ_ERR_CUDA: a CUDA launch failed";
    case TQ_ERR_TIMEOUT: return "TQ_ERR_TIMEOUT: a bounded device wait ran out";
    case TQ_ERR_SCRATCH:
      return "TQ_ERR_SCRATCH: the call needs more workspace than the static scratch of tq_linear_static (1 MiB)";
    case TQ_ERR_FORMAT: return "TQ_ERR_FORMAT: container magic, version, size or hash mismatch";
    case TQ_ERR_KEY: return "TQ_ERR_KEY: container name missing, unexpected, duplicate or malformed";
  }
  return "unknown tq_status";
}

}  // extern "C"
