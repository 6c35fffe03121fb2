// tq_static.cu - tq_linear_static: tq_linear with its workspace in a scratch
// array held by the library (declared and documented in include/tq.h).
//
// The array is a file-scope __device__ object, so its device memory comes
// with the module; the first call on a device looks its address up once
// (cudaGetSymbolAddress) and caches it per device.  Every call then forwards
// to tq_linear unchanged.
#include <mutex>

#include "tq_common.cuh"

namespace tq {
size_t call_ws_bytes(int M, int N, int K);
}

namespace {

static __device__ __align__(256) unsigned char g_tq_static_scratch[TQ_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void *g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up on
// the first call per device), or nullptr if the lookup failed.
void *scratch_for_current_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_tq_static_scratch) != cudaSuccess || p == nullptr) return nullptr;
    g_scratch_ptr[dev] = p;
  }
  return g_scratch_ptr[dev];
}

}  // namespace

extern "C" {

tq_status tq_linear_static(int32_t M, int32_t N, int32_t K, const tq_weight *w, const uint16_t *x, uint16_t *y,
                           void *stream) {
  if (M < 1 || N < 1 || K < TQ_GROUP || K % TQ_GROUP != 0) return TQ_ERR_SHAPE;
  if (tq::call_ws_bytes(M, N, K) > TQ_STATIC_SCRATCH_BYTES) return TQ_ERR_SCRATCH;
  void *ws = scratch_for_current_device();
  if (!ws) return TQ_ERR_CUDA;
  return tq_linear(M, N, K, w, x, y, ws, TQ_STATIC_SCRATCH_BYTES, stream);
}

}  // extern "C"
