// tq_selftest.cu - self-test of the failure path shared by the kernels: one
// bounded wait (mbar_wait, the wait the kernels drain their copies with) on
// an mbarrier phase that nothing completes.  The wait gives up after its
// time limit (2 s of the global timer), records the timeout in this unit's
// device status word and returns; the kernel ends and the context stays
// usable.  No fault, trap or endless loop is involved.
#include "tq_common.cuh"
#include "tq_sm100.cuh"

namespace tq {
namespace {

__global__ void wait_selftest_kernel(int32_t *result) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);  // phase 0 completes after one arrival; none is made
    mbar_fence_init();
    result[0] = mbar_wait(&bar, 0u) ? 1 : 0;
  }
}

}  // namespace

TQ_STATUS_ACCESSOR(read_status_selftest)

cudaError_t launch_wait_selftest(int32_t *result, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(result);
  return cudaGetLastError();
}

}  // namespace tq
