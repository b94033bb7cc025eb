// Self-test of the bounded waits that every tensor-core kernel of this library
// uses (sm100::mbar_wait): one block waits on an mbarrier that nothing ever
// arrives at, with a caller-given limit in SM clock cycles, and records
// kErrTimeout in the device error word when the wait gives up.  The failure
// is made on purpose without faulting or hanging the GPU: the wait ends by its
// own limit, the kernel returns, and the context stays usable.
#include "common.cuh"
#include "sm100.cuh"

namespace dck {
namespace {

__global__ void bounded_wait_selftest_kernel(long long limit_cycles, int* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    sm100::mbar_init(&bar, 1);
    abort_flag = 0;
    sm100::fence_mbar_init();
  }
  __syncthreads();
  // phase 0 never completes: no thread arrives and no copy is in flight
  if (threadIdx.x == 0 && !sm100::mbar_wait(&bar, 0, &abort_flag, limit_cycles)) atomicOr(err, kErrTimeout);
}

}  // namespace

cudaError_t launch_bounded_wait_selftest(long long limit_cycles, int* err, cudaStream_t s) {
  bounded_wait_selftest_kernel<<<1, 32, 0, s>>>(limit_cycles, err);
  return cudaGetLastError();
}

}  // namespace dck
