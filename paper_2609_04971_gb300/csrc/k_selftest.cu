// Diagnostic kernel: one bounded wait on an mbarrier that nothing completes,
// through the same wait routine the library's kernels use, so that the expiry
// path (error word set, kernel returns, context stays usable) can be checked
// without faulting or hanging the device.
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

__global__ void selftest_wait_kernel(int* err, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_sh;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);  // one arrival expected; none is ever made
    abort_sh = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait_for(&bar, 0, &abort_sh, err, kDevTimeoutSelftest, limit_ns);
  __syncthreads();
}

}  // namespace

cudaError_t launch_selftest_wait(int* err, unsigned long long limit_ns, cudaStream_t st) {
  selftest_wait_kernel<<<1, 32, 0, st>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace bkv
