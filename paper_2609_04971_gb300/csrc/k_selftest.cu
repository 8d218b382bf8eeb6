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

// One checked store at index 32 of a shared array of 64 words whose logical length is 32: with
// bounds checks compiled in (BKV_CHECKED) the check fails, records kDevBounds and the store is
// skipped; without them the store lands in the array's second half, which this kernel owns.
__global__ void selftest_bounds_kernel(int* err, int n) {
  __shared__ int buf[64];
  buf[threadIdx.x] = 0;
  buf[threadIdx.x + 32] = 0;
  __syncthreads();
  if (threadIdx.x == 0 && n <= 32 && in_bounds(n, 32, err)) buf[n] = 1;
  __syncthreads();
}

}  // namespace

cudaError_t launch_selftest_bounds(int* err, cudaStream_t st) {
  selftest_bounds_kernel<<<1, 32, 0, st>>>(err, 32);
  return cudaGetLastError();
}

cudaError_t launch_selftest_wait(int* err, unsigned long long limit_ns, cudaStream_t st) {
  selftest_wait_kernel<<<1, 32, 0, st>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace bkv
