// Per-instance cache lengths (bkv_compress_ragged): which instances one
// compress evicts from.  In batched decoding every sequence has its own cache
// length (Section 5.4; Algorithm 2 runs per sequence), so an instance is
// compressed only when its own length exceeds the budget.
//
// ragged_plan_kernel (one CTA): lists, in index order, the instances with
// budget < L <= capacity in work[0 .. *n_work); the compress kernels then take
// their instances from that list.  A length outside 1..capacity is recorded in
// the device error word (kDevBadLength) and that instance is left untouched.
// ragged_keep_kernel: the kept rows of every instance that is not compressed:
// 0 .. L - 1, then -1 (all -1 for a length outside the range).
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kPlanThreads = 1024;

__global__ void __launch_bounds__(kPlanThreads) ragged_plan_kernel(int n_inst, int cap, const int* __restrict__ Ls,
                                                                    int budget, int* __restrict__ work,
                                                                    int* __restrict__ n_work, int* err) {
  __shared__ int wsum[kPlanThreads / 32];
  __shared__ int base_sh;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) base_sh = 0;
  __syncthreads();
  for (int c0 = 0; c0 < n_inst; c0 += kPlanThreads) {
    const int e = c0 + static_cast<int>(threadIdx.x);
    const int L = e < n_inst ? Ls[e] : 0;
    const bool bad = e < n_inst && (L < 1 || L > cap);
    if (bad) record_error(err, kDevBadLength);
    const bool evict = e < n_inst && !bad && L > budget;
    const unsigned bal = __ballot_sync(0xffffffffu, evict);
    if (lane == 0) wsum[warp] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
#pragma unroll 4
    for (int w = 0; w < kPlanThreads / 32; ++w) {
      const int c = wsum[w];
      before += w < warp ? c : 0;
      total += c;
    }
    const int base = base_sh;
    if (evict) work[base + before + __popc(bal & ((1u << lane) - 1u))] = e;
    __syncthreads();  // every read of wsum and base_sh is done
    if (threadIdx.x == 0) base_sh = base + total;
    __syncthreads();
  }
  if (threadIdx.x == 0) *n_work = base_sh;
}

__global__ void ragged_keep_kernel(int n_inst, int cap, const int* __restrict__ Ls, int budget,
                                   int* __restrict__ kept) {
  const size_t n = static_cast<size_t>(n_inst) * budget;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int e = static_cast<int>(i / budget), j = static_cast<int>(i % budget);
    const int L = Ls[e];
    const bool ok = L >= 1 && L <= cap;
    if (ok && L > budget) continue;  // compressed: the selection writes this row
    kept[i] = ok && j < L ? j : -1;
  }
}

}  // namespace

cudaError_t launch_ragged_plan(const Shape& s, const int* Ls, int budget, int* work, int* n_work, int* kept, int* err,
                               cudaStream_t st) {
  ragged_plan_kernel<<<1, kPlanThreads, 0, st>>>(s.n_inst, s.cap, Ls, budget, work, n_work, err);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t n = static_cast<size_t>(s.n_inst) * budget;
  const int blocks = static_cast<int>(n / 256 + 1 < 4096 ? n / 256 + 1 : 4096);
  ragged_keep_kernel<<<blocks, 256, 0, st>>>(s.n_inst, s.cap, Ls, budget, kept);
  return cudaGetLastError();
}

}  // namespace bkv
