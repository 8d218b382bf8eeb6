// Beacon seeding by Farthest Point Sampling (Appendix D.1, Algorithm 1) over
// the prompt queries of every GQA group (Appendix D.2, prefill branch).
//
// One CTA per instance.  Runs once per sequence (not on the per-step path),
// so it favours exactness over speed: all similarities are fp64.  The
// farthest-point loop evaluates every cosine with the same operation order as
// the definition cos(a, b) = (a.b) / (|a| |b|) (sequential sums, no fused
// multiply-add), so its argmin decisions are exact.  The first pick uses the
// identity mean_j cos(q_i, q_j) = (q_i . sum_j q_j / |q_j|) / (N |q_i|), which
// needs O(N d) instead of O(N^2 d) work; it can only differ from the literal
// average at ties below ~1e-15 relative.
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kFpsThreads = 256;

__device__ __forceinline__ double bf(const __nv_bfloat16 v) { return static_cast<double>(__bfloat162float(v)); }

// Block-wide argmin of (value, index); ties go to the lower index.
__device__ void block_argmin(double v, int i, double* red_v, int* red_i, double& out_v, int& out_i) {
  const unsigned full = 0xffffffffu;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    double ov = __shfl_down_sync(full, v, o);
    int oi = __shfl_down_sync(full, i, o);
    if (ov < v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
    }
  }
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    red_v[w] = v;
    red_i[w] = i;
  }
  __syncthreads();
  if (w == 0) {
    const int nw = blockDim.x >> 5;
    v = lane < nw ? red_v[lane] : INFINITY;
    i = lane < nw ? red_i[lane] : 0x7fffffff;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      double ov = __shfl_down_sync(full, v, o);
      int oi = __shfl_down_sync(full, i, o);
      if (ov < v || (ov == v && oi < i)) {
        v = ov;
        i = oi;
      }
    }
    if (lane == 0) {
      red_v[0] = v;
      red_i[0] = i;
    }
  }
  __syncthreads();
  out_v = red_v[0];
  out_i = red_i[0];
  __syncthreads();
}

template <int D>
__global__ void __launch_bounds__(kFpsThreads) fps_init_kernel(const __nv_bfloat16* __restrict__ q, int N, int nb,
                                                                float* __restrict__ cent, double* __restrict__ sums,
                                                                long long* __restrict__ counts) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  double* nrm = reinterpret_cast<double*>(smem_raw);  // [N]
  double* S = nrm + N;                                 // [N]
  double* u = S + N;                                   // [D]
  int* picks = reinterpret_cast<int*>(u + D);          // [kMaxBeacons]
  unsigned char* sel = reinterpret_cast<unsigned char*>(picks + kMaxBeacons);  // [N]
  __shared__ double red_v[32];
  __shared__ int red_i[32];

  const int e = blockIdx.x;
  const __nv_bfloat16* x = q + static_cast<size_t>(e) * N * D;

  // |q_i| with the sequential sum of the definition
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    double a = 0.0;
    for (int k = 0; k < D; ++k) {
      const double v = bf(x[static_cast<size_t>(i) * D + k]);
      a = __dadd_rn(a, __dmul_rn(v, v));
    }
    nrm[i] = __dsqrt_rn(a);
    sel[i] = 0;
  }
  __syncthreads();

  // u = sum_j q_j / |q_j|
  for (int k = threadIdx.x; k < D; k += blockDim.x) {
    double a = 0.0;
    for (int j = 0; j < N; ++j)
      if (nrm[j] > 0.0) a = __dadd_rn(a, __ddiv_rn(bf(x[static_cast<size_t>(j) * D + k]), nrm[j]));
    u[k] = a;
  }
  __syncthreads();

  // first pick: argmin_i of the mean cosine (scaled by N, which keeps the order)
  double best_v = INFINITY;
  int best_i = 0x7fffffff;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    double t = 0.0;
    if (nrm[i] > 0.0) {
      double a = 0.0;
      for (int k = 0; k < D; ++k) a = __dadd_rn(a, __dmul_rn(bf(x[static_cast<size_t>(i) * D + k]), u[k]));
      t = __ddiv_rn(a, nrm[i]);
    }
    if (t < best_v || (t == best_v && i < best_i)) {
      best_v = t;
      best_i = i;
    }
  }
  int p;
  double pv;
  block_argmin(best_v, best_i, red_v, red_i, pv, p);
  if (threadIdx.x == 0) {
    picks[0] = p;
    sel[p] = 1;
  }
  __syncthreads();

  // S_j = max over picked r of cos(q_j, q_r), updated pick by pick
  int r = p;
  for (int k = 0; k < nb; ++k) {
    if (k > 0) {
      double v = INFINITY;
      int vi = 0x7fffffff;
      for (int j = threadIdx.x; j < N; j += blockDim.x)
        if (!sel[j] && (S[j] < v || (S[j] == v && j < vi))) {
          v = S[j];
          vi = j;
        }
      double rv;
      block_argmin(v, vi, red_v, red_i, rv, r);
      if (threadIdx.x == 0) {
        picks[k] = r;
        sel[r] = 1;
      }
      __syncthreads();
    }
    if (k == nb - 1) break;
    for (int j = threadIdx.x; j < N; j += blockDim.x) {
      if (sel[j]) continue;
      double c = 0.0;
      if (nrm[j] > 0.0 && nrm[r] > 0.0) {
        double a = 0.0;
        for (int kk = 0; kk < D; ++kk)
          a = __dadd_rn(a, __dmul_rn(bf(x[static_cast<size_t>(j) * D + kk]), bf(x[static_cast<size_t>(r) * D + kk])));
        c = __ddiv_rn(a, __dmul_rn(nrm[j], nrm[r]));
      }
      if (k == 0 || c > S[j]) S[j] = c;
    }
    __syncthreads();
  }

  // beacon k = k-th pick, count 1
  for (int idx = threadIdx.x; idx < nb * D; idx += blockDim.x) {
    const int k = idx / D, i = idx % D;
    const __nv_bfloat16 v = x[static_cast<size_t>(picks[k]) * D + i];
    cent[(static_cast<size_t>(e) * nb + k) * D + i] = __bfloat162float(v);
    if (sums) sums[(static_cast<size_t>(e) * nb + k) * D + i] = bf(v);
  }
  for (int k = threadIdx.x; k < nb; k += blockDim.x) counts[static_cast<size_t>(e) * nb + k] = 1;
}

}  // namespace

cudaError_t launch_fps_init(const Shape& s, const __nv_bfloat16* q_init, int n_init, float* cent, double* sums,
                            long long* counts, cudaStream_t st) {
  const int N = s.G * n_init;
  const size_t smem = sizeof(double) * (2 * static_cast<size_t>(N) + s.d) + sizeof(int) * kMaxBeacons + N;
  if (s.d == 128) {
    cudaFuncSetAttribute(fps_init_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    fps_init_kernel<128><<<s.n_inst, kFpsThreads, smem, st>>>(q_init, N, s.nb, cent, sums, counts);
  } else {
    cudaFuncSetAttribute(fps_init_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    fps_init_kernel<64><<<s.n_inst, kFpsThreads, smem, st>>>(q_init, N, s.nb, cent, sums, counts);
  }
  return cudaGetLastError();
}

}  // namespace bkv
