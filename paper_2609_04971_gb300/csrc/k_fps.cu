// Beacon seeding by Farthest Point Sampling (Appendix D.1, Algorithm 1) over
// the prompt queries of every GQA group (Appendix D.2, prefill branch).
//
// One CTA per instance (or query head), one thread per prompt query.  The
// similarities carry about 44 significant bits without fp64 arithmetic (which
// is slow on this part): a product of two bf16 values is exact in fp32, dot
// products are sums of those products in double-float arithmetic (TwoSum),
// 1 / |q| comes from a Newton step, and cos(q_j, q_r) = (q_j . q_r) (1 / |q_j|)
// (1 / |q_r|) in double-float.  Candidates are compared as the doubles those
// double-floats equal, so the argmin decisions equal those of the fp64
// definition except at ties below ~1e-13 relative (lowest index on exact
// ties).  The first pick uses the identity
// mean_j cos(q_i, q_j) = (q_i . sum_j q_j / |q_j|) / (N |q_i|), which needs
// O(N d) instead of O(N^2 d) work; it can only differ from the literal average
// at such ties.
#include "bkv_device.cuh"
#include "bkv_internal.h"
#include "k_update_math.cuh"

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

// Sum over this row's elements of x_k * y_k for bf16 rows (two 16-byte loads per 8
// elements): each product of two bf16 values is exact in fp32, and the products are
// summed in double-float arithmetic in two interleaved chains (even and odd groups of 8).
template <int D>
__device__ __forceinline__ DF dot_bf16(const __nv_bfloat16* x, const __nv_bfloat16* y) {
  DF a0{0.f, 0.f}, a1{0.f, 0.f};
#pragma unroll 2
  for (int k = 0; k < D; k += 16) {
    const uint4 xa = *reinterpret_cast<const uint4*>(x + k), xb = *reinterpret_cast<const uint4*>(x + k + 8);
    const uint4 ya = *reinterpret_cast<const uint4*>(y + k), yb = *reinterpret_cast<const uint4*>(y + k + 8);
    const uint32_t wx[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
    const uint32_t wy[8] = {ya.x, ya.y, ya.z, ya.w, yb.x, yb.y, yb.z, yb.w};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      DF& acc = i < 4 ? a0 : a1;
      acc = df_add(acc, DF{__fmul_rn(__uint_as_float(wx[i] << 16), __uint_as_float(wy[i] << 16)), 0.f});
      acc = df_add(acc, DF{__fmul_rn(__uint_as_float(wx[i] & 0xffff0000u), __uint_as_float(wy[i] & 0xffff0000u)), 0.f});
    }
  }
  return df_add(a0, a1);
}

// A double-float as the double it equals (hi + lo needs at most 48 significant bits).
__device__ __forceinline__ double df_to_double(DF v) {
  return __dadd_rn(static_cast<double>(v.hi), static_cast<double>(v.lo));
}

template <int D>
__global__ void __launch_bounds__(kFpsThreads) fps_init_kernel(const __nv_bfloat16* __restrict__ q, int N, int nb,
                                                                float* __restrict__ cent, double* __restrict__ sums,
                                                                long long* __restrict__ counts) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  DF* inv = reinterpret_cast<DF*>(smem_raw);                 // [N] 1 / |q_j| (0 for a zero query)
  double* S = reinterpret_cast<double*>(inv + N);            // [N]
  DF* u = reinterpret_cast<DF*>(S + N);                      // [D]
  int* picks = reinterpret_cast<int*>(u + D);                // [kMaxBeacons]
  unsigned char* sel = reinterpret_cast<unsigned char*>(picks + kMaxBeacons);  // [N]
  __shared__ double red_v[32];
  __shared__ int red_i[32];

  const int e = blockIdx.x;
  const __nv_bfloat16* x = q + static_cast<size_t>(e) * N * D;

  // 1 / |q_i|: the exact squares summed in double-float arithmetic, then one Newton step
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    const DF n2 = dot_bf16<D>(x + static_cast<size_t>(i) * D, x + static_cast<size_t>(i) * D);
    bool plain = true;
    inv[i] = n2.hi > 0.f ? centroid_inv_norm(n2, n2.hi, plain) : DF{0.f, 0.f};
    sel[i] = 0;
  }
  __syncthreads();

  // u = sum_j q_j / |q_j|
  for (int k = threadIdx.x; k < D; k += blockDim.x) {
    DF a{0.f, 0.f};
    for (int j = 0; j < N; ++j)
      a = df_add(a, df_mul(DF{__bfloat162float(x[static_cast<size_t>(j) * D + k]), 0.f}, inv[j]));
    u[k] = a;
  }
  __syncthreads();

  // first pick: argmin_i of the mean cosine (scaled by N, which keeps the order)
  double best_v = INFINITY;
  int best_i = 0x7fffffff;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    DF t{0.f, 0.f};
    if (inv[i].hi > 0.f) {
      DF a{0.f, 0.f};
      for (int k = 0; k < D; ++k) a = df_add(a, df_mul(DF{__bfloat162float(x[static_cast<size_t>(i) * D + k]), 0.f}, u[k]));
      t = df_mul(a, inv[i]);
    }
    const double tv = df_to_double(t);
    if (tv < best_v || (tv == best_v && i < best_i)) {
      best_v = tv;
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
    const DF inv_r = inv[r];
    const __nv_bfloat16* xr = x + static_cast<size_t>(r) * D;
    for (int j = threadIdx.x; j < N; j += blockDim.x) {
      if (sel[j]) continue;
      double c = 0.0;
      if (inv[j].hi > 0.f && inv_r.hi > 0.f)
        c = df_to_double(df_mul(df_mul(dot_bf16<D>(x + static_cast<size_t>(j) * D, xr), inv[j]), inv_r));
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
  const size_t smem = sizeof(DF) * N + sizeof(double) * N + sizeof(DF) * s.d + sizeof(int) * kMaxBeacons + N;
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
