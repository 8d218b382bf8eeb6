// Beacon maintenance: nearest-beacon assignment by cosine similarity and the
// running-mean centroid update, for every instance at once.
//
// One CTA of 256 threads per instance; its queries are processed in passes
// of up to 2048:
//   * Screening (4 threads per query, straight from global memory): fp32 dots
//     of the query with unit-length centroids, four independent FMA chains
//     per thread.  When the best and second-best dot differ by less than
//     1e-4 |q| (far above the ~1e-5 |q| worst-case error of a 128-term fp32
//     dot), the query is re-decided in fp64 by one warp: cos(q, c_b) =
//     (q . c_b) / (|q| |c_b|) with fp64 products and sums, which can differ
//     from a sequential fp64 evaluation only at ties below ~1e-15 (the lowest
//     beacon wins ties).
//   * Accumulation: each bf16 query element is converted to an int64 fixed
//     point value with 40 fractional bits (exact for |x| >= 2^-33).  The
//     queries are bucketed by beacon (counting sort); the thread that owns
//     (beacon, column) sums its bucket in a register and adds it to its
//     shared-memory cell, so the per-call sum is exact and independent of
//     ordering.  It is then added once to the fp64 running sum.
//   * Centroid: c = fp32(sum * (1 / count)) in fp64, within one fp32 ulp of
//     fp32(sum / count).
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kUpdThreads = 256;
constexpr int kUpdWarps = kUpdThreads / 32;
constexpr int kPass = 2048;  // queries per pass (assignment buffer size)

__device__ __forceinline__ long long to_fixed40(__nv_bfloat16 v) {
  return __float2ll_rn(__bfloat162float(v) * 0x1p40f);
}

__device__ __forceinline__ double warp_sum_f64(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <int D>
__global__ void __launch_bounds__(kUpdThreads) update_kernel(const __nv_bfloat16* __restrict__ q_new, int nq, int nb,
                                                              float* __restrict__ cent, double* __restrict__ sums,
                                                              long long* __restrict__ counts,
                                                              int* __restrict__ assign_out) {
  constexpr int kPer = D / 4;  // dims per screening thread
  extern __shared__ __align__(16) unsigned char smem_raw[];
  long long* acc = reinterpret_cast<long long*>(smem_raw);  // [nb][D]
  float* chat = reinterpret_cast<float*>(acc + nb * D);     // [nb][D] unit centroids
  __shared__ int asg[kPass];
  __shared__ short order[kPass];
  __shared__ int refine_idx[kPass];
  __shared__ int n_refine;
  __shared__ int bucket_start[kMaxBeacons + 1];
  __shared__ int bucket_fill[kMaxBeacons];
  __shared__ int add_cnt[kMaxBeacons];
  __shared__ int bvalid[kMaxBeacons];
  __shared__ double cn64[kMaxBeacons];
  __shared__ int degenerate;

  const int e = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float* cent_e = cent + static_cast<size_t>(e) * nb * D;
  const __nv_bfloat16* q_e = q_new + static_cast<size_t>(e) * nq * D;

  for (int idx = tid; idx < nb * D; idx += kUpdThreads) {
    chat[idx] = cent_e[idx];
    acc[idx] = 0;
  }
  if (tid < kMaxBeacons) add_cnt[tid] = 0;
  if (tid == 0) degenerate = 0;
  __syncthreads();

  // one warp per beacon: qualification, fp64 norm, unit-length fp32 copy
  for (int b = warp; b < nb; b += kUpdWarps) {
    float n2 = 0.f;
    double n2d = 0.0;
    int nz = 0;
    for (int i = lane; i < D; i += 32) {
      const float c = chat[b * D + i];
      n2 = fmaf(c, c, n2);
      n2d = fma(static_cast<double>(c), static_cast<double>(c), n2d);
      nz |= (c != 0.f);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      n2 += __shfl_xor_sync(0xffffffffu, n2, o);
      nz |= __shfl_xor_sync(0xffffffffu, nz, o);
    }
    n2d = warp_sum_f64(n2d);
    const int ok = (counts[static_cast<size_t>(e) * nb + b] > 0) && nz;
    const float inv = rsqrtf(n2);
    for (int i = lane; i < D; i += 32) chat[b * D + i] *= inv;
    if (lane == 0) {
      bvalid[b] = ok;
      cn64[b] = sqrt(n2d);
      if (ok && !(n2 > 1e-30f && n2 < 1e30f)) atomicExch(&degenerate, 1);
    }
  }
  __syncthreads();

  const int quad = tid >> 2, sub = tid & 3;
  for (int p0 = 0; p0 < nq; p0 += kPass) {
    const int rows = min(kPass, nq - p0);
    if (tid == 0) n_refine = 0;
    if (tid < kMaxBeacons) bucket_fill[tid] = 0;
    __syncthreads();

    // ---- screening: 64 queries per block-wide step, 4 threads each (warp-uniform trip count)
    for (int n0 = 0; n0 < rows; n0 += kUpdThreads / 4) {
      const int n = n0 + quad;
      const bool active = n < rows;
      const __nv_bfloat16* qrow = q_e + static_cast<size_t>(p0 + (active ? n : rows - 1)) * D + 4 * sub;
      float qv[kPer];
      unsigned nz = 0;
      float qa = 0.f, qb = 0.f;
#pragma unroll
      for (int k = 0; k < kPer / 4; ++k) {
        const uint2 raw = __ldg(reinterpret_cast<const uint2*>(qrow + 16 * k));
        nz |= (raw.x | raw.y) & 0x7fff7fffu;
        const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.x));
        const float2 c = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.y));
        qv[4 * k + 0] = a.x;
        qv[4 * k + 1] = a.y;
        qv[4 * k + 2] = c.x;
        qv[4 * k + 3] = c.y;
        qa = fmaf(a.x, a.x, fmaf(a.y, a.y, qa));
        qb = fmaf(c.x, c.x, fmaf(c.y, c.y, qb));
      }
      float qn2 = qa + qb;
      qn2 += __shfl_xor_sync(0xffffffffu, qn2, 1);
      qn2 += __shfl_xor_sync(0xffffffffu, qn2, 2);
      nz |= __shfl_xor_sync(0xffffffffu, nz, 1);
      nz |= __shfl_xor_sync(0xffffffffu, nz, 2);
      float best = -INFINITY, second = -INFINITY;
      int bi = -1;
      for (int b = 0; b < nb; ++b) {
        if (!bvalid[b]) continue;
        const float* cb = chat + b * D + 4 * sub;
        float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
        for (int k = 0; k < kPer / 4; ++k) {
          const float4 c4 = *reinterpret_cast<const float4*>(cb + 16 * k);
          d0 = fmaf(qv[4 * k + 0], c4.x, d0);
          d1 = fmaf(qv[4 * k + 1], c4.y, d1);
          d2 = fmaf(qv[4 * k + 2], c4.z, d2);
          d3 = fmaf(qv[4 * k + 3], c4.w, d3);
        }
        float dot = (d0 + d1) + (d2 + d3);
        dot += __shfl_xor_sync(0xffffffffu, dot, 1);
        dot += __shfl_xor_sync(0xffffffffu, dot, 2);
        if (dot > best) {
          second = best;
          best = dot;
          bi = b;
        } else if (dot > second) {
          second = dot;
        }
      }
      if (active && sub == 0) {
        int a;
        if (nz == 0 || bi < 0) {
          a = -1;
        } else if (degenerate || !(qn2 > 1e-30f && qn2 < 1e30f) || !(best - second > 1e-4f * sqrtf(qn2))) {
          a = -2;  // decided exactly below
          refine_idx[atomicAdd(&n_refine, 1)] = n;
        } else {
          a = bi;
        }
        asg[n] = a;
      }
    }
    __syncthreads();

    // ---- exact fp64 decisions for close calls: one warp per query
    for (int t = warp; t < n_refine; t += kUpdWarps) {
      const int n = refine_idx[t];
      const __nv_bfloat16* qrow = q_e + static_cast<size_t>(p0 + n) * D;
      double x[D / 32];
#pragma unroll
      for (int k = 0; k < D / 32; ++k) x[k] = __bfloat162float(qrow[lane + 32 * k]);
      double qq = 0.0;
#pragma unroll
      for (int k = 0; k < D / 32; ++k) qq = fma(x[k], x[k], qq);
      const double nqd = sqrt(warp_sum_f64(qq));
      double b1 = -INFINITY;
      int best_b = -1;
      for (int b = 0; b < nb; ++b) {
        if (!bvalid[b]) continue;
        double dt = 0.0;
#pragma unroll
        for (int k = 0; k < D / 32; ++k) dt = fma(x[k], static_cast<double>(cent_e[b * D + lane + 32 * k]), dt);
        const double cs = warp_sum_f64(dt) / (nqd * cn64[b]);
        if (cs > b1) {
          b1 = cs;
          best_b = b;
        }
      }
      if (lane == 0) asg[n] = best_b;
    }
    __syncthreads();

    // ---- bucket the pass's queries by beacon (order inside a bucket is irrelevant)
    for (int n = tid; n < rows; n += kUpdThreads) {
      const int b = asg[n];
      if (b >= 0) atomicAdd(&bucket_fill[b], 1);
      if (assign_out) assign_out[static_cast<size_t>(e) * nq + p0 + n] = b;
    }
    __syncthreads();
    if (tid == 0) {
      int run = 0;
      for (int b = 0; b < nb; ++b) {
        bucket_start[b] = run;
        run += bucket_fill[b];
        add_cnt[b] += bucket_fill[b];
        bucket_fill[b] = 0;
      }
      bucket_start[nb] = run;
    }
    __syncthreads();
    for (int n = tid; n < rows; n += kUpdThreads) {
      const int b = asg[n];
      if (b >= 0) order[bucket_start[b] + atomicAdd(&bucket_fill[b], 1)] = static_cast<short>(n);
    }
    __syncthreads();

    // ---- exact sums: thread (group g, column col) owns cells (b, col) of beacons b = g mod kGroups
    {
      constexpr int kGroups = kUpdThreads / D;
      const int col = tid % D, g = tid / D;
      const __nv_bfloat16* qc = q_e + static_cast<size_t>(p0) * D + col;
      for (int b = g; b < nb; b += kGroups) {
        const int r0 = bucket_start[b], r1 = bucket_start[b + 1];
        if (r0 == r1) continue;
        long long s0 = 0, s1 = 0;
        int r = r0;
        for (; r + 8 <= r1; r += 8) {  // eight independent loads in flight
          __nv_bfloat16 v[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) v[u] = qc[static_cast<size_t>(order[r + u]) * D];
#pragma unroll
          for (int u = 0; u < 8; u += 2) {
            s0 += to_fixed40(v[u]);
            s1 += to_fixed40(v[u + 1]);
          }
        }
        for (; r < r1; ++r) s0 += to_fixed40(qc[static_cast<size_t>(order[r]) * D]);
        acc[b * D + col] += s0 + s1;
      }
    }
    __syncthreads();
  }

  // ---- fold the call into the running state
  for (int idx = tid; idx < nb * D; idx += kUpdThreads) {
    const int b = idx / D;
    const int add = add_cnt[b];
    if (add == 0) continue;
    const size_t g = static_cast<size_t>(e) * nb * D + idx;
    const double s_new = __dadd_rn(sums[g], static_cast<double>(acc[idx]) * 0x1p-40);
    sums[g] = s_new;
    const long long cnt = counts[static_cast<size_t>(e) * nb + b] + add;
    cent[g] = __double2float_rn(__dmul_rn(s_new, __drcp_rn(static_cast<double>(cnt))));
  }
  __syncthreads();
  if (tid < nb) counts[static_cast<size_t>(e) * nb + tid] += add_cnt[tid];
}

}  // namespace

cudaError_t launch_update(const Shape& s, const __nv_bfloat16* q_new, int n_new, float* cent, double* sums,
                          long long* counts, int* assign_out, cudaStream_t st) {
  const int nq = s.G * n_new;
  const int nb = s.nb;
  const size_t smem = static_cast<size_t>(nb) * s.d * (sizeof(long long) + sizeof(float));
  if (s.d == 128) {
    cudaFuncSetAttribute(update_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    update_kernel<128><<<s.n_inst, kUpdThreads, smem, st>>>(q_new, nq, nb, cent, sums, counts, assign_out);
  } else {
    cudaFuncSetAttribute(update_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    update_kernel<64><<<s.n_inst, kUpdThreads, smem, st>>>(q_new, nq, nb, cent, sums, counts, assign_out);
  }
  return cudaGetLastError();
}

}  // namespace bkv
