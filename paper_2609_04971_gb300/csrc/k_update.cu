// Beacon maintenance: nearest-beacon assignment by cosine similarity and the
// running-mean centroid update, for every instance at once.
//
// One CTA per instance; queries are staged through shared memory in chunks
// of 64 and handled by four threads each.
//   * Screening: fp32 dots of the query with unit-length centroids.  When the
//     best and second-best dot differ by less than 1e-4 |q| (far above the
//     ~1e-5 |q| worst-case fp32 error of a 128-term dot), the query is re-decided
//     in fp64 with the operation order of the definition cos(a, b) =
//     (a.b) / (|a| |b|), so every assignment equals the exact argmax (ties to
//     the lowest beacon).
//   * Accumulation: each bf16 query element is converted to an int64 fixed
//     point value with 40 fractional bits (exact for |x| >= 2^-33) and added
//     with shared-memory integer atomics, so the per-call sum is exact and
//     independent of ordering; it is then added once to the fp64 running sum.
//   * Centroid: c = fp32(sum * (1 / count)) in fp64, within one fp32 ulp of
//     fp32(sum / count).
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kUpdThreads = 256;
constexpr int kChunk = 64;  // queries per staged chunk (4 threads per query)

__device__ __forceinline__ long long to_fixed40(__nv_bfloat16 v) {
  return __float2ll_rn(__bfloat162float(v) * 0x1p40f);
}

template <int D>
struct UpdSmem {
  static constexpr int kPitch = D + 16;  // bf16 per staged row: 32 bytes of padding
};

template <int D>
__global__ void __launch_bounds__(kUpdThreads) update_kernel(const __nv_bfloat16* __restrict__ q_new, int nq, int nb,
                                                              float* __restrict__ cent, double* __restrict__ sums,
                                                              long long* __restrict__ counts,
                                                              int* __restrict__ assign_out) {
  constexpr int kPitch = UpdSmem<D>::kPitch;
  constexpr int kPer = D / 4;  // dims per thread
  extern __shared__ __align__(16) unsigned char smem_raw[];
  long long* acc = reinterpret_cast<long long*>(smem_raw);                     // [nb][D]
  float* chat = reinterpret_cast<float*>(acc + nb * D);                        // [nb][D]
  __nv_bfloat16* qs = reinterpret_cast<__nv_bfloat16*>(chat + nb * D);         // [kChunk][kPitch]
  __shared__ int asg[kChunk];
  __shared__ int refine_idx[kChunk];
  __shared__ int n_refine;
  __shared__ int add_cnt[kMaxBeacons];
  __shared__ int bvalid[kMaxBeacons];
  __shared__ double cn64[kMaxBeacons];
  __shared__ int cn64_ready;
  __shared__ int degenerate;

  const int e = blockIdx.x;
  const int tid = threadIdx.x;
  const float* cent_e = cent + static_cast<size_t>(e) * nb * D;
  const __nv_bfloat16* q_e = q_new + static_cast<size_t>(e) * nq * D;

  for (int idx = tid; idx < nb * D; idx += kUpdThreads) {
    chat[idx] = cent_e[idx];
    acc[idx] = 0;
  }
  if (tid < kMaxBeacons) add_cnt[tid] = 0;
  if (tid == 0) {
    n_refine = 0;
    cn64_ready = 0;
    degenerate = 0;
  }
  __syncthreads();

  // unit-length screening copies; a beacon qualifies with count > 0 and a non-zero centroid
  {
    const int w = tid >> 5, lane = tid & 31;
    for (int b = w; b < nb; b += kUpdThreads / 32) {
      float n2 = 0.f;
      int nz = 0;
      for (int i = lane; i < D; i += 32) {
        const float c = chat[b * D + i];
        n2 = fmaf(c, c, n2);
        nz |= (c != 0.f);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        n2 += __shfl_xor_sync(0xffffffffu, n2, o);
        nz |= __shfl_xor_sync(0xffffffffu, nz, o);
      }
      const int ok = (counts[static_cast<size_t>(e) * nb + b] > 0) && nz;
      const float inv = rsqrtf(n2);
      for (int i = lane; i < D; i += 32) chat[b * D + i] *= inv;
      if (lane == 0) {
        bvalid[b] = ok;
        if (ok && !(n2 > 1e-30f && n2 < 1e30f)) degenerate = 1;
      }
    }
  }
  __syncthreads();

  const int quad = tid >> 2, sub = tid & 3;
  for (int r0 = 0; r0 < nq; r0 += kChunk) {
    const int rows = min(kChunk, nq - r0);
    // stage the chunk: 16-byte vectors, coalesced
    constexpr int kVecPerRow = D * 2 / 16;
    for (int v = tid; v < rows * kVecPerRow; v += kUpdThreads) {
      const int row = v / kVecPerRow, c = v % kVecPerRow;
      const uint4 x = *reinterpret_cast<const uint4*>(q_e + static_cast<size_t>(r0 + row) * D + c * 8);
      *reinterpret_cast<uint4*>(qs + row * kPitch + c * 8) = x;
    }
    __syncthreads();

    // screening: 4 threads per query, thread `sub` holds dims 4*sub + 16*k + {0..3}
    {
      const bool active = quad < rows;
      float qv[kPer];
      unsigned nz = 0;
      float qn2 = 0.f;
      const __nv_bfloat16* qrow = qs + (active ? quad : 0) * kPitch;
#pragma unroll
      for (int k = 0; k < kPer / 4; ++k) {
        const uint2 raw = *reinterpret_cast<const uint2*>(qrow + 4 * sub + 16 * k);
        nz |= (raw.x | raw.y) & 0x7fff7fffu;
        const __nv_bfloat162 lo = *reinterpret_cast<const __nv_bfloat162*>(&raw.x);
        const __nv_bfloat162 hi = *reinterpret_cast<const __nv_bfloat162*>(&raw.y);
        const float2 a = __bfloat1622float2(lo), b2 = __bfloat1622float2(hi);
        qv[4 * k + 0] = a.x;
        qv[4 * k + 1] = a.y;
        qv[4 * k + 2] = b2.x;
        qv[4 * k + 3] = b2.y;
        qn2 = fmaf(a.x, a.x, fmaf(a.y, a.y, fmaf(b2.x, b2.x, fmaf(b2.y, b2.y, qn2))));
      }
      qn2 += __shfl_xor_sync(0xffffffffu, qn2, 1);
      qn2 += __shfl_xor_sync(0xffffffffu, qn2, 2);
      nz |= __shfl_xor_sync(0xffffffffu, nz, 1);
      nz |= __shfl_xor_sync(0xffffffffu, nz, 2);

      float best = -INFINITY, second = -INFINITY;
      int bi = -1;
      for (int b = 0; b < nb; ++b) {
        if (!bvalid[b]) continue;
        const float* cb = chat + b * D + 4 * sub;
        float dot = 0.f;
#pragma unroll
        for (int k = 0; k < kPer / 4; ++k) {
          const float4 c4 = *reinterpret_cast<const float4*>(cb + 16 * k);
          dot = fmaf(qv[4 * k + 0], c4.x, dot);
          dot = fmaf(qv[4 * k + 1], c4.y, dot);
          dot = fmaf(qv[4 * k + 2], c4.z, dot);
          dot = fmaf(qv[4 * k + 3], c4.w, dot);
        }
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
          a = -2;  // decide exactly below
          refine_idx[atomicAdd(&n_refine, 1)] = quad;
        } else {
          a = bi;
        }
        asg[quad] = a;
      }
    }
    __syncthreads();

    // exact fp64 decisions for close calls (rare)
    if (n_refine > 0) {
      if (!cn64_ready) {
        if (tid < nb) {
          double a = 0.0;
          for (int i = 0; i < D; ++i) {
            const double c = cent_e[tid * D + i];
            a = __dadd_rn(a, __dmul_rn(c, c));
          }
          cn64[tid] = __dsqrt_rn(a);
        }
        __syncthreads();
        if (tid == 0) cn64_ready = 1;
      }
      __syncthreads();
      for (int t = tid; t < n_refine; t += kUpdThreads) {
        const int ql = refine_idx[t];
        const __nv_bfloat16* qrow = qs + ql * kPitch;
        double qq = 0.0;
        for (int i = 0; i < D; ++i) {
          const double x = __bfloat162float(qrow[i]);
          qq = __dadd_rn(qq, __dmul_rn(x, x));
        }
        const double nqd = __dsqrt_rn(qq);
        double b1 = -INFINITY;
        int best_b = -1;
        for (int b = 0; b < nb; ++b) {
          if (!bvalid[b]) continue;
          double dot = 0.0;
          for (int i = 0; i < D; ++i)
            dot = __dadd_rn(dot, __dmul_rn(static_cast<double>(__bfloat162float(qrow[i])),
                                           static_cast<double>(cent_e[b * D + i])));
          const double cs = __ddiv_rn(dot, __dmul_rn(nqd, cn64[b]));
          if (cs > b1) {
            b1 = cs;
            best_b = b;
          }
        }
        asg[ql] = best_b;
      }
      __syncthreads();
      if (tid == 0) n_refine = 0;
    }

    // exact per-call sums: column-owned int64 atomics (order-independent)
    {
      constexpr int kGroups = kUpdThreads / D;
      const int col = tid % D, g = tid / D;
      for (int ql = g; ql < rows; ql += kGroups) {
        const int b = asg[ql];
        if (b >= 0)
          atomicAdd(reinterpret_cast<unsigned long long*>(&acc[b * D + col]),
                    static_cast<unsigned long long>(to_fixed40(qs[ql * kPitch + col])));
      }
      if (tid < rows) {
        const int b = asg[tid];
        if (b >= 0) atomicAdd(&add_cnt[b], 1);
        if (assign_out) assign_out[static_cast<size_t>(e) * nq + r0 + tid] = b;
      }
    }
    __syncthreads();
  }

  // fold the call into the running state
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
  const size_t smem_base = static_cast<size_t>(nb) * s.d * (sizeof(long long) + sizeof(float));
  if (s.d == 128) {
    const size_t smem = smem_base + sizeof(__nv_bfloat16) * kChunk * UpdSmem<128>::kPitch;
    cudaFuncSetAttribute(update_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    update_kernel<128><<<s.n_inst, kUpdThreads, smem, st>>>(q_new, nq, nb, cent, sums, counts, assign_out);
  } else {
    const size_t smem = smem_base + sizeof(__nv_bfloat16) * kChunk * UpdSmem<64>::kPitch;
    cudaFuncSetAttribute(update_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    update_kernel<64><<<s.n_inst, kUpdThreads, smem, st>>>(q_new, nq, nb, cent, sums, counts, assign_out);
  }
  return cudaGetLastError();
}

}  // namespace bkv
