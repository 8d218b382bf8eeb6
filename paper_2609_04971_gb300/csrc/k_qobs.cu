// Observation queries of every GQA group (Section 4.3; Appendix D.2):
// recent queries rotated to their own positions, beacons rotated to the
// current step, each rounded to bf16 for the tensor-core scoring.
//
// Layout written: qobs bf16 [n_inst][n_obs_pad][d]; rows h*W + w are recent
// slot w of query head h, rows G*W + b are beacon b, rows >= n_obs are zero.
// valid [n_inst][4] is a 128-bit mask of rows that take part in the maximum
// (all recent rows, beacons with count > 0).
//
// Definition of each output element: y_i = x_i c - x_{i+d/2} s and
// y_{i+d/2} = x_{i+d/2} c + x_i s evaluated in fp64 (separately rounded
// products, host-computed fp64 cos / sin), then rounded fp64 -> fp32 -> bf16.
// The kernel first evaluates y in fp32 (one FMA, fp32 copies of cos / sin).
// The fp32 value v differs from the fp64 one by at most
//   delta = 2^-22 (|x_a| + |x_b| + |v|)
// (rounding of cos and sin to fp32, of the product and of the FMA, with a
// factor 2 of margin).  The composite rounding can only change where the fp32
// value crosses a bf16 rounding midpoint (low 16 bits 0x8000) or lands within
// one fp32 ulp of it; if v is farther than delta + 1 ulp from the nearest
// midpoint, bf16(v) is the defined value.  Otherwise (about 2e-4 of the
// elements) the element is recomputed in fp64 exactly as defined.
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kQobsThreads = 256;

// Exact definition: fp64 products, fp64 sum, then fp32, then bf16.
__device__ __forceinline__ __nv_bfloat16 rot_exact(double xa, double xb, double c, double s, bool plus) {
  const double y = plus ? __dadd_rn(__dmul_rn(xa, c), __dmul_rn(xb, s)) : __dsub_rn(__dmul_rn(xa, c), __dmul_rn(xb, s));
  return __float2bfloat16_rn(__double2float_rn(y));
}

// bf16 of (xa*c +- xb*s) through the fp32 fast path when provably equal to the definition; the
// fp64 (cos, sin) pair `cs` is read only on the exact path.
__device__ __forceinline__ __nv_bfloat16 rot_fast(float xa, float xb, float c32, float s32, const double2* cs,
                                                   bool plus) {
  const float p = xb * s32;
  const float v = fmaf(xa, c32, plus ? p : -p);
  const uint32_t t = __float_as_uint(v);
  const uint32_t ex = t & 0x7f800000u;
  if (ex >= (25u << 23) && ex != 0x7f800000u) {
    const float ulp = __uint_as_float(ex - (23u << 23));
    const float delta = 0x1p-22f * (fabsf(xa) + fabsf(xb) + fabsf(v));
    const int dist = abs(static_cast<int>(t & 0xffffu) - 0x8000);
    if (static_cast<float>(dist - 1) * ulp > delta) return __float2bfloat16_rn(v);
  }
  const double2 c = *cs;
  return rot_exact(xa, xb, c.x, c.y, plus);
}

// work / n_work (per-instance lengths): block w builds instance work[w] when w < *n_work; rope_row: the
// distance between two batch rows' rotary tables (0: one table for every instance).
__global__ void __launch_bounds__(kQobsThreads) qobs_kernel(Shape s, const __nv_bfloat16* __restrict__ q_recent,
                                                             const float* __restrict__ cent,
                                                             const long long* __restrict__ counts,
                                                             const double2* __restrict__ rope_all, size_t rope_row,
                                                             int rotate, const int* __restrict__ work,
                                                             const int* __restrict__ n_work,
                                                             __nv_bfloat16* __restrict__ qobs,
                                                             uint32_t* __restrict__ valid, int* err) {
  int e = blockIdx.x;
  if (work) {
    if (e >= *n_work) return;  // whole block
    e = work[e];
    if (!in_bounds(e, s.n_inst, err)) return;  // whole block: every thread read the same entry
  }
  const int d = s.d, h = d / 2, h4 = h / 4;
  const int GW = s.G * s.W;
  const double2* rope = rope_all + (rope_row ? static_cast<size_t>((e / s.n_kv) % s.batch) * rope_row : 0);
  const float2* rope32 = reinterpret_cast<const float2*>(rope + static_cast<size_t>(s.W + 1) * h);
  __nv_bfloat16* out = qobs + static_cast<size_t>(e) * s.n_obs_pad * d;
  for (int idx = threadIdx.x; idx < s.n_obs_pad * h4; idx += blockDim.x) {
    const int row = idx / h4, i = (idx % h4) * 4;
    float xa[4] = {0.f, 0.f, 0.f, 0.f}, xb[4] = {0.f, 0.f, 0.f, 0.f};
    int slot = 0;
    if (row < GW) {
      const __nv_bfloat16* src = q_recent + (static_cast<size_t>(e) * GW + row) * d;
      const uint2 a = *reinterpret_cast<const uint2*>(src + i);
      const uint2 b = *reinterpret_cast<const uint2*>(src + i + h);
      const float2 a0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&a.x));
      const float2 a1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&a.y));
      const float2 b0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&b.x));
      const float2 b1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&b.y));
      xa[0] = a0.x; xa[1] = a0.y; xa[2] = a1.x; xa[3] = a1.y;
      xb[0] = b0.x; xb[1] = b0.y; xb[2] = b1.x; xb[3] = b1.y;
      slot = row % s.W;
    } else if (row < s.n_obs) {
      const float* src = cent + (static_cast<size_t>(e) * s.nb + (row - GW)) * d;
      const float4 a = *reinterpret_cast<const float4*>(src + i);
      const float4 b = *reinterpret_cast<const float4*>(src + i + h);
      xa[0] = a.x; xa[1] = a.y; xa[2] = a.z; xa[3] = a.w;
      xb[0] = b.x; xb[1] = b.y; xb[2] = b.z; xb[3] = b.w;
      slot = s.W;
    }
    __nv_bfloat16 y1[4], y2[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (row < s.n_obs && rotate) {
        const float2 cs32 = rope32[slot * h + i + k];
        const double2* cs64 = rope + slot * h + i + k;
        y1[k] = rot_fast(xa[k], xb[k], cs32.x, cs32.y, cs64, false);
        y2[k] = rot_fast(xb[k], xa[k], cs32.x, cs32.y, cs64, true);
      } else {
        y1[k] = __float2bfloat16_rn(xa[k]);
        y2[k] = __float2bfloat16_rn(xb[k]);
      }
    }
    *reinterpret_cast<uint2*>(out + row * d + i) = *reinterpret_cast<const uint2*>(y1);
    *reinterpret_cast<uint2*>(out + row * d + i + h) = *reinterpret_cast<const uint2*>(y2);
  }
  if (threadIdx.x < 128) {  // warp w builds mask word w: one row per lane, loads in parallel
    const int row = threadIdx.x;
    bool v = row < GW;
    if (!v && row < s.n_obs) v = counts[static_cast<size_t>(e) * s.nb + (row - GW)] > 0;
    const uint32_t m = __ballot_sync(0xffffffffu, v);
    if ((threadIdx.x & 31) == 0) valid[e * 4 + (threadIdx.x >> 5)] = m;
  }
}

// Copies one compress's rotary table from pinned host memory, read through its
// device mapping, into device memory.  The copy is made by the SMs rather than
// a copy engine, so the stream's kernels never wait in a copy-engine queue
// behind bulk host transfers that other streams have issued.
__global__ void __launch_bounds__(256) rope_stage_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst,
                                                         int n16) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n16) dst[i] = src[i];
}

}  // namespace

cudaError_t launch_rope_stage(const void* src, void* dst, size_t bytes, cudaStream_t st) {
  if (bytes == 0) return cudaSuccess;
  if (bytes % 16 != 0 || (reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) % 16 != 0)
    return cudaErrorInvalidValue;
  const int n16 = static_cast<int>(bytes / 16);
  rope_stage_kernel<<<(n16 + 255) / 256, 256, 0, st>>>(static_cast<const uint4*>(src), static_cast<uint4*>(dst), n16);
  return cudaGetLastError();
}

cudaError_t launch_qobs(const Shape& s, const __nv_bfloat16* q_recent, const float* cent, const long long* counts,
                        const double2* rope, int rotate, __nv_bfloat16* qobs, uint32_t* valid, int* err,
                        cudaStream_t st) {
  qobs_kernel<<<s.n_inst, kQobsThreads, 0, st>>>(s, q_recent, cent, counts, rope, 0, rotate, nullptr, nullptr, qobs,
                                                 valid, err);
  return cudaGetLastError();
}

cudaError_t launch_qobs_ragged(const Shape& s, const __nv_bfloat16* q_recent, const float* cent,
                               const long long* counts, const double2* rope, size_t rope_row, int rotate,
                               const int* work, const int* n_work, __nv_bfloat16* qobs, uint32_t* valid, int* err,
                               cudaStream_t st) {
  qobs_kernel<<<s.n_inst, kQobsThreads, 0, st>>>(s, q_recent, cent, counts, rope, rope_row, rotate, work, n_work,
                                                 qobs, valid, err);
  return cudaGetLastError();
}

}  // namespace bkv
