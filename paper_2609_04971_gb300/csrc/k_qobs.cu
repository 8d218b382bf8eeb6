// Observation queries of every GQA group (Section 4.3; Appendix D.2):
// recent queries rotated to their own positions, beacons rotated to the
// current step, each rounded to bf16 for the tensor-core scoring.
//
// Layout written: qobs bf16 [n_inst][n_obs_pad][d]; rows h*W + w are recent
// slot w of query head h, rows G*W + b are beacon b, rows >= n_obs are zero.
// valid [n_inst][4] is a 128-bit mask of rows that take part in the maximum
// (all recent rows, beacons with count > 0).
//
// The rotation y_i = x_i c - x_{i+d/2} s, y_{i+d/2} = x_{i+d/2} c + x_i s is
// evaluated in fp64 with separately rounded products (no fused
// multiply-add) from host-computed fp64 cos / sin, then rounded fp64 -> fp32
// -> bf16, so every scoring query is the correctly defined bf16 value.
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kQobsThreads = 256;

__global__ void __launch_bounds__(kQobsThreads) qobs_kernel(Shape s, const __nv_bfloat16* __restrict__ q_recent,
                                                             const float* __restrict__ cent,
                                                             const long long* __restrict__ counts,
                                                             const double2* __restrict__ rope, int rotate,
                                                             __nv_bfloat16* __restrict__ qobs,
                                                             uint32_t* __restrict__ valid) {
  const int e = blockIdx.x;
  const int d = s.d, h = d / 2;
  const int GW = s.G * s.W;
  __nv_bfloat16* out = qobs + static_cast<size_t>(e) * s.n_obs_pad * d;
  for (int idx = threadIdx.x; idx < s.n_obs_pad * h; idx += blockDim.x) {
    const int row = idx / h, i = idx % h;
    float y1 = 0.f, y2 = 0.f;
    if (row < s.n_obs) {
      double x1, x2;
      int slot;
      if (row < GW) {
        const __nv_bfloat16* src = q_recent + (static_cast<size_t>(e) * GW + row) * d;
        x1 = __bfloat162float(src[i]);
        x2 = __bfloat162float(src[i + h]);
        slot = row % s.W;
      } else {
        const float* src = cent + (static_cast<size_t>(e) * s.nb + (row - GW)) * d;
        x1 = src[i];
        x2 = src[i + h];
        slot = s.W;
      }
      if (rotate) {
        const double2 cs = rope[slot * h + i];
        y1 = __double2float_rn(__dsub_rn(__dmul_rn(x1, cs.x), __dmul_rn(x2, cs.y)));
        y2 = __double2float_rn(__dadd_rn(__dmul_rn(x2, cs.x), __dmul_rn(x1, cs.y)));
      } else {
        y1 = static_cast<float>(x1);
        y2 = static_cast<float>(x2);
      }
    }
    out[row * d + i] = __float2bfloat16_rn(y1);
    out[row * d + i + h] = __float2bfloat16_rn(y2);
  }
  if (threadIdx.x < 4) {
    uint32_t m = 0;
    for (int bit = 0; bit < 32; ++bit) {
      const int row = threadIdx.x * 32 + bit;
      bool v = row < GW;
      if (!v && row < s.n_obs) v = counts[static_cast<size_t>(e) * s.nb + (row - GW)] > 0;
      if (v) m |= 1u << bit;
    }
    valid[e * 4 + threadIdx.x] = m;
  }
}

}  // namespace

cudaError_t launch_qobs(const Shape& s, const __nv_bfloat16* q_recent, const float* cent, const long long* counts,
                        const double2* rope, int rotate, __nv_bfloat16* qobs, uint32_t* valid, cudaStream_t st) {
  qobs_kernel<<<s.n_inst, kQobsThreads, 0, st>>>(s, q_recent, cent, counts, rope, rotate, qobs, valid);
  return cudaGetLastError();
}

}  // namespace bkv
