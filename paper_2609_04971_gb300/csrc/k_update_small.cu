// Beacon maintenance for a few queries per instance (Section 3.2, Appendix D):
// the decode-step pattern, where each call brings the queries of one or a few
// generated tokens (Algorithm 2's decode branch), G * n_new <= 32 per instance.
//
// One warp per instance, kSmallWarps instances per CTA, no tensor cores: at a
// handful of rows an instance is too small for the batched kernel's pipeline
// (TMA ring, MMA screening, accumulator and bookkeeping warps), whose
// per-instance handoffs then bound the call.  The warp copies the instance's
// centroids to shared memory, takes each centroid's norm data, and walks the
// queries in order:
//   screening: fp32 dots of q with the unit centroids c / |c| (rsqrtf), summed
//     over the lanes by a butterfly; error far below 1e-4 |q|;
//   decision: the best valid beacon, ties to the lower one; when best and
//     second best differ by at most 1e-4 |q| (or a norm is extreme) the query
//     is re-decided exactly, with the same double-float arithmetic as the
//     batched kernel, so both kernels take the same decisions;
//   sums: per beacon, the rows assigned to it are added as the same three
//     exact fp32 parts, turned into round(sum * 2^40), added once to the fp64
//     running sum, and c = fp32(sum / count) to within one ulp from double-float
//     arithmetic, as in the batched kernel's fold.
// All queries of the call see the centroids as they were at call start.
#include "bkv_device.cuh"
#include "bkv_internal.h"
#include "k_update_math.cuh"

namespace bkv {
namespace {

constexpr int kSmallWarps = 8;

struct SmallArgs {
  int n_inst, nq, nb;
  const __nv_bfloat16* q;  // [n_inst * nq][D] (the G query heads of an instance are adjacent)
  float* cent;             // [n_inst][nb][D]
  double* sums;            // [n_inst][nb][D]
  long long* counts;       // [n_inst][nb]
  int* assign_out;         // [n_inst * nq] or nullptr
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <int D>
__global__ void __launch_bounds__(32 * kSmallWarps) update_small_kernel(SmallArgs a) {
  extern __shared__ __align__(16) float small_cent[];  // [kSmallWarps][nb][D]
  __shared__ DF cninv_sh[kSmallWarps][kMaxBeacons];
  __shared__ float inv_sh[kSmallWarps][kMaxBeacons];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int e = blockIdx.x * kSmallWarps + w;
  if (e >= a.n_inst) return;  // whole warp
  const int nb = a.nb, nq = a.nq;
  float* cs = small_cent + static_cast<size_t>(w) * nb * D;
  const size_t cbase = static_cast<size_t>(e) * nb * D;
  const __nv_bfloat16* qe = a.q + static_cast<size_t>(e) * nq * D;
  const long long cnt_lane = lane < nb ? a.counts[static_cast<size_t>(e) * nb + lane] : 0;  // lane b: beacon b's count
  for (int i = lane; i < nb * D / 4; i += 32)
    reinterpret_cast<float4*>(cs)[i] = reinterpret_cast<const float4*>(a.cent + cbase)[i];
  __syncwarp();

  // ---- norm data of every centroid (the operations of the batched kernel's operand build)
  uint32_t vmask = 0;  // valid beacons: count > 0 and a nonzero centroid
  bool degenerate = false;
  for (int b = 0; b < nb; ++b) {
    float n2 = 0.f;
    DF n2d{0.f, 0.f};
    int nz = 0;
#pragma unroll
    for (int k = 0; k < D / 32; ++k) {
      const float c = cs[b * D + lane + 32 * k];
      n2 = fmaf(c, c, n2);
      n2d = df_add(n2d, df_two_prod(c, c));
      nz |= (c != 0.f);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      n2 += __shfl_xor_sync(0xffffffffu, n2, o);
      nz |= __shfl_xor_sync(0xffffffffu, nz, o);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
      n2d = df_add(n2d, DF{__shfl_xor_sync(0xffffffffu, n2d.hi, o), __shfl_xor_sync(0xffffffffu, n2d.lo, o)});
    const bool ok = __shfl_sync(0xffffffffu, cnt_lane, b) > 0 && nz;
    bool plain = true;
    DF inv_df{0.f, 0.f};
    if (ok) inv_df = centroid_inv_norm(n2d, n2, plain);
    if (lane == 0) {
      cninv_sh[w][b] = inv_df;
      inv_sh[w][b] = ok ? rsqrtf(n2) : 0.f;
    }
    if (ok) vmask |= 1u << b;
    if (!plain) degenerate = true;
  }
  __syncwarp();

  // ---- decisions, against the centroids at call start; lane r keeps query r's beacon
  int my_b = -1;
  for (int r = 0; r < nq; ++r) {
    float x[D / 32];
#pragma unroll
    for (int j = 0; j < D / 32; ++j) x[j] = __bfloat162float(qe[static_cast<size_t>(r) * D + lane + 32 * j]);
    float qn2 = 0.f;
#pragma unroll
    for (int j = 0; j < D / 32; ++j) qn2 = fmaf(x[j], x[j], qn2);
    qn2 = warp_sum(qn2);
    float best = -INFINITY, second = -INFINITY;
    int bi = -1;
    for (int b = 0; b < nb; ++b) {
      if (!((vmask >> b) & 1u)) continue;
      const float inv = inv_sh[w][b];
      float p = 0.f;
#pragma unroll
      for (int j = 0; j < D / 32; ++j) p = fmaf(x[j], cs[b * D + lane + 32 * j] * inv, p);
      p = warp_sum(p);
      if (p > best) {
        second = best;
        best = p;
        bi = b;
      } else if (p > second) {
        second = p;
      }
    }
    int dec = bi;
    if (bi >= 0 && (degenerate || !(qn2 > 1e-30f && qn2 < 1e30f) || !(best - second > kMarginRel * sqrtf(qn2))))
      dec = exact_decision<D>(
          x, nb, [&](int b, int col) { return cs[b * D + col]; }, [&](int b) { return ((vmask >> b) & 1u) != 0; },
          cninv_sh[w]);
    if (a.assign_out && lane == 0) a.assign_out[static_cast<size_t>(e) * nq + r] = dec;
    if (lane == r) my_b = dec;
  }

  // ---- per beacon: exact sum of its rows, added once to the running sum
  for (int b = 0; b < nb; ++b) {
    const uint32_t rows = __ballot_sync(0xffffffffu, lane < nq && my_b == b);
    if (!rows) continue;
    Parts p[D / 32];
#pragma unroll
    for (int j = 0; j < D / 32; ++j) p[j] = Parts{0.f, 0.f, 0.f};
    for (uint32_t m = rows; m; m &= m - 1) {
      const int r = __ffs(m) - 1;
#pragma unroll
      for (int j = 0; j < D / 32; ++j) parts_add(p[j], __bfloat162float(qe[static_cast<size_t>(r) * D + lane + 32 * j]));
    }
    const size_t ci = static_cast<size_t>(e) * nb + b;
    const long long cnt = __shfl_sync(0xffffffffu, cnt_lane, b) + __popc(rows);
    const DF rcp = count_reciprocal(cnt);
#pragma unroll
    for (int j = 0; j < D / 32; ++j) {
      const size_t gi = cbase + static_cast<size_t>(b) * D + lane + 32 * j;
      const double s_new = __dadd_rn(a.sums[gi], fixed40_to_double(fixed40(p[j])));
      a.sums[gi] = s_new;
      a.cent[gi] = centroid_value(s_new, rcp);
    }
    if (lane == 0) a.counts[ci] = cnt;
  }
}

template <int D>
cudaError_t launch_small_d(const SmallArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(float) * kSmallWarps * a.nb * D;
  cudaError_t e = cudaFuncSetAttribute(update_small_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  update_small_kernel<D><<<(a.n_inst + kSmallWarps - 1) / kSmallWarps, 32 * kSmallWarps, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_update_small(const Shape& s, const __nv_bfloat16* q_new, int n_new, float* cent, double* sums,
                                long long* counts, int* assign_out, cudaStream_t st) {
  SmallArgs a{s.n_inst, s.G * n_new, s.nb, q_new, cent, sums, counts, assign_out};
  if (a.n_inst == 0 || a.nq == 0 || a.nb == 0) return cudaSuccess;
  if (a.nq > kUpdateSmallMaxRows || a.nb > kMaxBeacons) return cudaErrorInvalidValue;
  return s.d == 128 ? launch_small_d<128>(a, st) : launch_small_d<64>(a, st);
}

}  // namespace bkv
