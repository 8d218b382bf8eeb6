// Beacon maintenance for a few queries per instance (Section 3.2, Appendix D):
// the decode-step pattern, where each call brings the queries of one or a few
// generated tokens (Algorithm 2's decode branch), G * n_new <= 32 per instance.
//
// One warp per instance, no tensor cores: at a handful of rows an instance is
// too small for the batched kernel's pipeline (TMA ring, MMA screening,
// accumulator and bookkeeping warps), whose per-instance handoffs then bound
// the call.  The warp stages the call's queries in shared memory as fp32 and
// gives each centroid row R = 32 / nb lanes (nb rounded up to a power of two):
//   screening: the R lanes of beacon b stream its row from HBM once, in
//     interleaved 16-byte chunks (adjacent lanes read adjacent chunks), and
//     form its squared norm and its dot with every query (packed fp32
//     multiply-adds, two columns per instruction), added over the R lanes at
//     the end; the screened value of (query r, beacon b) is
//     dot * rsqrtf(|c_b|^2), whose error is far below 1e-4 |q|.  The
//     centroids are never held in shared memory, so every instance of a
//     decode step fits in one wave;
//   decision: lane r scans the screened values of query r in beacon order for
//     the best valid beacon, ties to the lower one; when best and second best
//     differ by at most 1e-4 |q| (or a norm is extreme) the query is re-decided
//     exactly, with the same double-float arithmetic and the same centroid
//     norm data as the batched kernel (built only when a call needs it), so
//     both kernels take the same decisions.  Only beacons screened within
//     2e-4 |q| of the best enter the exact comparison: the screening error is
//     far below 5e-5 |q|, so the exact maximum (and any exact tie with it)
//     lies among them;
//   sums: per touched beacon, the rows assigned to it are added as the same
//     three exact fp32 parts, turned into round(sum * 2^40), added once to the
//     fp64 running sum (fold_sum: exact integer addition and one rounding, no
//     fp64 arithmetic in the common case), and c = fp32(sum / count) to within
//     one ulp from double-float arithmetic, as in the batched kernel's fold.  The running
//     sums of every touched beacon are prefetched into L2 at once.
// All queries of the call see the centroids as they were at call start.
#include "bkv_device.cuh"
#include "bkv_internal.h"
#include "k_update_math.cuh"

namespace bkv {
namespace {

struct SmallArgs {
  int n_inst, nq, nb;
  int lg_rows;             // log2 of the lanes that share one centroid row (32 / nb rounded up to a power of 2)
  const __nv_bfloat16* q;  // [n_inst * nq][D] (the G query heads of an instance are adjacent)
  float* cent;             // [n_inst][nb][D]
  double* sums;            // [n_inst][nb][D]
  long long* counts;       // [n_inst][nb]
  int* assign_out;         // [n_inst * nq] or nullptr
};

// Per-warp shared memory (floats), for at most NQ queries of head_dim D:
//   qs    [NQ][D + 4]   the queries as fp32; the 4-float pad makes the row-per-lane
//                       16-byte reads of the norm pass conflict-free
//   sc    [NQ][33]      screened value of (query r, beacon b) at r * 33 + b
//   cninv [kMaxBeacons] double-float 1 / |c_b| (exact re-decisions only)
//   qn2   [NQ]          the queries' squared norms
template <int D, int NQ>
struct SmallLayout {
  static constexpr int kPitch = D + 4;
  static constexpr int kScPitch = 33;
  static constexpr int kQs = 0;
  static constexpr int kSc = NQ * kPitch;
  static constexpr int kCninv = kSc + NQ * kScPitch;             // even: DF-aligned
  static constexpr int kQn2 = kCninv + 2 * kMaxBeacons;
  static constexpr int kPerWarp = kQn2 + NQ;                      // a multiple of 4: float4-aligned warps
  static constexpr int kWarps = NQ <= 8 ? 8 : 4;
  static_assert(kSc % 4 == 0 && kCninv % 2 == 0 && kPerWarp % 4 == 0, "shared-memory alignment");
};

// Up to this many touched beacons have their running sums loaded at once (all of them are
// prefetched into L2 first).
constexpr int kFoldChunk = 2;

// Packed fp32 (two columns per instruction, low word first): d = a * b + c.
__device__ __forceinline__ unsigned long long fma2(unsigned long long a, unsigned long long b, unsigned long long c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ unsigned long long pack2(float lo, float hi) {
  return static_cast<unsigned long long>(__float_as_uint(lo)) |
         (static_cast<unsigned long long>(__float_as_uint(hi)) << 32);
}
__device__ __forceinline__ float sum2(unsigned long long v) {
  return __uint_as_float(static_cast<uint32_t>(v)) + __uint_as_float(static_cast<uint32_t>(v >> 32));
}

template <int D, int NQ>
__global__ void __launch_bounds__(32 * SmallLayout<D, NQ>::kWarps, NQ <= 8 ? 4 : 2)
    update_small_kernel(SmallArgs a) {
  using Lay = SmallLayout<D, NQ>;
  constexpr int P = Lay::kPitch, SP = Lay::kScPitch;
  extern __shared__ __align__(16) float small_sh[];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int e = blockIdx.x * Lay::kWarps + w;
  if (e >= a.n_inst) return;  // whole warp
  const int nb = a.nb, nq = a.nq;
  float* qs = small_sh + static_cast<size_t>(w) * Lay::kPerWarp + Lay::kQs;
  float* sc = small_sh + static_cast<size_t>(w) * Lay::kPerWarp + Lay::kSc;
  DF* cninv = reinterpret_cast<DF*>(small_sh + static_cast<size_t>(w) * Lay::kPerWarp + Lay::kCninv);
  float* qn2s = small_sh + static_cast<size_t>(w) * Lay::kPerWarp + Lay::kQn2;
  const size_t cbase = static_cast<size_t>(e) * nb * D;
  const __nv_bfloat16* qe = a.q + static_cast<size_t>(e) * nq * D;
  const long long cnt_lane = lane < nb ? a.counts[static_cast<size_t>(e) * nb + lane] : 0;  // lane b: beacon b's count

  // ---- the call's queries, bf16 -> fp32 (exact), 8 values per 16-byte load; rows nq..NQ-1 are zero.
  // A row is D / 8 consecutive lanes' loads, so its squared norm (for the screening margin) is a sum
  // over those lanes: a butterfly over D / 8 lanes, written to qn2 by the row's first lane.
  static_assert(32 % (D / 8) == 0, "a row's loads stay inside one warp");
  for (int i = lane; i < NQ * D / 8; i += 32) {
    const int r = i / (D / 8), c = (i % (D / 8)) * 8;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (r < nq) v = reinterpret_cast<const uint4*>(qe)[i];
    const float4 x0 = make_float4(__uint_as_float(v.x << 16), __uint_as_float(v.x & 0xffff0000u),
                                  __uint_as_float(v.y << 16), __uint_as_float(v.y & 0xffff0000u));
    const float4 x1 = make_float4(__uint_as_float(v.z << 16), __uint_as_float(v.z & 0xffff0000u),
                                  __uint_as_float(v.w << 16), __uint_as_float(v.w & 0xffff0000u));
    float4* dst = reinterpret_cast<float4*>(qs + r * P + c);
    dst[0] = x0;
    dst[1] = x1;
    float p = x0.x * x0.x;
    p = fmaf(x0.y, x0.y, p);
    p = fmaf(x0.z, x0.z, p);
    p = fmaf(x0.w, x0.w, p);
    p = fmaf(x1.x, x1.x, p);
    p = fmaf(x1.y, x1.y, p);
    p = fmaf(x1.z, x1.z, p);
    p = fmaf(x1.w, x1.w, p);
#pragma unroll
    for (int o = 1; o < D / 8; o <<= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
    if ((i % (D / 8)) == 0) qn2s[r] = p;
  }
  __syncwarp();

  // ---- R lanes per centroid row (R = 32 / nb rounded up to a power of two): lane l takes row
  // l / R and its 16-byte chunks l % R, l % R + R, ... (adjacent lanes read adjacent chunks), forming
  // the row's squared norm and its dot with every query; the R partial sums are then added
  const int lg_r = a.lg_rows;
  const int R = 1 << lg_r;
  const int row = lane >> lg_r, part = lane & (R - 1);
  const bool has_row = row < nb;
  const float4* crow = reinterpret_cast<const float4*>(a.cent + cbase + static_cast<size_t>(has_row ? row : 0) * D);
  // packed fp32 accumulators: even columns in the low word, odd ones in the high word
  unsigned long long acc2[NQ];
#pragma unroll
  for (int r = 0; r < NQ; ++r) acc2[r] = 0ull;
  unsigned long long n2p = 0ull;
  int nz = 0;
#pragma unroll(NQ <= 4 ? 4 : 2)
  for (int k = part; k < D / 4; k += R) {
    const float4 c = has_row ? crow[k] : make_float4(0.f, 0.f, 0.f, 0.f);
    const unsigned long long c01 = pack2(c.x, c.y), c23 = pack2(c.z, c.w);
    n2p = fma2(c01, c01, n2p);
    n2p = fma2(c23, c23, n2p);
    nz |= (c.x != 0.f) | (c.y != 0.f) | (c.z != 0.f) | (c.w != 0.f);
#pragma unroll
    for (int r = 0; r < NQ; ++r) {
      const ulonglong2 x = *reinterpret_cast<const ulonglong2*>(qs + r * P + 4 * k);  // R distinct addresses
      acc2[r] = fma2(x.x, c01, acc2[r]);
      acc2[r] = fma2(x.y, c23, acc2[r]);
    }
  }
  float acc[NQ];
#pragma unroll
  for (int r = 0; r < NQ; ++r) acc[r] = sum2(acc2[r]);
  float n2 = sum2(n2p);
  for (int o = 1; o < R; o <<= 1) {
    n2 += __shfl_xor_sync(0xffffffffu, n2, o);
    nz |= __shfl_xor_sync(0xffffffffu, nz, o);
#pragma unroll
    for (int r = 0; r < NQ; ++r) acc[r] += __shfl_xor_sync(0xffffffffu, acc[r], o);
  }
  const long long cnt_row = __shfl_sync(0xffffffffu, cnt_lane, row & 31);  // lane b holds beacon b's count
  const bool valid = has_row && cnt_row > 0 && nz;  // count > 0 and a nonzero centroid
  // every lane takes part in the shuffle (row b's validity from its first lane); lane b < nb votes it
  const bool valid_b = __shfl_sync(0xffffffffu, valid, (lane << lg_r) & 31);
  const uint32_t vmask = __ballot_sync(0xffffffffu, lane < nb && valid_b);
  const bool degenerate = __any_sync(0xffffffffu, valid && !(n2 > 1e-30f && n2 < 1e30f));
  const float inv = valid ? rsqrtf(n2) : 0.f;
  if (part == 0) {
#pragma unroll
    for (int r = 0; r < NQ; ++r)
      if (r < nq) sc[r * SP + row] = valid ? acc[r] * inv : -INFINITY;
  }
  __syncwarp();

  // ---- lane r: decision for query r against the centroids at call start
  int dec = -1;
  bool need_exact = false;
  uint32_t cand = 0;  // candidate beacons of an exact re-decision (lane r: query r)
  if (lane < nq) {
    const float qn2 = qn2s[lane];
    float best = -INFINITY, second = -INFINITY;
    for (int b = 0; b < nb; ++b) {
      if (!((vmask >> b) & 1u)) continue;
      const float p = sc[lane * SP + b];
      if (p > best) {
        second = best;
        best = p;
        dec = b;
      } else if (p > second) {
        second = p;
      }
    }
    const bool wild = degenerate || !(qn2 > 1e-30f && qn2 < 1e30f);
    // with a valid beacon but no screened best (every value NaN: an extreme norm), best - second is NaN
    need_exact = vmask != 0u && (wild || !(best - second > kMarginRel * sqrtf(qn2)));
    // Candidates for the exact decision: a screened value is within kMarginRel |q| / 2 of the exact
    // one, so only beacons screened within 2 kMarginRel |q| of the best can have the largest exact
    // value (or tie with it); with an extreme norm every valid beacon is a candidate.
    if (need_exact) {
      if (wild) {
        cand = vmask;
      } else {
        const float floor_v = best - 2.f * kMarginRel * sqrtf(qn2);
        for (int b = 0; b < nb; ++b)
          if (((vmask >> b) & 1u) && sc[lane * SP + b] >= floor_v) cand |= 1u << b;
      }
    }
  }

  // ---- close calls: exact re-decisions, with the batched kernel's centroid norm data
  const uint32_t need = __ballot_sync(0xffffffffu, need_exact);
  const uint32_t cand_any = __reduce_or_sync(0xffffffffu, cand);  // beacons whose norm data is needed
  if (need) {
    for (int b = 0; b < nb; ++b) {
      if (!((cand_any >> b) & 1u)) continue;  // warp-uniform
      float n2b = 0.f;
      DF n2d{0.f, 0.f};
#pragma unroll
      for (int k = 0; k < D / 32; ++k) {
        const float c = a.cent[cbase + static_cast<size_t>(b) * D + lane + 32 * k];
        n2b = fmaf(c, c, n2b);
        n2d = df_add(n2d, df_two_prod(c, c));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) n2b += __shfl_xor_sync(0xffffffffu, n2b, o);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1)
        n2d = df_add(n2d, DF{__shfl_xor_sync(0xffffffffu, n2d.hi, o), __shfl_xor_sync(0xffffffffu, n2d.lo, o)});
      bool plain = true;
      const DF inv_df = centroid_inv_norm(n2d, n2b, plain);
      if (lane == 0) cninv[b] = inv_df;
    }
    __syncwarp();
    for (uint32_t m = need; m; m &= m - 1) {
      const int r = __ffs(m) - 1;
      const uint32_t cand_r = __shfl_sync(0xffffffffu, cand, r);
      float x[D / 32];
#pragma unroll
      for (int j = 0; j < D / 32; ++j) x[j] = qs[r * P + lane + 32 * j];
      const int d = exact_decision<D>(
          x, nb, [&](int b, int col) { return a.cent[cbase + static_cast<size_t>(b) * D + col]; },
          [&](int b) { return ((cand_r >> b) & 1u) != 0; }, cninv);
      if (lane == r) dec = d;
    }
  }
  if (a.assign_out && lane < nq) a.assign_out[static_cast<size_t>(e) * nq + lane] = dec;

  // ---- per touched beacon: exact sum of its rows, added once to the running sum
  uint32_t touched = __reduce_or_sync(0xffffffffu, dec >= 0 ? (1u << dec) : 0u);
  for (uint32_t m = touched; m; m &= m - 1) {
    const double* srow = a.sums + cbase + static_cast<size_t>(__ffs(m) - 1) * D + lane;
#pragma unroll
    for (int j = 0; j < D / 32; ++j) asm volatile("prefetch.global.L2 [%0];" ::"l"(srow + 32 * j));
  }
  while (touched) {
    int bs[kFoldChunk];
    int nbk = 0;
#pragma unroll
    for (int i = 0; i < kFoldChunk; ++i) {
      bs[i] = touched ? __ffs(touched) - 1 : 0;
      if (touched) {
        touched &= touched - 1;
        nbk = i + 1;
      }
    }
    double s_old[kFoldChunk][D / 32];
#pragma unroll
    for (int i = 0; i < kFoldChunk; ++i)
#pragma unroll
      for (int j = 0; j < D / 32; ++j)
        s_old[i][j] = i < nbk ? a.sums[cbase + static_cast<size_t>(bs[i]) * D + lane + 32 * j] : 0.0;
#pragma unroll
    for (int i = 0; i < kFoldChunk; ++i) {
      if (i >= nbk) break;  // warp-uniform
      const int b = bs[i];
      const uint32_t rows = __ballot_sync(0xffffffffu, lane < nq && dec == b);
      long long acc[D / 32];
      if (__popc(rows) == 1) {  // one query (the common case): its fixed-point value directly
        const int r = __ffs(rows) - 1;
#pragma unroll
        for (int j = 0; j < D / 32; ++j) acc[j] = fixed40_one(qs[r * P + lane + 32 * j]);
      } else {
        Parts p[D / 32];
#pragma unroll
        for (int j = 0; j < D / 32; ++j) p[j] = Parts{0.f, 0.f, 0.f};
        for (uint32_t m = rows; m; m &= m - 1) {
          const int r = __ffs(m) - 1;
#pragma unroll
          for (int j = 0; j < D / 32; ++j) parts_add(p[j], qs[r * P + lane + 32 * j]);
        }
#pragma unroll
        for (int j = 0; j < D / 32; ++j) acc[j] = fixed40_few(p[j]);
      }
      const long long cnt = __shfl_sync(0xffffffffu, cnt_lane, b) + __popc(rows);
      const DF rcp = count_reciprocal(cnt);
#pragma unroll
      for (int j = 0; j < D / 32; ++j) {
        const size_t gi = cbase + static_cast<size_t>(b) * D + lane + 32 * j;
        const double s_new = fold_sum(s_old[i][j], acc[j]);
        a.sums[gi] = s_new;
        a.cent[gi] = centroid_value(s_new, rcp);
      }
      if (lane == 0) a.counts[static_cast<size_t>(e) * nb + b] = cnt;
    }
  }
}

template <int D, int NQ>
cudaError_t launch_small_dq(const SmallArgs& a, cudaStream_t st) {
  using Lay = SmallLayout<D, NQ>;
  const size_t smem = sizeof(float) * Lay::kWarps * Lay::kPerWarp;
  cudaError_t e = cudaFuncSetAttribute(update_small_kernel<D, NQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  update_small_kernel<D, NQ><<<(a.n_inst + Lay::kWarps - 1) / Lay::kWarps, 32 * Lay::kWarps, smem, st>>>(a);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_small_d(const SmallArgs& a, cudaStream_t st) {
  if (a.nq <= 4) return launch_small_dq<D, 4>(a, st);
  if (a.nq <= 8) return launch_small_dq<D, 8>(a, st);
  if (a.nq <= 16) return launch_small_dq<D, 16>(a, st);
  return launch_small_dq<D, 32>(a, st);
}

}  // namespace

cudaError_t launch_update_small(const Shape& s, const __nv_bfloat16* q_new, int n_new, float* cent, double* sums,
                                long long* counts, int* assign_out, cudaStream_t st) {
  int lg = 0;
  while ((32 >> (lg + 1)) >= s.nb && lg < 3) ++lg;  // 2^lg lanes per row, 2^lg * nb <= 32
  SmallArgs a{s.n_inst, s.G * n_new, s.nb, lg, q_new, cent, sums, counts, assign_out};
  if (a.n_inst == 0 || a.nq == 0 || a.nb == 0) return cudaSuccess;
  if (a.nq > kUpdateSmallMaxRows || a.nb > kMaxBeacons) return cudaErrorInvalidValue;
  return s.d == 128 ? launch_small_d<128>(a, st) : launch_small_d<64>(a, st);
}

}  // namespace bkv
