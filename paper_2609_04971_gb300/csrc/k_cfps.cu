// Continual FPS beacon maintenance (Section 4.2, Eq. 9): each query head keeps
// a bounded buffer of pre-RoPE queries that is compressed by Farthest Point
// Sampling (Appendix D.1, Algorithm 1) whenever it fills; Algorithm 2's
// decode branch, its beacon freeze and its post-eviction merge.
//
// One warp per query head, kHeadsPerCta heads per CTA.  A head's buffer (at
// most 32 rows) sits transposed in shared memory as bf16 [d][kPitch] with its
// fp32 Gram matrix; lane j owns buffer row j.  The dot product of a new row
// with row j is a fused multiply-add chain in element order, run by lane j;
// the similarities are fp32 (cos = dot / (|a| |b|), 0 when a norm is 0) and
// the farthest-point loop takes its argmins in the same precision and order
// as the definition, ties to the lowest row.  These are the operations the
// fp32 decisions of the reference are defined by, so both pick the same rows.
//
// The same warp routine serves three calls:
//   update   append the call's queries in order; whenever the buffer holds
//            b_max = b_min + window rows, replace it by the FPS selection of
//            b_min of them, in pick order;
//   beacons  the beacons of a compress: the FPS selection of min(b_min, size)
//            buffer rows, written as fp32 rows with count 1 (count 0 and a
//            zero row for an empty slot) for the scoring-query build;
//   merge    after an eviction the buffer becomes the FPS selection of b_min
//            rows of (the beacons, then the head's window queries in order).
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kHeadsPerCta = 8;
constexpr int kMaxRows = kCfpsMaxRows;  // 32: one buffer row per lane
constexpr int kChunk = 16;              // rows added to the Gram matrix per pass
constexpr int kPitch = 34;              // bf16 elements per transposed row (even; spreads banks)

template <int D>
struct WarpSmem {
  __nv_bfloat16 xt[D][kPitch];          // buffer, transposed: xt[k][j] = element k of row j
  __align__(16) float xn[D][kChunk];    // the rows being added, fp32, for broadcast reads
  float G[kMaxRows][kMaxRows + 1];      // Gram matrix of the buffer rows
  int picks[kMaxRows];
};

__device__ __forceinline__ float cos_of(float dot, float ni, float nj) {
  return (ni == 0.f || nj == 0.f) ? 0.f : __fdiv_rn(dot, __fmul_rn(ni, nj));
}

// Warp-wide argmin of (v, lane), ties to the lower lane.
__device__ __forceinline__ int warp_argmin(float v) {
  int i = threadIdx.x & 31;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (ov < v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
    }
  }
  return i;
}

// Row `slot` of the buffer from `kPer` = D / 32 consecutive bf16 (or fp32) values per lane.
template <int D>
__device__ __forceinline__ void put_row(WarpSmem<D>& w, int slot, int u, const float (&v)[D / 32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int e = 0; e < D / 32; ++e) {
    const int k = lane * (D / 32) + e;
    w.xt[k][slot] = __float2bfloat16_rn(v[e]);  // exact: v holds a bf16 value
    w.xn[k][u] = v[e];
  }
}

template <int D>
__device__ __forceinline__ void load_bf16_row(const __nv_bfloat16* src, float (&v)[D / 32]) {
  const int lane = threadIdx.x & 31;
  if constexpr (D == 128) {
    const uint2 p = *reinterpret_cast<const uint2*>(src + lane * 4);
    v[0] = __uint_as_float(p.x << 16);
    v[1] = __uint_as_float(p.x & 0xffff0000u);
    v[2] = __uint_as_float(p.y << 16);
    v[3] = __uint_as_float(p.y & 0xffff0000u);
  } else {
    const uint32_t p = *reinterpret_cast<const uint32_t*>(src + lane * 2);
    v[0] = __uint_as_float(p << 16);
    v[1] = __uint_as_float(p & 0xffff0000u);
  }
}

template <int D>
__device__ __forceinline__ void load_f32_row(const float* src, float (&v)[D / 32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int e = 0; e < D / 32; ++e) v[e] = src[lane * (D / 32) + e];
}

// Gram entries of the staged rows [sz0, sz0 + cnt) with every row [0, sz0 + cnt).
template <int D>
__device__ void gram_add(WarpSmem<D>& w, int sz0, int cnt) {
  const int j = threadIdx.x & 31;
  __syncwarp();
  float acc[kChunk];
#pragma unroll
  for (int u = 0; u < kChunk; ++u) acc[u] = 0.f;
#pragma unroll 4
  for (int k = 0; k < D; ++k) {
    const float xj = __bfloat162float(w.xt[k][j]);
    const float4* xr = reinterpret_cast<const float4*>(&w.xn[k][0]);
#pragma unroll
    for (int q = 0; q < kChunk / 4; ++q) {
      const float4 a = xr[q];
      acc[4 * q + 0] = __fmaf_rn(a.x, xj, acc[4 * q + 0]);
      acc[4 * q + 1] = __fmaf_rn(a.y, xj, acc[4 * q + 1]);
      acc[4 * q + 2] = __fmaf_rn(a.z, xj, acc[4 * q + 2]);
      acc[4 * q + 3] = __fmaf_rn(a.w, xj, acc[4 * q + 3]);
    }
  }
  if (j < sz0 + cnt) {
#pragma unroll
    for (int u = 0; u < kChunk; ++u)
      if (u < cnt) {
        w.G[sz0 + u][j] = acc[u];
        w.G[j][sz0 + u] = acc[u];
      }
  }
  __syncwarp();
}

// Algorithm 1 on the first n buffer rows; picks min(m, n) rows into w.picks.
template <int D>
__device__ int fps_rows(WarpSmem<D>& w, int n, int m) {
  const int j = threadIdx.x & 31;
  if (m > n) m = n;
  const float nj = j < n ? __fsqrt_rn(w.G[j][j]) : 0.f;
  float sum = 0.f;
  for (int i = 0; i < n; ++i) {
    const float ni = __shfl_sync(0xffffffffu, nj, i);
    sum = __fadd_rn(sum, cos_of(w.G[i][j], ni, nj));
  }
  const float avg = j < n ? __fdiv_rn(sum, static_cast<float>(n)) : INFINITY;
  int r = warp_argmin(avg);
  if (j == 0) w.picks[0] = r;
  bool sel = j == r;
  float nr = __shfl_sync(0xffffffffu, nj, r);
  float S = cos_of(w.G[r][j], nr, nj);
  for (int k = 1; k < m; ++k) {
    r = warp_argmin((j < n && !sel) ? S : INFINITY);
    if (j == 0) w.picks[k] = r;
    if (j == r) sel = true;
    nr = __shfl_sync(0xffffffffu, nj, r);
    const float c = cos_of(w.G[r][j], nr, nj);
    if (!sel && c > S) S = c;
  }
  __syncwarp();
  return m;
}

// The buffer becomes its rows picks[0 .. m), in that order (rows and Gram entries).
template <int D>
__device__ void keep_picks(WarpSmem<D>& w, int m) {
  const int t = threadIdx.x & 31;
  const int src = t < m ? w.picks[t] : 0;
  for (int k = 0; k < D; ++k) {
    const __nv_bfloat16 v = w.xt[k][src];
    __syncwarp();
    if (t < m) w.xt[k][t] = v;
    __syncwarp();
  }
  float g[kMaxRows];
#pragma unroll
  for (int q = 0; q < kMaxRows; ++q) g[q] = (q < m && t < m) ? w.G[w.picks[q]][src] : 0.f;
  __syncwarp();
  if (t < m)
#pragma unroll
    for (int q = 0; q < kMaxRows; ++q)
      if (q < m) w.G[q][t] = g[q];
  __syncwarp();
}

template <int D>
__device__ void store_buffer(WarpSmem<D>& w, int n, __nv_bfloat16* dst) {
  const int lane = threadIdx.x & 31;
  for (int t = 0; t < n; ++t) {
    if constexpr (D == 128) {
      const int k = lane * 4;
      const uint32_t a = __bfloat16_as_ushort(w.xt[k][t]) | (static_cast<uint32_t>(__bfloat16_as_ushort(w.xt[k + 1][t])) << 16);
      const uint32_t b =
          __bfloat16_as_ushort(w.xt[k + 2][t]) | (static_cast<uint32_t>(__bfloat16_as_ushort(w.xt[k + 3][t])) << 16);
      *reinterpret_cast<uint2*>(dst + static_cast<size_t>(t) * D + k) = make_uint2(a, b);
    } else {
      const int k = lane * 2;
      const uint32_t a = __bfloat16_as_ushort(w.xt[k][t]) | (static_cast<uint32_t>(__bfloat16_as_ushort(w.xt[k + 1][t])) << 16);
      *reinterpret_cast<uint32_t*>(dst + static_cast<size_t>(t) * D + k) = a;
    }
  }
}

template <int D>
__global__ void __launch_bounds__(32 * kHeadsPerCta) cfps_kernel(CfpsArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x * kHeadsPerCta + wid;
  if (h >= a.H) return;  // whole warp
  WarpSmem<D>& w = reinterpret_cast<WarpSmem<D>*>(smem_raw)[wid];
  __nv_bfloat16* buf = a.buf + static_cast<size_t>(h) * a.b_max * D;
  float* bcn = a.bcn + static_cast<size_t>(h) * a.b_min * D;
  long long* bcnt = a.bcnt + static_cast<size_t>(h) * a.b_min;
  float v[D / 32];

  if (a.mode == kCfpsUpdate) {
    // rows to append, in order: the buffer's own rows (its Gram is rebuilt), then the new queries
    const int n_old = a.size[h];
    const int total = n_old + a.n_q;
    const __nv_bfloat16* qn = a.q + static_cast<size_t>(h) * a.n_q * D;
    int sz = 0, next = 0;
    while (next < total) {
      const int add = min(a.b_max - sz, total - next);
      for (int c0 = 0; c0 < add; c0 += kChunk) {
        const int cnt = min(kChunk, add - c0);
        for (int u = 0; u < kChunk; ++u) {
          const int src = next + c0 + u;
          if (u < cnt) {
            load_bf16_row<D>(src < n_old ? buf + static_cast<size_t>(src) * D : qn + static_cast<size_t>(src - n_old) * D,
                             v);
          } else {
#pragma unroll
            for (int e = 0; e < D / 32; ++e) v[e] = 0.f;
          }
          if (u < cnt) {
            put_row<D>(w, sz + c0 + u, u, v);
          } else {
#pragma unroll
            for (int e = 0; e < D / 32; ++e) w.xn[lane * (D / 32) + e][u] = 0.f;
          }
        }
        gram_add<D>(w, sz + c0, cnt);
      }
      sz += add;
      next += add;
      if (sz == a.b_max) {
        const int m = fps_rows<D>(w, sz, a.b_min);
        keep_picks<D>(w, m);
        sz = m;
      }
    }
    store_buffer<D>(w, sz, buf);
    if (lane == 0) a.size[h] = sz;
    return;
  }

  // beacons / merge: gather the candidate rows (at most b_max of them)
  int n = 0;
  if (a.mode == kCfpsBeacons) {
    n = a.size[h];
  } else {
    int nbc = 0;
    for (int t = 0; t < a.b_min; ++t) nbc += bcnt[t] != 0;
    n = nbc + a.n_q;
  }
  const __nv_bfloat16* qr = a.q ? a.q + static_cast<size_t>(h) * a.n_q * D : nullptr;
  const int nbc = n - (a.mode == kCfpsMerge ? a.n_q : 0);
  for (int c0 = 0; c0 < n; c0 += kChunk) {
    const int cnt = min(kChunk, n - c0);
    for (int u = 0; u < kChunk; ++u) {
      const int src = c0 + u;
      if (u < cnt) {
        if (a.mode == kCfpsBeacons) {
          load_bf16_row<D>(buf + static_cast<size_t>(src) * D, v);
        } else if (src < nbc) {
          load_f32_row<D>(bcn + static_cast<size_t>(src) * D, v);
        } else {
          load_bf16_row<D>(qr + static_cast<size_t>(src - nbc) * D, v);
        }
        put_row<D>(w, src, u, v);
      } else {
#pragma unroll
        for (int e = 0; e < D / 32; ++e) w.xn[lane * (D / 32) + e][u] = 0.f;
      }
    }
    gram_add<D>(w, c0, cnt);
  }
  const int m = n > 0 ? fps_rows<D>(w, n, a.b_min) : 0;
  if (a.mode == kCfpsBeacons) {
    for (int t = 0; t < a.b_min; ++t) {
      const int row = t < m ? w.picks[t] : 0;
#pragma unroll
      for (int e = 0; e < D / 32; ++e) {
        const int k = lane * (D / 32) + e;
        bcn[static_cast<size_t>(t) * D + k] = t < m ? __bfloat162float(w.xt[k][row]) : 0.f;
      }
      if (lane == 0) bcnt[t] = t < m ? 1 : 0;
    }
  } else {
    keep_picks<D>(w, m);
    store_buffer<D>(w, m, buf);
    if (lane == 0) a.size[h] = m;
  }
}

// Buffer seeded from FPS picks written as fp32 rows by the prefill seeding kernel.
template <int D>
__global__ void cfps_seed_kernel(const float* __restrict__ rows, int H, int b_min, int b_max,
                                 __nv_bfloat16* __restrict__ buf, int* __restrict__ size) {
  const size_t n = static_cast<size_t>(H) * b_min * D;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const size_t h = i / (static_cast<size_t>(b_min) * D), r = i % (static_cast<size_t>(b_min) * D);
    buf[h * b_max * D + r] = __float2bfloat16_rn(rows[i]);  // exact: the rows are bf16 queries
  }
  for (int h = blockIdx.x * blockDim.x + threadIdx.x; h < H; h += gridDim.x * blockDim.x) size[h] = b_min;
}

template <int D>
cudaError_t launch_cfps_d(const CfpsArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(WarpSmem<D>) * kHeadsPerCta;
  cudaError_t e = cudaFuncSetAttribute(cfps_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int grid = (a.H + kHeadsPerCta - 1) / kHeadsPerCta;
  cfps_kernel<D><<<grid, 32 * kHeadsPerCta, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_cfps(int d, const CfpsArgs& a, cudaStream_t st) {
  if (a.H == 0) return cudaSuccess;
  return d == 128 ? launch_cfps_d<128>(a, st) : launch_cfps_d<64>(a, st);
}

cudaError_t launch_cfps_seed(int d, const float* rows, int H, int b_min, int b_max, __nv_bfloat16* buf, int* size,
                             cudaStream_t st) {
  if (H == 0) return cudaSuccess;
  const int grid = 4 * 152;
  if (d == 128)
    cfps_seed_kernel<128><<<grid, 256, 0, st>>>(rows, H, b_min, b_max, buf, size);
  else
    cfps_seed_kernel<64><<<grid, 256, 0, st>>>(rows, H, b_min, b_max, buf, size);
  return cudaGetLastError();
}

}  // namespace bkv
