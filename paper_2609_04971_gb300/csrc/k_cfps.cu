// Continual FPS beacon maintenance (Section 4.2, Eq. 9): each query head keeps
// a bounded buffer of pre-RoPE queries that is compressed by Farthest Point
// Sampling (Appendix D.1, Algorithm 1) whenever it fills; Algorithm 2's
// decode branch, its beacon freeze and its post-eviction merge.
//
// One warp per query head, kHeadsPerCta heads per CTA.  A head's buffer (at
// most 32 rows) sits transposed in shared memory as bf16 [d][kPitch], one
// physical slot per column, with the fp32 cosines between slots; the buffer
// order (which the FPS ties and the output follow) is a list of slots held
// one per lane, so an FPS compression only permutes that list.  The dot
// product of a new row with slot p is a fused multiply-add chain in element
// order, run by lane p; the norms are fp32 square roots of the self dots and
// each cosine dot / (|a| |b|) (0 when a norm is 0) is taken once, when its
// later row arrives.  The farthest-point loop sums and compares those
// cosines in the definition's order, ties to the lowest row.  These are the
// operations the fp32 decisions of the reference are defined by, so both
// pick the same rows.
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

constexpr int kHeadsPerCta = 12;
constexpr int kMaxRows = kCfpsMaxRows;  // 32: one slot per lane
constexpr int kChunk = 8;               // rows added per pass over the elements
constexpr int kPitch = 34;              // bf16 elements per transposed row (even; spreads banks)

template <int D>
struct WarpSmem {
  __nv_bfloat16 xt[D][kPitch];          // slots, transposed: xt[k][p] = element k of slot p
  __align__(16) float xn[D][kChunk];    // the rows being added, fp32, for broadcast reads
  float C[kMaxRows][kMaxRows + 1];      // cosines between slots
};

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

// One head's buffer: the list of slots in buffer order (lane t holds row t's slot), the norm
// of every slot (lane p holds slot p's), the set of slots in use and the number of rows.
struct Buf {
  int slot;
  float nrm;
  uint32_t used;
  int n;
};

// A row to append: bf16 values, or fp32 values that hold bf16 numbers.
struct RowSrc {
  const void* p;
  bool f32;
};

// Appends cnt <= kChunk rows, whose sources `src(u)` gives, to the end of the buffer.
template <int D, typename Src>
__device__ void add_rows(WarpSmem<D>& w, Buf& b, int cnt, Src src) {
  const int lane = threadIdx.x & 31;
  int q[kChunk];  // slots of the new rows: the lowest free ones
  uint32_t taken = b.used;
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    q[u] = u < cnt ? __ffs(~taken) - 1 : 0;
    if (u < cnt) taken |= 1u << q[u];
  }
  // all the chunk's loads are in flight together (a global load takes about a microsecond)
  RowSrc rs[kChunk];
#pragma unroll
  for (int u = 0; u < kChunk; ++u) rs[u] = u < cnt ? src(u) : RowSrc{nullptr, false};
  uint4 raw[kChunk];
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    raw[u] = make_uint4(0u, 0u, 0u, 0u);
    if (rs[u].p) {
      const char* base = static_cast<const char*>(rs[u].p);
      if constexpr (D == 128) {
        if (rs[u].f32)
          asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
                       : "=r"(raw[u].x), "=r"(raw[u].y), "=r"(raw[u].z), "=r"(raw[u].w) : "l"(base + lane * 16));
        else
          asm volatile("ld.global.nc.v2.u32 {%0,%1}, [%2];" : "=r"(raw[u].x), "=r"(raw[u].y) : "l"(base + lane * 8));
      } else {
        if (rs[u].f32)
          asm volatile("ld.global.nc.v2.u32 {%0,%1}, [%2];" : "=r"(raw[u].x), "=r"(raw[u].y) : "l"(base + lane * 8));
        else
          asm volatile("ld.global.nc.u32 %0, [%1];" : "=r"(raw[u].x) : "l"(base + lane * 4));
      }
    }
  }
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    float v[D / 32];
    if (rs[u].f32) {
      const uint32_t r4[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
#pragma unroll
      for (int e = 0; e < D / 32; ++e) v[e] = __uint_as_float(r4[e]);
    } else {
      const uint32_t r2[2] = {raw[u].x, raw[u].y};
#pragma unroll
      for (int e = 0; e < D / 32; ++e) v[e] = __uint_as_float((e & 1) ? (r2[e >> 1] & 0xffff0000u) : (r2[e >> 1] << 16));
    }
#pragma unroll
    for (int e = 0; e < D / 32; ++e) {
      const int k = lane * (D / 32) + e;
      if (u < cnt) w.xt[k][q[u]] = __float2bfloat16_rn(v[e]);  // exact: v holds a bf16 value
      w.xn[k][u] = u < cnt ? v[e] : 0.f;
    }
  }
  __syncwarp();
  // lane p: dots of the new rows with slot p, element order
  float acc[kChunk];
#pragma unroll
  for (int u = 0; u < kChunk; ++u) acc[u] = 0.f;
#pragma unroll 4
  for (int k = 0; k < D; ++k) {
    const float xp = __bfloat162float(w.xt[k][lane]);
    const float4 a0 = *reinterpret_cast<const float4*>(&w.xn[k][0]);
    const float4 a1 = *reinterpret_cast<const float4*>(&w.xn[k][4]);
    acc[0] = __fmaf_rn(a0.x, xp, acc[0]);
    acc[1] = __fmaf_rn(a0.y, xp, acc[1]);
    acc[2] = __fmaf_rn(a0.z, xp, acc[2]);
    acc[3] = __fmaf_rn(a0.w, xp, acc[3]);
    acc[4] = __fmaf_rn(a1.x, xp, acc[4]);
    acc[5] = __fmaf_rn(a1.y, xp, acc[5]);
    acc[6] = __fmaf_rn(a1.z, xp, acc[6]);
    acc[7] = __fmaf_rn(a1.w, xp, acc[7]);
  }
  // norms of the new slots (their self dots), then every cosine with a new row
#pragma unroll
  for (int u = 0; u < kChunk; ++u)
    if (u < cnt && lane == q[u]) b.nrm = __fsqrt_rn(acc[u]);
  const bool mine = (taken >> lane) & 1u;
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    if (u < cnt) {
      const float nq = __shfl_sync(0xffffffffu, b.nrm, q[u]);
      const float c = (nq == 0.f || b.nrm == 0.f) ? 0.f : __fdiv_rn(acc[u], __fmul_rn(nq, b.nrm));
      if (mine) {
        w.C[q[u]][lane] = c;
        w.C[lane][q[u]] = c;
      }
    }
  }
#pragma unroll
  for (int u = 0; u < kChunk; ++u)
    if (u < cnt && lane == b.n + u) b.slot = q[u];
  b.used = taken;
  b.n += cnt;
  __syncwarp();
}

// Algorithm 1 on the buffer's rows; the buffer becomes its min(m, n) picks in pick order.
template <int D>
__device__ void fps_keep(WarpSmem<D>& w, Buf& b, int m) {
  const int t = threadIdx.x & 31;
  const int n = b.n;
  if (m > n) m = n;
  if (m <= 0) {
    b.n = 0;
    b.used = 0;
    return;
  }
  const bool row = t < n;
  const int pt = row ? b.slot : 0;
  float sum = 0.f;
  for (int i = 0; i < n; ++i) sum = __fadd_rn(sum, w.C[__shfl_sync(0xffffffffu, b.slot, i)][pt]);
  const float avg = row ? __fdiv_rn(sum, static_cast<float>(n)) : INFINITY;
  int r = warp_argmin(avg);
  int pick = r;  // lane k ends up with the k-th pick
  bool sel = t == r;
  float S = w.C[__shfl_sync(0xffffffffu, b.slot, r)][pt];
  for (int k = 1; k < m; ++k) {
    r = warp_argmin((row && !sel) ? S : INFINITY);
    if (t == k) pick = r;
    if (t == r) sel = true;
    const float c = w.C[__shfl_sync(0xffffffffu, b.slot, r)][pt];
    if (!sel && c > S) S = c;
  }
  const int ns = __shfl_sync(0xffffffffu, b.slot, pick);
  b.slot = t < m ? ns : 0;
  b.used = __reduce_or_sync(0xffffffffu, t < m ? (1u << ns) : 0u);
  b.n = m;
  __syncwarp();
}

// Rows of the buffer, in order, as bf16 rows at dst.
template <int D>
__device__ void store_rows(const WarpSmem<D>& w, const Buf& b, __nv_bfloat16* dst) {
  const int lane = threadIdx.x & 31;
  for (int t = 0; t < b.n; ++t) {
    const int p = __shfl_sync(0xffffffffu, b.slot, t);
    if constexpr (D == 128) {
      const int k = lane * 4;
      const uint32_t x0 = __bfloat16_as_ushort(w.xt[k][p]) | (static_cast<uint32_t>(__bfloat16_as_ushort(w.xt[k + 1][p])) << 16);
      const uint32_t x1 =
          __bfloat16_as_ushort(w.xt[k + 2][p]) | (static_cast<uint32_t>(__bfloat16_as_ushort(w.xt[k + 3][p])) << 16);
      *reinterpret_cast<uint2*>(dst + static_cast<size_t>(t) * D + k) = make_uint2(x0, x1);
    } else {
      const int k = lane * 2;
      const uint32_t x0 = __bfloat16_as_ushort(w.xt[k][p]) | (static_cast<uint32_t>(__bfloat16_as_ushort(w.xt[k + 1][p])) << 16);
      *reinterpret_cast<uint32_t*>(dst + static_cast<size_t>(t) * D + k) = x0;
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
  const __nv_bfloat16* qh = a.q ? a.q + static_cast<size_t>(h) * a.n_q * D : nullptr;
  Buf b{0, 0.f, 0u, 0};

  if (a.mode == kCfpsUpdate) {
    // rows in order: the buffer's own rows (their cosines are rebuilt), then the new queries
    const int n_old = a.size[h];
    const int total = n_old + a.n_q;
    int next = 0;
    while (next < total) {
      const int add = min(a.b_max - b.n, total - next);
      for (int c0 = 0; c0 < add; c0 += kChunk) {
        const int base = next + c0;
        add_rows<D>(w, b, min(kChunk, add - c0), [&](int u) {
          const int src = base + u;
          return RowSrc{src < n_old ? buf + static_cast<size_t>(src) * D : qh + static_cast<size_t>(src - n_old) * D,
                        false};
        });
      }
      next += add;
      if (b.n == a.b_max) fps_keep<D>(w, b, a.b_min);
    }
    store_rows<D>(w, b, buf);
    if (lane == 0) a.size[h] = b.n;
    return;
  }

  // beacons: the buffer's rows; merge: this compress's beacons, then the head's window queries
  int n = 0, nbc = 0;
  if (a.mode == kCfpsBeacons) {
    n = a.size[h];
  } else {
    for (int t = 0; t < a.b_min; ++t) nbc += bcnt[t] != 0;
    n = nbc + a.n_q;
  }
  for (int c0 = 0; c0 < n; c0 += kChunk) {
    add_rows<D>(w, b, min(kChunk, n - c0), [&](int u) {
      const int src = c0 + u;
      if (a.mode == kCfpsBeacons) return RowSrc{buf + static_cast<size_t>(src) * D, false};
      if (src < nbc) return RowSrc{bcn + static_cast<size_t>(src) * D, true};
      return RowSrc{qh + static_cast<size_t>(src - nbc) * D, false};
    });
  }
  fps_keep<D>(w, b, a.b_min);
  if (a.mode == kCfpsBeacons) {
    for (int t = 0; t < a.b_min; ++t) {
      const int p = __shfl_sync(0xffffffffu, b.slot, t < b.n ? t : 0);
#pragma unroll
      for (int e = 0; e < D / 32; ++e) {
        const int k = lane * (D / 32) + e;
        bcn[static_cast<size_t>(t) * D + k] = t < b.n ? __bfloat162float(w.xt[k][p]) : 0.f;
      }
      if (lane == 0) bcnt[t] = t < b.n ? 1 : 0;
    }
  } else {
    store_rows<D>(w, b, buf);
    if (lane == 0) a.size[h] = b.n;
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
