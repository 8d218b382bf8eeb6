// Continual FPS beacon maintenance (Section 4.2, Eq. 9): each query head keeps
// a bounded buffer of pre-RoPE queries that is compressed by Farthest Point
// Sampling (Appendix D.1, Algorithm 1) whenever it fills; Algorithm 2's
// decode branch, its beacon freeze and its post-eviction merge.
//
// One warp per query head, kHeadsPerCta heads per CTA.  A head's buffer (at
// most R = 16 or 32 rows, one physical slot each) sits transposed in shared
// memory as bf16 pairs [d/2][R + 1], with the fp32 cosines between slots; the
// buffer order (which the FPS ties and the output follow) is a list of slots
// held one per lane, so an FPS compression only permutes that list.  Rows are
// added in chunks of 8: lane l loads the pairs (2l, 2l+1) (and 64 + 2l,
// 65 + 2l when d = 128), so the transposing stores hit 32 distinct banks, and
// the chunk is also staged as fp32 rows for broadcast reads.  The dot product
// of a new row with slot p is a fused multiply-add chain in element order; with
// R = 16 the two half-warps take 4 new rows each (their staged rows sit 16
// banks apart), with R = 32 lane p takes all 8.  The norms are fp32 square
// roots of the self dots and each cosine dot / (|a| |b|) (0 when a norm is 0)
// is taken once, when its later row arrives.  The farthest-point loop sums and
// compares those cosines in the definition's order, ties to the lowest row
// (an argmin by warp min-reduction of an order-preserving key, then the lowest
// lane holding it).  These are the operations the fp32 decisions of the
// reference are defined by, so both pick the same rows.  Each chunk's global
// loads are issued before the previous chunk's products and FPS run, so their
// latency is hidden.
//
// The same warp routine serves three calls:
//   update   append the call's queries in order (a call that does not fill the
//            buffer only copies them behind its rows); whenever the buffer holds
//            b_max = b_min + window rows, replace it by the FPS selection of
//            b_min of them, in pick order;
//   beacons  the beacons of a compress: the FPS selection of min(b_min, size)
//            buffer rows, written as fp32 rows with count 1 (count 0 and a
//            zero row for an empty slot) for the scoring-query build;
//   merge    after an eviction the buffer becomes the FPS selection of b_min
//            rows of (the beacons, then the head's window queries in order).
// Inputs are finite bf16 queries; a stored size outside 0..b_max is clamped.
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kHeadsPerCta = 12;
constexpr int kChunk = 8;  // rows added per pass over the elements
constexpr uint32_t kFull = 0xffffffffu;
constexpr uint32_t kNotCandidate = 0xffffffffu;  // argmin key above every float's

template <int D, int R>
struct WarpSmem {
  uint32_t xt[D / 2][R + 1];           // xt[kk][p]: elements 2kk, 2kk+1 of slot p (bf16 pair)
  __align__(16) float xn[kChunk][D];   // the rows being added, fp32; element k of row u at column xn_col(u, k)
  float C[R][R + 1];                   // cosines between slots
};

// With R = 16 the rows 4..7 read by the upper half-warp are stored 16 columns
// (banks) away from rows 0..3, so both halves' broadcast reads go in one pass.
template <int R>
__device__ __forceinline__ int xn_swz(int u) {
  return (R == 16 && u >= 4) ? 16 : 0;
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Order-preserving unsigned key of a float (-0 taken as +0, NaN ranked with +inf).
__device__ __forceinline__ uint32_t fkey(float v) {
  v = __fadd_rn(v, 0.f);
  if (v != v) v = INFINITY;
  const uint32_t b = __float_as_uint(v);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Lowest lane holding the warp's minimum key.
__device__ __forceinline__ int warp_argmin_key(uint32_t k) {
  const uint32_t mn = __reduce_min_sync(kFull, k);
  return __ffs(__ballot_sync(kFull, k == mn)) - 1;
}

// One head's buffer: the list of slots in buffer order (lane t holds row t's slot), the norm
// of every slot (lane l holds slot l mod R's), the set of slots in use and the number of rows.
struct Buf {
  int slot;
  float nrm;
  uint32_t used;
  int n;
};

// A row to add: bf16 values, or fp32 values that hold bf16 numbers.
struct RowSrc {
  const void* p;
  bool f32;
};

// Words per lane and row of a chunk in flight: bf16 pairs, or fp32 pairs of values.
template <int D, bool F32>
struct RawWords {
  static constexpr int n = (D / 64) * (F32 ? 2 : 1);
};

// Issues the global loads of cnt <= kChunk rows: lane l takes elements 2l, 2l+1 (+ 64 when d = 128).
template <int D, bool F32, typename Src>
__device__ __forceinline__ void load_rows(uint32_t (&raw)[kChunk][RawWords<D, F32>::n], bool (&f32)[kChunk], int cnt,
                                          Src src) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
#pragma unroll
    for (int i = 0; i < RawWords<D, F32>::n; ++i) raw[u][i] = 0u;
    f32[u] = false;
    if (u < cnt) {
      const RowSrc rs = src(u);
      const char* base = static_cast<const char*>(rs.p);
      if constexpr (F32) {
        f32[u] = rs.f32;
        if (rs.f32) {
#pragma unroll
          for (int h = 0; h < D / 64; ++h)
            asm volatile("ld.global.nc.v2.u32 {%0,%1}, [%2];"
                         : "=r"(raw[u][2 * h]), "=r"(raw[u][2 * h + 1])
                         : "l"(base + h * 256 + lane * 8));
          continue;
        }
      }
#pragma unroll
      for (int h = 0; h < D / 64; ++h)
        asm volatile("ld.global.nc.u32 %0, [%1];" : "=r"(raw[u][h]) : "l"(base + h * 128 + lane * 4));
    }
  }
}

// The bf16 pair h (elements 64h + 2l, 64h + 2l + 1) of a loaded row.
template <int D, bool F32>
__device__ __forceinline__ uint32_t pair_of(const uint32_t (&r)[RawWords<D, F32>::n], bool f32, int h) {
  if constexpr (F32) {
    if (f32) return (r[2 * h] >> 16) | (r[2 * h + 1] & 0xffff0000u);  // exact: the values are bf16 numbers
    return r[h];
  } else {
    (void)f32;
    return r[h];
  }
}

// Appends the cnt <= kChunk loaded rows to the end of the buffer; next() issues the loads of the
// following chunk once this one's registers are in shared memory.
template <int D, int R, bool F32, typename Next>
__device__ __forceinline__ void add_rows(WarpSmem<D, R>& w, Buf& b, int cnt, uint32_t (&raw)[kChunk][RawWords<D, F32>::n],
                                         bool (&f32)[kChunk], Next next) {
  constexpr int NR = R == 16 ? 4 : 8;  // new rows per lane in the products
  const int lane = threadIdx.x & 31;
  const int p = lane & (R - 1);        // the slot this lane multiplies
  const int half = R == 16 ? lane >> 4 : 0;
  int q[kChunk];  // slots of the new rows: the lowest free ones
  uint32_t taken = b.used;
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    q[u] = u < cnt ? __ffs(~taken) - 1 : 0;
    if (u < cnt) taken |= 1u << q[u];
  }
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    if (u < cnt) {
#pragma unroll
      for (int h = 0; h < D / 64; ++h) {
        const uint32_t pr = pair_of<D, F32>(raw[u], f32[u], h);
        w.xt[32 * h + lane][q[u]] = pr;
        const int k = 64 * h + 2 * lane;
        *reinterpret_cast<float2*>(&w.xn[u][k ^ xn_swz<R>(u)]) = make_float2(bf_lo(pr), bf_hi(pr));
      }
    }
  }
  next();
  __syncwarp();
  // products of the new rows half * NR + j with slot p, element order
  float acc[NR];
#pragma unroll
  for (int j = 0; j < NR; ++j) acc[j] = 0.f;
  const float* xr = &w.xn[half * NR][0];
  const int sw = R == 16 ? 16 * half : 0;
#pragma unroll 2
  for (int k4 = 0; k4 < D / 4; ++k4) {
    const uint32_t w0 = w.xt[2 * k4][p], w1 = w.xt[2 * k4 + 1][p];
    const float x0 = bf_lo(w0), x1 = bf_hi(w0), x2 = bf_lo(w1), x3 = bf_hi(w1);
#pragma unroll
    for (int j = 0; j < NR; ++j) {
      const float4 a = *reinterpret_cast<const float4*>(xr + j * D + ((4 * k4) ^ sw));
      acc[j] = __fmaf_rn(a.x, x0, acc[j]);
      acc[j] = __fmaf_rn(a.y, x1, acc[j]);
      acc[j] = __fmaf_rn(a.z, x2, acc[j]);
      acc[j] = __fmaf_rn(a.w, x3, acc[j]);
    }
  }
  // norms of the new slots (their self dots), then every cosine with a new row
  float nq[kChunk];
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    const int owner = q[u] + (R == 16 ? 16 * (u >> 2) : 0);
    nq[u] = __fsqrt_rn(__shfl_sync(kFull, acc[u % NR], owner));
    if (u < cnt && p == q[u]) b.nrm = nq[u];
  }
  const bool mine = (taken >> p) & 1u;
#pragma unroll
  for (int j = 0; j < NR; ++j) {
    const int u = half * NR + j;
    const int qu = (R == 16 && half) ? q[(j + 4) % kChunk] : q[j];
    const float nu = (R == 16 && half) ? nq[(j + 4) % kChunk] : nq[j];
    if (u < cnt && mine) {
      const float c = (nu == 0.f || b.nrm == 0.f) ? 0.f : __fdiv_rn(acc[j], __fmul_rn(nu, b.nrm));
      w.C[qu][p] = c;
      w.C[p][qu] = c;
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
template <int D, int R>
__device__ void fps_keep(WarpSmem<D, R>& w, Buf& b, int m) {
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
  // avg_t = (sum over rows i in order of cos(i, t)) / n
  float sum = 0.f;
#pragma unroll
  for (int i0 = 0; i0 < R; i0 += 8) {
    if (i0 < n) {
      float cv[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) cv[i] = w.C[__shfl_sync(kFull, b.slot, i0 + i)][pt];
#pragma unroll
      for (int i = 0; i < 8; ++i)
        if (i0 + i < n) sum = __fadd_rn(sum, cv[i]);
    }
  }
  int r = warp_argmin_key(row ? fkey(__fdiv_rn(sum, static_cast<float>(n))) : kNotCandidate);
  int pick = r;  // lane k ends up with the k-th pick
  bool sel = t == r;
  float S = w.C[__shfl_sync(kFull, b.slot, r)][pt];
  for (int k = 1; k < m; ++k) {
    r = warp_argmin_key((row && !sel) ? fkey(S) : kNotCandidate);
    if (t == k) pick = r;
    if (t == r) sel = true;
    const float c = w.C[__shfl_sync(kFull, b.slot, r)][pt];
    if (!sel && c > S) S = c;
  }
  const int ns = __shfl_sync(kFull, b.slot, pick);
  b.slot = t < m ? ns : 0;
  b.used = __reduce_or_sync(kFull, t < m ? (1u << ns) : 0u);
  b.n = m;
  __syncwarp();
}

// Rows of the buffer, in order, as bf16 rows at dst.
template <int D, int R>
__device__ void store_rows(const WarpSmem<D, R>& w, const Buf& b, __nv_bfloat16* dst) {
  const int lane = threadIdx.x & 31;
  for (int t = 0; t < b.n; ++t) {
    const int p = __shfl_sync(kFull, b.slot, t);
#pragma unroll
    for (int h = 0; h < D / 64; ++h)
      *reinterpret_cast<uint32_t*>(dst + static_cast<size_t>(t) * D + 64 * h + 2 * lane) = w.xt[32 * h + lane][p];
  }
}

template <int D, int R, int MODE>
__global__ void __launch_bounds__(32 * kHeadsPerCta, R == 16 ? 2 : 1) cfps_kernel(CfpsArgs a) {
  constexpr bool F32 = MODE == kCfpsMerge;  // the merge reads the fp32 beacon rows
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x * kHeadsPerCta + wid;
  if (h >= a.H) return;  // whole warp
  if (MODE == kCfpsMerge && a.Ls) {  // per-instance lengths: no eviction in this instance, nothing to merge
    const int L = a.Ls[h / a.group];
    if (L <= a.budget || L > a.cap) return;
  }
  WarpSmem<D, R>& w = reinterpret_cast<WarpSmem<D, R>*>(smem_raw)[wid];
  __nv_bfloat16* buf = a.buf + static_cast<size_t>(h) * a.b_max * D;
  float* bcn = a.bcn + static_cast<size_t>(h) * a.b_min * D;
  long long* bcnt = a.bcnt + static_cast<size_t>(h) * a.b_min;
  const __nv_bfloat16* qh = a.q ? a.q + static_cast<size_t>(h) * a.n_q * D : nullptr;
  Buf b{0, 0.f, 0u, 0};

  // the rows to add, in order: update: the buffer's own rows (their cosines are rebuilt), then
  // the new queries; beacons: the buffer's rows; merge: this compress's beacons, then the window
  const int n_old = min(max(a.size[h], 0), a.b_max);
  in_bounds(a.size[h], a.b_max, a.err);  // a stored size is 0 .. b_max - 1; the clamp above keeps accesses in range
  if (MODE == kCfpsUpdate && n_old + a.n_q < a.b_max) {
    // the buffer does not fill: the new queries are appended in order and nothing is compressed
    const int words = a.n_q * D / 2;  // 32-bit words of the new rows
    const uint32_t* src = reinterpret_cast<const uint32_t*>(qh);
    uint32_t* dst = reinterpret_cast<uint32_t*>(buf + static_cast<size_t>(n_old) * D);
    for (int i = lane; i < words; i += 32) dst[i] = src[i];
    if (lane == 0) a.size[h] = n_old + a.n_q;
    return;
  }
  int nbc = 0;
  if (MODE == kCfpsMerge)
    for (int t = 0; t < a.b_min; ++t) nbc += bcnt[t] != 0;
  const int total = MODE == kCfpsUpdate ? n_old + a.n_q : MODE == kCfpsBeacons ? n_old : nbc + a.n_q;
  auto src = [&](int i) -> RowSrc {
    if (MODE == kCfpsMerge) {
      if (i < nbc) return RowSrc{bcn + static_cast<size_t>(i) * D, true};
      return RowSrc{qh + static_cast<size_t>(i - nbc) * D, false};
    }
    if (i < n_old) return RowSrc{buf + static_cast<size_t>(i) * D, false};
    return RowSrc{qh + static_cast<size_t>(i - n_old) * D, false};
  };
  // chunks: at most kChunk rows and never past b_max rows in the buffer; in an update the buffer
  // is compressed to b_min rows whenever it reaches b_max
  uint32_t raw[kChunk][RawWords<D, F32>::n];
  bool f32[kChunk];
  int pos = 0, n = 0;
  int cnt = min(min(kChunk, a.b_max - n), total - pos);
  load_rows<D, F32>(raw, f32, cnt, [&](int u) { return src(pos + u); });
  while (cnt > 0) {
    const bool full = MODE == kCfpsUpdate && n + cnt == a.b_max;
    const int n_next = full ? a.b_min : n + cnt;
    const int pos_next = pos + cnt;
    const int cnt_next = min(min(kChunk, a.b_max - n_next), total - pos_next);
    add_rows<D, R, F32>(w, b, cnt, raw, f32, [&] {
      load_rows<D, F32>(raw, f32, cnt_next, [&](int u) { return src(pos_next + u); });
    });
    if (full) fps_keep<D, R>(w, b, a.b_min);
    pos = pos_next;
    n = n_next;
    cnt = cnt_next;
  }

  if (MODE == kCfpsUpdate) {
    store_rows<D, R>(w, b, buf);
    if (lane == 0) a.size[h] = b.n;
    return;
  }
  fps_keep<D, R>(w, b, a.b_min);
  if (MODE == kCfpsBeacons) {
    for (int t = 0; t < a.b_min; ++t) {
      const int p = __shfl_sync(kFull, b.slot, t < b.n ? t : 0);
#pragma unroll
      for (int hh = 0; hh < D / 64; ++hh) {
        const uint32_t pr = w.xt[32 * hh + lane][p];
        *reinterpret_cast<float2*>(bcn + static_cast<size_t>(t) * D + 64 * hh + 2 * lane) =
            t < b.n ? make_float2(bf_lo(pr), bf_hi(pr)) : make_float2(0.f, 0.f);
      }
      if (lane == 0) bcnt[t] = t < b.n ? 1 : 0;
    }
  } else {
    store_rows<D, R>(w, b, buf);
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

template <int D, int R, int MODE>
cudaError_t launch_cfps_m(const CfpsArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(WarpSmem<D, R>) * kHeadsPerCta;
  cudaError_t e = cudaFuncSetAttribute(cfps_kernel<D, R, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  // the largest shared-memory carveout, so that two CTAs of the 16-row form share an SM
  e = cudaFuncSetAttribute(cfps_kernel<D, R, MODE>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  if (e != cudaSuccess) return e;
  const int grid = (a.H + kHeadsPerCta - 1) / kHeadsPerCta;
  cfps_kernel<D, R, MODE><<<grid, 32 * kHeadsPerCta, smem, st>>>(a);
  return cudaGetLastError();
}

template <int D, int R>
cudaError_t launch_cfps_r(const CfpsArgs& a, cudaStream_t st) {
  if (a.mode == kCfpsUpdate) return launch_cfps_m<D, R, kCfpsUpdate>(a, st);
  if (a.mode == kCfpsBeacons) return launch_cfps_m<D, R, kCfpsBeacons>(a, st);
  return launch_cfps_m<D, R, kCfpsMerge>(a, st);
}

template <int D>
cudaError_t launch_cfps_d(const CfpsArgs& a, cudaStream_t st) {
  return a.b_max <= 16 ? launch_cfps_r<D, 16>(a, st) : launch_cfps_r<D, 32>(a, st);
}

}  // namespace

cudaError_t launch_cfps(int d, const CfpsArgs& a, cudaStream_t st) {
  if (a.H == 0) return cudaSuccess;
  if (a.b_max > kCfpsMaxRows || a.b_min >= a.b_max || a.b_min < 1) return cudaErrorInvalidValue;
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
