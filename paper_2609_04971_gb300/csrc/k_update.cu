// Beacon maintenance (Section 3.2, Appendix D): every new query is assigned to
// the beacon of highest cosine similarity and that beacon's centroid becomes
// the running mean of the queries assigned to it.
//
// Persistent kernel, one CTA per SM; CTA k takes instances k, k + grid, ...
// An instance's queries stream through a ring of shared-memory stages in
// tiles of up to 128 (TMA, 128-byte swizzle) and are read from HBM once.
//
// Screening on the tensor cores: per tile, D1 = Q x [c_hi ; c_lo]^T where
// c_hi = bf16(c / |c|) and c_lo = bf16(c / |c| - c_hi), so dot_b = D1[:, b] +
// D1[:, nbp + b] carries the unit-centroid dot to about 2^-16 |q| (bf16 x bf16
// products are exact, the accumulation is fp32); D2 = Q x Q^T gives |q|^2 on
// its diagonal.  When best and second-best dots differ by at most 1e-4 |q|
// (about twice the bound on their difference's error: 2^-17 |q| per dot from
// the hi/lo split, 128 fp32 accumulation steps), the query is re-decided
// exactly: the beacon maximising (q . c_b) / |c_b| in double-float arithmetic
// (exact products, TwoSum accumulation, 1 / |c_b| from a double-float sum of
// squares and one Newton step, to about 2^-44 relative), which
// agrees with the cosine (q . c_b) / (|q| |c_b|) evaluated in fp64 except at
// ties below ~1e-12 (the lowest beacon wins ties).  Zero queries and instances
// without a valid beacon give -1.
//
// Sums: int64 fixed point with 40 fractional bits.  A tile's screened rows
// are sorted by beacon (ballot counting sort); each accumulator warp takes an
// equal slice of that order, its lanes owning D / 32 columns each, and keeps
// three fp32 part sums per column that are exact by construction (see Parts;
// exact for 2^-31 <= |x| < 2^14, the conversion to fixed point per beacon
// change rather than per element); re-decided rows are converted directly.
// The per-call sum is exact and independent of the order.  It is then
// added once to the fp64 running sum, correctly rounded (fold_sum_fp64: one
// fp64 addition while the call's sum is exact in fp64, fold_sum's exact
// integer addition beyond; the bookkeeping warps that fold have the fp64 pipe
// to themselves), and c = fp32(sum / count) to within one fp32 ulp from
// double-float arithmetic on the sum's bits.
//
// Warp roles (26 warps): warp 0 TMA producer; warp 1 TMEM allocation and MMA
// issue; warps 2..5 screeners (one per TMEM lane quarter: decisions, the
// sorted row list of the tile, exact re-decisions); warps 6..21 accumulators
// (the sums of a tile, while the screeners work on the next one; the row
// lists are double-buffered); warps 22..25 bookkeeping: they build the
// unit-centroid operand of the next instance and fold the finished one into
// the running state, from centroids and sums brought in by bulk copies
// (accumulators double-buffered by instance).  All waits are bounded.
#include "bkv_device.cuh"
#include "bkv_internal.h"
#include "k_update_math.cuh"

namespace bkv {
namespace {

constexpr int kScreeners = 4;
constexpr int kAccum = 16;
constexpr int kKeepers = 4;
constexpr int kUThreads = 32 * (2 + kScreeners + kAccum + kKeepers);
constexpr int kQTile = 128;                 // queries per tile (MMA M)
constexpr uint32_t kQBox = 128 * 128;       // [128 rows][64 bf16] swizzled box slot
constexpr int kUMaxStages = 8;
constexpr size_t kUSmemBudget = 216 * 1024;
constexpr int kGroup = 4;  // rows an accumulator lane sums per step when they share a beacon

struct UpdArgs {
  int n_inst, nq, nb, nbp;  // instances, queries per instance, beacons, beacons padded to 8
  int box_rows;             // rows of one TMA box of queries (<= 128)
  float* cent;
  double* sums;
  long long* counts;
  int* assign_out;
  int* err;
};

template <int D>
struct UpdCfg {
  static constexpr int kBoxes = D / 64;
  static constexpr uint32_t kStageBytes = kBoxes * kQBox;
  __host__ __device__ static size_t bmat_bytes(int nbp) { return static_cast<size_t>(kBoxes) * 2 * nbp * 128; }
  __host__ __device__ static size_t state_bytes(int nb, int nbp) {
    // bmat[2], acc[2] (int64), cent[2] (fp32), sums (fp64)
    return 2 * bmat_bytes(nbp) + 2 * static_cast<size_t>(nb) * D * 8 + 2 * static_cast<size_t>(nb) * D * 4 +
           static_cast<size_t>(nb) * D * 8;
  }
  static int stages(int nb, int nbp) {
    const size_t room = kUSmemBudget - 1024 - state_bytes(nb, nbp);
    const int n = static_cast<int>(room / kStageBytes);
    return n < kUMaxStages ? n : kUMaxStages;
  }
  static size_t smem_bytes(int nb, int nbp) {
    return 1024 + static_cast<size_t>(stages(nb, nbp)) * kStageBytes + state_bytes(nb, nbp);
  }
};

__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, int* err) {
  int never = 0;
  mbar_wait(bar, parity, &never, err, kDevTimeoutDrain);
}

__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Contiguous global -> shared copy by the TMA unit, completing on `bar`.
__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// round(x * 2^40) of the bf16 value whose bits sit in the upper half of
// `hi16` (lower half zero): the scale is added to the fp32 exponent field
// (exact for |x| < 2^88; a zero or subnormal x becomes a value below 2^-80,
// which rounds to 0 as x * 2^40 would), then one round-to-nearest conversion.
__device__ __forceinline__ long long bf16_fixed40(uint32_t hi16) {
  return __float2ll_rn(__uint_as_float(hi16 + (40u << 23)));
}

// Byte offset of element (row, col) in a [rows][D] bf16 tile stored as D / 64
// boxes of [rows][64] with the 128-byte swizzle (box_bytes apart).
__device__ __forceinline__ uint32_t sw128_offset(int row, int col, uint32_t box_bytes) {
  return (col >> 6) * box_bytes + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4) + ((col & 7) << 1);
}

// Adds the kCols bf16 values at p (columns col0 ..) to s as fixed point.
template <int kCols>
__device__ __forceinline__ void add_fixed(long long (&s)[kCols], const unsigned char* p) {
  if constexpr (kCols == 4) {
    const uint2 w = *reinterpret_cast<const uint2*>(p);
    s[0] += bf16_fixed40(w.x << 16);
    s[1] += bf16_fixed40(w.x & 0xffff0000u);
    s[2] += bf16_fixed40(w.y << 16);
    s[3] += bf16_fixed40(w.y & 0xffff0000u);
  } else {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(p);
    s[0] += bf16_fixed40(w << 16);
    s[1] += bf16_fixed40(w & 0xffff0000u);
  }
}

// *cell += v on a shared int64 cell, as two 32-bit atomic additions: the low word's carry-out is
// decided by the value that addition found, so concurrent additions still sum exactly (a 64-bit
// shared-memory atomic addition is a compare-and-swap loop on this part).
__device__ __forceinline__ void shared_add_i64(long long* cell, long long v) {
  uint32_t* w = reinterpret_cast<uint32_t*>(cell);
  const uint32_t lo = static_cast<uint32_t>(v);
  const uint32_t old = atomicAdd(w, lo);
  const uint32_t carry = old + lo < old ? 1u : 0u;
  const uint32_t hi = static_cast<uint32_t>(static_cast<unsigned long long>(v) >> 32) + carry;
  if (hi != 0u) atomicAdd(w + 1, hi);
}

// The same split for two adjacent columns at once, on packed f32x2 values
// (low word: the first column), with Blackwell's paired fp32 adds.
struct Parts2 {
  unsigned long long h, m, l;
};

__device__ __forceinline__ unsigned long long f2_add(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ unsigned long long f2_sub(unsigned long long a, unsigned long long b) {
  unsigned long long d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// w holds two bf16 values (low half: the first column).
__device__ __forceinline__ void parts2_add(Parts2& p, uint32_t w) {
  constexpr unsigned long long kM1 = 0x49C0000049C00000ull;  // {1.5 * 2^20, 1.5 * 2^20}
  constexpr unsigned long long kM2 = 0x4140000041400000ull;  // {12, 12}
  const unsigned long long x = static_cast<unsigned long long>(w << 16) |
                               (static_cast<unsigned long long>(w & 0xffff0000u) << 32);
  const unsigned long long xh = f2_sub(f2_add(x, kM1), kM1);
  const unsigned long long r = f2_sub(x, xh);
  const unsigned long long xm = f2_sub(f2_add(r, kM2), kM2);
  p.h = f2_add(p.h, xh);
  p.m = f2_add(p.m, xm);
  p.l = f2_add(p.l, f2_sub(r, xm));
}

// Column `second` (0 or 1) of a packed pair of part sums.
__device__ __forceinline__ Parts parts2_get(const Parts2& p, int second) {
  const int sh = second ? 32 : 0;
  return Parts{__uint_as_float(static_cast<uint32_t>(p.h >> sh)), __uint_as_float(static_cast<uint32_t>(p.m >> sh)),
               __uint_as_float(static_cast<uint32_t>(p.l >> sh))};
}

template <int D>
__global__ void __launch_bounds__(kUThreads, 1)
    update_kernel(const __grid_constant__ CUtensorMap qmap, UpdArgs a, int n_stages) {
  using C = UpdCfg<D>;
  constexpr int kCols = D / 32;  // columns per lane in the accumulation
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kUMaxStages], empty_bar[kUMaxStages];
  __shared__ __align__(8) uint64_t accfull[2], accfree[2], bready[2], bfree[2], drain_bar;
  __shared__ __align__(8) uint64_t accdone[2], accclear[2], cbar[2], sbar, sfull[2], sempty[2];
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;
  __shared__ int order_t[2][kQTile];  // row | beacon << 8, sorted by beacon (by tile parity)
  __shared__ int refine_t[2][kQTile];
  __shared__ int n_refine[2], n_asg_sh[2];
  __shared__ int cnt_w[2][4][kMaxBeacons];
  __shared__ int add_cnt[2][kMaxBeacons];
  __shared__ int bvalid[2][kMaxBeacons];
  __shared__ DF cninv[2][kMaxBeacons];  // 1 / |c_b| as a double-float
  __shared__ long long cnt_old[2][kMaxBeacons];
  __shared__ DF rcp_sh[kMaxBeacons];  // 1 / count after this call, as a double-float
  __shared__ int degenerate[2];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nq = a.nq, nb = a.nb, nbp = a.nbp;
  const int cells = nb * D;
  const int n_my = blockIdx.x < a.n_inst ? (a.n_inst - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  const int T = (nq + kQTile - 1) / kQTile;  // tiles per instance
  const int ncols1 = 2 * nbp;                 // screening columns (hi, lo)
  const int acc_cols = ncols1 + kQTile;       // + the Q Q^T block
  const uint32_t bbox = static_cast<uint32_t>(ncols1) * 128;  // bytes of one 64-column box of bmat

  // 1024-byte aligned (the 128-byte swizzle pattern repeats every 1024 bytes);
  // offset from the __shared__ array itself so that accesses stay shared-space
  unsigned char* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  unsigned char* stage_smem = base;                                             // [n_stages][kBoxes][128 x 128 B]
  unsigned char* bmat = base + static_cast<size_t>(n_stages) * C::kStageBytes;  // [2][kBoxes][2 nbp x 128 B]
  // [2][nb][D]; column 4 l + c of a beacon row (l = lane, c < D / 32) sits at
  // c * 32 + l, so that the 64-bit updates of a warp hit consecutive words
  long long* acc = reinterpret_cast<long long*>(bmat + 2 * C::bmat_bytes(nbp));
  float* cent_sm = reinterpret_cast<float*>(acc + 2 * cells);                     // [2][nb][D]
  double* sums_sm = reinterpret_cast<double*>(cent_sm + 2 * cells);               // [nb][D]

  if (threadIdx.x == 0) {
    for (int i = 0; i < n_stages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accfull[i], 1);
      mbar_init(&accfree[i], 4);  // the four screening warps
      mbar_init(&bready[i], 1);
      mbar_init(&bfree[i], 1);
      mbar_init(&accdone[i], 1);
      mbar_init(&accclear[i], 1);
      mbar_init(&cbar[i], 1);
      mbar_init(&sfull[i], 1);
      mbar_init(&sempty[i], 1);
    }
    mbar_init(&sbar, 1);
    mbar_init(&drain_bar, 1);
    abort_sh = 0;
    n_refine[0] = n_refine[1] = 0;
    fence_mbar_init();
  }
  for (int c = threadIdx.x; c < 2 * cells; c += kUThreads) acc[c] = 0;
  if (threadIdx.x < 2 * kMaxBeacons) add_cnt[threadIdx.x >> 5][threadIdx.x & 31] = 0;
  if (warp == 1) {
    tmem_alloc(&tmem_base_sh, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_sh;
  volatile int* abort_flag = &abort_sh;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0 && n_my > 0) {
      const uint64_t once = l2_policy_evict_first();
      prefetch_tmap(&qmap);
      int g = 0;
      bool ok = true;
      for (int i = 0; ok && i < n_my; ++i) {
        const int e = blockIdx.x + i * gridDim.x;
        for (int t = 0; t < T; ++t, ++g) {
          const int st = g % n_stages;
          if (g >= n_stages &&
              !mbar_wait(&empty_bar[st], ((g / n_stages) - 1) & 1, abort_flag, a.err, kDevTimeoutProducer)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full_bar[st], static_cast<uint32_t>(C::kBoxes * a.box_rows * 128));
          for (int b = 0; b < C::kBoxes; ++b)
            tma_load_2d(stage_smem + st * C::kStageBytes + b * kQBox, &qmap, &full_bar[st], b * 64,
                        e * nq + t * kQTile, once);
        }
      }
      if (!ok || *abort_flag)
        for (int j = (g > n_stages ? g - n_stages : 0); j < g; ++j)
          drain_wait(&full_bar[j % n_stages], (j / n_stages) & 1, a.err);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0 && n_my > 0) {
      const uint32_t idesc1 = idesc_bf16_f32(128, ncols1), idesc2 = idesc_bf16_f32(128, kQTile);
      int g = 0;
      bool ok = true;
      for (int i = 0; ok && i < n_my; ++i) {
        const int pb = i & 1;
        if (!mbar_wait(&bready[pb], (i >> 1) & 1, abort_flag, a.err, kDevTimeoutMma)) break;
        for (int t = 0; t < T; ++t, ++g) {
          const int st = g % n_stages, ab = g & 1;
          if (!mbar_wait(&full_bar[st], (g / n_stages) & 1, abort_flag, a.err, kDevTimeoutMma) ||
              (g >= 2 && !mbar_wait(&accfree[ab], ((g >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutMma))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + ab * acc_cols;
          const uint32_t q_addr = smem_u32(stage_smem + st * C::kStageBytes);
          const uint32_t b_addr = smem_u32(bmat + pb * C::bmat_bytes(nbp));
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t qoff = (kk >> 2) * kQBox + (kk & 3) * 32;
            const uint32_t boff = (kk >> 2) * bbox + (kk & 3) * 32;
            mma_bf16_ss(d, sdesc_kmajor_sw128(q_addr + qoff), sdesc_kmajor_sw128(b_addr + boff), idesc1, kk > 0);
          }
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t qoff = (kk >> 2) * kQBox + (kk & 3) * 32;
            mma_bf16_ss(d + ncols1, sdesc_kmajor_sw128(q_addr + qoff), sdesc_kmajor_sw128(q_addr + qoff), idesc2,
                        kk > 0);
          }
          mma_commit(&accfull[ab]);
        }
        if (ok) mma_commit(&bfree[pb]);  // this instance's centroid operand is no longer read
      }
      mma_commit(&drain_bar);
      drain_wait(&drain_bar, 0, a.err);
    }
    __syncwarp();
  } else if (warp < 2 + kScreeners) {
    // ---------------------------------------------------------------- screeners
    const int ws = warp - 2;          // 0 .. 3
    const int quarter = warp & 3;     // TMEM lane quarter (warps 2..5 cover all four)
    const int ts = threadIdx.x - 64;  // 0 .. 127
    const uint32_t lane_addr = static_cast<uint32_t>(quarter * 32) << 16;
    const int n = quarter * 32 + lane;  // this thread's query row in the tile
    const int col0 = lane * kCols;
    const unsigned lt = (1u << lane) - 1u;
    int g = 0;
    for (int i = 0; i < n_my; ++i) {
      const int e = blockIdx.x + i * gridDim.x;
      const int pb = i & 1;
      long long* acc_i = acc + pb * cells;
      const float* cent_i = cent_sm + pb * cells;
      // re-decided rows go straight into acc_i: wait until the fold two instances back cleared it
      if (i >= 2) mbar_wait(&accclear[pb], ((i >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
      for (int t = 0; t < T; ++t, ++g) {
        const int st = g % n_stages, ab = g & 1, ob = g & 1;
        const int rows = min(kQTile, nq - t * kQTile);
        const unsigned char* qs = stage_smem + st * C::kStageBytes;
        int* assign_t = a.assign_out ? a.assign_out + static_cast<size_t>(e) * nq + t * kQTile : nullptr;

        // ---- dots and norm of this thread's query from tensor memory
        bool have = !*abort_flag && mbar_wait(&accfull[ab], (g >> 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
        have = __all_sync(0xffffffffu, have);
        float best = -INFINITY, second = -INFINITY, qn2 = 0.f;
        int bi = -1;
        bool any_valid = false;  // a valid beacon (screened values that are all NaN leave bi at -1)
        if (have) {
          tc_fence_after();
          const uint32_t d = tmem + ab * acc_cols + lane_addr;
          float v[32];
          tmem_ld32(d + ncols1 + quarter * 32, v);  // Q Q^T columns of this quarter: the diagonal is v[lane]
          tmem_wait_ld();
#pragma unroll
          for (int k = 0; k < 32; ++k) qn2 = (k == lane) ? v[k] : qn2;
          for (int c0 = 0; c0 < nbp; c0 += 8) {
            uint32_t h[8], l[8];
            asm volatile(
                "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                : "=r"(h[0]), "=r"(h[1]), "=r"(h[2]), "=r"(h[3]), "=r"(h[4]), "=r"(h[5]), "=r"(h[6]), "=r"(h[7])
                : "r"(d + c0));
            asm volatile(
                "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                : "=r"(l[0]), "=r"(l[1]), "=r"(l[2]), "=r"(l[3]), "=r"(l[4]), "=r"(l[5]), "=r"(l[6]), "=r"(l[7])
                : "r"(d + nbp + c0));
            tmem_wait_ld();
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              const int b = c0 + u;
              if (b < nb && bvalid[pb][b]) {
                any_valid = true;
                const float dot = __uint_as_float(h[u]) + __uint_as_float(l[u]);
                if (dot > best) {
                  second = best;
                  best = dot;
                  bi = b;
                } else if (dot > second) {
                  second = dot;
                }
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&accfree[ab]);

        // ---- decision; close calls go to the exact list; counts per beacon by ballot
        int my_b = -1, my_pos = 0;
        if (have && n < rows) {
          if (any_valid && (degenerate[pb] || !(qn2 > 1e-30f && qn2 < 1e30f) ||
                          !(best - second > kMarginRel * sqrtf(qn2)))) {
            refine_t[ob][atomicAdd(&n_refine[ob], 1)] = n;
          } else {
            my_b = bi;
            if (assign_t) assign_t[n] = bi;
          }
        }
        for (int b = 0; b < nb; ++b) {
          const unsigned m = __ballot_sync(0xffffffffu, my_b == b);
          if (lane == b) cnt_w[ob][quarter][b] = __popc(m);
          if (my_b == b) my_pos = __popc(m & lt);
        }
        named_barrier(1, 32 * kScreeners);

        // ---- sorted row list for the accumulators (its buffer is free once they are done with tile g - 2)
        if (g >= 2) mbar_wait(&sempty[ob], ((g >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
        if (ts == 0) n_refine[ob ^ 1] = 0;  // the next tile's list; its previous readers finished a tile ago
        {
          int tot = 0, mine = 0;
          if (lane < nb)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int c = cnt_w[ob][q][lane];
              tot += c;
              mine += (q < quarter) ? c : 0;
            }
          int incl = tot;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
          }
          const int off = incl - tot + mine;  // where this warp's rows of beacon `lane` start
          const int my_off = __shfl_sync(0xffffffffu, off, my_b < 0 ? 0 : my_b);
          if (my_b >= 0) order_t[ob][my_off + my_pos] = n | (my_b << 8);
          if (quarter == 0) {
            if (lane == 31) n_asg_sh[ob] = incl;
            if (lane < nb && tot > 0) atomicAdd(&add_cnt[pb][lane], tot);  // refinements add concurrently
          }
        }

        // ---- exact decisions for close calls, one warp per query; the row is added here
        const int nr = n_refine[ob];
        for (int k = ws; k < nr; k += kScreeners) {
          const int r = refine_t[ob][k];
          float x[D / 32];
#pragma unroll
          for (int j = 0; j < D / 32; ++j)
            x[j] = __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(qs + sw128_offset(r, lane + 32 * j, kQBox)));
          const int best_b = exact_decision<D>(
              x, nb, [&](int b, int col) { return cent_i[b * D + col]; }, [&](int b) { return bvalid[pb][b] != 0; },
              cninv[pb]);
          if (lane == 0) {
            if (assign_t) assign_t[r] = best_b;
            if (best_b >= 0) atomicAdd(&add_cnt[pb][best_b], 1);
          }
          if (best_b >= 0) {
            long long sr[kCols];
#pragma unroll
            for (int c = 0; c < kCols; ++c) sr[c] = 0;
            add_fixed<kCols>(sr, qs + sw128_offset(r, col0, kQBox));
#pragma unroll
            for (int c = 0; c < kCols; ++c)
              shared_add_i64(&acc_i[best_b * D + c * 32 + lane], sr[c]);
          }
        }
        named_barrier(1, 32 * kScreeners);
        if (ts == 0) mbar_arrive(&sfull[ob]);
      }
    }
  } else if (warp < 2 + kScreeners + kAccum) {
    // ---------------------------------------------------------------- accumulators
    const int wa = warp - 2 - kScreeners;               // 0 .. kAccum - 1
    const int ta = threadIdx.x - 32 * (2 + kScreeners);  // 0 .. 32 * kAccum - 1
    const int col0 = lane * kCols;
    const int chunk = (col0 & 63) >> 3;
    const uint32_t lane_off = (col0 >> 6) * kQBox + ((col0 & 7) << 1);
    int g = 0;
    for (int i = 0; i < n_my; ++i) {
      const int pb = i & 1;
      long long* acc_i = acc + pb * cells;
      if (i >= 2) mbar_wait(&accclear[pb], ((i >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
      for (int t = 0; t < T; ++t, ++g) {
        const int st = g % n_stages, ob = g & 1;
        const unsigned char* qs = stage_smem + st * C::kStageBytes + lane_off;
        const bool ready = mbar_wait(&sfull[ob], (g >> 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
        const int n_asg = ready ? n_asg_sh[ob] : 0;
        const int* ord = order_t[ob];
        const int p1 = (wa + 1) * n_asg / kAccum;
        int p = wa * n_asg / kAccum;
        auto row_ptr = [&](int en) {
          const int r = en & 0xff;
          return qs + r * 128 + ((chunk ^ (r & 7)) << 4);
        };
        constexpr int kPairs = kCols / 2;
        Parts2 s[kPairs];
#pragma unroll
        for (int h = 0; h < kPairs; ++h) s[h] = Parts2{0ull, 0ull, 0ull};
        int cur = -1;
        auto flush = [&]() {
#pragma unroll
          for (int c = 0; c < kCols; ++c)
            shared_add_i64(&acc_i[cur * D + c * 32 + lane], fixed40(parts2_get(s[c >> 1], c & 1)));
#pragma unroll
          for (int h = 0; h < kPairs; ++h) s[h] = Parts2{0ull, 0ull, 0ull};
        };
        auto add_row = [&](const unsigned char* rp) {
          if constexpr (kCols == 4) {
            const uint2 v = *reinterpret_cast<const uint2*>(rp);
            parts2_add(s[0], v.x);
            parts2_add(s[1 % kPairs], v.y);
          } else {
            parts2_add(s[0], *reinterpret_cast<const uint32_t*>(rp));
          }
        };
        while (p < p1) {
          if (p + kGroup <= p1 && (ord[p] >> 8) == cur && (ord[p + kGroup - 1] >> 8) == cur) {
            // sorted: the group's rows share the beacon
#pragma unroll
            for (int r = 0; r < kGroup; ++r) add_row(row_ptr(ord[p + r]));
            p += kGroup;
            continue;
          }
          const int en = ord[p];
          const int b = en >> 8;
          if (b != cur) {
            if (cur >= 0) flush();
            cur = b;
          }
          add_row(row_ptr(en));
          ++p;
        }
        if (cur >= 0) flush();
        named_barrier(2, 32 * kAccum);
        if (ta == 0) {
          mbar_arrive(&empty_bar[st]);  // the stage's queries are no longer read
          mbar_arrive(&sempty[ob]);
          if (t == T - 1) mbar_arrive(&accdone[pb]);  // this instance's sums are complete
        }
      }
    }
  } else {
    // ---------------------------------------------------------------- bookkeeping
    const int wk = warp - 2 - kScreeners - kAccum;  // 0 .. 3
    const int tk = threadIdx.x - 32 * (2 + kScreeners + kAccum);
    const uint32_t cbytes = static_cast<uint32_t>(cells) * 4, sbytes = static_cast<uint32_t>(cells) * 8;
    auto inst = [&](int idx) { return blockIdx.x + idx * gridDim.x; };
    auto issue_cent = [&](int idx) {  // centroids of instance idx into cent_sm[idx & 1]
      fence_proxy_async_smem();
      mbar_arrive_expect_tx(&cbar[idx & 1], cbytes);
      bulk_copy_g2s(cent_sm + (idx & 1) * cells, a.cent + static_cast<size_t>(inst(idx)) * cells, cbytes,
                    &cbar[idx & 1]);
    };
    auto issue_sums = [&](int idx) {
      fence_proxy_async_smem();
      mbar_arrive_expect_tx(&sbar, sbytes);
      bulk_copy_g2s(sums_sm, a.sums + static_cast<size_t>(inst(idx)) * cells, sbytes, &sbar);
    };
    auto build = [&](int idx) {
      const int pb = idx & 1;
      const int e = inst(idx);
      if (tk < nb) cnt_old[pb][tk] = a.counts[static_cast<size_t>(e) * nb + tk];
      if (tk == 0) degenerate[pb] = 0;
      mbar_wait(&cbar[pb], (idx >> 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
      if (idx >= 2) mbar_wait(&bfree[pb], ((idx >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
      named_barrier(3, 32 * kKeepers);
      const float* cs = cent_sm + pb * cells;
      unsigned char* bm = bmat + pb * C::bmat_bytes(nbp);
      for (int b = wk; b < nbp; b += kKeepers) {
        float c[D / 32];
        float n2 = 0.f;
        DF n2d{0.f, 0.f};  // the exact products c^2 summed in double-float arithmetic
        int nz = 0;
#pragma unroll
        for (int k = 0; k < D / 32; ++k) {
          c[k] = b < nb ? cs[b * D + lane + 32 * k] : 0.f;
          n2 = fmaf(c[k], c[k], n2);
          n2d = df_add(n2d, df_two_prod(c[k], c[k]));
          nz |= (c[k] != 0.f);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          n2 += __shfl_xor_sync(0xffffffffu, n2, o);
          nz |= __shfl_xor_sync(0xffffffffu, nz, o);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
          n2d = df_add(n2d, DF{__shfl_xor_sync(0xffffffffu, n2d.hi, o), __shfl_xor_sync(0xffffffffu, n2d.lo, o)});
        const bool ok = b < nb && cnt_old[pb][b] > 0 && nz;
        const float inv = ok ? rsqrtf(n2) : 0.f;
#pragma unroll
        for (int k = 0; k < D / 32; ++k) {
          const int col = lane + 32 * k;
          const float u = c[k] * inv;
          const __nv_bfloat16 hi = __float2bfloat16_rn(u);
          const __nv_bfloat16 lo = __float2bfloat16_rn(u - __bfloat162float(hi));
          *reinterpret_cast<__nv_bfloat16*>(bm + sw128_offset(b, col, bbox)) = hi;
          *reinterpret_cast<__nv_bfloat16*>(bm + sw128_offset(nbp + b, col, bbox)) = lo;
        }
        if (lane == 0 && b < nb) {
          bvalid[pb][b] = ok;
          bool plain = true;
          DF inv_df{0.f, 0.f};
          if (ok) inv_df = centroid_inv_norm(n2d, n2, plain);
          cninv[pb][b] = inv_df;
          if (!plain) degenerate[pb] = 1;
        }
      }
      fence_proxy_async_smem();  // generic-proxy writes, read next by the tensor cores
      named_barrier(3, 32 * kKeepers);
      if (tk == 0) mbar_arrive(&bready[pb]);
    };
    auto fold = [&](int idx) {
      const int pb = idx & 1;
      const int e = inst(idx);
      long long* acc_i = acc + pb * cells;
      mbar_wait(&accdone[pb], (idx >> 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
      mbar_wait(&sbar, idx & 1, abort_flag, a.err, kDevTimeoutEpilogue);
      if (tk < nb) rcp_sh[tk] = count_reciprocal(cnt_old[pb][tk] + add_cnt[pb][tk]);
      named_barrier(3, 32 * kKeepers);
      for (int c = tk; c < cells; c += 32 * kKeepers) {
        const int b = c / D, col = c - b * D;
        const int ai = b * D + (col % kCols) * 32 + col / kCols;  // the accumulator cell of (b, col)
        if (add_cnt[pb][b] > 0) {
          const size_t gi = static_cast<size_t>(e) * cells + c;
          const double s_new = fold_sum_fp64(sums_sm[c], acc_i[ai]);
          a.sums[gi] = s_new;
          a.cent[gi] = centroid_value(s_new, rcp_sh[b]);
        }
        acc_i[ai] = 0;  // the cell this thread read: no other thread touches it
      }
      named_barrier(3, 32 * kKeepers);
      if (tk < nb) {
        if (add_cnt[pb][tk] > 0) a.counts[static_cast<size_t>(e) * nb + tk] = cnt_old[pb][tk] + add_cnt[pb][tk];
        add_cnt[pb][tk] = 0;
      }
      named_barrier(3, 32 * kKeepers);
      if (tk == 0) {
        mbar_arrive(&accclear[pb]);
        if (idx + 1 < n_my) issue_sums(idx + 1);
        if (idx + 2 < n_my) issue_cent(idx + 2);
      }
    };

    if (n_my > 0) {
      if (tk == 0) {
        issue_cent(0);
        issue_sums(0);
        if (n_my > 1) issue_cent(1);
      }
      build(0);
      for (int i = 0; i < n_my; ++i) {
        if (i + 1 < n_my) build(i + 1);
        fold(i);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace

cudaError_t launch_update(const Shape& s, const CUtensorMap& qmap, int box_rows, int n_new, float* cent,
                          double* sums, long long* counts, int* assign_out, int* err, cudaStream_t st) {
  UpdArgs a;
  a.n_inst = s.n_inst;
  a.nq = s.G * n_new;
  a.box_rows = box_rows;
  a.nb = s.nb;
  a.nbp = (s.nb + 7) / 8 * 8;
  a.cent = cent;
  a.sums = sums;
  a.counts = counts;
  a.assign_out = assign_out;
  a.err = err;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int grid = s.n_inst < sms ? s.n_inst : sms;
  if (s.d == 128) {
    using C = UpdCfg<128>;
    const size_t smem = C::smem_bytes(a.nb, a.nbp);
    cudaError_t e =
        cudaFuncSetAttribute(update_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    update_kernel<128><<<grid, kUThreads, smem, st>>>(qmap, a, C::stages(a.nb, a.nbp));
  } else {
    using C = UpdCfg<64>;
    const size_t smem = C::smem_bytes(a.nb, a.nbp);
    cudaError_t e =
        cudaFuncSetAttribute(update_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    update_kernel<64><<<grid, kUThreads, smem, st>>>(qmap, a, C::stages(a.nb, a.nbp));
  }
  return cudaGetLastError();
}

}  // namespace bkv
