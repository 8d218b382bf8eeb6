// Scoring of every cached key (Eq. 4 softmax over the whole cache, Eq. 6 max
// form, maximum over the GQA group's observation queries; Section 4.3).
//
// Persistent kernel, one CTA per SM.  Instances are processed by
// thread-block clusters of C CTAs; cluster k takes instances k,
// k + n_clusters, ...; CTA r of a cluster owns the same contiguous range of
// keys of every instance, the cache split in 32-key units as evenly as
// possible, and walks it in 128-key tiles (a ragged last tile is loaded in
// 32-row boxes; the MMA lanes past the range are ignored).
//
// Each tile goes through the tensor cores once: D = K_tile x Qobs^T with
// M = 128 keys (TMEM lanes) and N = padded query count (TMEM columns),
// bf16 x bf16 -> fp32 (tcgen05.mma, operands staged by TMA with 128-byte
// swizzle).  The fp32 logits of every tile a CTA owns stay resident in
// tensor memory, in a ring of N-column slots that successive instances fill
// in turn (slots left over by one instance let the next one's tiles land
// while it finishes), so K is read from HBM exactly once.  y = logit * log2(e) is the base-2 logit.
//   Pass 1 (statistics, as tiles land): each thread owns one key of the tile
//     and keeps, for the query columns it owns, a reference m_q and the sum
//     s_q of 2^(y - m_q) over the keys it has seen (m_q follows the maximum
//     lazily, so that the terms stay below 2^64).  After the CTA's last tile the partials are merged
//     (recursive halving inside each warp, shared memory across warps) and
//     the CTAs of a cluster exchange theirs through distributed shared memory;
//     every CTA combines them in rank order and gets the same
//     lse2_q = log2 sum_j 2^(y_qj) over all L keys.
//   Pass 2 (scores, from tensor memory): r_j = max over valid q of
//     (y_qj - lse2_q) = log2 Score_j, or under mean aggregation
//     r_j = log2 of the mean over the valid q of 2^(y_qj - lse2_q).
// When a CTA owns more tiles than tensor memory holds (very long caches), the
// tiles past the resident ones cycle through two streaming slots in pass 1
// and are loaded and multiplied a second time for pass 2, into one slot per
// pass-2 warp half.  Every slot barrier thus has a fixed set of warps that
// waits on each of its uses in order, which keeps the parity waits exact.
//
// Warp roles (10 warps): warp 0 TMA producer (queries into one of two
// buffers, K tiles through a ring of shared-memory stages); warp 1 TMEM
// allocation and MMA issue; warps 2..9 epilogue, two warps per TMEM lane
// quarter: in pass 1 each owns half of the query columns, in pass 2 each
// takes every other tile with all columns.
//
// Cross-CTA exchange (all waits bounded): barriers are initialised, then a
// cluster barrier.  Per instance every CTA pushes its (m, s) column partials
// into each peer's receive buffer with st.async, whose bytes complete on the
// peer's receive barrier; the receiver arms that barrier with the byte count
// of all csize senders.  Receive buffers and barriers alternate between two
// copies by instance parity: a sender can be at most one instance ahead of
// any receiver, since it needs every peer's partials of the instance before.
// No release fence at cluster scope sits on this path (one would wait for the
// CTA's score stores, queued behind the K stream).  The exchange runs for
// every instance even after a timeout, and the kernel ends with a cluster
// barrier, so no CTA leaves while a peer may still write to its shared memory.
// Outputs: r (log2 scores, for selection) and optionally 2^r.
//
// Column split: a launch takes at most 64 scoring queries, Q_obs rows
// [col0, col0 + N).  Each query's normaliser lse2_q depends on its own column
// only, so with more queries the caller runs one launch per 64 rows and every
// later launch folds its r into the previous one (max: the larger; mean: the
// log2 of the sum of the two powers of 2, both scaled by the count of all
// valid queries).  K is then read once per launch, and the tensor memory ring
// keeps spare slots at every query count.
//
// Causal form (CAUSAL): recent slot w must not see window rows after its own
// position (row j >= L - W is masked for it when j > thr[w]); beacons and
// older rows are never masked.  Only tiles that hold window rows take the
// masked paths: pass 1 skips the masked (row, column) terms of the
// statistics, pass 2 leaves them out of the maximum or the mean (a masked
// weight is 0 and still counts in the mean's query count).
//
// This header holds the kernel template; k_score.cu instantiates the max
// form, k_score_mean.cu the mean form and k_score_causal*.cu their causal
// forms, so that they compile in parallel.
#pragma once
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kEpiWarps = 8;
constexpr int kScThreads = 32 * (2 + kEpiWarps);
constexpr int kTile = 128;                  // keys per tile (MMA M)
constexpr uint32_t kBoxBytes = 128 * 128;   // [128 rows][64 bf16] swizzled box
constexpr uint32_t kTmemCols = 512;
constexpr int kMaxStages = 12;
constexpr int kMaxSlots = 32;               // tensor-memory slots (resident + streaming)
constexpr size_t kSmemBudget = 220 * 1024;  // dynamic shared memory of the one CTA per SM

template <int D>
struct ScoreCfg {
  static constexpr int kBoxes = D / 64;                  // 64-column boxes per row
  static constexpr uint32_t kTileBytes = kTile * D * 2;  // one K tile
  static size_t q_bytes(int n_cols) { return 2 * static_cast<size_t>(kBoxes) * n_cols * 128; }
  // two receive buffers of csize x n_cols (m, s) pairs
  static size_t recv_bytes(int n_cols, int csize) {
    return csize > 1 ? 2 * static_cast<size_t>(csize) * n_cols * 8 : 0;
  }
  // as many K stages as fit next to the query and receive buffers
  static int stages(int n_cols, int csize) {
    const size_t room = kSmemBudget - 1024 - q_bytes(n_cols) - recv_bytes(n_cols, csize);
    const int n = static_cast<int>(room / (static_cast<size_t>(kBoxes) * kBoxBytes));
    return n < kMaxStages ? n : kMaxStages;
  }
  static size_t smem_bytes(int n_cols, int csize) {
    return 1024 + q_bytes(n_cols) + static_cast<size_t>(stages(n_cols, csize)) * kBoxes * kBoxBytes +
           recv_bytes(n_cols, csize);
  }
};

// Placement of one instance's tiles: cluster size and resident ring slots;
// `stream` adds four streaming slots after the ring (two rotating pass-1
// slots, one pass-2 slot per epilogue half).
struct Plan {
  int csize, slots, stream;
};

// This CTA's share of one instance of L keys: keys [k0, k1), T tiles, the first R of them resident
// in the ring and n_str streaming.  The producer, the MMA issuer and the epilogue all derive it from
// the same L, so they agree on every instance's job list.
struct Geom {
  int k0, k1, T, R, n_str;
};

__device__ __forceinline__ Geom inst_geom(int L, int crank, int csize, int slots) {
  Geom g;
  const int U = (L + 31) / 32;  // 32-key units of the cache
  g.k0 = (crank * U / csize) * 32;
  g.k1 = min(L, ((crank + 1) * U / csize) * 32);
  g.T = (g.k1 - g.k0 + kTile - 1) / kTile;
  g.R = g.T < slots ? g.T : slots;
  g.n_str = g.T - g.R;
  return g;
}

// Instance of work item w and its number of keys: the compact list of a per-instance-length
// compress, or every instance with the launch's L.
// In a BKV_CHECKED build an entry outside 0 .. n_inst - 1 is recorded and replaced by instance 0, and a
// length outside 1 .. L (the launch's longest) by L, identically in every role, so that the roles still agree on
// each instance's job list (the outputs are then flagged invalid by the error word).
__device__ __forceinline__ int item_inst(const ScoreArgs& a, int w, int n_inst) {
  if (!a.work) return w;
  const int e = a.work[w];
  return in_bounds(e, n_inst, a.err) ? e : 0;
}
__device__ __forceinline__ int inst_len(const ScoreArgs& a, int e) {
  if (!a.Ls) return a.L;
  const int L = a.Ls[e];
  return in_bounds(L - 1, a.L, a.err) ? L : a.L;
}

// Wait used while draining after an abort: ignores the abort flag.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, int* err) {
  int never = 0;
  mbar_wait(bar, parity, &never, err, kDevTimeoutDrain);
}

// Read-only global load emitted exactly here (the compiler may not sink it
// towards its first use, where its latency behind the K stream would show).
__device__ __forceinline__ uint32_t ld_nc_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.global.nc.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}

// Asynchronous store of (m, s) into a peer CTA's shared memory; its 8 bytes
// complete on the peer's barrier `bar` (both shared::cluster addresses).
__device__ __forceinline__ void st_async_pair(uint32_t dst, float m, float s, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(dst),
               "f"(m), "f"(s), "r"(bar)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive_cnt(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// Merge of two base-2 log-sum-exp partials (m, s) -> (max, rescaled sum).
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  const float a = (m == M) ? s : s * ex2_approx(m - M);
  const float b = (m2 == M) ? s2 : s2 * ex2_approx(m2 - M);
  m = M;
  s = a + b;
}

// Merge of NQ per-lane column partials across the 32 lanes of a warp.  Steps
// halve the columns a lane holds while their count is even and exchange all of
// them otherwise.  Returns the first column of the lane's result block (the
// block is m[0 .. count-1]); `writer` is true for one lane per block.
template <int NQ>
__device__ __forceinline__ int warp_merge_columns(float (&m)[NQ], float (&s)[NQ], int lane, bool& writer) {
  int first = 0;
  writer = true;
  int cols = NQ;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    if (cols % 2 == 0) {
      const int half = cols / 2;
      const bool upper = (lane & o) != 0;
#pragma unroll
      for (int i = 0; i < NQ / 2; ++i) {
        if (i < half) {
          const float send_m = upper ? m[i] : m[i + half];
          const float send_s = upper ? s[i] : s[i + half];
          const float keep_m = upper ? m[i + half] : m[i];
          const float keep_s = upper ? s[i + half] : s[i];
          const float got_m = __shfl_xor_sync(0xffffffffu, send_m, o);
          const float got_s = __shfl_xor_sync(0xffffffffu, send_s, o);
          m[i] = keep_m;
          s[i] = keep_s;
          lse_merge(m[i], s[i], got_m, got_s);
        }
      }
      if (upper) first += half;
      cols = half;
    } else {
#pragma unroll
      for (int i = 0; i < NQ; ++i) {
        if (i < cols) {
          const float got_m = __shfl_xor_sync(0xffffffffu, m[i], o);
          const float got_s = __shfl_xor_sync(0xffffffffu, s[i], o);
          lse_merge(m[i], s[i], got_m, got_s);
        }
      }
      if (lane & o) writer = false;
    }
  }
  return first;
}

// r = max over the N columns of (v * sc - lse2), columns read from tensor
// memory in chunks of 32 (16 for a ragged last chunk).
template <int N>
__device__ __forceinline__ float tile_score(uint32_t taddr, const float* lse2, float sc) {
  float r0 = -INFINITY, r1 = -INFINITY;
#pragma unroll
  for (int c0 = 0; c0 < N; c0 += 32) {
    float v[32];
    if (c0 + 32 <= N) {
      tmem_ld32(taddr + c0, v);
    } else {
      tmem_ld16(taddr + c0, v);
    }
    tmem_wait_ld();
#pragma unroll
    for (int u = 0; u < 32; u += 4) {
      if (c0 + u < N) {
        const float4 l = *reinterpret_cast<const float4*>(lse2 + c0 + u);
        r0 = fmaxf(r0, fmaf(v[u], sc, -l.x));
        r1 = fmaxf(r1, fmaf(v[u + 1], sc, -l.y));
        r0 = fmaxf(r0, fmaf(v[u + 2], sc, -l.z));
        r1 = fmaxf(r1, fmaf(v[u + 3], sc, -l.w));
      }
    }
  }
  return fmaxf(r0, r1);
}

// The N (<= 64) columns of this thread's lane of a slot, all loaded before one wait: the slot can be
// released before the arithmetic.
template <int N>
__device__ __forceinline__ void tile_load(uint32_t taddr, float (&v)[64]) {
  static_assert(N <= 64 && N % 16 == 0, "columns in loads of 32 and 16");
#pragma unroll
  for (int c0 = 0; c0 < N; c0 += 32) {
    if (c0 + 32 <= N) {
      tmem_ld32(taddr + c0, *reinterpret_cast<float(*)[32]>(v + c0));
    } else {
      tmem_ld16(taddr + c0, v + c0);
    }
  }
  tmem_wait_ld();
}

// tile_score on loaded columns.
template <int N>
__device__ __forceinline__ float tile_score_regs(const float (&v)[64], const float* lse2, float sc) {
  float r0 = -INFINITY, r1 = -INFINITY;
#pragma unroll
  for (int u = 0; u < N; u += 4) {
    const float4 l = *reinterpret_cast<const float4*>(lse2 + u);
    r0 = fmaxf(r0, fmaf(v[u], sc, -l.x));
    r1 = fmaxf(r1, fmaf(v[u + 1], sc, -l.y));
    r0 = fmaxf(r0, fmaf(v[u + 2], sc, -l.z));
    r1 = fmaxf(r1, fmaf(v[u + 3], sc, -l.w));
  }
  return fmaxf(r0, r1);
}

// r = log2 of inv_m times the sum over the N columns of 2^(v * sc - lse2)
// (mean aggregation; a column with lse2 = +inf adds nothing).
template <int N>
__device__ __forceinline__ float tile_mean(uint32_t taddr, const float* lse2, float sc, float inv_m) {
  float s0 = 0.f, s1 = 0.f;
#pragma unroll
  for (int c0 = 0; c0 < N; c0 += 32) {
    float v[32];
    if (c0 + 32 <= N) {
      tmem_ld32(taddr + c0, v);
    } else {
      tmem_ld16(taddr + c0, v);
    }
    tmem_wait_ld();
#pragma unroll
    for (int u = 0; u < 32; u += 4) {
      if (c0 + u < N) {
        const float4 l = *reinterpret_cast<const float4*>(lse2 + c0 + u);
        s0 += ex2_approx(fmaf(v[u], sc, -l.x));
        s1 += ex2_approx(fmaf(v[u + 1], sc, -l.y));
        s0 += ex2_approx(fmaf(v[u + 2], sc, -l.z));
        s1 += ex2_approx(fmaf(v[u + 3], sc, -l.w));
      }
    }
  }
  return lg2_approx((s0 + s1) * inv_m);
}

template <int N, bool MEAN>
__device__ __forceinline__ float tile_agg(uint32_t taddr, const float* lse2, float sc, float inv_m) {
  if constexpr (MEAN) {
    return tile_mean<N>(taddr, lse2, sc, inv_m);
  } else {
    return tile_score<N>(taddr, lse2, sc);
  }
}

// r of a key over the columns of two launches (column split): the max form
// keeps the larger, the mean form adds the two powers of 2 (both launches
// scale by the count of all valid queries).
template <bool MEAN>
__device__ __forceinline__ float fold_split(float r_prev, float r) {
  if constexpr (MEAN) {
    const float hi = fmaxf(r_prev, r), lo = fminf(r_prev, r);
    return hi == -INFINITY ? hi : hi + lg2_approx(1.f + ex2_approx(lo - hi));
  } else {
    return fmaxf(r_prev, r);
  }
}

// tile_agg for a tile that holds window rows: column c is left out for key
// `key` when key >= win0 and key > thr[c].
template <int N, bool MEAN>
__device__ __forceinline__ float tile_agg_causal(uint32_t taddr, const float* lse2, float sc, float inv_m, int key,
                                                 int win0, const int* thr) {
  const bool in_win = key >= win0;
  float r = -INFINITY, sum = 0.f;
#pragma unroll
  for (int c0 = 0; c0 < N; c0 += 32) {
    float v[32];
    if (c0 + 32 <= N) {
      tmem_ld32(taddr + c0, v);
    } else {
      tmem_ld16(taddr + c0, v);
    }
    tmem_wait_ld();
#pragma unroll
    for (int u = 0; u < 32; ++u) {
      const int c = c0 + u;
      if (c < N && !(in_win && key > thr[c])) {
        const float x = fmaf(v[u], sc, -lse2[c]);
        if constexpr (MEAN) {
          sum += ex2_approx(x);
        } else {
          r = fmaxf(r, x);
        }
      }
    }
  }
  if constexpr (MEAN) {
    return lg2_approx(sum * inv_m);
  } else {
    return r;
  }
}

template <int D, int NQ, bool MEAN, bool CAUSAL, bool COMBINE>
__global__ void __launch_bounds__(kScThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap kmap32,
                 const __grid_constant__ CUtensorMap qmap, Shape s, ScoreArgs a, Plan plan, int n_stages) {
  using C = ScoreCfg<D>;
  constexpr int N = 2 * NQ;  // padded query columns
  static_assert(NQ % 8 == 0 && NQ <= 32, "query columns per pass-1 warp");
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages], empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t slot_full[kMaxSlots], slot_free[kMaxSlots];
  __shared__ __align__(8) uint64_t qfull_bar[2], qempty_bar[2], drain_bar;
  __shared__ __align__(8) uint64_t recv_bar[2];
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;
  __shared__ __align__(16) float lse2_sh[128];
  __shared__ int vcount_sh[4];  // valid queries per 32-column group of the instance (mean aggregation)
  __shared__ int thr_sh[CAUSAL ? 2 : 1][CAUSAL ? 128 : 1];  // causal form: last visible window row per column
  __shared__ float wred_m[kEpiWarps][64], wred_s[kEpiWarps][64];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int csize = plan.csize;
  const int crank = csize > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int cluster_id = blockIdx.x / csize;
  const int n_clusters = gridDim.x / csize;
  int n_items = a.work ? *a.n_work : s.n_inst;  // instances to compress
  if (!in_bounds(n_items, s.n_inst + 1, a.err)) n_items = 0;
  const int n_my = cluster_id < n_items ? (n_items - cluster_id + n_clusters - 1) / n_clusters : 0;
  const int ring = plan.slots;                       // resident slots, used in cyclic order
  const int str_slot = ring;                         // pass-1 streaming slots; +2, +3: pass-2 slots
  const uint32_t qbox = static_cast<uint32_t>(a.n_cols) * 128;  // one 64-column box of this launch's queries (N rows)
  const int col0 = COMBINE ? a.col0 : 0;  // only a later launch of a column split starts past row 0

  // 1024-byte aligned (the 128-byte swizzle pattern repeats every 1024 bytes);
  // offset from the __shared__ array itself so that accesses stay shared-space
  unsigned char* base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  unsigned char* q_smem = base;                         // [2 buffers][kBoxes][N rows x 128 B]
  unsigned char* k_smem = base + 2 * C::kBoxes * qbox;  // [n_stages][kBoxes][128 rows x 128 B]
  float2* recv = reinterpret_cast<float2*>(k_smem + n_stages * C::kBoxes * kBoxBytes);  // [2][csize][N]

  if (threadIdx.x == 0) {
    for (int i = 0; i < n_stages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < kMaxSlots; ++i) {
      mbar_init(&slot_full[i], 1);
      mbar_init(&slot_free[i], kEpiWarps);  // eight warp arrivals per use
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&qfull_bar[i], 1);
      mbar_init(&qempty_bar[i], 1);
    }
    mbar_init(&drain_bar, 1);
    mbar_init(&recv_bar[0], 1);
    mbar_init(&recv_bar[1], 1);
    abort_sh = 0;
    fence_mbar_init();
  }
  if constexpr (CAUSAL) {
    if (threadIdx.x < 128 && !a.gaps) {  // one call-wide table; with per-instance lengths see the epilogue
      const int c = col0 + threadIdx.x;  // Q_obs row: recent slot c % W of head c / W, or a beacon / padding
      thr_sh[0][threadIdx.x] = c < s.G * s.W ? a.thr[c % s.W] : 0x7fffffff;
    }
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base_sh, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (csize > 1) cluster_sync_all();  // peers' barriers exist before anyone arrives on them
  const uint32_t tmem = tmem_base_sh;
  volatile int* abort_flag = &abort_sh;

  // Job order of an instance (producer, MMA and epilogue agree on it):
  // pass-1 jobs for tiles 0 .. T-1, then pass-2 jobs for the streaming tiles.
  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      const uint64_t once = l2_policy_evict_first(), again = l2_policy_evict_last();
      prefetch_tmap(&kmap);
      prefetch_tmap(&kmap32);
      prefetch_tmap(&qmap);
      int g = 0;  // ring iteration
      bool ok = true;
      int q_issued = 0;
      for (int i = 0; ok && i < n_my; ++i) {
        const int e = item_inst(a, cluster_id + i * n_clusters, s.n_inst);
        const Geom gm = inst_geom(inst_len(a, e), crank, csize, ring);
        const int k0 = gm.k0, k1 = gm.k1, T = gm.T, R = gm.R, n_str = gm.n_str;
        const int qb = i & 1;
        if (i >= 2 && !mbar_wait(&qempty_bar[qb], ((i >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutProducer)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&qfull_bar[qb], static_cast<uint32_t>(a.n_cols) * D * 2);
        for (int b = 0; b < C::kBoxes; ++b)
          tma_load_2d(q_smem + (qb * C::kBoxes + b) * qbox, &qmap, &qfull_bar[qb], b * 64,
                      e * s.n_obs_pad + col0, again);
        q_issued = i + 1;
        for (int j = 0; j < T + n_str; ++j) {
          const int t = j < T ? j : R + (j - T);
          const int st = g % n_stages;
          if (g >= n_stages &&
              !mbar_wait(&empty_bar[st], ((g / n_stages) - 1) & 1, abort_flag, a.err, kDevTimeoutProducer)) {
            ok = false;
            break;
          }
          const uint64_t pol = (j < T && t >= R) ? again : once;
          const int row = e * s.cap + k0 + t * kTile;
          const int rows = min(kTile, k1 - k0 - t * kTile);
          unsigned char* dst = k_smem + st * C::kBoxes * kBoxBytes;
          if (rows == kTile) {
            mbar_arrive_expect_tx(&full_bar[st], C::kTileBytes);
            for (int b = 0; b < C::kBoxes; ++b) tma_load_2d(dst + b * kBoxBytes, &kmap, &full_bar[st], b * 64, row, pol);
          } else {  // ragged tile: 32-row boxes at 4 KB steps keep the 128-row swizzled layout
            const int chunks = (rows + 31) / 32;
            mbar_arrive_expect_tx(&full_bar[st], static_cast<uint32_t>(chunks * 32 * D * 2));
            for (int q = 0; q < chunks; ++q)
              for (int b = 0; b < C::kBoxes; ++b)
                tma_load_2d(dst + b * kBoxBytes + q * 4096, &kmap32, &full_bar[st], b * 64, row + q * 32, pol);
          }
          ++g;
        }
      }
      if (!ok || *abort_flag) {  // let every copy already issued land before the CTA exits
        for (int p = (q_issued > 2 ? q_issued - 2 : 0); p < q_issued; ++p)
          drain_wait(&qfull_bar[p & 1], (p >> 1) & 1, a.err);
        for (int j = (g > n_stages ? g - n_stages : 0); j < g; ++j)
          drain_wait(&full_bar[j % n_stages], (j / n_stages) & 1, a.err);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, N);
      int g = 0, ks = 0, kp2_0 = 0, kp2_1 = 0;  // pass-1 streaming uses; pass-2 uses per half
      int rs = 0, ru = 0;                        // next ring slot and its use count
      bool ok = true;
      for (int i = 0; ok && i < n_my; ++i) {
        const int e = item_inst(a, cluster_id + i * n_clusters, s.n_inst);
        const Geom gm = inst_geom(inst_len(a, e), crank, csize, ring);
        const int T = gm.T, R = gm.R, n_str = gm.n_str;
        if (!mbar_wait(&qfull_bar[i & 1], (i >> 1) & 1, abort_flag, a.err, kDevTimeoutMma)) break;
        for (int j = 0; j < T + n_str; ++j) {
          const int st = g % n_stages;
          int slot, u;
          if (j < R) {
            slot = rs;
            u = ru;
          } else if (j < T) {
            slot = str_slot + (ks & 1);
            u = ks >> 1;
          } else {
            const int h = (j - T) & 1;
            slot = str_slot + 2 + h;
            u = h ? kp2_1 : kp2_0;
          }
          if (!mbar_wait(&full_bar[st], (g / n_stages) & 1, abort_flag, a.err, kDevTimeoutMma) ||
              (u >= 1 && !mbar_wait(&slot_free[slot], (u - 1) & 1, abort_flag, a.err, kDevTimeoutMma))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem + slot * N;
          const uint32_t k_addr = smem_u32(k_smem + st * C::kBoxes * kBoxBytes);
          const uint32_t q_addr = smem_u32(q_smem + (i & 1) * C::kBoxes * qbox);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t qoff = (kk >> 2) * qbox + (kk & 3) * 32;
            const uint32_t koff = (kk >> 2) * kBoxBytes + (kk & 3) * 32;
            mma_bf16_ss(d_tmem, sdesc_kmajor_sw128(k_addr + koff), sdesc_kmajor_sw128(q_addr + qoff), idesc, kk > 0);
          }
          mma_commit(&empty_bar[st]);
          mma_commit(&slot_full[slot]);
          ++g;
          if (j < R && ++rs == ring) {
            rs = 0;
            ++ru;
          }
          if (j >= T) {
            if ((j - T) & 1) ++kp2_1;
            else ++kp2_0;
          }
          else if (j >= R) ++ks;
        }
        if (ok) mma_commit(&qempty_bar[i & 1]);  // this instance's queries are no longer read
      }
      mma_commit(&drain_bar);  // every MMA issued above has finished once this arrives
      drain_wait(&drain_bar, 0, a.err);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------------- epilogue
    const int we = warp - 2;                 // 0 .. 7
    const int quarter = warp & 3;            // TMEM lane quarter
    const int half = we >> 2;                // pass 1: column half; pass 2: tile parity
    const int key_row = quarter * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(quarter * 32) << 16;
    const int te = threadIdx.x - 64;         // 0 .. 255
    const bool leader = te == 0;
    const float sc = a.scale_log2;
    int ks = 0, kp2 = 0;  // uses of the pass-1 streaming slots / of this half's pass-2 slot
    int rs = 0, ru = 0;   // ring slot and use count of this instance's first tile
    // valid-row words are fetched one instance ahead: a global load queues
    // behind the K stream for microseconds.  Thread te < N reads the word of
    // its column (Q_obs row col0 + te); the four words that threads 0, 32, 64
    // and 96 read are all of the instance's words in some order (their total
    // is the valid count of the mean form).
    const int vw = COMBINE ? ((col0 >> 5) + (te >> 5)) & 3 : te >> 5;  // this thread's valid word
    int e_next = n_my > 0 ? item_inst(a, cluster_id, s.n_inst) : 0;
    uint32_t vnext = (te < 128 && n_my > 0) ? ld_nc_u32(&a.valid[e_next * 4 + vw]) : 0u;
    for (int i = 0; i < n_my; ++i) {
      const int e = e_next;
      const uint32_t vword = vnext;
      if (i + 1 < n_my) {
        e_next = item_inst(a, cluster_id + (i + 1) * n_clusters, s.n_inst);
        if (te < 128) vnext = ld_nc_u32(&a.valid[e_next * 4 + vw]);
      }
      const int L_e = inst_len(a, e);
      const Geom gm = inst_geom(L_e, crank, csize, ring);
      const int k0 = gm.k0, k1 = gm.k1, T = gm.T, R = gm.R;
      const int win0 = a.gaps ? L_e - s.W : a.win0;  // first window row
      const int* thr = thr_sh[0];
      if constexpr (CAUSAL) {
        if (a.gaps) {  // per-instance lengths: this instance's table, in the buffer of its parity
          thr = thr_sh[i & 1];
          if (te < 128) {
            const int c = col0 + te;
            int t = 0x7fffffff;
            if (c < s.G * s.W) {
              const int g = a.gaps[((e / s.n_kv) % s.batch) * s.W + c % s.W];
              t = g == 0 ? L_e : (g > L_e ? -1 : L_e - 1 - g);
            }
            thr_sh[i & 1][te] = t;
          }
          named_barrier(1, 32 * kEpiWarps);  // the table is written before pass 1 reads it
        }
      }
      float m[NQ], sm[NQ];
#pragma unroll
      for (int c = 0; c < NQ; ++c) {
        m[c] = -INFINITY;
        sm[c] = 0.f;
      }
      bool resident_ok = true;
      // ---- pass 1
      for (int j = 0; j < T; ++j) {
        int slot, u;
        if (j < R) {
          slot = rs + j;
          u = ru;
          if (slot >= ring) {
            slot -= ring;
            ++u;
          }
        } else {
          slot = str_slot + (ks & 1);
          u = ks >> 1;
        }
        bool have = !*abort_flag && mbar_wait(&slot_full[slot], u & 1, abort_flag, a.err, kDevTimeoutEpilogue);
        have = __all_sync(0xffffffffu, have);
        if (j < R) resident_ok = resident_ok && have;
        float v[NQ];
        if (have) {
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < NQ; c += 8) {
            uint32_t r[8];
            asm volatile(
                "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                : "r"(tmem + slot * N + half * NQ + c + lane_addr));
#pragma unroll
            for (int q = 0; q < 8; ++q) v[c + q] = __uint_as_float(r[q]);
          }
          tmem_wait_ld();
        }
        if (j >= R) {  // a streaming slot is free once every warp has its columns
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&slot_free[slot]);
          ++ks;
        }
        // Running sums relative to a reference m that moves only when a base-2
        // logit exceeds it by more than 64, so the terms stay below 2^64 and
        // the common step is one FFMA, one ex2 and one add per column.
        const int tile0 = k0 + j * kTile;
        if (have && CAUSAL && tile0 + kTile > win0) {
          // a tile with window rows: the careful path, without the masked (row, column) terms
          const int key = tile0 + key_row;
          if (key < k1) {
            const bool in_win = key >= win0;
#pragma unroll
            for (int c = 0; c < NQ; ++c) {
              if (in_win && key > thr[half * NQ + c]) continue;
              const float t = fmaf(v[c], sc, -m[c]);
              if (t > 64.f) {
                const float y = v[c] * sc;
                sm[c] = fmaf(sm[c], ex2_approx(m[c] - y), 1.f);
                m[c] = y;
              } else {
                sm[c] += ex2_approx(t);
              }
            }
          }
        } else if (have) {
          const bool key_ok = tile0 + key_row < k1;
          float t[NQ];
          bool rebase = !__all_sync(0xffffffffu, key_ok);  // a ragged tile takes the careful path
#pragma unroll
          for (int c = 0; c < NQ; ++c) {
            t[c] = fmaf(v[c], sc, -m[c]);
            rebase |= t[c] > 64.f;
          }
          if (__any_sync(0xffffffffu, rebase)) {
            if (key_ok) {
#pragma unroll
              for (int c = 0; c < NQ; ++c) {
                if (t[c] > 64.f) {  // also the first key: m = -inf gives t = +inf
                  const float y = v[c] * sc;
                  sm[c] = fmaf(sm[c], ex2_approx(m[c] - y), 1.f);
                  m[c] = y;
                } else {
                  sm[c] += ex2_approx(t[c]);
                }
              }
            }
          } else {
#pragma unroll
            for (int c = 0; c < NQ; ++c) sm[c] += ex2_approx(t[c]);
          }
        }
      }

      // ---- merge: lanes, then the four warps of this column half, then the cluster
      bool writer;
      const int first = warp_merge_columns<NQ>(m, sm, lane, writer);
      constexpr int kKeep = NQ % 32 == 0 ? NQ / 32 : (NQ % 16 == 0 ? NQ / 16 : NQ / 8);
      if (writer)
#pragma unroll
        for (int c = 0; c < kKeep; ++c) {
          wred_m[we][first + c] = m[c];
          wred_s[we][first + c] = sm[c];
        }
      named_barrier(1, 32 * kEpiWarps);  // also: every pass-2 read of the previous lse2 is done
      const bool col_thread = te < N;
      float cm = -INFINITY, cs = 0.f;
      if (col_thread) {
        const int h = te / NQ, cc = te % NQ;  // column te lives in the warps of half h
        for (int w = 0; w < 4; ++w) lse_merge(cm, cs, wred_m[h * 4 + w][cc], wred_s[h * 4 + w][cc]);
      }
      const bool my_valid = col_thread && ((vword >> (te & 31)) & 1u);
      float lse = INFINITY;
      if (csize == 1) {
        if (my_valid && cm > -INFINITY) lse = cm + lg2_approx(cs);
      } else if (col_thread) {
        const int b = i & 1;
        if (leader) mbar_arrive_expect_tx(&recv_bar[b], static_cast<uint32_t>(csize * N * 8));
        const uint32_t dst = smem_u32(&recv[(b * csize + crank) * N + te]), bar = smem_u32(&recv_bar[b]);
        for (int c = 0; c < csize; ++c) st_async_pair(mapa_shared(dst, c), cm, cs, mapa_shared(bar, c));
        const bool ok = mbar_wait_cluster(&recv_bar[b], (i >> 1) & 1, a.err, kDevTimeoutCluster);
        float M = -INFINITY, S = 0.f;
        if (ok)
          for (int c = 0; c < csize; ++c) {  // rank order: every CTA gets the same lse2
            const float2 p = recv[(b * csize + c) * N + te];
            lse_merge(M, S, p.x, p.y);
          }
        if (!ok) *abort_flag = 1;
        if (ok && my_valid && M > -INFINITY) lse = M + lg2_approx(S);
      }
      if (te < 128) lse2_sh[te] = lse;
      if (MEAN && te < 128 && (te & 31) == 0) vcount_sh[te >> 5] = __popc(vword);
      named_barrier(1, 32 * kEpiWarps);  // lse2 written; every read of wred is done
      float inv_m = 0.f;  // 1 / (valid queries), 0 when there are none
      if constexpr (MEAN) {
        const int mv = vcount_sh[0] + vcount_sh[1] + vcount_sh[2] + vcount_sh[3];
        if (mv > 0) inv_m = 1.f / static_cast<float>(mv);
      }

      // ---- pass 2: warps of half h take the tiles with parity h, all columns
      float* r_e = a.r_out + static_cast<size_t>(e) * s.cap;
      float* s_e = a.scores_out ? a.scores_out + static_cast<size_t>(e) * s.cap : nullptr;
      tc_fence_after();
      for (int j = half; j < R; j += 2) {
        const int slot = rs + j < ring ? rs + j : rs + j - ring;
        float r = -INFINITY;
        const int key = k0 + j * kTile + key_row;
        const bool window_tile = CAUSAL && k0 + j * kTile + kTile > win0;  // warp-uniform
        if (!MEAN && N <= 64 && resident_ok && !window_tile) {
          // max form: the columns into registers, the slot released, then the arithmetic
          float v[64];
          tile_load<N>(tmem + slot * N + lane_addr, v);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cnt(&slot_free[slot], 2);  // two arrivals: this warp stands for its pair
          r = tile_score_regs<N>(v, lse2_sh, sc);
        } else {
          if (resident_ok)
            r = window_tile
                    ? tile_agg_causal<N, MEAN>(tmem + slot * N + lane_addr, lse2_sh, sc, inv_m, key, win0, thr)
                    : tile_agg<N, MEAN>(tmem + slot * N + lane_addr, lse2_sh, sc, inv_m);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cnt(&slot_free[slot], 2);
        }
        if (resident_ok && key < k1) {
          if constexpr (COMBINE) r = fold_split<MEAN>(r_e[key], r);
          r_e[key] = r;
          if (s_e) s_e[key] = ex2_approx(r);
        }
      }
      for (int j = R + half; j < T; j += 2) {  // streaming tiles come back from HBM / L2
        const int slot = str_slot + 2 + half;
        const int u = kp2++;
        bool have = !*abort_flag && mbar_wait(&slot_full[slot], u & 1, abort_flag, a.err, kDevTimeoutEpilogue);
        have = __all_sync(0xffffffffu, have);
        float r = -INFINITY;
        const int key = k0 + j * kTile + key_row;
        if (have) {
          tc_fence_after();
          r = (CAUSAL && k0 + j * kTile + kTile > win0)
                  ? tile_agg_causal<N, MEAN>(tmem + slot * N + lane_addr, lse2_sh, sc, inv_m, key, win0, thr)
                  : tile_agg<N, MEAN>(tmem + slot * N + lane_addr, lse2_sh, sc, inv_m);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cnt(&slot_free[slot], 2);
        if (have && key < k1) {
          if constexpr (COMBINE) r = fold_split<MEAN>(r_e[key], r);
          r_e[key] = r;
          if (s_e) s_e[key] = ex2_approx(r);
        }
      }
      rs += R;  // the next instance starts where this one ended
      if (rs >= ring) {
        rs -= ring;
        ++ru;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (csize > 1) cluster_sync_all();  // no CTA leaves while a peer may still access its shared memory
}

// Cluster size and tensor-memory placement.  sms[c] (c = 1..kMaxCluster) is how many SMs clusters
// of c CTAs keep busy at once (0: not available).  Among the sizes whose tiles all fit the slot ring,
// the one keeping the most SMs busy wins (ties: more spare slots, then fewer CTAs); one spare slot
// lets the next instance's first tile land while an instance finishes.  When no size fits, the size
// keeping the most SMs busy streams its extra tiles through four slots after the ring.  Slot
// barriers exist for kMaxSlots slots, and tensor memory holds kTmemCols / n_cols of them (at least 8:
// a launch has n_cols <= 64).
constexpr int kMaxCluster = 16;  // 9 and more need the non-portable cluster-size attribute
constexpr int kMaxDevicesScore = 64;

Plan plan_score(int L, int n_cols, const int* sms) {
  const int U = (L + 31) / 32;
  int cap = static_cast<int>(kTmemCols) / n_cols;
  if (cap > kMaxSlots) cap = kMaxSlots;
  const int cmax = U < kMaxCluster ? U : kMaxCluster;  // every CTA owns at least one 32-key unit
  int best = 0, best_sms = 0, best_slack = -1;
  for (int c = 1; c <= cmax; ++c) {
    const int tiles = ((U + c - 1) / c + 3) / 4;  // tiles of the CTA with the most units
    const int slack = cap - tiles;
    if (slack < 0 || sms[c] <= 0) continue;
    const int sl = slack > 0 ? 1 : 0;
    if (sms[c] > best_sms || (sms[c] == best_sms && sl > best_slack)) {
      best = c;
      best_sms = sms[c];
      best_slack = sl;
    }
  }
  if (best > 0) return Plan{best, cap, 0};
  int sc = 1;
  for (int c = 2; c <= cmax; ++c)
    if (sms[c] > sms[sc]) sc = c;
  return Plan{sc, cap - 4, 1};
}

template <int D, int NQ, bool MEAN, bool CAUSAL, bool COMBINE>
cudaError_t launch_score_dq(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32,
                            const CUtensorMap& qmap, const ScoreArgs& a, cudaStream_t st) {
  using C = ScoreCfg<D>;
  auto kern = score_kernel<D, NQ, MEAN, CAUSAL, COMBINE>;
  int dev = 0, sms = 0, max_clusters = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // SMs that clusters of each size keep busy, queried once per device for this kernel (the shared
  // memory of a cluster's CTAs grows with its size by a few bytes only, so the largest is used)
  static int busy[kMaxDevicesScore][kMaxCluster + 1] = {};
  cudaError_t err = cudaSuccess;
  if (dev < kMaxDevicesScore && busy[dev][0] == 0) {
    const size_t smem_q = C::smem_bytes(2 * NQ, kMaxCluster);
    if ((err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem_q))) !=
            cudaSuccess ||
        (err = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) != cudaSuccess)
      return err;
    for (int c = 1; c <= kMaxCluster; ++c) {
      cudaLaunchConfig_t q = {};
      q.blockDim = dim3(kScThreads);
      q.dynamicSmemBytes = smem_q;
      q.gridDim = dim3(static_cast<unsigned>(c * sms));
      cudaLaunchAttribute qa[1];
      qa[0].id = cudaLaunchAttributeClusterDimension;
      qa[0].val.clusterDim.x = static_cast<unsigned>(c);
      qa[0].val.clusterDim.y = 1;
      qa[0].val.clusterDim.z = 1;
      q.attrs = qa;
      q.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, kern, &q) != cudaSuccess) {
        cudaGetLastError();
        n = c <= 8 ? sms / c : 0;
      }
      busy[dev][c] = n * c;
    }
    busy[dev][0] = 1;
  }
  int fallback[kMaxCluster + 1] = {};
  for (int c = 1; c <= 8; ++c) fallback[c] = (sms / c) * c;
  const Plan plan = plan_score(a.L, 2 * NQ, dev < kMaxDevicesScore ? busy[dev] : fallback);
  const size_t smem = C::smem_bytes(2 * NQ, plan.csize);
  const int n_stages = C::stages(2 * NQ, plan.csize);
  err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  if (plan.csize > 8 && (err = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) !=
                            cudaSuccess)
    return err;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kScThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(plan.csize);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // one resident wave of clusters, each looping over its share of the instances
  cfg.gridDim = dim3(static_cast<unsigned>(plan.csize * sms));
  if (cudaOccupancyMaxActiveClusters(&max_clusters, score_kernel<D, NQ, MEAN, CAUSAL, COMBINE>, &cfg) != cudaSuccess || max_clusters < 1) {
    cudaGetLastError();
    max_clusters = sms / plan.csize > 0 ? sms / plan.csize : 1;
  }
  const int n_clusters = max_clusters < s.n_inst ? max_clusters : s.n_inst;
  cfg.gridDim = dim3(static_cast<unsigned>(n_clusters * plan.csize));
  return cudaLaunchKernelEx(&cfg, score_kernel<D, NQ, MEAN, CAUSAL, COMBINE>, kmap, kmap32, qmap, s, a, plan, n_stages);
}

template <int D, bool MEAN, bool CAUSAL>
cudaError_t launch_score_d(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32, const CUtensorMap& qmap,
                           const ScoreArgs& a, cudaStream_t st) {
  // query columns of each pass-1 warp: half of this launch's padded query count; a launch after
  // the first of a column split folds into the scores before it
  if (a.combine) {
    switch (a.n_cols) {
      case 16: return launch_score_dq<D, 8, MEAN, CAUSAL, true>(s, kmap, kmap32, qmap, a, st);
      case 32: return launch_score_dq<D, 16, MEAN, CAUSAL, true>(s, kmap, kmap32, qmap, a, st);
      case 48: return launch_score_dq<D, 24, MEAN, CAUSAL, true>(s, kmap, kmap32, qmap, a, st);
      case 64: return launch_score_dq<D, 32, MEAN, CAUSAL, true>(s, kmap, kmap32, qmap, a, st);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (a.n_cols) {
    case 16: return launch_score_dq<D, 8, MEAN, CAUSAL, false>(s, kmap, kmap32, qmap, a, st);
    case 32: return launch_score_dq<D, 16, MEAN, CAUSAL, false>(s, kmap, kmap32, qmap, a, st);
    case 48: return launch_score_dq<D, 24, MEAN, CAUSAL, false>(s, kmap, kmap32, qmap, a, st);
    case 64: return launch_score_dq<D, 32, MEAN, CAUSAL, false>(s, kmap, kmap32, qmap, a, st);
    default: return cudaErrorInvalidValue;
  }
}

// Dispatch on head_dim and the padded query count for one aggregation and mask.
template <bool MEAN, bool CAUSAL>
cudaError_t launch_score_agg(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32,
                             const CUtensorMap& qmap, const ScoreArgs& a, cudaStream_t st) {
  return s.d == 128 ? launch_score_d<128, MEAN, CAUSAL>(s, kmap, kmap32, qmap, a, st)
                    : launch_score_d<64, MEAN, CAUSAL>(s, kmap, kmap32, qmap, a, st);
}

}  // namespace
}  // namespace bkv
