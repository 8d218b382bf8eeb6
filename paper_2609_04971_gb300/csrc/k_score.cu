// Scoring of every cached key (Eq. 4 softmax over the whole cache, Eq. 6 max
// form, maximum over the GQA group's observation queries; Section 4.3).
//
// Persistent kernel, one CTA per SM.  Instances are processed by
// thread-block clusters of C CTAs (C = 1 or more, chosen from the cache
// length); cluster k takes instances k, k + n_clusters, ...; CTA r of a
// cluster owns the same contiguous range of 128-key tiles of every instance.
// Each CTA is warp-specialised:
//   warp 0      TMA producer: per instance the observation queries (into one
//               of two buffers) and the CTA's K tiles (128 keys x d, 128-byte
//               swizzle) twice, through a ring of shared-memory stages;
//   warp 1      allocates TMEM and issues tcgen05.mma (bf16 x bf16 -> fp32):
//               D = K_tile x Qobs^T, M = 128 keys (TMEM lanes), N = padded
//               query count (TMEM columns), for both passes;
//   warps 2..9  two epilogue groups of four warps (one TMEM lane quarter
//               per warp).  With at most 64 query columns the groups take
//               alternate tiles; with more, both read every tile of pass 1
//               and each group owns 64 query columns.
// Pass 1: each thread owns one key of the tile and keeps, for every query
// column it owns, a running maximum m_q and sum s_q of 2^(y - m_q) over the
// keys it has seen (y = logit * log2(e), one ex2 per element).  At the end of
// the CTA's tiles the per-thread partials are merged (recursive halving
// inside each warp, then shared memory across warps and groups) and the CTAs
// of a cluster exchange theirs through distributed shared memory; every CTA
// combines them in rank order, giving the same lse2_q = log2 sum_j 2^(y_qj)
// over all L keys.  Pass 2 recomputes the tile (the K bytes are still in L2)
// and takes r_j = max over valid q of (y_qj - lse2_q) = log2 Score_j.
//
// Cross-CTA protocol (all waits bounded): barriers are initialised, then a
// cluster barrier.  Per instance each CTA publishes its partials and arrives
// on every peer's `part_ready`; after reading every peer it arrives on every
// peer's `read_done`; it overwrites its partials for the next instance only
// after its own `read_done` phase completed.  The exchange runs for every
// instance even after a timeout, and the kernel ends with a cluster barrier,
// so no CTA leaves while a peer may still touch its shared memory.
// Outputs: r (log2 scores, for selection) and optionally Score = 2^r.
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kEpiGroups = 2;
constexpr int kScThreads = 64 + 128 * kEpiGroups;
constexpr int kTile = 128;                 // keys per tile (MMA M)
constexpr uint32_t kBoxBytes = 128 * 128;  // [128 rows][64 bf16] swizzled box
constexpr int kAcc = 4;                    // fp32 accumulators of 128 TMEM columns each
constexpr uint32_t kTmemCols = 128 * kAcc;
constexpr int kMaxStages = 12;
constexpr size_t kSmemBudget = 220 * 1024;  // dynamic shared memory of the one CTA per SM

template <int D>
struct ScoreCfg {
  static constexpr int kBoxes = D / 64;                  // 64-column boxes per row
  static constexpr uint32_t kTileBytes = kTile * D * 2;  // one K tile
  static size_t q_bytes(int n_obs_pad) { return 2 * static_cast<size_t>(kBoxes) * n_obs_pad * 128; }
  // as many K stages as fit next to the two query buffers
  static int stages(int n_obs_pad) {
    const size_t room = kSmemBudget - 1024 - q_bytes(n_obs_pad);
    const int n = static_cast<int>(room / (static_cast<size_t>(kBoxes) * kBoxBytes));
    return n < kMaxStages ? n : kMaxStages;
  }
  static size_t smem_bytes(int n_obs_pad) {
    return 1024 + q_bytes(n_obs_pad) + static_cast<size_t>(stages(n_obs_pad)) * kBoxes * kBoxBytes;
  }
};

// Wait used while draining after an abort: ignores the abort flag.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, int* err) {
  int never = 0;
  mbar_wait(bar, parity, &never, err, kDevTimeoutDrain);
}

__device__ __forceinline__ void mbar_arrive_n(uint64_t* bar, uint32_t n) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(n) : "memory");
}

// Merge of two base-2 log-sum-exp partials (m, s) -> (max, rescaled sum).
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  const float a = (m == M) ? s : s * ex2_approx(m - M);
  const float b = (m2 == M) ? s2 : s2 * ex2_approx(m2 - M);
  m = M;
  s = a + b;
}

// Recursive-halving merge across the 32 lanes of a warp for NQ columns held
// by every lane; afterwards lane l holds the warp's merge of columns
// l * (NQ / 32) .. + NQ / 32 - 1 in m[0 .. NQ/32 - 1], s[...].
template <int NQ>
__device__ __forceinline__ void warp_reduce_scatter(float (&m)[NQ], float (&s)[NQ], int lane) {
#pragma unroll
  for (int half = NQ / 2, o = 16; half >= NQ / 32; half /= 2, o /= 2) {
    const bool upper = (lane & o) != 0;  // keeps the upper half of its current columns
#pragma unroll
    for (int i = 0; i < half; ++i) {
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
}

template <int D, int NQ>
__global__ void __launch_bounds__(kScThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap, Shape s,
                 ScoreArgs a, int csize, int n_stages) {
  using C = ScoreCfg<D>;
  constexpr int kPer = NQ / 32;  // columns per lane after the warp merge
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages], empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t accf_bar[kAcc], acce_bar[kAcc], qfull_bar[2], qempty_bar[2], drain_bar;
  __shared__ __align__(8) uint64_t part_ready_bar, read_done_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;
  __shared__ float lse2_sh[128];
  __shared__ float part_m[128], part_s[128];
  __shared__ float wred_m[kEpiGroups * 4][64], wred_s[kEpiGroups * 4][64];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int crank = csize > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int cluster_id = blockIdx.x / csize;
  const int n_clusters = gridDim.x / csize;
  const int n_my = cluster_id < s.n_inst ? (s.n_inst - cluster_id + n_clusters - 1) / n_clusters : 0;
  const int T_all = (a.L + kTile - 1) / kTile;
  const int t0 = crank * T_all / csize;
  const int T = (crank + 1) * T_all / csize - t0;  // tiles this CTA owns in every instance
  const uint32_t qbox = static_cast<uint32_t>(s.n_obs_pad) * 128;
  const bool split = s.n_obs_pad > 64;  // pass 1: both groups read every tile, 64 columns each

  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* q_smem = base;                         // [2 buffers][kBoxes][n_obs_pad rows x 128 B]
  unsigned char* k_smem = base + 2 * C::kBoxes * qbox;  // [n_stages][kBoxes][128 rows x 128 B]

  if (threadIdx.x == 0) {
    for (int i = 0; i < n_stages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < kAcc; ++i) {
      mbar_init(&accf_bar[i], 1);
      mbar_init(&acce_bar[i], split ? 8 : 4);  // warp arrivals that free an accumulator
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&qfull_bar[i], 1);
      mbar_init(&qempty_bar[i], 1);
    }
    mbar_init(&drain_bar, 1);
    mbar_init(&part_ready_bar, csize);
    mbar_init(&read_done_bar, csize);
    abort_sh = 0;
    fence_mbar_init();
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

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      const uint64_t keep = l2_policy_evict_last(), stream = l2_policy_evict_first();
      prefetch_tmap(&kmap);
      prefetch_tmap(&qmap);
      int g = 0;  // ring iteration over all instances
      bool ok = true;
      int q_issued = 0;
      for (int li = 0; ok && li < n_my; ++li) {
        const int e = cluster_id + li * n_clusters;
        const int qb = li & 1;
        if (li >= 2 && !mbar_wait(&qempty_bar[qb], ((li >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutProducer)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&qfull_bar[qb], static_cast<uint32_t>(s.n_obs_pad) * D * 2);
        for (int b = 0; b < C::kBoxes; ++b)
          tma_load_2d(q_smem + (qb * C::kBoxes + b) * qbox, &qmap, &qfull_bar[qb], b * 64, e * s.n_obs_pad, keep);
        q_issued = li + 1;
        for (int it = 0; it < 2 * T; ++it, ++g) {
          const int st = g % n_stages;
          if (g >= n_stages &&
              !mbar_wait(&empty_bar[st], ((g / n_stages) - 1) & 1, abort_flag, a.err, kDevTimeoutProducer)) {
            ok = false;
            break;
          }
          const int t = t0 + (it < T ? it : it - T);
          mbar_arrive_expect_tx(&full_bar[st], C::kTileBytes);
          for (int b = 0; b < C::kBoxes; ++b)
            tma_load_2d(k_smem + (st * C::kBoxes + b) * kBoxBytes, &kmap, &full_bar[st], b * 64,
                        e * s.cap + t * kTile, it < T ? keep : stream);
        }
      }
      if (!ok || *abort_flag) {  // let every copy already issued land before the CTA exits
        for (int li = (q_issued > 2 ? q_issued - 2 : 0); li < q_issued; ++li)
          drain_wait(&qfull_bar[li & 1], (li >> 1) & 1, a.err);
        for (int j = (g > n_stages ? g - n_stages : 0); j < g; ++j)
          drain_wait(&full_bar[j % n_stages], (j / n_stages) & 1, a.err);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, s.n_obs_pad);
      int g = 0, ga = 0;
      bool ok = true;
      for (int li = 0; ok && li < n_my; ++li) {
        const int qb = li & 1;
        if (!mbar_wait(&qfull_bar[qb], (li >> 1) & 1, abort_flag, a.err, kDevTimeoutMma)) break;
        const uint32_t q_addr = smem_u32(q_smem + qb * C::kBoxes * qbox);
        for (int it = 0; it < 2 * T; ++it, ++g, ++ga) {
          const int st = g % n_stages, acc = ga % kAcc;
          if (!mbar_wait(&full_bar[st], (g / n_stages) & 1, abort_flag, a.err, kDevTimeoutMma) ||
              (ga >= kAcc && !mbar_wait(&acce_bar[acc], ((ga / kAcc) - 1) & 1, abort_flag, a.err, kDevTimeoutMma))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem + acc * 128;
          const uint32_t k_addr = smem_u32(k_smem + st * C::kBoxes * kBoxBytes);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t qoff = (kk >> 2) * qbox + (kk & 3) * 32;
            const uint32_t koff = (kk >> 2) * kBoxBytes + (kk & 3) * 32;
            mma_bf16_ss(d_tmem, sdesc_kmajor_sw128(k_addr + koff), sdesc_kmajor_sw128(q_addr + qoff), idesc, kk > 0);
          }
          mma_commit(&empty_bar[st]);
          mma_commit(&accf_bar[acc]);
        }
        if (ok) mma_commit(&qempty_bar[qb]);  // this query buffer is free once its MMAs finish
      }
      mma_commit(&drain_bar);  // every MMA issued above has finished once this arrives
      drain_wait(&drain_bar, 0, a.err);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------------- epilogue
    const int group = (warp - 2) >> 2;
    const int wig = warp & 3;                 // TMEM lane quarter of this warp
    const int key_row = wig * 32 + lane;      // key of the tile owned by this thread
    const uint32_t lane_addr = static_cast<uint32_t>(wig * 32) << 16;
    const int col0 = split ? 64 * group : 0;  // first query column of this group in pass 1
    const bool leader = threadIdx.x == 64;
    const int n_epi = 128 * kEpiGroups;
    const int wslot = group * 4 + wig;        // slot of this warp in the cross-warp merge
    const float sc = a.scale_log2;
    int ga = 0;
    for (int li = 0; li < n_my; ++li) {
      const int e = cluster_id + li * n_clusters;

      // ---- pass 1: per-thread running (max, sum) of every owned query column
      float m[NQ], sm[NQ];
#pragma unroll
      for (int i = 0; i < NQ; ++i) {
        m[i] = -INFINITY;
        sm[i] = 0.f;
      }
      for (int t = 0; t < T; ++t, ++ga) {
        if (!split && (ga & 1) != group) continue;
        const int acc = ga % kAcc;
        const bool have = !*abort_flag &&
                          mbar_wait(&accf_bar[acc], (ga / kAcc) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
        const bool key_ok = (t0 + t) * kTile + key_row < a.L;
        if (have) tc_fence_after();
#pragma unroll
        for (int c = 0; c < NQ / 32; ++c) {
          float v[32];
          if (have) {
            tmem_ld32(tmem + acc * 128 + col0 + c * 32 + lane_addr, v);
            tmem_wait_ld();
          }
          if (c == NQ / 32 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acce_bar[acc]);  // all columns are in registers
          }
          if (have && key_ok) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float y = v[i] * sc;
              const float dlt = y - m[c * 32 + i];
              const float u = ex2_approx(-fabsf(dlt));
              const bool up = dlt > 0.f;
              sm[c * 32 + i] = up ? fmaf(sm[c * 32 + i], u, 1.f) : sm[c * 32 + i] + u;
              m[c * 32 + i] = up ? y : m[c * 32 + i];
            }
          }
        }
      }

      // ---- merge: warp lanes, then warps and groups, then the CTAs of the cluster
      warp_reduce_scatter<NQ>(m, sm, lane);
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        wred_m[wslot][lane * kPer + k] = m[k];
        wred_s[wslot][lane * kPer + k] = sm[k];
      }
      named_barrier(1, n_epi);  // also: every thread finished the previous instance's pass 2
      const int tq = threadIdx.x - 64;  // 0 .. 255: thread of the column merge
      const bool col_thread = tq < s.n_obs_pad;
      float cm = -INFINITY, cs = 0.f;
      if (col_thread) {
        // column tq lives in group (tq / 64) when split, else in every group
        const int g_lo = split ? tq / 64 : 0, g_hi = split ? g_lo + 1 : kEpiGroups;
        const int cc = split ? tq % 64 : tq;
        for (int g = g_lo; g < g_hi; ++g)
          for (int w = 0; w < 4; ++w) lse_merge(cm, cs, wred_m[g * 4 + w][cc], wred_s[g * 4 + w][cc]);
      }
      const bool my_valid = col_thread && ((a.valid[e * 4 + (tq >> 5)] >> (tq & 31)) & 1u);
      if (csize == 1) {
        if (tq < 128) lse2_sh[tq] = (my_valid && cm > -INFINITY) ? cm + lg2_approx(cs) : INFINITY;
      } else {
        // the peers have read this CTA's previous partials before they are overwritten
        if (li > 0 && tq < 128) mbar_wait_cluster(&read_done_bar, (li - 1) & 1, a.err, kDevTimeoutCluster);
        if (tq < 128) {
          part_m[tq] = cm;
          part_s[tq] = cs;
        }
        named_barrier(1, n_epi);
        if (leader)
          for (int c = 0; c < csize; ++c) mbar_arrive_remote(mapa_shared(smem_u32(&part_ready_bar), c));
        if (tq < 128) {
          const bool ok = mbar_wait_cluster(&part_ready_bar, li & 1, a.err, kDevTimeoutCluster);
          float M = -INFINITY, S = 0.f;
          if (ok && col_thread) {
            const uint32_t am = smem_u32(&part_m[tq]), as = smem_u32(&part_s[tq]);
            for (int c = 0; c < csize; ++c)
              lse_merge(M, S, ld_shared_cluster_f32(mapa_shared(am, c)), ld_shared_cluster_f32(mapa_shared(as, c)));
          }
          if (!ok) *abort_flag = 1;
          lse2_sh[tq] = (ok && my_valid && M > -INFINITY) ? M + lg2_approx(S) : INFINITY;
        }
      }
      named_barrier(1, n_epi);  // lse2 complete; in a cluster, every peer read is done
      if (csize > 1 && leader)
        for (int c = 0; c < csize; ++c) mbar_arrive_remote(mapa_shared(smem_u32(&read_done_bar), c));

      // ---- pass 2: thread = key; r_j = max_q (y_qj - lse2_q); groups take alternate tiles
      float* r_e = a.r_out + static_cast<size_t>(e) * s.cap;
      float* s_e = a.scores_out ? a.scores_out + static_cast<size_t>(e) * s.cap : nullptr;
      for (int t = 0; t < T; ++t, ++ga) {
        if ((ga & 1) != group) continue;
        const int acc = ga % kAcc;
        const bool have = !*abort_flag &&
                          mbar_wait(&accf_bar[acc], (ga / kAcc) & 1, abort_flag, a.err, kDevTimeoutEpilogue);
        if (have) tc_fence_after();
        float r0 = -INFINITY, r1 = -INFINITY;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const bool used = c * 32 < s.n_obs_pad;
          float v[32];
          if (have && used) {
            tmem_ld32(tmem + acc * 128 + c * 32 + lane_addr, v);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              r0 = fmaxf(r0, fmaf(v[i], sc, -lse2_sh[c * 32 + i]));
              r1 = fmaxf(r1, fmaf(v[i + 1], sc, -lse2_sh[c * 32 + i + 1]));
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_n(&acce_bar[acc], split ? 2 : 1);
        const int j = (t0 + t) * kTile + key_row;
        if (have && j < a.L) {
          const float r = fmaxf(r0, r1);
          r_e[j] = r;
          if (s_e) s_e[j] = ex2_approx(r);
        }
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

// CTAs per instance: enough that the instances in flight (one per cluster,
// one CTA per SM) hold about 90 MB of K between the two passes; at most 8.
int cluster_size(int L, int d, int sms) {
  const double bytes = static_cast<double>(sms) * L * d * 2;
  int c = static_cast<int>(bytes / 90e6 + 0.999);
  const int tiles = (L + kTile - 1) / kTile;
  if (c > tiles) c = tiles;
  return c < 1 ? 1 : (c > 8 ? 8 : c);
}

template <int D, int NQ>
cudaError_t launch_score_dq(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreArgs& a,
                            cudaStream_t st) {
  using C = ScoreCfg<D>;
  const size_t smem = C::smem_bytes(s.n_obs_pad);
  const int n_stages = C::stages(s.n_obs_pad);
  cudaError_t err = cudaFuncSetAttribute(score_kernel<D, NQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  int dev = 0, sms = 0, max_clusters = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int csize = cluster_size(a.L, s.d, sms);
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kScThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(csize);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // one resident wave of clusters, each looping over its share of the instances
  cfg.gridDim = dim3(static_cast<unsigned>(csize * sms));
  if (cudaOccupancyMaxActiveClusters(&max_clusters, score_kernel<D, NQ>, &cfg) != cudaSuccess || max_clusters < 1) {
    cudaGetLastError();
    max_clusters = sms / csize > 0 ? sms / csize : 1;
  }
  const int n_clusters = max_clusters < s.n_inst ? max_clusters : s.n_inst;
  cfg.gridDim = dim3(static_cast<unsigned>(n_clusters * csize));
  return cudaLaunchKernelEx(&cfg, score_kernel<D, NQ>, kmap, qmap, s, a, csize, n_stages);
}

template <int D>
cudaError_t launch_score_d(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreArgs& a,
                           cudaStream_t st) {
  // query columns each epilogue thread tracks in pass 1
  if (s.n_obs_pad <= 32) return launch_score_dq<D, 32>(s, kmap, qmap, a, st);
  return launch_score_dq<D, 64>(s, kmap, qmap, a, st);
}

}  // namespace

cudaError_t launch_score(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreArgs& a,
                         cudaStream_t st) {
  return s.d == 128 ? launch_score_d<128>(s, kmap, qmap, a, st) : launch_score_d<64>(s, kmap, qmap, a, st);
}

}  // namespace bkv
