// Scoring of every cached key (Eq. 4 softmax over the whole cache, Eq. 6 max
// form, maximum over the GQA group's observation queries; Section 4.3).
//
// One CTA per instance, warp-specialised:
//   warp 0      TMA producer: the instance's observation queries once, then
//               its K tiles (128 keys x d, 128-byte swizzle) twice, through a
//               ring of shared-memory stages;
//   warp 1      allocates TMEM and issues tcgen05.mma (bf16 x bf16 -> fp32);
//   warps 2..5  epilogue, one TMEM lane quarter each.
// Pass 1 computes D1 = Qobs x K_tile^T (M = 128 query rows, N = 128 keys),
// so each epilogue thread owns one query and folds the tile into its running
// (max, sum of 2^(y - max)) without any cross-thread reduction; at the end
// lse2_q = max + log2(sum).  Pass 2 computes D2 = K_tile x Qobs^T (M = 128
// key rows, N = padded query count), so each thread owns one key and takes
// r_j = max over valid q of (y_qj - lse2_q).  y = logit * log2(e) is the
// base-2 logit, r_j = log2 Score_j.  The second pass re-reads K with an L2
// evict-first hint after the first pass read it with evict-last.
// Outputs: r (log2 scores, for selection) and optionally Score = 2^r.
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kScThreads = 192;
constexpr int kTile = 128;                 // keys per tile (MMA M in pass 2, N in pass 1)
constexpr uint32_t kBoxBytes = 128 * 128;  // [128 rows][64 bf16] swizzled box
constexpr uint32_t kTmemCols = 256;        // two fp32 accumulators of 128 columns

template <int D>
struct ScoreCfg {
  static constexpr int kBoxes = D / 64;                  // 64-column boxes per row
  static constexpr int kStages = D == 128 ? 2 : 4;       // K ring depth (2 CTAs per SM)
  static constexpr uint32_t kTileBytes = kTile * D * 2;  // one K tile
  static constexpr size_t kSmem = 1024 + static_cast<size_t>(kBoxBytes) * kBoxes * (1 + kStages);
};

// Wait used while draining after an abort: ignores the abort flag.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, int* err) {
  int never = 0;
  mbar_wait(bar, parity, &never, err, kDevTimeoutDrain);
}

template <int D>
__global__ void __launch_bounds__(kScThreads, 2)
    score_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap qmap, Shape s,
                 ScoreArgs a) {
  using C = ScoreCfg<D>;
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[C::kStages], empty_bar[C::kStages];
  __shared__ __align__(8) uint64_t accf_bar[2], acce_bar[2], q_bar, drain_bar;
  __shared__ uint32_t tmem_base_sh;
  __shared__ int abort_sh;
  __shared__ float lse2_sh[128];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int e = blockIdx.x;
  const int T = (a.L + kTile - 1) / kTile;
  const int n_it = 2 * T;

  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  unsigned char* q_smem = base;
  unsigned char* k_smem = base + kBoxBytes * C::kBoxes;

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accf_bar[i], 1);
      mbar_init(&acce_bar[i], 4);
    }
    mbar_init(&q_bar, 1);
    mbar_init(&drain_bar, 1);
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
  const uint32_t tmem = tmem_base_sh;
  volatile int* abort_flag = &abort_sh;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      const uint64_t keep = l2_policy_evict_last(), stream = l2_policy_evict_first();
      prefetch_tmap(&kmap);
      prefetch_tmap(&qmap);
      mbar_arrive_expect_tx(&q_bar, static_cast<uint32_t>(s.n_obs_pad) * D * 2);
      for (int b = 0; b < C::kBoxes; ++b)
        tma_load_2d(q_smem + b * kBoxBytes, &qmap, &q_bar, b * 64, e * s.n_obs_pad, keep);
      int it = 0;
      for (; it < n_it; ++it) {
        const int st = it % C::kStages;
        if (it >= C::kStages &&
            !mbar_wait(&empty_bar[st], ((it / C::kStages) - 1) & 1, abort_flag, a.err, kDevTimeoutProducer))
          break;
        const int t = it < T ? it : it - T;
        mbar_arrive_expect_tx(&full_bar[st], C::kTileBytes);
        for (int b = 0; b < C::kBoxes; ++b)
          tma_load_2d(k_smem + (st * C::kBoxes + b) * kBoxBytes, &kmap, &full_bar[st], b * 64,
                      e * s.cap + t * kTile, it < T ? keep : stream);
      }
      if (*abort_flag) {  // let every copy already issued land before the CTA exits
        drain_wait(&q_bar, 0, a.err);
        for (int j = (it > C::kStages ? it - C::kStages : 0); j < it; ++j)
          drain_wait(&full_bar[j % C::kStages], (j / C::kStages) & 1, a.err);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc1 = idesc_bf16_f32(128, kTile);
      const uint32_t idesc2 = idesc_bf16_f32(128, s.n_obs_pad);
      const uint32_t q_addr = smem_u32(q_smem);
      bool ok = mbar_wait(&q_bar, 0, abort_flag, a.err, kDevTimeoutMma);
      for (int it = 0; ok && it < n_it; ++it) {
        const int st = it % C::kStages, acc = it & 1;
        if (!mbar_wait(&full_bar[st], (it / C::kStages) & 1, abort_flag, a.err, kDevTimeoutMma)) break;
        if (it >= 2 && !mbar_wait(&acce_bar[acc], ((it >> 1) - 1) & 1, abort_flag, a.err, kDevTimeoutMma)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem + acc * 128;
        const uint32_t k_addr = smem_u32(k_smem + st * C::kBoxes * kBoxBytes);
        const bool pass1 = it < T;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kBoxBytes + (kk & 3) * 32;
          const uint64_t qd = sdesc_kmajor_sw128(q_addr + off);
          const uint64_t kd = sdesc_kmajor_sw128(k_addr + off);
          if (pass1)
            mma_bf16_ss(d_tmem, qd, kd, idesc1, kk > 0);
          else
            mma_bf16_ss(d_tmem, kd, qd, idesc2, kk > 0);
        }
        mma_commit(&empty_bar[st]);
        mma_commit(&accf_bar[acc]);
      }
      mma_commit(&drain_bar);  // every MMA issued above has finished once this arrives
      drain_wait(&drain_bar, 0, a.err);
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(quarter * 32) << 16;
    const bool my_valid = (a.valid[e * 4 + quarter] >> lane) & 1u;
    const bool rows_exist = quarter * 32 < s.n_obs_pad;
    const float sc = a.scale_log2;

    // pass 1: thread = query row; running base-2 log-sum-exp over all keys
    float m = -INFINITY, ssum = 0.f;
    for (int t = 0; t < T; ++t) {
      const int acc = t & 1;
      if (!mbar_wait(&accf_bar[acc], (t >> 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue)) break;
      tc_fence_after();
      if (rows_exist) {
        const int kbase = t * kTile;
#pragma unroll 1
        for (int c = 0; c < kTile / 32; ++c) {
          const int nvalid = min(32, a.L - (kbase + c * 32));
          if (nvalid <= 0) break;
          float v[32];
          tmem_ld32(tmem + acc * 128 + c * 32 + lane_addr, v);
          tmem_wait_ld();
          float cmax = -INFINITY;
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (i < nvalid) cmax = fmaxf(cmax, v[i]);
          const float mn = fmaxf(m, cmax * sc);
          ssum *= ex2_approx(m - mn);
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (i < nvalid) ssum += ex2_approx(fmaf(v[i], sc, -mn));
          m = mn;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce_bar[acc]);
    }
    lse2_sh[row] = (my_valid && rows_exist && m > -INFINITY) ? m + lg2_approx(ssum) : INFINITY;
    named_barrier(1, 128);

    // pass 2: thread = key; r_j = max_q (y_qj - lse2_q)
    float* r_e = a.r_out + static_cast<size_t>(e) * s.cap;
    float* s_e = a.scores_out ? a.scores_out + static_cast<size_t>(e) * s.cap : nullptr;
    for (int t = 0; t < T && !*abort_flag; ++t) {
      const int it = T + t, acc = it & 1;
      if (!mbar_wait(&accf_bar[acc], (it >> 1) & 1, abort_flag, a.err, kDevTimeoutEpilogue)) break;
      tc_fence_after();
      float r = -INFINITY;
      int c = 0;
#pragma unroll 1
      for (; c + 32 <= s.n_obs_pad; c += 32) {
        float v[32];
        tmem_ld32(tmem + acc * 128 + c + lane_addr, v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) r = fmaxf(r, fmaf(v[i], sc, -lse2_sh[c + i]));
      }
      if (c < s.n_obs_pad) {
        float v[16];
        tmem_ld16(tmem + acc * 128 + c + lane_addr, v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 16; ++i) r = fmaxf(r, fmaf(v[i], sc, -lse2_sh[c + i]));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce_bar[acc]);
      const int j = t * kTile + row;
      if (j < a.L) {
        r_e[j] = r;
        if (s_e) s_e[j] = ex2_approx(r);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

template <int D>
cudaError_t launch_score_d(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreArgs& a,
                           cudaStream_t st) {
  using C = ScoreCfg<D>;
  cudaError_t err =
      cudaFuncSetAttribute(score_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(C::kSmem));
  if (err != cudaSuccess) return err;
  score_kernel<D><<<s.n_inst, kScThreads, C::kSmem, st>>>(kmap, qmap, s, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& qmap, const ScoreArgs& a,
                         cudaStream_t st) {
  return s.d == 128 ? launch_score_d<128>(s, kmap, qmap, a, st) : launch_score_d<64>(s, kmap, qmap, a, st);
}

}  // namespace bkv
