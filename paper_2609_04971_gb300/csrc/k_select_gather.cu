// Selection (Eq. 7 with the keep set of Algorithm 2) and in-place compaction
// of K and V (Eq. 8), one CTA of 256 threads per instance.
//
// Selection: the log2 scores of the candidates [n_prefix, L - W) are mapped to
// order-preserving uint32 keys in shared memory; a 4-pass MSB-first radix
// select (8-bit digits, per-warp histograms) finds the exact key T of the
// k_sel-th best candidate and how many candidates equal to T are needed.
// One pass over the cache in index order then keeps every row of the keep
// set, every candidate with key > T, and the first needed candidates with key
// == T (ties go to the lower index), writing kept indices in ascending order
// with block-wide ballot scans.  No sort is needed.
//
// Compaction: row i of K and V receives row kept[i].  kept is ascending with
// kept[i] >= i, so destinations are processed in ascending chunks: all loads
// of a chunk are issued before the barrier that precedes its stores, and a
// chunk's loads only touch rows at or beyond its own first destination,
// which no earlier chunk writes.  Rows below the first evicted row already
// hold their final contents and are skipped.  Transfers are 16-byte vectors,
// coalesced along each 2*d-byte row; the kept indices are read from shared
// memory (they overwrite the score keys once compaction has consumed them).
#include "bkv_device.cuh"
#include "bkv_internal.h"

namespace bkv {
namespace {

constexpr int kSgThreads = 256;
constexpr int kSgWarps = kSgThreads / 32;

// Exclusive block-wide prefix count of `flag`; also returns the block total.
__device__ __forceinline__ void block_count_scan(bool flag, int* wsum, int& excl, int& total) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const unsigned bal = __ballot_sync(0xffffffffu, flag);
  if (lane == 0) wsum[warp] = __popc(bal);
  __syncthreads();
  int before = 0, all = 0;
#pragma unroll
  for (int w = 0; w < kSgWarps; ++w) {
    const int c = wsum[w];
    before += (w < warp) ? c : 0;
    all += c;
  }
  excl = before + __popc(bal & ((1u << lane) - 1u));
  total = all;
  __syncthreads();
}

// work / n_work (per-instance lengths): block w compresses instance work[w], with Ls[work[w]] rows,
// when w < *n_work; otherwise every block compresses its own instance from L rows.
template <int D>
__global__ void __launch_bounds__(kSgThreads) select_gather_kernel(Shape s, const float* __restrict__ r, int L,
                                                                    int budget, __nv_bfloat16* K, __nv_bfloat16* V,
                                                                    int* kept, const int* __restrict__ Ls,
                                                                    const int* __restrict__ work,
                                                                    const int* __restrict__ n_work, int* err) {
  extern __shared__ __align__(16) uint32_t keys[];  // [L]
  __shared__ uint32_t hist[kSgWarps][256];
  __shared__ uint32_t tot[256];
  __shared__ int wsum[kSgWarps];
  __shared__ uint32_t sh_prefix, sh_k;
  __shared__ int sh_first_evicted;

  int e = blockIdx.x;
  if (work) {
    if (e >= *n_work) return;  // whole block
    e = work[e];
    if (!in_bounds(e, s.n_inst, err)) return;  // whole block: every thread read the same entries
    L = Ls[e];
    if (!in_bounds(L - 1, s.cap, err)) return;
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c_lo = s.n_prefix, c_hi = L - s.W;
  const int k_sel = budget - s.n_prefix - s.W;
  const float* r_e = r + static_cast<size_t>(e) * s.cap;
  int* kept_e = kept + static_cast<size_t>(e) * budget;

  for (int j = tid; j < L; j += kSgThreads) keys[j] = float_order_key(r_e[j]);
  if (tid == 0) {
    sh_prefix = 0;
    sh_k = static_cast<uint32_t>(k_sel);
    sh_first_evicted = L;
  }
  __syncthreads();

  // ---------------------------------------------------------------- radix select
  uint32_t prefix = 0, pmask = 0;
  if (k_sel > 0) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < kSgWarps * 256; i += kSgThreads) (&hist[0][0])[i] = 0;
      __syncthreads();
      for (int j = c_lo + tid; j < c_hi; j += kSgThreads) {
        const uint32_t key = keys[j];
        if ((key & pmask) == prefix) atomicAdd(&hist[warp][(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (tid < 256) {
        uint32_t t = 0;
#pragma unroll
        for (int w = 0; w < kSgWarps; ++w) t += hist[w][tid];
        tot[tid] = t;
      }
      __syncthreads();
      if (warp == 0) {
        // lane l scans bins 255 - 8l - i (i = 0..7), i.e. descending digit order
        uint32_t loc[8], lsum = 0;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          loc[i] = tot[255 - 8 * lane - i];
          lsum += loc[i];
        }
        uint32_t incl = lsum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t n = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += n;
        }
        uint32_t above = incl - lsum;
        const uint32_t k = sh_k;
        if (above < k && k <= above + lsum) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            if (above + loc[i] >= k) {
              sh_prefix = prefix | (static_cast<uint32_t>(255 - 8 * lane - i) << shift);
              sh_k = k - above;
              break;
            }
            above += loc[i];
          }
        }
      }
      __syncthreads();
      prefix = sh_prefix;
      pmask |= 0xFFu << shift;
    }
  }
  const uint32_t T = k_sel > 0 ? prefix : 0xFFFFFFFFu;
  const int k_ties = k_sel > 0 ? static_cast<int>(sh_k) : 0;

  // ---------------------------------------------------------------- index-order compaction
  // kept indices go to global memory and, in place of the consumed keys, to shared memory
  int* kept_s = reinterpret_cast<int*>(keys);
  int run_tie = 0, run_keep = 0;
  for (int base = 0; base < L; base += kSgThreads) {
    const int j = base + tid;
    const bool in = j < L;
    const bool cand = in && j >= c_lo && j < c_hi;
    const uint32_t key = cand ? keys[j] : 0u;
    const bool tie = cand && key == T;
    int tie_excl, tie_total;
    block_count_scan(tie, wsum, tie_excl, tie_total);  // also orders every read of keys[base..] before the writes
    const bool keep = in && (!cand || key > T || (tie && run_tie + tie_excl < k_ties));
    int keep_excl, keep_total;
    block_count_scan(keep, wsum, keep_excl, keep_total);
    if (keep && in_bounds(run_keep + keep_excl, budget, err)) {
      kept_e[run_keep + keep_excl] = j;
      kept_s[run_keep + keep_excl] = j;  // position <= j: that key has been read already
    } else if (in && !keep) {
      atomicMin(&sh_first_evicted, j);
    }
    run_tie += tie_total;
    run_keep += keep_total;
  }
  __syncthreads();
  // the selection keeps exactly `budget` rows; a checked build verifies it (block-uniform)
  if (!in_bounds(run_keep - budget, 1, err) || !in_bounds(budget - run_keep, 1, err)) return;

  // ---------------------------------------------------------------- in-place gather
  constexpr int kVpr = D * 2 / 16;                 // 16-byte vectors per row of one tensor
  constexpr int kRowVec = 2 * kVpr;                // K row then V row
  constexpr int kPer = 8;                          // vectors per thread per chunk
  constexpr int kRowsPerPass = kSgThreads / kRowVec;
  constexpr int kChunkRows = kRowsPerPass * kPer;
  const int col = tid % kRowVec;                   // fixed 16-byte column of this thread
  const int row0 = tid / kRowVec;                  // first row of this thread inside a chunk
  uint4* base_t = reinterpret_cast<uint4*>((col < kVpr ? K : V) + static_cast<size_t>(e) * s.cap * D) +
                  (col < kVpr ? col : col - kVpr);
  const int first = sh_first_evicted;

  uint4 cur[kPer], nxt[kPer];
  auto load_chunk = [&](int i0, uint4 (&R)[kPer]) {
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int row = i0 + row0 + kRowsPerPass * u;
      if (row < budget) {
        int src = kept_s[row];
        if (!in_bounds(src - row, L - row, err)) src = row;  // kept rows satisfy row <= kept[row] < L
        R[u] = __ldcg(base_t + static_cast<size_t>(src) * kVpr);
      }
    }
  };
  auto store_chunk = [&](int i0, const uint4 (&R)[kPer]) {
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int row = i0 + row0 + kRowsPerPass * u;
      if (row < budget) base_t[static_cast<size_t>(row) * kVpr] = R[u];
    }
  };
  if (first < budget) load_chunk(first, cur);
  for (int i0 = first; i0 < budget; i0 += kChunkRows) {
    __syncthreads();  // every load of this chunk was issued before any of its stores
    const int i1 = i0 + kChunkRows;
    if (i1 < budget) load_chunk(i1, nxt);
    store_chunk(i0, cur);
#pragma unroll
    for (int u = 0; u < kPer; ++u) cur[u] = nxt[u];
  }
}

__global__ void keep_all_kernel(int n_inst, int L, int budget, int* kept) {
  const size_t n = static_cast<size_t>(n_inst) * budget;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int j = static_cast<int>(i % budget);
    kept[i] = j < L ? j : -1;
  }
}

template <int D>
cudaError_t launch_sg_d(const Shape& s, const float* r, int L, int budget, __nv_bfloat16* K, __nv_bfloat16* V,
                        int* kept, int* err, cudaStream_t st) {
  const size_t smem = sizeof(uint32_t) * static_cast<size_t>(L);
  const cudaError_t ce = cudaFuncSetAttribute(select_gather_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(smem));
  if (ce != cudaSuccess) return ce;
  select_gather_kernel<D><<<s.n_inst, kSgThreads, smem, st>>>(s, r, L, budget, K, V, kept, nullptr, nullptr, nullptr,
                                                              err);
  return cudaGetLastError();
}

// L_max sizes the shared-memory key array (every instance has at most that many rows).
template <int D>
cudaError_t launch_sg_ragged_d(const Shape& s, const float* r, const int* Ls, const int* work, const int* n_work,
                               int L_max, int budget, __nv_bfloat16* K, __nv_bfloat16* V, int* kept, int* err,
                               cudaStream_t st) {
  const size_t smem = sizeof(uint32_t) * static_cast<size_t>(L_max);
  const cudaError_t ce = cudaFuncSetAttribute(select_gather_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(smem));
  if (ce != cudaSuccess) return ce;
  select_gather_kernel<D><<<s.n_inst, kSgThreads, smem, st>>>(s, r, L_max, budget, K, V, kept, Ls, work, n_work, err);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_select_gather(const Shape& s, const float* r, int L, int budget, __nv_bfloat16* K,
                                 __nv_bfloat16* V, int* kept, int* err, cudaStream_t st) {
  return s.d == 128 ? launch_sg_d<128>(s, r, L, budget, K, V, kept, err, st)
                    : launch_sg_d<64>(s, r, L, budget, K, V, kept, err, st);
}

cudaError_t launch_select_gather_ragged(const Shape& s, const float* r, const int* Ls, const int* work,
                                        const int* n_work, int budget, __nv_bfloat16* K, __nv_bfloat16* V, int* kept,
                                        int* err, cudaStream_t st) {
  return s.d == 128 ? launch_sg_ragged_d<128>(s, r, Ls, work, n_work, s.cap, budget, K, V, kept, err, st)
                    : launch_sg_ragged_d<64>(s, r, Ls, work, n_work, s.cap, budget, K, V, kept, err, st);
}

cudaError_t launch_keep_all(const Shape& s, int L, int budget, int* kept, cudaStream_t st) {
  const size_t n = static_cast<size_t>(s.n_inst) * budget;
  const int blocks = static_cast<int>(n / 256 + 1 < 4096 ? n / 256 + 1 : 4096);
  keep_all_kernel<<<blocks, 256, 0, st>>>(s.n_inst, L, budget, kept);
  return cudaGetLastError();
}

}  // namespace bkv
