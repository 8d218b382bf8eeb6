// Host-side declarations shared between the C-ABI layer (bkv_api.cu) and the
// kernel translation units.  Not part of the public interface.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace bkv {

// Per-context shape, derived once from bkv_config.
struct Shape {
  int n_inst;      // layers * batch * kv_heads
  int G;           // query heads per KV head
  int d;           // head_dim (64 or 128)
  int nb;          // beacons per KV head
  int W;           // recent window
  int n_prefix;    // always-kept leading rows
  int cap;         // rows per instance in K / V
  int n_obs;       // G * W + nb scoring queries
  int n_obs_pad;   // n_obs rounded up to 16
  int batch;       // batch rows: instance e belongs to batch row (e / n_kv) % batch
  int n_kv;        // KV heads
};

constexpr int kMaxBeacons = 32;
constexpr int kMaxObs = 128;
constexpr int kMaxWindow = 64;
constexpr int kMaxCapacity = 32768;
constexpr int kMaxFpsRows = 4096;

// ---- Continual FPS buffers (k_cfps.cu)
constexpr int kCfpsMaxRows = 32;  // b_max = n_beacons + window per query head
enum { kCfpsUpdate = 0, kCfpsBeacons = 1, kCfpsMerge = 2 };
struct CfpsArgs {
  int mode;                 // kCfpsUpdate / kCfpsBeacons / kCfpsMerge
  int H;                    // query heads: n_layers * batch * n_q_heads
  int b_min, b_max;         // n_beacons, n_beacons + window
  const __nv_bfloat16* q;   // update: q_new [H][n_q][d]; merge: q_recent [H][n_q][d]; beacons: unused
  int n_q;                  // n_new (update) or window (merge)
  __nv_bfloat16* buf;       // [H][b_max][d] buffers
  int* size;                // [H] rows in use
  float* bcn;               // [H][b_min][d] beacons of a compress (fp32 copies of bf16 queries)
  long long* bcnt;          // [H][b_min] 1 for a beacon, 0 for an empty slot
  // merge after a per-instance-length compress: only heads of instances with budget < Ls[h / group]
  // <= cap were evicted from and merge; the others keep their buffers
  const int* Ls = nullptr;
  int budget = 0, cap = 0, group = 1;
  int* err = nullptr;  // device error word (bounds checks of BKV_CHECKED builds)
};
cudaError_t launch_cfps(int d, const CfpsArgs& a, cudaStream_t st);
// Buffers seeded with b_min fp32 rows per head (FPS picks of the prompt), size b_min.
cudaError_t launch_cfps_seed(int d, const float* rows, int H, int b_min, int b_max, __nv_bfloat16* buf, int* size,
                             cudaStream_t st);

// ---- beacon maintenance (k_fps.cu, k_update.cu); fps_init's sums may be NULL
cudaError_t launch_fps_init(const Shape& s, const __nv_bfloat16* q_init, int n_init, float* cent, double* sums,
                            long long* counts, cudaStream_t st);

// qmap: the new queries as [n_inst * G * n_new][d] bf16 in boxes of
// [box_rows][64] (128-byte swizzle), box_rows = min(128, rows); err: device
// error word.
cudaError_t launch_update(const Shape& s, const CUtensorMap& qmap, int box_rows, int n_new, float* cent,
                          double* sums, long long* counts, int* assign_out, int* err, cudaStream_t st);
// A few queries per instance (G * n_new <= kUpdateSmallMaxRows, e.g. one decode step): one warp
// per instance, the same decisions and sums as launch_update (k_update_small.cu).
constexpr int kUpdateSmallMaxRows = 32;
cudaError_t launch_update_small(const Shape& s, const __nv_bfloat16* q_new, int n_new, float* cent, double* sums,
                                long long* counts, int* assign_out, cudaStream_t st);
// n_steps decode steps of one query per query head, applied in order (k_update_seq.cu): the result of
// one launch_update_small(n_new = 1) per step, bit for bit.  q_steps: [n_steps][n_inst * G][d];
// assign_out: [n_steps][n_inst * G] or nullptr.  cudaErrorInvalidValue when G > kUpdateSmallMaxRows or
// one instance's state does not fit in shared memory (the caller then goes step by step).
cudaError_t launch_update_seq(const Shape& s, const __nv_bfloat16* q_steps, int n_steps, float* cent, double* sums,
                              long long* counts, int* assign_out, cudaStream_t st);

// ---- compression (k_qobs.cu, k_score.cu, k_select_gather.cu)
// rope: [W + 1][d / 2] fp64 (cos, sin) pairs, immediately followed by the same
// [W + 1][d / 2] table as fp32 pairs; entry w < W is recent slot w, entry W
// is the beacon position.  rotate == 0 leaves vectors unrotated.
// Device copy of `bytes` (a multiple of 16, both ends 16-byte aligned) from a
// device-mapped pinned host buffer, by a kernel on `st`.
cudaError_t launch_rope_stage(const void* src, void* dst, size_t bytes, cudaStream_t st);
cudaError_t launch_qobs(const Shape& s, const __nv_bfloat16* q_recent, const float* cent, const long long* counts,
                        const double2* rope, int rotate, __nv_bfloat16* qobs, uint32_t* valid, int* err,
                        cudaStream_t st);
// Per-instance cache lengths (bkv_compress_ragged): the same build for the instances work[0 .. *n_work)
// only, batch row b taking its own rotary table at rope + b * rope_row (double2 units).
cudaError_t launch_qobs_ragged(const Shape& s, const __nv_bfloat16* q_recent, const float* cent,
                               const long long* counts, const double2* rope, size_t rope_row, int rotate,
                               const int* work, const int* n_work, __nv_bfloat16* qobs, uint32_t* valid, int* err,
                               cudaStream_t st);

// ---- per-instance cache lengths (k_ragged.cu)
// Instances whose length Ls[e] exceeds `budget` are listed in index order in work[0 .. *n_work); every
// other instance gets kept = 0 .. L - 1 and -1 after (its K and V are not touched).  A length outside
// 1..cap records kDevBadLength in err and leaves that instance's kept row at -1.
cudaError_t launch_ragged_plan(const Shape& s, const int* Ls, int budget, int* work, int* n_work, int* kept, int* err,
                               cudaStream_t st);

struct ScoreArgs {
  int L = 0;
  float scale_log2 = 0.f;          // log2(e) / sqrt(d)
  const uint32_t* valid = nullptr; // [n_inst][4] bitmask of valid scoring rows
  bool mean = false;               // mean over the valid queries instead of the maximum
  bool causal = false;             // causal mask inside the recent window (set_causal)
  int win0 = 0;                    // first window row, L - W
  int thr[kMaxWindow] = {};        // recent slot w sees window row j only if j <= thr[w]
  int col0 = 0;                    // column split: first Q_obs row of this launch (a multiple of 64)
  int n_cols = 0;                  // padded query rows of this launch: 16, 32, 48 or 64
  bool combine = false;            // fold into r_out of the launch of the rows before col0
  float* r_out = nullptr;          // [n_inst][cap] log2-domain scores (log2 of the aggregated weight)
  float* scores_out = nullptr;     // [n_inst][cap] probabilities, or nullptr
  int* err = nullptr;              // device error word
  // per-instance lengths (bkv_compress_ragged): the instances work[0 .. *n_work), instance e with
  // Ls[e] rows; L above is then the longest possible (it sizes the plan).  Causal form: gaps[b][w] is
  // t_pos - recent_pos[w] of batch row b, clamped to [0, cap + 1] (0: the slot sees every window row).
  const int* Ls = nullptr;
  const int* work = nullptr;
  const int* n_work = nullptr;
  const int* gaps = nullptr;
};
// Causal mask inside the recent window: recent slot w sits at recent_pos[w] and window row j
// (L - W <= j < L) at t_pos - (L - 1 - j), so slot w sees window row j only if
// j <= L - 1 - (t_pos - recent_pos[w]); beacons (at t_pos) and older rows are never masked.
inline void set_causal(ScoreArgs& a, int L, int W, long long t_pos, const int64_t* recent_pos) {
  a.causal = W > 0;
  a.win0 = L - W;
  for (int w = 0; w < W; ++w) {
    if (recent_pos[w] >= t_pos) {
      a.thr[w] = L;  // at or after every window row
    } else {
      const unsigned long long gap = static_cast<unsigned long long>(t_pos) - static_cast<unsigned long long>(recent_pos[w]);
      a.thr[w] = gap > static_cast<unsigned long long>(L) ? -1 : (L - 1) - static_cast<int>(gap);
    }
  }
}
// Tensor map of a bf16 matrix [rows][d] (row pitch d * 2 bytes) in boxes of [box_rows][64] with the
// 128-byte swizzle; CUDA_ERROR_NOT_FOUND when the driver has no cuTensorMapEncodeTiled.
CUresult encode_rows_bf16(CUtensorMap* map, const void* base, uint64_t rows, int d, uint32_t box_rows);

constexpr int kScoreMaxCols = 64;  // scoring queries per score launch (column split beyond)
// kmap / kmap32: K as [n_inst * cap][d] in 128-row and 32-row boxes of [64]
// columns (128-byte swizzle); qmap: Qobs as [n_inst * n_obs_pad][d] in boxes
// of n_cols rows (the launch's Q_obs rows start at row e * n_obs_pad + col0).
cudaError_t launch_score(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32, const CUtensorMap& qmap,
                         const ScoreArgs& a, cudaStream_t st);
// The mean form (a.mean) and the causal forms (a.causal), each compiled in its own translation
// unit; launch_score forwards to them.
cudaError_t launch_score_mean(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32,
                              const CUtensorMap& qmap, const ScoreArgs& a, cudaStream_t st);
cudaError_t launch_score_causal(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32,
                                const CUtensorMap& qmap, const ScoreArgs& a, cudaStream_t st);
cudaError_t launch_score_causal_mean(const Shape& s, const CUtensorMap& kmap, const CUtensorMap& kmap32,
                                     const CUtensorMap& qmap, const ScoreArgs& a, cudaStream_t st);

cudaError_t launch_select_gather(const Shape& s, const float* r, int L, int budget, __nv_bfloat16* K,
                                 __nv_bfloat16* V, int* kept, int* err, cudaStream_t st);
// Per-instance lengths: the instances work[0 .. *n_work), instance e with Ls[e] rows (at most cap).
cudaError_t launch_select_gather_ragged(const Shape& s, const float* r, const int* Ls, const int* work,
                                        const int* n_work, int budget, __nv_bfloat16* K, __nv_bfloat16* V, int* kept,
                                        int* err, cudaStream_t st);

cudaError_t launch_keep_all(const Shape& s, int L, int budget, int* kept, cudaStream_t st);

// ---- diagnostics (k_selftest.cu): a bounded wait that expires after limit_ns
cudaError_t launch_selftest_wait(int* err, unsigned long long limit_ns, cudaStream_t st);
// One checked access at an index one past the logical end of a buffer that is twice that long, so
// that the access stays in memory this kernel owns whether or not bounds checks are compiled in.
cudaError_t launch_selftest_bounds(int* err, cudaStream_t st);

}  // namespace bkv
