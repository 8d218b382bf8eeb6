/*
 * bkv.h - C ABI of the BeaconKV KV-cache compression step on GB300 (sm_103a).
 *
 * BeaconKV (arXiv 2609.04971) keeps a KV cache within budget by scoring every
 * cached key with the attention weights of a set of observation queries -
 * "beacon" queries that represent recurring global query clusters plus the
 * most recent queries - and keeping the best keys together with the recent
 * window (Sections 4.1-4.3, Appendix D.2).  This library implements the two
 * data-parallel parts of that step for a whole model (all layers, batch rows
 * and KV heads at once):
 *
 *   beacon maintenance  - FPS seeding from prompt queries (Appendix D.1,
 *                         Algorithm 1) and, per decode query, nearest-beacon
 *                         assignment by cosine similarity followed by a
 *                         running-mean centroid update;
 *   compression         - observation queries (beacons rotated to the current
 *                         step, recent queries at their own positions;
 *                         Section 4.3), scoring (Eq. 4 softmax over the whole
 *                         cache, Eq. 6 max form, maximum over the GQA group),
 *                         selection (keep set + TopK, Eq. 7, Algorithm 2) and
 *                         in-place compaction of K and V (Eq. 8).
 *
 * Terms.  An *instance* is one (layer, batch row, KV head).  G = n_q_heads /
 * n_kv_heads query heads share a KV head; their queries all feed that KV
 * head's beacons.  n_inst = n_layers * batch * n_kv_heads.  Instances are
 * numbered (layer * batch + b) * n_kv_heads + g, which is also the row order
 * of every per-instance array below.
 *
 * Memory.  Every tensor argument is a DEVICE pointer owned by the caller,
 * row-major and contiguous, aligned to 16 bytes, unless the description says
 * "host".  bf16 tensors hold IEEE binary32 values truncated to their top 16
 * bits (bfloat16).  The library owns only what bkv_create allocates (beacon
 * state and scratch) and frees it in bkv_destroy.
 *
 * Streams.  All work is enqueued on the CUDA stream given to bkv_create (or
 * bkv_set_stream); calls return before it completes.  Outputs are valid once
 * that stream has been synchronised (bkv_sync does so and reports device-side
 * errors).  bkv_compress stages its rotary table in one of four pinned host
 * buffers, which a kernel on the stream copies to the device (no copy-engine
 * transfer, so the stream does not queue behind other streams' bulk host
 * copies), and waits only when the stream is more than four compress calls
 * behind.  One context must not be used from two host threads at once.
 *
 * Errors.  Every call returns BKV_OK (0) or a negative code; nothing throws.
 * Argument errors are detected on the host before any work is enqueued and
 * leave all buffers untouched.  Kernels whose internal waits expire record
 * BKV_ETIMEOUT in a device error word that the next bkv_sync returns.
 * bkv_last_error(ctx) gives a one-line description of the last failure.
 */
#ifndef BKV_H
#define BKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BKV_OK 0
#define BKV_EINVAL (-1)   /* bad shape, size, alignment, null pointer or range   */
#define BKV_ENOMEM (-2)   /* device allocation failed                            */
#define BKV_ECUDA (-3)    /* a CUDA runtime / driver call failed                 */
#define BKV_ETIMEOUT (-4) /* a bounded device-side wait expired (kernel aborted) */
#define BKV_ESTATE (-5)   /* call order violated (e.g. update before init)       */
#define BKV_EBOUNDS (-6)  /* a device-side bounds check failed (checked builds)  */

/* bkv_config.flags (bitwise OR). */
#define BKV_F_NONE 0u
/*
 * Mean aggregation (the mean form of Eq. 6, the paper's ablation of its max
 * pooling, Section 4.3): Score[j] = the mean of the softmax weights of key j
 * over the group's valid observation queries instead of their maximum (0
 * when no query is valid).  Selection, the keep set and compaction are
 * unchanged.
 */
#define BKV_F_MEAN_AGG 1u
/*
 * Continual FPS beacons (Section 4.2, Eq. 9; Algorithm 2), the paper's own
 * beacon maintenance, instead of running-mean centroids.  n_beacons is then
 * B_Q^min per QUERY head and every query head keeps a buffer of at most
 * B_Q^max = n_beacons + window pre-RoPE queries:
 *   bkv_init_beacons    buffer = FPS (Algorithm 1, fp64 similarities) of the
 *                       head's n_init prompt queries down to n_beacons rows;
 *   bkv_update_beacons  each new query is appended in order; whenever the
 *                       buffer holds B_Q^max rows it is replaced by its FPS
 *                       selection of n_beacons rows (Eq. 9);
 *   bkv_compress        the beacons of head h are the FPS selection of
 *                       min(n_beacons, size) buffer rows, rotated to t_pos;
 *                       the group scores with its G * n_beacons beacons and
 *                       G * window recent queries; after an eviction each
 *                       buffer becomes the FPS selection of n_beacons rows of
 *                       (its beacons, then its window queries in order).
 * The FPS of the buffer steps takes its similarities in fp32: fused
 * multiply-add dot products in element order, cos = dot / (|a| |b|) (0 for a
 * zero vector), the averages summed in row order, ties to the lowest row.
 * Requires n_beacons >= 1, window >= 1, n_beacons + window <= 32 and
 * G * (n_beacons + window) <= 128.  The centroid state functions do not apply.
 */
#define BKV_F_CONTINUAL_FPS 2u
/*
 * Causal mask inside the recent window (AttnWeight's mask, which the paper
 * leaves open; Algorithm 2, Section 4.3).  Positions: recent slot w sits at
 * recent_pos[w], beacons at t_pos, and the last `window` cache rows j
 * (L - window <= j < L) at t_pos - (L - 1 - j); older rows come before every
 * window position.  A recent query then takes no part in the softmax of the
 * window rows after its own position: those rows are left out of its
 * normaliser and its weight on them is 0 (it still counts in the mean of
 * BKV_F_MEAN_AGG).  Beacons and older rows are never masked.  Selection, the
 * keep set and compaction are unchanged.  Applies to bkv_compress and
 * bkv_compress_static; no effect when window = 0.
 */
#define BKV_F_CAUSAL_WINDOW 4u

typedef struct bkv_ctx bkv_ctx;

/*
 * Model / cache shape, fixed for the life of a context.
 *   head_dim    64 or 128.
 *   n_beacons   beacons per KV head, 0..32 (0 = recent queries only).
 *   window      recent queries per query head kept for scoring AND number of
 *               most recent cache rows that are always kept, 0..64.
 *   n_prefix    number of leading cache rows that are always kept (>= 0).
 *   capacity    rows allocated per instance in K and V (1..32768).
 *   rope_theta  rotary base; 0 disables rotation.
 * Limits: G * window + n_beacons must be in 1..128.
 */
typedef struct {
  int32_t n_layers, batch, n_q_heads, n_kv_heads, head_dim;
  int32_t n_beacons, window, n_prefix;
  int32_t capacity;
  double rope_theta;
  uint32_t flags; /* BKV_F_* options; unknown bits are rejected */
} bkv_config;

/*
 * Creates a context on the current CUDA device and allocates its beacon state
 * (fp32 centroids, fp64 sums, int64 counts; all zero, i.e. no beacon yet) and
 * scratch.  `stream` is a cudaStream_t (NULL = legacy default stream).
 * Returns BKV_EINVAL for a bad config, BKV_ENOMEM / BKV_ECUDA on failure.
 */
int bkv_create(const bkv_config* cfg, void* stream, bkv_ctx** out);

/* Frees everything the context owns (after synchronising its stream). NULL is ignored. */
void bkv_destroy(bkv_ctx* ctx);

/* Changes the stream used by later calls.  The new stream is made to wait
 * (cudaStreamWaitEvent) for the work already enqueued on the old one, so a
 * switch never lets two calls of one context run concurrently.  Returns
 * BKV_ECUDA if the event record or the wait fails (the stream is then
 * unchanged). */
int bkv_set_stream(bkv_ctx* ctx, void* stream);

/*
 * Prefill seeding (Appendix D.2: FPS over the prompt's pre-RoPE queries;
 * Algorithm 1).  For every instance, FPS runs over the G * n_init queries of
 * its group (head-major order h * n_init + i, cosine similarity, ties to the
 * lowest index) and beacon k becomes the k-th selected query with count 1.
 *   q_init  bf16 [n_layers][batch][n_q_heads][n_init][head_dim], pre-RoPE.
 * Requires G * n_init >= n_beacons and G * n_init <= 4096.
 * Replaces any previous beacon state.
 */
int bkv_init_beacons(bkv_ctx* ctx, const void* q_init, int32_t n_init);

/*
 * Beacon maintenance for n_new decode queries per query head.  Each query q
 * is assigned to argmax_b cos(q, c_b) over the beacons with count > 0 and a
 * non-zero centroid, using the centroids as they were when the call started
 * (ties go to the lowest b; a zero query is skipped).  Then for each beacon
 * sums_b += sum of its assigned queries, counts_b += their number and
 * c_b = fp32(sums_b / counts_b) to within one fp32 ulp.  Query elements must be finite with
 * |x| < 2^14, and one call's sum for a beacon must stay below 2^23 in every
 * element (int64 fixed point with 40 fractional bits); that sum is then
 * exact, except that elements below 2^-31 in magnitude are rounded to
 * multiples of 2^-38.  Assignments equal the exact cosine argmax except at
 * ties below about 1e-12 relative.
 *   q_new       bf16 [n_layers][batch][n_q_heads][n_new][head_dim], pre-RoPE.
 *   assign_out  int32 [n_layers][batch][n_q_heads][n_new] or NULL: the beacon
 *               chosen for each query, -1 when it was skipped (all -1 under
 *               BKV_F_CONTINUAL_FPS, which assigns nothing).
 * n_new == 0 is a no-op.  BKV_ESTATE if bkv_init_beacons / bkv_set_state was
 * never called.
 */
int bkv_update_beacons(bkv_ctx* ctx, const void* q_new, int32_t n_new, int32_t* assign_out);

/*
 * A run of decode steps in one call: step t brings one query per query head
 * (Algorithm 2's decode branch, one generated token), and the steps are
 * applied in order, each against the centroids the steps before it left.
 * The state afterwards and every assignment are bit-identical to those of
 * n_steps calls of bkv_update_beacons(q_steps + t * step, n_new = 1), under
 * every flag.  Nothing reads the beacons between two compressions, so a
 * decode loop may hold a period's queries and hand them over at once; the
 * state is then read from and written back to device memory once per call
 * instead of once per step.  The paper has no such call: it is a batching of
 * Algorithm 2's per-token updates.
 *   q_steps     bf16 [n_steps][n_layers][batch][n_q_heads][head_dim], pre-RoPE
 *               (step-major: each step is the q_new of a one-query call).
 *   assign_out  int32 [n_steps][n_layers][batch][n_q_heads] or NULL.
 * Same element limits as bkv_update_beacons, per step.  n_steps == 0 is a
 * no-op.  BKV_ESTATE as bkv_update_beacons.
 */
int bkv_update_beacons_seq(bkv_ctx* ctx, const void* q_steps, int32_t n_steps, int32_t* assign_out);

/*
 * One compression of every instance's cache from L rows to `budget` rows.
 * Observation queries (Section 4.3): for each instance, the recent queries of
 * its G query heads, query (h, w) rotated to position recent_pos[w], and its
 * beacons with count > 0 rotated to t_pos; each is rounded to bf16 after the
 * rotation.  Score[j] = max over those queries of the softmax weight of key
 * j over all L cached keys (Eq. 4, Eq. 6 max form; logits q.k / sqrt(d)), or
 * their mean under BKV_F_MEAN_AGG; under BKV_F_CAUSAL_WINDOW a recent query
 * leaves out the window rows after its own position.
 * Kept rows = [0, n_prefix) U [L - window, L) U the (budget - n_prefix -
 * window) other rows with the largest Score (ties to the lower index), in
 * ascending order (Eq. 7, Algorithm 2).  Row i of K and V then holds what row
 * kept[i] held (Eq. 8); rows >= budget are left unspecified.
 *   K, V          bf16 [n_layers][batch][n_kv_heads][capacity][head_dim]; rows
 *                 [0, L) are read, rows [0, budget) rewritten in place.  Keys
 *                 are taken as already rotated (post-RoPE).
 *   L             current rows per instance, 1..capacity.
 *   budget        rows to keep, >= n_prefix + window.  L <= budget: nothing
 *                 is evicted, K/V are not touched and kept_idx_out[i] = i for
 *                 i < L, -1 for L <= i < budget.
 *   t_pos         absolute position of the current decode step (beacons).
 *   q_recent      bf16 [n_layers][batch][n_q_heads][window][head_dim], pre-RoPE.
 *   recent_pos    HOST int64 [window]: absolute position of recent slot w.
 *   kept_idx_out  int32 [n_layers][batch][n_kv_heads][budget].
 *   scores_out    fp32 [n_layers][batch][n_kv_heads][capacity] or NULL:
 *                 Score[j] for j < L (only written when L > budget).
 * BKV_ESTATE if n_beacons > 0 and no beacon state was set.
 */
int bkv_compress(bkv_ctx* ctx, void* K, void* V, int32_t L, int32_t budget, int64_t t_pos,
                 const void* q_recent, const int64_t* recent_pos, int32_t* kept_idx_out, float* scores_out);

/*
 * bkv_compress with a cache length of its own for every instance: in batched
 * decoding each sequence of the batch has its own length and position
 * (Section 5.4), and Algorithm 2 runs per sequence.  Everything is as in
 * bkv_compress, instance by instance, except:
 *   L           DEVICE int32 [n_layers][batch][n_kv_heads]: rows of each
 *               instance.  An instance with L <= budget is not touched and
 *               gets kept_idx_out[i] = i for i < L, -1 after; an instance with
 *               budget < L is compressed to budget rows from its own L (its
 *               softmax runs over its L keys, its window is its last
 *               `window` rows).  A length outside 1..capacity leaves that
 *               instance untouched with kept_idx_out all -1, and the next
 *               bkv_sync returns BKV_EINVAL.
 *   t_pos       HOST int64 [batch]: position of each batch row's current
 *               decode step (its beacons are rotated there).
 *   recent_pos  HOST int64 [batch][window]: positions of each batch row's
 *               recent slots.
 *   scores_out  written for j < L of the instances that are compressed.
 * Under BKV_F_CONTINUAL_FPS only the heads of compressed instances merge
 * (Algorithm 2's post-eviction step).
 */
int bkv_compress_ragged(bkv_ctx* ctx, void* K, void* V, const int32_t* L, int32_t budget, const int64_t* t_pos,
                        const void* q_recent, const int64_t* recent_pos, int32_t* kept_idx_out, float* scores_out);

/*
 * Copies the beacon state to / from caller buffers (checkpoint / resume):
 *   centroids fp32 [n_inst][n_beacons][head_dim]
 *   sums      fp64 [n_inst][n_beacons][head_dim]
 *   counts    int64 [n_inst][n_beacons]
 * Each pointer may be device memory or host memory (pinned or pageable): the
 * direction of each copy is taken from the pointer (unified addressing).  The
 * copies are ordered on the context's stream; host results of bkv_get_state
 * are valid once the stream has been synchronised (bkv_sync), and host
 * sources of bkv_set_state may be reused when the call returns (a copy from
 * pageable memory is staged before the call returns).  Any pointer may be
 * NULL to skip that array (get only).  bkv_set_state needs all three and
 * marks the state as initialised.
 */
int bkv_get_state(bkv_ctx* ctx, float* centroids, double* sums, int64_t* counts);
int bkv_set_state(bkv_ctx* ctx, const float* centroids, const double* sums, const int64_t* counts);

/*
 * Continual FPS contexts: copies the buffers to / from caller memory (device
 * or host, as for bkv_get_state).
 *   buffers  bf16 [n_layers][batch][n_q_heads][n_beacons + window][head_dim];
 *            rows [0, size) of each head are in use, in buffer order.
 *   sizes    int32 [n_layers][batch][n_q_heads], each in 0..n_beacons + window - 1.
 * bkv_set_cfps_state needs both and marks the state as initialised.
 * BKV_EINVAL on a context without BKV_F_CONTINUAL_FPS.
 */
int bkv_get_cfps_state(bkv_ctx* ctx, void* buffers, int32_t* sizes);
int bkv_set_cfps_state(bkv_ctx* ctx, const void* buffers, const int32_t* sizes);

/*
 * Waits for the context's stream, then reads and clears the device error
 * word.  Returns BKV_OK, BKV_ETIMEOUT (a kernel gave up a bounded wait and
 * its outputs are invalid), BKV_EINVAL (a per-instance length of
 * bkv_compress_ragged outside 1..capacity), BKV_EBOUNDS (a library built with
 * BKV_CHECKED found an index from device data out of range, skipped that
 * access, and the outputs are invalid) or BKV_ECUDA.
 */
int bkv_sync(bkv_ctx* ctx);

/*
 * Diagnostic with no counterpart in the paper: checks the expiry path of the
 * library's bounded device waits.  After a bkv_sync of earlier work, launches
 * on the context's stream one kernel that waits on a barrier nothing
 * completes, through the same wait routine the other kernels use, with the
 * limit limit_ns (1e3 .. 1e10 ns) instead of the kernels' 1 s; the wait
 * expires, the kernel records the timeout in the device error word and
 * returns.  Returns what bkv_sync then reports: BKV_ETIMEOUT when the path
 * works, with the error word cleared and the context usable; BKV_EINVAL for
 * a NULL context or a limit out of range; BKV_ECUDA on a CUDA error.
 */
int bkv_selftest_wait_timeout(bkv_ctx* ctx, int64_t limit_ns);

/*
 * Checked builds (diagnostic; no counterpart in the paper).  A library
 * compiled with BKV_CHECKED defined checks every index that its kernels take
 * from device data before using it: work-list entries and per-instance
 * lengths of a ragged compress, the positions and source rows of the kept
 * set in the selection and gather, and the stored Continual FPS buffer
 * sizes.  A failing check records BKV_EBOUNDS in the device error word (see
 * bkv_sync) and the access is skipped or redirected in range; nothing traps.
 * The default build compiles the checks out.
 *
 * bkv_checked_build returns 1 for a library built with BKV_CHECKED, else 0.
 * bkv_selftest_bounds, after a bkv_sync of earlier work, launches one kernel
 * that makes a checked store one past the logical end of a shared-memory
 * array twice that long (so the store stays in memory the kernel owns with
 * or without checks) and returns what bkv_sync then reports: BKV_EBOUNDS in
 * a checked build, BKV_OK in the default one, with the error word cleared
 * and the context usable either way.
 */
int bkv_checked_build(void);
int bkv_selftest_bounds(bkv_ctx* ctx);

/*
 * Allocation-failure hook (test diagnostic).  With nth > 0, the nth device
 * or pinned host allocation that later bkv_create calls attempt (counted
 * from this call, across contexts) fails as if memory ran out, without
 * allocating: that bkv_create releases what it had allocated, leaves *out
 * NULL and returns BKV_ENOMEM.  The hook disarms itself after that one
 * failure; nth = 0 disarms it.  Not thread-safe with concurrent bkv_create
 * calls.  Returns BKV_OK, or BKV_EINVAL for nth < 0.
 */
int bkv_debug_fail_alloc(int32_t nth);

/*
 * Per-kernel timing (tracing).  While enabled, every kernel launch made by
 * this context is bracketed by CUDA events on the context's stream.
 * bkv_profile_read synchronises the stream, then writes for each kernel k
 * (BKV_K_* below, n_kernels entries at most) the summed device time in
 * milliseconds (ms[k]) and the number of launches (launches[k]) since the
 * previous read, and resets the totals.  Either output may be NULL.
 */
#define BKV_K_FPS 0
#define BKV_K_UPDATE 1
#define BKV_K_QOBS 2
#define BKV_K_SCORE 3
#define BKV_K_SELECT_GATHER 4
#define BKV_K_KEEP_ALL 5
#define BKV_K_CFPS 6 /* Continual FPS buffer update, beacon selection and merge */
#define BKV_K_ROPE 7 /* rotary table of a compress, copied from pinned host memory */
#define BKV_NUM_KERNELS 8
int bkv_profile_enable(bkv_ctx* ctx, int on);
int bkv_profile_read(bkv_ctx* ctx, double* ms, int64_t* launches, int32_t n_kernels);

/*
 * bkv_compress_static - bkv_compress for callers that must not allocate
 * device memory.  The paper has no counterpart: this entry point exists for
 * integrations that cannot call cudaMalloc, such as a serving engine that has
 * given all of HBM to its own KV-cache page allocator, or a plugin whose host
 * framework owns every device allocation (cudaMalloc may also synchronise
 * the device, which a decode loop on a latency budget cannot afford).
 *
 * Computes exactly what bkv_compress computes, with the same kernels, but
 * takes everything from the caller: the shape (cfg, same limits as
 * bkv_create), the beacon state (centroids fp32 [n_inst][n_beacons][d] and
 * counts int64 [n_inst][n_beacons], device; may be NULL when n_beacons = 0)
 * and the stream; cfg->flags may hold BKV_F_MEAN_AGG and BKV_F_CAUSAL_WINDOW
 * (the Continual FPS mode needs a context and is rejected here).  It needs no
 * context and allocates or frees nothing.  Its
 * scratch is one library-owned device array of 16 MiB (resident on every
 * device that loads the library until the process exits); a call whose
 * scratch exceeds it - n_inst * (4 * capacity + 2 * n_obs_pad * head_dim +
 * 16) bytes plus the rotary table, each part rounded up to 256 bytes - is
 * rejected with BKV_EINVAL and a message.
 *   dev_status  device int32 or NULL: cleared by the call, set non-zero if a
 *               kernel's bounded wait expires or, in a checked build, a
 *               device-side bounds check fails (outputs are then invalid).
 *   err_msg     host buffer of err_len bytes or NULL: reason of a failure.
 * The rotary table (rope_theta != 0) reaches the device inside the
 * parameters of small kernels on `stream`, 16 KB per launch: no copy from
 * host memory, and the call does not wait for earlier work on the stream.
 * All calls share the scratch array and it keeps the previous call's
 * contents; calls that overlap on the GPU (other streams, other threads
 * without ordering) race on it.  The array's device address is looked up
 * with cudaGetSymbolAddress during the first call on each device (any call
 * that passes argument validation, with that device current), so make that
 * first call before any stream capture.
 */
int bkv_compress_static(const bkv_config* cfg, const float* centroids, const int64_t* counts, void* K, void* V,
                        int32_t L, int32_t budget, int64_t t_pos, const void* q_recent, const int64_t* recent_pos,
                        int32_t* kept_idx_out, float* scores_out, int32_t* dev_status, void* stream, char* err_msg,
                        size_t err_len);

/* Static description of an error code. */
const char* bkv_strerror(int code);

/* One-line description of the last error on this context ("" if none). */
const char* bkv_last_error(const bkv_ctx* ctx);

/* Version string of the library build. */
const char* bkv_version(void);

#ifdef __cplusplus
}
#endif
#endif /* BKV_H */
