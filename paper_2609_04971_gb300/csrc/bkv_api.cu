// C ABI of the BeaconKV compression step (declared in include/bkv.h):
// argument validation, context and scratch ownership, tensor-map encoding,
// the rotary table, and kernel launches on the context's stream.

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "bkv.h"
#include "bkv_device.cuh"
#include "bkv_internal.h"

using bkv::Shape;

struct bkv_ctx {
  bkv_config cfg{};
  Shape shape{};
  cudaStream_t stream = nullptr;
  int device = 0;
  // beacon state
  float* cent = nullptr;
  double* sums = nullptr;
  long long* counts = nullptr;
  bool state_ready = false;
  // Continual FPS (BKV_F_CONTINUAL_FPS): per-query-head buffers; cent / counts then hold each
  // compress's beacons ([n_inst][G * n_beacons] rows, count 1 or 0) for the scoring-query build
  bool cfps = false;
  int b_min = 0, b_max = 0, n_heads = 0;
  __nv_bfloat16* cbuf = nullptr;  // [n_heads][b_max][d]
  int* csize = nullptr;           // [n_heads]
  // scratch
  __nv_bfloat16* qobs = nullptr;  // [n_inst][n_obs_pad][d]
  uint32_t* valid = nullptr;      // [n_inst][4]
  float* rscore = nullptr;        // [n_inst][cap]
  double2* rope = nullptr;        // [W + 1][d / 2] fp64 (cos, sin), then the same table in fp32
  int* err = nullptr;             // device error word
  // pinned host staging of the rotary table, a ring of kRopeSlots: a compress fills the next slot,
  // a kernel on the stream copies it to `rope` through the slot's device mapping, and the slot is
  // refilled only after that copy's event completed
  static constexpr int kRopeSlots = 4;
  double2* rope_pinned[kRopeSlots] = {};
  void* rope_mapped[kRopeSlots] = {};  // device address of rope_pinned[i]
  cudaEvent_t rope_ev[kRopeSlots] = {};
  bool rope_used[kRopeSlots] = {};
  int rope_next = 0;
  // per-instance lengths (bkv_compress_ragged): the instances a compress evicts from, and a rotary
  // table per batch row followed by the causal gaps [batch][W] (int32), staged like `rope`
  int* work = nullptr;            // [n_inst]
  int* n_work = nullptr;          // [1]
  unsigned char* rag = nullptr;   // device copy of the per-row tables and gaps
  size_t rag_bytes = 0, rag_row = 0, rag_gaps_off = 0;  // total bytes; one row's table (double2 units); gaps offset
  void* rag_pinned[kRopeSlots] = {};
  void* rag_mapped[kRopeSlots] = {};
  cudaEvent_t rag_ev[kRopeSlots] = {};
  bool rag_used[kRopeSlots] = {};
  int rag_next = 0;
  cudaEvent_t switch_ev = nullptr;  // orders a new stream after the previous one (bkv_set_stream)
  std::string last_error;
  // per-kernel timing
  struct Rec {
    cudaEvent_t start, stop;
    int kernel;
  };
  bool prof = false;
  std::vector<Rec> pending;
  std::vector<cudaEvent_t> spare;
  double prof_ms[BKV_NUM_KERNELS] = {};
  long long prof_n[BKV_NUM_KERNELS] = {};
};

namespace {

int fail(bkv_ctx* c, int code, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    c->last_error = buf;
  }
  return code;
}

int cuda_fail(bkv_ctx* c, cudaError_t e, const char* what) {
  return fail(c, BKV_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

cudaEvent_t take_event(bkv_ctx* c) {
  if (!c->spare.empty()) {
    cudaEvent_t ev = c->spare.back();
    c->spare.pop_back();
    return ev;
  }
  cudaEvent_t ev = nullptr;
  cudaEventCreate(&ev);
  return ev;
}

// Brackets one kernel launch with events when timing is enabled.
struct ProfScope {
  bkv_ctx* c;
  int kernel;
  cudaEvent_t start = nullptr;
  ProfScope(bkv_ctx* ctx, int k) : c(ctx), kernel(k) {
    if (c->prof && (start = take_event(c))) cudaEventRecord(start, c->stream);
  }
  ~ProfScope() {
    if (!start) return;
    cudaEvent_t stop = take_event(c);
    if (!stop) return;
    cudaEventRecord(stop, c->stream);
    c->pending.push_back({start, stop, kernel});
  }
};

void fold_profile(bkv_ctx* c) {
  for (auto& r : c->pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.start, r.stop) == cudaSuccess) {
      c->prof_ms[r.kernel] += ms;
      c->prof_n[r.kernel] += 1;
    }
    c->spare.push_back(r.start);
    c->spare.push_back(r.stop);
  }
  c->pending.clear();
}

// 2-D bf16 tensor [rows][d] viewed in boxes of [box_rows][64] with 128-byte swizzle.
int encode_rows(bkv_ctx* c, CUtensorMap* map, const void* base, uint64_t rows, int d, uint32_t box_rows) {
  const CUresult r = bkv::encode_rows_bf16(map, base, rows, d, box_rows);
  if (r == CUDA_ERROR_NOT_FOUND) return fail(c, BKV_ECUDA, "cuTensorMapEncodeTiled is unavailable");
  if (r != CUDA_SUCCESS) return fail(c, BKV_ECUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return BKV_OK;
}

int validate_config(const bkv_config* cfg, std::string& why) {
  char buf[256];
  auto bad = [&](const char* m) {
    why = m;
    return BKV_EINVAL;
  };
  if (!cfg) return bad("config is NULL");
  if (cfg->n_layers < 1 || cfg->batch < 1 || cfg->n_q_heads < 1 || cfg->n_kv_heads < 1)
    return bad("n_layers, batch, n_q_heads and n_kv_heads must be >= 1");
  if (cfg->n_q_heads % cfg->n_kv_heads != 0) return bad("n_q_heads must be a multiple of n_kv_heads");
  if (cfg->head_dim != 64 && cfg->head_dim != 128) return bad("head_dim must be 64 or 128");
  if (cfg->n_beacons < 0 || cfg->n_beacons > bkv::kMaxBeacons) return bad("n_beacons must be in 0..32");
  if (cfg->window < 0 || cfg->window > bkv::kMaxWindow) return bad("window must be in 0..64");
  if (cfg->n_prefix < 0) return bad("n_prefix must be >= 0");
  if (cfg->capacity < 1 || cfg->capacity > bkv::kMaxCapacity) return bad("capacity must be in 1..32768");
  if (!(cfg->rope_theta >= 0.0) || !std::isfinite(cfg->rope_theta)) return bad("rope_theta must be finite and >= 0");
  if (cfg->flags & ~(BKV_F_MEAN_AGG | BKV_F_CONTINUAL_FPS | BKV_F_CAUSAL_WINDOW))
    return bad("flags holds an unknown option");
  const long long G = cfg->n_q_heads / cfg->n_kv_heads;
  const bool cfps = (cfg->flags & BKV_F_CONTINUAL_FPS) != 0;
  if (cfps && (cfg->n_beacons < 1 || cfg->window < 1 || cfg->n_beacons + cfg->window > bkv::kCfpsMaxRows))
    return bad("continual FPS needs n_beacons >= 1, window >= 1 and n_beacons + window <= 32");
  const long long n_obs = G * cfg->window + (cfps ? G * cfg->n_beacons : cfg->n_beacons);
  if (n_obs < 1 || n_obs > bkv::kMaxObs) {
    snprintf(buf, sizeof buf, "scoring queries per KV head (G * window + beacons) = %lld must be in 1..128", n_obs);
    why = buf;
    return BKV_EINVAL;
  }
  const long long n_inst = 1LL * cfg->n_layers * cfg->batch * cfg->n_kv_heads;
  if (n_inst * cfg->capacity >= (1LL << 31) || n_inst * 128 >= (1LL << 31))
    return bad("n_layers * batch * n_kv_heads * capacity must be below 2^31");
  return BKV_OK;
}

// Allocation-failure hook (bkv_debug_fail_alloc): once armed with n > 0, the n-th device or pinned
// host allocation that bkv_create attempts reports cudaErrorMemoryAllocation without allocating,
// and the hook disarms itself.
std::atomic<int> g_fail_nth{0};
std::atomic<int> g_alloc_seen{0};

bool fail_this_alloc() {
  const int nth = g_fail_nth.load();
  if (nth <= 0 || g_alloc_seen.fetch_add(1) + 1 != nth) return false;
  g_fail_nth.store(0);
  return true;
}

template <typename T>
cudaError_t dmalloc(T** p, size_t n) {
  if (fail_this_alloc()) return cudaErrorMemoryAllocation;
  return cudaMalloc(reinterpret_cast<void**>(p), sizeof(T) * (n ? n : 1));
}

template <typename T>
cudaError_t hmalloc(T** p, size_t bytes) {
  if (fail_this_alloc()) return cudaErrorMemoryAllocation;
  return cudaMallocHost(reinterpret_cast<void**>(p), bytes);
}

void free_all(bkv_ctx* c) {
  for (auto& r : c->pending) {
    cudaEventDestroy(r.start);
    cudaEventDestroy(r.stop);
  }
  c->pending.clear();
  for (auto ev : c->spare) cudaEventDestroy(ev);
  c->spare.clear();
  cudaFree(c->cent);
  cudaFree(c->sums);
  cudaFree(c->counts);
  cudaFree(c->cbuf);
  cudaFree(c->csize);
  cudaFree(c->qobs);
  cudaFree(c->valid);
  cudaFree(c->rscore);
  cudaFree(c->rope);
  cudaFree(c->err);
  for (int i = 0; i < bkv_ctx::kRopeSlots; ++i) {
    if (c->rope_pinned[i]) cudaFreeHost(c->rope_pinned[i]);
    if (c->rope_ev[i]) cudaEventDestroy(c->rope_ev[i]);
    if (c->rag_pinned[i]) cudaFreeHost(c->rag_pinned[i]);
    if (c->rag_ev[i]) cudaEventDestroy(c->rag_ev[i]);
  }
  cudaFree(c->work);
  cudaFree(c->n_work);
  cudaFree(c->rag);
  if (c->switch_ev) cudaEventDestroy(c->switch_ev);
}

}  // namespace

extern "C" {

int bkv_debug_fail_alloc(int32_t nth) {
  if (nth < 0) return BKV_EINVAL;
  g_alloc_seen.store(0);
  g_fail_nth.store(nth);
  return BKV_OK;
}

const char* bkv_version(void) { return "bkv 0.1.0 (sm_103a, tcgen05)"; }

const char* bkv_strerror(int code) {
  switch (code) {
    case BKV_OK: return "ok";
    case BKV_EINVAL: return "invalid argument";
    case BKV_ENOMEM: return "device allocation failed";
    case BKV_ECUDA: return "CUDA error";
    case BKV_ETIMEOUT: return "device wait timed out; outputs are invalid";
    case BKV_ESTATE: return "beacon state not initialised";
    case BKV_EBOUNDS: return "device-side bounds check failed (checked build); outputs are invalid";
    default: return "unknown error";
  }
}

const char* bkv_last_error(const bkv_ctx* ctx) { return ctx ? ctx->last_error.c_str() : ""; }

int bkv_create(const bkv_config* cfg, void* stream, bkv_ctx** out) {
  if (!out) return BKV_EINVAL;
  *out = nullptr;
  std::string why;
  if (validate_config(cfg, why) != BKV_OK) return BKV_EINVAL;
  auto* c = new (std::nothrow) bkv_ctx();
  if (!c) return BKV_ENOMEM;
  c->cfg = *cfg;
  Shape& s = c->shape;
  s.G = cfg->n_q_heads / cfg->n_kv_heads;
  s.n_inst = cfg->n_layers * cfg->batch * cfg->n_kv_heads;
  s.d = cfg->head_dim;
  c->cfps = (cfg->flags & BKV_F_CONTINUAL_FPS) != 0;
  s.nb = c->cfps ? s.G * cfg->n_beacons : cfg->n_beacons;  // beacon scoring rows per instance
  s.W = cfg->window;
  c->b_min = cfg->n_beacons;
  c->b_max = cfg->n_beacons + cfg->window;
  c->n_heads = c->cfps ? cfg->n_layers * cfg->batch * cfg->n_q_heads : 0;
  s.n_prefix = cfg->n_prefix;
  s.cap = cfg->capacity;
  s.n_obs = s.G * s.W + s.nb;
  s.n_obs_pad = (s.n_obs + 15) / 16 * 16;
  s.batch = cfg->batch;
  s.n_kv = cfg->n_kv_heads;
  c->stream = static_cast<cudaStream_t>(stream);
  // per-row rotary tables ([W + 1][d / 2] fp64 pairs, then fp32 pairs) and causal gaps of a ragged compress
  c->rag_row = static_cast<size_t>(s.W + 1) * (s.d / 2) * 3 / 2;  // double2 units (a multiple of 2: 16-byte rows)
  c->rag_gaps_off = sizeof(double2) * c->rag_row * static_cast<size_t>(s.batch);
  c->rag_bytes = c->rag_gaps_off + (sizeof(int32_t) * static_cast<size_t>(s.batch) * (s.W > 0 ? s.W : 1) + 15) / 16 * 16;
  cudaGetDevice(&c->device);

  const size_t ni = static_cast<size_t>(s.n_inst);
  cudaError_t e = cudaSuccess;
  const size_t nh = static_cast<size_t>(c->n_heads);
  if ((e = dmalloc(&c->cent, ni * s.nb * s.d)) != cudaSuccess ||
      (e = dmalloc(&c->sums, c->cfps ? 0 : ni * s.nb * s.d)) != cudaSuccess ||
      (e = dmalloc(&c->counts, ni * s.nb)) != cudaSuccess ||
      (e = dmalloc(&c->cbuf, nh * c->b_max * s.d)) != cudaSuccess ||
      (e = dmalloc(&c->csize, nh)) != cudaSuccess ||
      (e = dmalloc(&c->qobs, ni * s.n_obs_pad * s.d)) != cudaSuccess ||
      (e = dmalloc(&c->valid, ni * 4)) != cudaSuccess ||
      (e = dmalloc(&c->rscore, ni * s.cap)) != cudaSuccess ||
      (e = dmalloc(&c->rope, static_cast<size_t>(s.W + 1) * (s.d / 2) * 3 / 2 + 1)) != cudaSuccess ||
      (e = dmalloc(&c->work, ni)) != cudaSuccess || (e = dmalloc(&c->n_work, 1)) != cudaSuccess ||
      (e = dmalloc(&c->rag, c->rag_bytes)) != cudaSuccess ||
      (e = dmalloc(&c->err, 1)) != cudaSuccess) {
    const int code = (e == cudaErrorMemoryAllocation) ? BKV_ENOMEM : BKV_ECUDA;
    cudaGetLastError();
    free_all(c);
    delete c;
    return code;
  }
  if ((e = cudaMemsetAsync(c->cent, 0, sizeof(float) * ni * s.nb * s.d + 0, c->stream)) != cudaSuccess ||
      (e = cudaMemsetAsync(c->sums, 0, sizeof(double) * (c->cfps ? 1 : ni * s.nb * s.d), c->stream)) != cudaSuccess ||
      (e = cudaMemsetAsync(c->csize, 0, sizeof(int) * (nh ? nh : 1), c->stream)) != cudaSuccess ||
      (e = cudaMemsetAsync(c->counts, 0, sizeof(long long) * ni * s.nb, c->stream)) != cudaSuccess ||
      (e = cudaMemsetAsync(c->err, 0, sizeof(int), c->stream)) != cudaSuccess) {
    free_all(c);
    delete c;
    return BKV_ECUDA;
  }
  const size_t rope_bytes = sizeof(double2) * (static_cast<size_t>(s.W + 1) * (s.d / 2) * 3 / 2 + 1);
  for (int i = 0; i < bkv_ctx::kRopeSlots; ++i) {
    if ((e = hmalloc(&c->rope_pinned[i], rope_bytes)) != cudaSuccess ||
        (e = cudaHostGetDevicePointer(&c->rope_mapped[i], c->rope_pinned[i], 0)) != cudaSuccess ||
        (e = cudaEventCreateWithFlags(&c->rope_ev[i], cudaEventDisableTiming)) != cudaSuccess ||
        (e = hmalloc(&c->rag_pinned[i], c->rag_bytes)) != cudaSuccess ||
        (e = cudaHostGetDevicePointer(&c->rag_mapped[i], c->rag_pinned[i], 0)) != cudaSuccess ||
        (e = cudaEventCreateWithFlags(&c->rag_ev[i], cudaEventDisableTiming)) != cudaSuccess) {
      const int code = (e == cudaErrorMemoryAllocation) ? BKV_ENOMEM : BKV_ECUDA;
      cudaGetLastError();
      free_all(c);
      delete c;
      return code;
    }
  }
  if ((e = cudaEventCreateWithFlags(&c->switch_ev, cudaEventDisableTiming)) != cudaSuccess) {
    cudaGetLastError();
    free_all(c);
    delete c;
    return BKV_ECUDA;
  }
  *out = c;
  return BKV_OK;
}

void bkv_destroy(bkv_ctx* ctx) {
  if (!ctx) return;
  cudaStreamSynchronize(ctx->stream);
  free_all(ctx);
  delete ctx;
}

int bkv_set_stream(bkv_ctx* ctx, void* stream) {
  if (!ctx) return BKV_EINVAL;
  const cudaStream_t next = static_cast<cudaStream_t>(stream);
  if (next != ctx->stream) {
    // the context's scratch and state are reused by the next call: its work on the new stream
    // starts after everything already enqueued on the old one
    cudaError_t e = cudaEventRecord(ctx->switch_ev, ctx->stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(next, ctx->switch_ev, 0);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "stream switch");
  }
  ctx->stream = next;
  return BKV_OK;
}

int bkv_init_beacons(bkv_ctx* ctx, const void* q_init, int32_t n_init) {
  if (!ctx) return BKV_EINVAL;
  const Shape& s = ctx->shape;
  if (s.nb == 0) {
    ctx->state_ready = true;
    return BKV_OK;
  }
  if (!q_init || !aligned16(q_init)) return fail(ctx, BKV_EINVAL, "q_init must be a non-NULL 16-byte aligned pointer");
  if (ctx->cfps) {
    // per query head: FPS of its n_init prompt queries down to n_beacons rows (the buffer)
    if (n_init < ctx->b_min || n_init > bkv::kMaxFpsRows)
      return fail(ctx, BKV_EINVAL, "n_init = %d must be in n_beacons..4096", n_init);
    Shape hs = s;
    hs.n_inst = ctx->n_heads;
    hs.G = 1;
    hs.nb = ctx->b_min;
    ProfScope ps(ctx, BKV_K_FPS);
    cudaError_t e = bkv::launch_fps_init(hs, static_cast<const __nv_bfloat16*>(q_init), n_init, ctx->cent, nullptr,
                                         ctx->counts, ctx->stream);
    if (e == cudaSuccess)
      e = bkv::launch_cfps_seed(s.d, ctx->cent, ctx->n_heads, ctx->b_min, ctx->b_max, ctx->cbuf, ctx->csize,
                                ctx->stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "continual FPS seeding launch");
    ctx->state_ready = true;
    return BKV_OK;
  }
  const long long N = 1LL * s.G * n_init;
  if (n_init < 1 || N < s.nb || N > bkv::kMaxFpsRows)
    return fail(ctx, BKV_EINVAL, "G * n_init = %lld must be in n_beacons..4096", N);
  ProfScope ps(ctx, BKV_K_FPS);
  cudaError_t e = bkv::launch_fps_init(s, static_cast<const __nv_bfloat16*>(q_init), n_init, ctx->cent, ctx->sums,
                                       ctx->counts, ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "fps_init launch");
  ctx->state_ready = true;
  return BKV_OK;
}

int bkv_update_beacons(bkv_ctx* ctx, const void* q_new, int32_t n_new, int32_t* assign_out) {
  if (!ctx) return BKV_EINVAL;
  const Shape& s = ctx->shape;
  if (n_new < 0) return fail(ctx, BKV_EINVAL, "n_new must be >= 0");
  if (n_new == 0) return BKV_OK;
  if (!q_new || !aligned16(q_new)) return fail(ctx, BKV_EINVAL, "q_new must be a non-NULL 16-byte aligned pointer");
  if (assign_out && (reinterpret_cast<uintptr_t>(assign_out) & 3u))
    return fail(ctx, BKV_EINVAL, "assign_out must be 4-byte aligned");
  if (1LL * s.n_inst * s.G * n_new >= (1LL << 31)) return fail(ctx, BKV_EINVAL, "n_new too large");
  if (s.nb == 0) {
    if (assign_out) {
      cudaError_t e =
          cudaMemsetAsync(assign_out, 0xff, sizeof(int32_t) * s.n_inst * s.G * static_cast<size_t>(n_new), ctx->stream);
      if (e != cudaSuccess) return cuda_fail(ctx, e, "assign_out memset");
    }
    return BKV_OK;
  }
  if (!ctx->state_ready) return fail(ctx, BKV_ESTATE, "update before bkv_init_beacons / bkv_set_state");
  if (ctx->cfps) {
    if (assign_out) {  // nothing is assigned in this mode
      cudaError_t e =
          cudaMemsetAsync(assign_out, 0xff, sizeof(int32_t) * s.n_inst * s.G * static_cast<size_t>(n_new), ctx->stream);
      if (e != cudaSuccess) return cuda_fail(ctx, e, "assign_out memset");
    }
    bkv::CfpsArgs ca{};
    ca.mode = bkv::kCfpsUpdate;
    ca.H = ctx->n_heads;
    ca.b_min = ctx->b_min;
    ca.b_max = ctx->b_max;
    ca.q = static_cast<const __nv_bfloat16*>(q_new);
    ca.n_q = n_new;
    ca.buf = ctx->cbuf;
    ca.size = ctx->csize;
    ca.bcn = ctx->cent;
    ca.bcnt = ctx->counts;
    ca.err = ctx->err;
    ProfScope ps(ctx, BKV_K_CFPS);
    cudaError_t e = bkv::launch_cfps(s.d, ca, ctx->stream);
    return e == cudaSuccess ? BKV_OK : cuda_fail(ctx, e, "continual FPS update launch");
  }
  if (s.G * n_new <= bkv::kUpdateSmallMaxRows) {  // a decode step or a few: one warp per instance
    ProfScope ps(ctx, BKV_K_UPDATE);
    cudaError_t e = bkv::launch_update_small(s, static_cast<const __nv_bfloat16*>(q_new), n_new, ctx->cent, ctx->sums,
                                             ctx->counts, assign_out, ctx->stream);
    return e == cudaSuccess ? BKV_OK : cuda_fail(ctx, e, "update launch");
  }
  // a tile is at most 128 queries of one instance: boxes no taller than that
  const uint64_t q_rows = static_cast<uint64_t>(s.n_inst) * s.G * n_new;
  uint64_t box_rows = (static_cast<uint64_t>(s.G) * n_new + 7) / 8 * 8;
  if (box_rows > 128) box_rows = 128;
  if (box_rows > q_rows) box_rows = q_rows;
  CUtensorMap qmap;
  const int rc = encode_rows(ctx, &qmap, q_new, q_rows, s.d, static_cast<uint32_t>(box_rows));
  if (rc != BKV_OK) return rc;
  ProfScope ps(ctx, BKV_K_UPDATE);
  cudaError_t e = bkv::launch_update(s, qmap, static_cast<int>(box_rows), n_new, ctx->cent, ctx->sums, ctx->counts,
                                     assign_out, ctx->err, ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "update launch");
  return BKV_OK;
}

int bkv_update_beacons_seq(bkv_ctx* ctx, const void* q_steps, int32_t n_steps, int32_t* assign_out) {
  if (!ctx) return BKV_EINVAL;
  const Shape& s = ctx->shape;
  if (n_steps < 0) return fail(ctx, BKV_EINVAL, "n_steps must be >= 0");
  if (n_steps == 0) return BKV_OK;
  if (!q_steps || !aligned16(q_steps)) return fail(ctx, BKV_EINVAL, "q_steps must be a non-NULL 16-byte aligned pointer");
  if (assign_out && (reinterpret_cast<uintptr_t>(assign_out) & 3u))
    return fail(ctx, BKV_EINVAL, "assign_out must be 4-byte aligned");
  const size_t per_step = static_cast<size_t>(s.n_inst) * s.G;  // queries (and assignments) of one step
  if (1LL * s.n_inst * s.G * n_steps >= (1LL << 31)) return fail(ctx, BKV_EINVAL, "n_steps too large");
  if (s.nb > 0 && !ctx->state_ready) return fail(ctx, BKV_ESTATE, "update before bkv_init_beacons / bkv_set_state");
  if (s.nb > 0 && !ctx->cfps && s.G <= bkv::kUpdateSmallMaxRows) {
    ProfScope ps(ctx, BKV_K_UPDATE);
    cudaError_t e = bkv::launch_update_seq(s, static_cast<const __nv_bfloat16*>(q_steps), n_steps, ctx->cent,
                                           ctx->sums, ctx->counts, assign_out, ctx->stream);
    if (e == cudaSuccess) return BKV_OK;
    if (e != cudaErrorInvalidValue) return cuda_fail(ctx, e, "update launch");
    cudaGetLastError();  // the state does not fit in shared memory: step by step below
  }
  // step by step: no beacons, Continual FPS buffers, or more query heads per group than one warp takes
  const char* q = static_cast<const char*>(q_steps);
  for (int32_t t = 0; t < n_steps; ++t) {
    const int rc = bkv_update_beacons(ctx, q + t * per_step * s.d * 2, 1, assign_out ? assign_out + t * per_step : nullptr);
    if (rc != BKV_OK) return rc;
  }
  return BKV_OK;
}

int bkv_compress(bkv_ctx* ctx, void* K, void* V, int32_t L, int32_t budget, int64_t t_pos, const void* q_recent,
                 const int64_t* recent_pos, int32_t* kept_idx_out, float* scores_out) {
  if (!ctx) return BKV_EINVAL;
  const Shape& s = ctx->shape;
  if (!K || !V || !kept_idx_out) return fail(ctx, BKV_EINVAL, "K, V and kept_idx_out must be non-NULL");
  if (!aligned16(K) || !aligned16(V)) return fail(ctx, BKV_EINVAL, "K and V must be 16-byte aligned");
  if (reinterpret_cast<uintptr_t>(kept_idx_out) & 3u) return fail(ctx, BKV_EINVAL, "kept_idx_out must be 4-byte aligned");
  if (scores_out && (reinterpret_cast<uintptr_t>(scores_out) & 3u))
    return fail(ctx, BKV_EINVAL, "scores_out must be 4-byte aligned");
  if (L < 1 || L > s.cap) return fail(ctx, BKV_EINVAL, "L = %d must be in 1..capacity (%d)", L, s.cap);
  if (budget < s.n_prefix + s.W)
    return fail(ctx, BKV_EINVAL, "budget = %d is below n_prefix + window = %d", budget, s.n_prefix + s.W);
  if (budget < 1) return fail(ctx, BKV_EINVAL, "budget must be >= 1");
  if (1LL * s.n_inst * budget >= (1LL << 31)) return fail(ctx, BKV_EINVAL, "budget too large");
  cudaError_t e;
  if (L <= budget) {
    ProfScope ps(ctx, BKV_K_KEEP_ALL);
    e = bkv::launch_keep_all(s, L, budget, kept_idx_out, ctx->stream);
    return e == cudaSuccess ? BKV_OK : cuda_fail(ctx, e, "keep_all launch");
  }
  if (s.W > 0 && (!q_recent || !aligned16(q_recent) || !recent_pos))
    return fail(ctx, BKV_EINVAL, "q_recent (16-byte aligned) and recent_pos are required when window > 0");
  if (s.nb > 0 && !ctx->state_ready) return fail(ctx, BKV_ESTATE, "compress before bkv_init_beacons / bkv_set_state");

  // rotary table: slot w < W is recent_pos[w], slot W is t_pos
  const int h = s.d / 2;
  const double theta = ctx->cfg.rope_theta;
  const int rotate = theta != 0.0;
  if (rotate) {
    const size_t n = static_cast<size_t>(s.W + 1) * h;
    const int rs = ctx->rope_next;
    ctx->rope_next = (rs + 1) % bkv_ctx::kRopeSlots;
    if (ctx->rope_used[rs] && (e = cudaEventSynchronize(ctx->rope_ev[rs])) != cudaSuccess)
      return cuda_fail(ctx, e, "rope staging wait");
    double2* tab = ctx->rope_pinned[rs];
    float2* tab32 = reinterpret_cast<float2*>(tab + n);
    for (int slot = 0; slot <= s.W; ++slot) {
      const double pos = static_cast<double>(slot < s.W ? recent_pos[slot] : t_pos);
      for (int i = 0; i < h; ++i) {
        const double inv_freq = std::pow(theta, -static_cast<double>(2 * i) / static_cast<double>(s.d));
        const double ang = pos * inv_freq;
        const double c = std::cos(ang), sn = std::sin(ang);
        tab[static_cast<size_t>(slot) * h + i] = make_double2(c, sn);
        tab32[static_cast<size_t>(slot) * h + i] = make_float2(static_cast<float>(c), static_cast<float>(sn));
      }
    }
    {  // the slot is not refilled before this copy's event
      ProfScope ps(ctx, BKV_K_ROPE);
      e = bkv::launch_rope_stage(ctx->rope_mapped[rs], ctx->rope, sizeof(double2) * n + sizeof(float2) * n,
                                 ctx->stream);
    }
    if (e == cudaSuccess) e = cudaEventRecord(ctx->rope_ev[rs], ctx->stream);
    ctx->rope_used[rs] = true;
    if (e != cudaSuccess) return cuda_fail(ctx, e, "rope table upload");
  }
  bkv::CfpsArgs ca{};
  if (ctx->cfps) {  // this compress's beacons: FPS of each head's buffer, into cent / counts
    ca.H = ctx->n_heads;
    ca.b_min = ctx->b_min;
    ca.b_max = ctx->b_max;
    ca.buf = ctx->cbuf;
    ca.size = ctx->csize;
    ca.bcn = ctx->cent;
    ca.bcnt = ctx->counts;
    ca.err = ctx->err;
    ca.mode = bkv::kCfpsBeacons;
    ProfScope ps(ctx, BKV_K_CFPS);
    e = bkv::launch_cfps(s.d, ca, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "continual FPS beacon launch");
  }
  {
    ProfScope ps(ctx, BKV_K_QOBS);
    e = bkv::launch_qobs(s, static_cast<const __nv_bfloat16*>(q_recent), ctx->cent, ctx->counts, ctx->rope, rotate,
                         ctx->qobs, ctx->valid, ctx->err, ctx->stream);
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "qobs launch");

  CUtensorMap kmap, kmap32;
  int rc = encode_rows(ctx, &kmap, K, static_cast<uint64_t>(s.n_inst) * s.cap, s.d, 128);
  if (rc != BKV_OK) return rc;
  rc = encode_rows(ctx, &kmap32, K, static_cast<uint64_t>(s.n_inst) * s.cap, s.d, 32);
  if (rc != BKV_OK) return rc;
  bkv::ScoreArgs sa;
  sa.L = L;
  sa.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(s.d)));
  sa.valid = ctx->valid;
  sa.mean = (ctx->cfg.flags & BKV_F_MEAN_AGG) != 0;
  if (ctx->cfg.flags & BKV_F_CAUSAL_WINDOW) bkv::set_causal(sa, L, s.W, t_pos, recent_pos);
  sa.r_out = ctx->rscore;
  sa.err = ctx->err;
  // one launch per 64 scoring queries; later launches fold into the first's scores
  for (int col0 = 0; col0 < s.n_obs_pad; col0 += bkv::kScoreMaxCols) {
    CUtensorMap qmap;
    sa.col0 = col0;
    sa.n_cols = std::min(bkv::kScoreMaxCols, s.n_obs_pad - col0);
    sa.combine = col0 > 0;
    sa.scores_out = col0 + sa.n_cols == s.n_obs_pad ? scores_out : nullptr;
    rc = encode_rows(ctx, &qmap, ctx->qobs, static_cast<uint64_t>(s.n_inst) * s.n_obs_pad, s.d,
                     static_cast<uint32_t>(sa.n_cols));
    if (rc != BKV_OK) return rc;
    {
      ProfScope ps(ctx, BKV_K_SCORE);
      e = bkv::launch_score(s, kmap, kmap32, qmap, sa, ctx->stream);
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "score launch");
  }
  {
    ProfScope ps(ctx, BKV_K_SELECT_GATHER);
    e = bkv::launch_select_gather(s, ctx->rscore, L, budget, static_cast<__nv_bfloat16*>(K),
                                  static_cast<__nv_bfloat16*>(V), kept_idx_out, ctx->err, ctx->stream);
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "select_gather launch");
  if (ctx->cfps) {  // after the eviction: buffer = FPS of (beacons, then the window queries)
    ca.mode = bkv::kCfpsMerge;
    ca.q = static_cast<const __nv_bfloat16*>(q_recent);
    ca.n_q = s.W;
    ProfScope ps(ctx, BKV_K_CFPS);
    e = bkv::launch_cfps(s.d, ca, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "continual FPS merge launch");
  }
  return BKV_OK;
}

int bkv_compress_ragged(bkv_ctx* ctx, void* K, void* V, const int32_t* L, int32_t budget, const int64_t* t_pos,
                        const void* q_recent, const int64_t* recent_pos, int32_t* kept_idx_out, float* scores_out) {
  if (!ctx) return BKV_EINVAL;
  const Shape& s = ctx->shape;
  if (!K || !V || !kept_idx_out || !L) return fail(ctx, BKV_EINVAL, "K, V, L and kept_idx_out must be non-NULL");
  if (!aligned16(K) || !aligned16(V)) return fail(ctx, BKV_EINVAL, "K and V must be 16-byte aligned");
  if ((reinterpret_cast<uintptr_t>(kept_idx_out) | reinterpret_cast<uintptr_t>(L)) & 3u)
    return fail(ctx, BKV_EINVAL, "L and kept_idx_out must be 4-byte aligned");
  if (scores_out && (reinterpret_cast<uintptr_t>(scores_out) & 3u))
    return fail(ctx, BKV_EINVAL, "scores_out must be 4-byte aligned");
  if (budget < 1 || budget < s.n_prefix + s.W)
    return fail(ctx, BKV_EINVAL, "budget = %d must be >= max(1, n_prefix + window = %d)", budget, s.n_prefix + s.W);
  if (1LL * s.n_inst * budget >= (1LL << 31)) return fail(ctx, BKV_EINVAL, "budget too large");
  if (!t_pos) return fail(ctx, BKV_EINVAL, "t_pos (host, one per batch row) is required");
  if (s.W > 0 && (!q_recent || !aligned16(q_recent) || !recent_pos))
    return fail(ctx, BKV_EINVAL, "q_recent (16-byte aligned) and recent_pos are required when window > 0");
  if (s.nb > 0 && !ctx->state_ready) return fail(ctx, BKV_ESTATE, "compress before bkv_init_beacons / bkv_set_state");
  cudaError_t e;
  if (budget >= s.cap) {  // no instance can hold more rows than the budget: nothing is evicted anywhere
    ProfScope ps(ctx, BKV_K_KEEP_ALL);
    e = bkv::launch_ragged_plan(s, L, budget, ctx->work, ctx->n_work, kept_idx_out, ctx->err, ctx->stream);
    return e == cudaSuccess ? BKV_OK : cuda_fail(ctx, e, "ragged plan launch");
  }

  // per batch row: the rotary table (slot w < W at recent_pos[b][w], slot W at t_pos[b]), then the
  // causal gaps t_pos[b] - recent_pos[b][w], clamped to [0, capacity + 1]
  const int h = s.d / 2;
  const double theta = ctx->cfg.rope_theta;
  const int rotate = theta != 0.0;
  {
    const int rs = ctx->rag_next;
    ctx->rag_next = (rs + 1) % bkv_ctx::kRopeSlots;
    if (ctx->rag_used[rs] && (e = cudaEventSynchronize(ctx->rag_ev[rs])) != cudaSuccess)
      return cuda_fail(ctx, e, "ragged staging wait");
    unsigned char* host = static_cast<unsigned char*>(ctx->rag_pinned[rs]);
    const size_t n = static_cast<size_t>(s.W + 1) * h;
    for (int b = 0; b < s.batch; ++b) {
      double2* tab = reinterpret_cast<double2*>(host) + static_cast<size_t>(b) * ctx->rag_row;
      float2* tab32 = reinterpret_cast<float2*>(tab + n);
      for (int slot = 0; rotate && slot <= s.W; ++slot) {
        const double pos = static_cast<double>(slot < s.W ? recent_pos[static_cast<size_t>(b) * s.W + slot] : t_pos[b]);
        for (int i = 0; i < h; ++i) {
          const double inv_freq = std::pow(theta, -static_cast<double>(2 * i) / static_cast<double>(s.d));
          const double ang = pos * inv_freq;
          const double c = std::cos(ang), sn = std::sin(ang);
          tab[static_cast<size_t>(slot) * h + i] = make_double2(c, sn);
          tab32[static_cast<size_t>(slot) * h + i] = make_float2(static_cast<float>(c), static_cast<float>(sn));
        }
      }
      int32_t* gaps = reinterpret_cast<int32_t*>(host + ctx->rag_gaps_off) + static_cast<size_t>(b) * s.W;
      for (int w = 0; w < s.W; ++w) {
        const int64_t rp = recent_pos[static_cast<size_t>(b) * s.W + w];
        const int64_t g = rp >= t_pos[b] ? 0 : static_cast<int64_t>(static_cast<uint64_t>(t_pos[b]) - static_cast<uint64_t>(rp));
        gaps[w] = static_cast<int32_t>(g > s.cap + 1LL || g < 0 ? s.cap + 1LL : g);
      }
    }
    {
      ProfScope ps(ctx, BKV_K_ROPE);
      e = bkv::launch_rope_stage(ctx->rag_mapped[rs], ctx->rag, ctx->rag_bytes, ctx->stream);
    }
    if (e == cudaSuccess) e = cudaEventRecord(ctx->rag_ev[rs], ctx->stream);
    ctx->rag_used[rs] = true;
    if (e != cudaSuccess) return cuda_fail(ctx, e, "ragged table upload");
  }
  {
    ProfScope ps(ctx, BKV_K_KEEP_ALL);
    e = bkv::launch_ragged_plan(s, L, budget, ctx->work, ctx->n_work, kept_idx_out, ctx->err, ctx->stream);
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "ragged plan launch");
  bkv::CfpsArgs ca{};
  if (ctx->cfps) {  // this compress's beacons: FPS of each head's buffer, into cent / counts
    ca.H = ctx->n_heads;
    ca.b_min = ctx->b_min;
    ca.b_max = ctx->b_max;
    ca.buf = ctx->cbuf;
    ca.size = ctx->csize;
    ca.bcn = ctx->cent;
    ca.bcnt = ctx->counts;
    ca.err = ctx->err;
    ca.mode = bkv::kCfpsBeacons;
    ProfScope ps(ctx, BKV_K_CFPS);
    e = bkv::launch_cfps(s.d, ca, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "continual FPS beacon launch");
  }
  const double2* rope_rows = reinterpret_cast<const double2*>(ctx->rag);
  {
    ProfScope ps(ctx, BKV_K_QOBS);
    e = bkv::launch_qobs_ragged(s, static_cast<const __nv_bfloat16*>(q_recent), ctx->cent, ctx->counts, rope_rows,
                                ctx->rag_row, rotate, ctx->work, ctx->n_work, ctx->qobs, ctx->valid, ctx->err,
                                ctx->stream);
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "qobs launch");

  CUtensorMap kmap, kmap32;
  int rc = encode_rows(ctx, &kmap, K, static_cast<uint64_t>(s.n_inst) * s.cap, s.d, 128);
  if (rc != BKV_OK) return rc;
  rc = encode_rows(ctx, &kmap32, K, static_cast<uint64_t>(s.n_inst) * s.cap, s.d, 32);
  if (rc != BKV_OK) return rc;
  bkv::ScoreArgs sa;
  sa.L = s.cap;  // the plan is made for the longest possible cache
  sa.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(s.d)));
  sa.valid = ctx->valid;
  sa.mean = (ctx->cfg.flags & BKV_F_MEAN_AGG) != 0;
  sa.causal = (ctx->cfg.flags & BKV_F_CAUSAL_WINDOW) != 0 && s.W > 0;
  sa.r_out = ctx->rscore;
  sa.err = ctx->err;
  sa.Ls = L;
  sa.work = ctx->work;
  sa.n_work = ctx->n_work;
  sa.gaps = sa.causal ? reinterpret_cast<const int*>(ctx->rag + ctx->rag_gaps_off) : nullptr;
  for (int col0 = 0; col0 < s.n_obs_pad; col0 += bkv::kScoreMaxCols) {
    CUtensorMap qmap;
    sa.col0 = col0;
    sa.n_cols = std::min(bkv::kScoreMaxCols, s.n_obs_pad - col0);
    sa.combine = col0 > 0;
    sa.scores_out = col0 + sa.n_cols == s.n_obs_pad ? scores_out : nullptr;
    rc = encode_rows(ctx, &qmap, ctx->qobs, static_cast<uint64_t>(s.n_inst) * s.n_obs_pad, s.d,
                     static_cast<uint32_t>(sa.n_cols));
    if (rc != BKV_OK) return rc;
    {
      ProfScope ps(ctx, BKV_K_SCORE);
      e = bkv::launch_score(s, kmap, kmap32, qmap, sa, ctx->stream);
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "score launch");
  }
  {
    ProfScope ps(ctx, BKV_K_SELECT_GATHER);
    e = bkv::launch_select_gather_ragged(s, ctx->rscore, L, ctx->work, ctx->n_work, budget,
                                         static_cast<__nv_bfloat16*>(K), static_cast<__nv_bfloat16*>(V), kept_idx_out,
                                         ctx->err, ctx->stream);
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "select_gather launch");
  if (ctx->cfps) {  // after the eviction, in the instances evicted from: buffer = FPS of (beacons, window)
    ca.mode = bkv::kCfpsMerge;
    ca.q = static_cast<const __nv_bfloat16*>(q_recent);
    ca.n_q = s.W;
    ca.Ls = L;
    ca.budget = budget;
    ca.cap = s.cap;
    ca.group = s.G;
    ProfScope ps(ctx, BKV_K_CFPS);
    e = bkv::launch_cfps(s.d, ca, ctx->stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "continual FPS merge launch");
  }
  return BKV_OK;
}

int bkv_get_state(bkv_ctx* ctx, float* centroids, double* sums, int64_t* counts) {
  if (!ctx) return BKV_EINVAL;
  if (ctx->cfps) return fail(ctx, BKV_EINVAL, "a continual FPS context has no centroid state");
  const Shape& s = ctx->shape;
  const size_t n = static_cast<size_t>(s.n_inst) * s.nb;
  cudaError_t e = cudaSuccess;
  if (centroids && (e = cudaMemcpyAsync(centroids, ctx->cent, sizeof(float) * n * s.d, cudaMemcpyDefault,
                                        ctx->stream)) != cudaSuccess)
    return cuda_fail(ctx, e, "get_state centroids");
  if (sums && (e = cudaMemcpyAsync(sums, ctx->sums, sizeof(double) * n * s.d, cudaMemcpyDefault,
                                   ctx->stream)) != cudaSuccess)
    return cuda_fail(ctx, e, "get_state sums");
  if (counts && (e = cudaMemcpyAsync(counts, ctx->counts, sizeof(int64_t) * n, cudaMemcpyDefault,
                                     ctx->stream)) != cudaSuccess)
    return cuda_fail(ctx, e, "get_state counts");
  return BKV_OK;
}

int bkv_set_state(bkv_ctx* ctx, const float* centroids, const double* sums, const int64_t* counts) {
  if (!ctx) return BKV_EINVAL;
  if (ctx->cfps) return fail(ctx, BKV_EINVAL, "a continual FPS context has no centroid state");
  const Shape& s = ctx->shape;
  if (!centroids || !sums || !counts) return fail(ctx, BKV_EINVAL, "set_state needs all three arrays");
  const size_t n = static_cast<size_t>(s.n_inst) * s.nb;
  cudaError_t e;
  if ((e = cudaMemcpyAsync(ctx->cent, centroids, sizeof(float) * n * s.d, cudaMemcpyDefault, ctx->stream)) !=
          cudaSuccess ||
      (e = cudaMemcpyAsync(ctx->sums, sums, sizeof(double) * n * s.d, cudaMemcpyDefault, ctx->stream)) !=
          cudaSuccess ||
      (e = cudaMemcpyAsync(ctx->counts, counts, sizeof(int64_t) * n, cudaMemcpyDefault, ctx->stream)) !=
          cudaSuccess)
    return cuda_fail(ctx, e, "set_state copy");
  ctx->state_ready = true;
  return BKV_OK;
}

int bkv_get_cfps_state(bkv_ctx* ctx, void* buffers, int32_t* sizes) {
  if (!ctx) return BKV_EINVAL;
  if (!ctx->cfps) return fail(ctx, BKV_EINVAL, "not a continual FPS context");
  const size_t nh = static_cast<size_t>(ctx->n_heads);
  cudaError_t e = cudaSuccess;
  if (buffers && (e = cudaMemcpyAsync(buffers, ctx->cbuf, sizeof(__nv_bfloat16) * nh * ctx->b_max * ctx->shape.d,
                                      cudaMemcpyDefault, ctx->stream)) != cudaSuccess)
    return cuda_fail(ctx, e, "get_cfps_state buffers");
  if (sizes && (e = cudaMemcpyAsync(sizes, ctx->csize, sizeof(int32_t) * nh, cudaMemcpyDefault, ctx->stream)) !=
                   cudaSuccess)
    return cuda_fail(ctx, e, "get_cfps_state sizes");
  return BKV_OK;
}

int bkv_set_cfps_state(bkv_ctx* ctx, const void* buffers, const int32_t* sizes) {
  if (!ctx) return BKV_EINVAL;
  if (!ctx->cfps) return fail(ctx, BKV_EINVAL, "not a continual FPS context");
  if (!buffers || !sizes) return fail(ctx, BKV_EINVAL, "set_cfps_state needs buffers and sizes");
  const size_t nh = static_cast<size_t>(ctx->n_heads);
  cudaError_t e;
  if ((e = cudaMemcpyAsync(ctx->cbuf, buffers, sizeof(__nv_bfloat16) * nh * ctx->b_max * ctx->shape.d,
                           cudaMemcpyDefault, ctx->stream)) != cudaSuccess ||
      (e = cudaMemcpyAsync(ctx->csize, sizes, sizeof(int32_t) * nh, cudaMemcpyDefault, ctx->stream)) !=
          cudaSuccess)
    return cuda_fail(ctx, e, "set_cfps_state");
  ctx->state_ready = true;
  return BKV_OK;
}

int bkv_profile_enable(bkv_ctx* ctx, int on) {
  if (!ctx) return BKV_EINVAL;
  ctx->prof = on != 0;
  return BKV_OK;
}

int bkv_profile_read(bkv_ctx* ctx, double* ms, int64_t* launches, int32_t n_kernels) {
  if (!ctx || n_kernels < 0) return BKV_EINVAL;
  cudaError_t e = cudaStreamSynchronize(ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "stream synchronize");
  fold_profile(ctx);
  for (int k = 0; k < BKV_NUM_KERNELS && k < n_kernels; ++k) {
    if (ms) ms[k] = ctx->prof_ms[k];
    if (launches) launches[k] = ctx->prof_n[k];
  }
  for (int k = 0; k < BKV_NUM_KERNELS; ++k) {
    ctx->prof_ms[k] = 0.0;
    ctx->prof_n[k] = 0;
  }
  return BKV_OK;
}

int bkv_selftest_wait_timeout(bkv_ctx* ctx, int64_t limit_ns) {
  if (!ctx) return BKV_EINVAL;
  if (limit_ns < 1000 || limit_ns > 10000000000LL) return fail(ctx, BKV_EINVAL, "limit_ns must be in 1e3..1e10");
  int rc = bkv_sync(ctx);  // report earlier work first
  if (rc != BKV_OK) return rc;
  cudaError_t e = bkv::launch_selftest_wait(ctx->err, static_cast<unsigned long long>(limit_ns), ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "selftest launch");
  return bkv_sync(ctx);
}

int bkv_selftest_bounds(bkv_ctx* ctx) {
  if (!ctx) return BKV_EINVAL;
  int rc = bkv_sync(ctx);  // report earlier work first
  if (rc != BKV_OK) return rc;
  cudaError_t e = bkv::launch_selftest_bounds(ctx->err, ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "selftest launch");
  return bkv_sync(ctx);
}

int bkv_checked_build(void) {
#ifdef BKV_CHECKED
  return 1;
#else
  return 0;
#endif
}

int bkv_sync(bkv_ctx* ctx) {
  if (!ctx) return BKV_EINVAL;
  cudaError_t e = cudaStreamSynchronize(ctx->stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "stream synchronize");
  int h = 0;
  if ((e = cudaMemcpy(&h, ctx->err, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(ctx, e, "error word read");
  if (h != 0) {
    cudaMemset(ctx->err, 0, sizeof(int));
    if (h == bkv::kDevBadLength)
      return fail(ctx, BKV_EINVAL, "a per-instance cache length was outside 1..capacity; that instance was left untouched");
    if (h == bkv::kDevBounds)
      return fail(ctx, BKV_EBOUNDS, "a device-side bounds check failed; the access was skipped and the outputs are invalid");
    return fail(ctx, BKV_ETIMEOUT, "device wait expired (code %d)", h);
  }
  return BKV_OK;
}

}  // extern "C"
