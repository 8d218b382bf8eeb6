// bkv_compress_static: the compression step without any device allocation.
//
// Some callers cannot call cudaMalloc: a serving engine that has handed all
// of HBM to its own paged KV-cache allocator and forbids allocations behind
// its back, or a plugin hosted by a framework that owns every allocation on
// the device.  cudaMalloc can also synchronise the device, which a decode
// loop on a latency budget may not afford.  For them this entry point runs the
// same kernels as bkv_compress, but its scratch (observation queries, their
// valid mask, the per-key scores and the rotary table) lives in one
// file-scope device array of fixed size, and the beacon state comes from the
// caller instead of a context.  No device memory is allocated or freed here.
//
// Shared-array rules:
//   * the array holds kStaticScratchBytes (16 MiB) and stays resident on
//     every device that loads this library until the process exits;
//   * every call uses the same array and it keeps the previous call's
//     contents; nothing in it needs to start at zero (each call writes every
//     byte it later reads), only the caller's status word is cleared per call;
//   * two calls whose work overlaps on the GPU (different streams, or the
//     same device from two threads without ordering) race on the array and
//     produce undefined results; calls on one stream are ordered and safe;
//   * the device address of the array is looked up with cudaGetSymbolAddress
//     the first time this entry point runs on a device (with that device
//     current), so that first call should come before any stream capture.
//
// The rotary table of a call (at most 65 positions x 64 frequency pairs, in
// fp64 and fp32) reaches the device as by-value kernel parameters, in chunks
// of 16 KB that a small kernel writes into the array: no copy from pageable
// host memory, so the call never waits for the stream.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>


#include "bkv.h"
#include "bkv_internal.h"

namespace {

constexpr size_t kStaticScratchBytes = 16u << 20;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_static_scratch on the current device (set up once per device).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

void message(char* buf, size_t len, const char* text) {
  if (buf && len) {
    std::strncpy(buf, text, len - 1);
    buf[len - 1] = '\0';
  }
}

bool encode(CUtensorMap* map, const void* base, uint64_t rows, int d, uint32_t box_rows) {
  return bkv::encode_rows_bf16(map, base, rows, d, box_rows) == CUDA_SUCCESS;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

// One chunk of the rotary table, passed by value: 16-byte units [first, first + count).
constexpr int kRopeChunkUnits = 1024;
struct RopeChunk {
  uint32_t first, count;
  uint4 unit[kRopeChunkUnits];
};

__global__ void __launch_bounds__(256) rope_param_kernel(const __grid_constant__ RopeChunk c, uint4* table) {
  for (uint32_t i = threadIdx.x; i < c.count; i += blockDim.x) table[c.first + i] = c.unit[i];
}

// 16-byte unit u of the table laid out as bkv_compress lays it out: units [0, n) are the fp64
// (cos, sin) entries, units [n, 3n/2) two fp32 (cos, sin) entries each (n is even: d/2 is 32 or 64).
// Entry k is slot k / h (recent slot w < W at recent_pos[w], slot W at t_pos), frequency k % h.
struct RopeTable {
  double theta;
  int d, h, W;
  int64_t t_pos;
  const int64_t* recent_pos;
  size_t n;
  void entry(size_t k, double& c, double& s) const {
    const int slot = static_cast<int>(k / h), i = static_cast<int>(k % h);
    const double pos = static_cast<double>(slot < W ? recent_pos[slot] : t_pos);
    const double inv_freq = std::pow(theta, -static_cast<double>(2 * i) / static_cast<double>(d));
    const double ang = pos * inv_freq;
    c = std::cos(ang);
    s = std::sin(ang);
  }
  uint4 unit(size_t u) const {
    uint4 out;
    double c, s;
    if (u < n) {
      entry(u, c, s);
      const double2 v = make_double2(c, s);
      std::memcpy(&out, &v, sizeof out);
    } else {
      float2 v[2];
      for (int j = 0; j < 2; ++j) {
        entry(2 * (u - n) + j, c, s);
        v[j] = make_float2(static_cast<float>(c), static_cast<float>(s));
      }
      std::memcpy(&out, v, sizeof out);
    }
    return out;
  }
};

}  // namespace

extern "C" int bkv_compress_static(const bkv_config* cfg, const float* centroids, const int64_t* counts, void* K,
                                   void* V, int32_t L, int32_t budget, int64_t t_pos, const void* q_recent,
                                   const int64_t* recent_pos, int32_t* kept_idx_out, float* scores_out,
                                   int32_t* dev_status, void* stream, char* err_msg, size_t err_len) {
  message(err_msg, err_len, "");
  auto bad = [&](const char* why) {
    message(err_msg, err_len, why);
    return BKV_EINVAL;
  };
  // ---- configuration (same limits as bkv_create)
  if (!cfg) return bad("cfg is NULL");
  if (cfg->n_layers < 1 || cfg->batch < 1 || cfg->n_q_heads < 1 || cfg->n_kv_heads < 1 ||
      cfg->n_q_heads % cfg->n_kv_heads != 0)
    return bad("bad head / batch / layer counts");
  if (cfg->head_dim != 64 && cfg->head_dim != 128) return bad("head_dim must be 64 or 128");
  if (cfg->n_beacons < 0 || cfg->n_beacons > bkv::kMaxBeacons) return bad("n_beacons must be in 0..32");
  if (cfg->window < 0 || cfg->window > bkv::kMaxWindow) return bad("window must be in 0..64");
  if (cfg->n_prefix < 0) return bad("n_prefix must be >= 0");
  if (cfg->flags & ~(BKV_F_MEAN_AGG | BKV_F_CAUSAL_WINDOW)) return bad("flags holds an unknown option");
  if (cfg->capacity < 1 || cfg->capacity > bkv::kMaxCapacity) return bad("capacity must be in 1..32768");
  if (!(cfg->rope_theta >= 0.0) || !std::isfinite(cfg->rope_theta)) return bad("rope_theta must be finite, >= 0");
  bkv::Shape s{};
  s.G = cfg->n_q_heads / cfg->n_kv_heads;
  s.n_inst = cfg->n_layers * cfg->batch * cfg->n_kv_heads;
  s.d = cfg->head_dim;
  s.nb = cfg->n_beacons;
  s.W = cfg->window;
  s.n_prefix = cfg->n_prefix;
  s.cap = cfg->capacity;
  s.n_obs = s.G * s.W + s.nb;
  s.n_obs_pad = (s.n_obs + 15) / 16 * 16;
  s.batch = cfg->batch;
  s.n_kv = cfg->n_kv_heads;
  if (s.n_obs < 1 || s.n_obs > bkv::kMaxObs) return bad("G * window + n_beacons must be in 1..128");

  // ---- call arguments (same rules as bkv_compress)
  if (!K || !V || !kept_idx_out) return bad("K, V and kept_idx_out must be non-NULL");
  if (!aligned(K, 16) || !aligned(V, 16) || !aligned(kept_idx_out, 4) || (scores_out && !aligned(scores_out, 4)) ||
      (dev_status && !aligned(dev_status, 4)))
    return bad("K and V must be 16-byte aligned, kept_idx_out / scores_out / dev_status 4-byte aligned");
  if (L < 1 || L > s.cap) return bad("L must be in 1..capacity");
  if (budget < 1 || budget < s.n_prefix + s.W) return bad("budget must be >= max(1, n_prefix + window)");
  if (1LL * s.n_inst * budget >= (1LL << 31) || 1LL * s.n_inst * s.cap >= (1LL << 31)) return bad("too many rows");

  // ---- fixed scratch budget
  const size_t off_qobs = 0;
  const size_t off_valid = off_qobs + align256(sizeof(__nv_bfloat16) * s.n_inst * s.n_obs_pad * s.d);
  const size_t off_score = off_valid + align256(sizeof(uint32_t) * 4 * s.n_inst);
  const size_t off_rope = off_score + align256(sizeof(float) * static_cast<size_t>(s.n_inst) * s.cap);
  const size_t need = off_rope + align256((sizeof(double2) + sizeof(float2)) * static_cast<size_t>(s.W + 1) * (s.d / 2));
  if (need > kStaticScratchBytes) {
    char buf[160];
    std::snprintf(buf, sizeof buf, "needs %zu bytes of scratch; the static scratch holds %zu", need,
                  kStaticScratchBytes);
    return bad(buf);
  }

  // the scoring inputs matter only when rows are evicted; checked before anything is enqueued
  if (L > budget && s.W > 0 && (!q_recent || !aligned(q_recent, 16) || !recent_pos))
    return bad("q_recent (16-byte aligned) and recent_pos are required when window > 0");
  if (L > budget && s.nb > 0 && (!centroids || !counts || !aligned(centroids, 4) || !aligned(counts, 8)))
    return bad("centroids and counts are required when n_beacons > 0");

  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  // the set-up of this device (the array's address) happens on its first call, whatever that call keeps
  void* base = nullptr;
  if ((e = scratch_address(&base)) != cudaSuccess) {
    message(err_msg, err_len, cudaGetErrorString(e));
    return BKV_ECUDA;
  }
  if (dev_status && (e = cudaMemsetAsync(dev_status, 0, sizeof(int32_t), st)) != cudaSuccess) {
    message(err_msg, err_len, cudaGetErrorString(e));
    return BKV_ECUDA;
  }
  if (L <= budget) {
    e = bkv::launch_keep_all(s, L, budget, kept_idx_out, st);
    if (e != cudaSuccess) message(err_msg, err_len, cudaGetErrorString(e));
    return e == cudaSuccess ? BKV_OK : BKV_ECUDA;
  }

  unsigned char* b = static_cast<unsigned char*>(base);
  auto* qobs = reinterpret_cast<__nv_bfloat16*>(b + off_qobs);
  auto* valid = reinterpret_cast<uint32_t*>(b + off_valid);
  auto* rscore = reinterpret_cast<float*>(b + off_score);
  auto* rope = reinterpret_cast<double2*>(b + off_rope);

  const int h = s.d / 2;
  const double theta = cfg->rope_theta;
  const int rotate = theta != 0.0;
  if (rotate) {
    // fp64 (cos, sin) entries followed by the same entries in fp32, as kernel parameters
    const RopeTable tab{theta, s.d, h, s.W, t_pos, recent_pos, static_cast<size_t>(s.W + 1) * h};
    const size_t units = tab.n + tab.n / 2;
    RopeChunk chunk;
    for (size_t u0 = 0; u0 < units; u0 += kRopeChunkUnits) {
      chunk.first = static_cast<uint32_t>(u0);
      chunk.count = static_cast<uint32_t>(std::min<size_t>(kRopeChunkUnits, units - u0));
      for (uint32_t i = 0; i < chunk.count; ++i) chunk.unit[i] = tab.unit(u0 + i);
      rope_param_kernel<<<1, 256, 0, st>>>(chunk, reinterpret_cast<uint4*>(rope));
      if ((e = cudaGetLastError()) != cudaSuccess) {
        message(err_msg, err_len, cudaGetErrorString(e));
        return BKV_ECUDA;
      }
    }
  }
  e = bkv::launch_qobs(s, static_cast<const __nv_bfloat16*>(q_recent), centroids,
                       reinterpret_cast<const long long*>(counts), rope, rotate, qobs, valid,
                       reinterpret_cast<int*>(dev_status), st);
  CUtensorMap kmap, kmap32;
  if (e == cudaSuccess && (!encode(&kmap, K, static_cast<uint64_t>(s.n_inst) * s.cap, s.d, 128) ||
                           !encode(&kmap32, K, static_cast<uint64_t>(s.n_inst) * s.cap, s.d, 32))) {
    message(err_msg, err_len, "cuTensorMapEncodeTiled failed");
    return BKV_ECUDA;
  }
  if (e == cudaSuccess) {
    bkv::ScoreArgs sa;
    sa.L = L;
    sa.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(s.d)));
    sa.valid = valid;
    sa.mean = (cfg->flags & BKV_F_MEAN_AGG) != 0;
    if (cfg->flags & BKV_F_CAUSAL_WINDOW) bkv::set_causal(sa, L, s.W, t_pos, recent_pos);
    sa.r_out = rscore;
    sa.err = reinterpret_cast<int*>(dev_status);
    // one launch per 64 scoring queries; later launches fold into the first's scores
    for (int col0 = 0; e == cudaSuccess && col0 < s.n_obs_pad; col0 += bkv::kScoreMaxCols) {
      CUtensorMap qmap;
      sa.col0 = col0;
      sa.n_cols = std::min(bkv::kScoreMaxCols, s.n_obs_pad - col0);
      sa.combine = col0 > 0;
      sa.scores_out = col0 + sa.n_cols == s.n_obs_pad ? scores_out : nullptr;
      if (!encode(&qmap, qobs, static_cast<uint64_t>(s.n_inst) * s.n_obs_pad, s.d, static_cast<uint32_t>(sa.n_cols))) {
        message(err_msg, err_len, "cuTensorMapEncodeTiled failed");
        return BKV_ECUDA;
      }
      e = bkv::launch_score(s, kmap, kmap32, qmap, sa, st);
    }
  }
  if (e == cudaSuccess)
    e = bkv::launch_select_gather(s, rscore, L, budget, static_cast<__nv_bfloat16*>(K),
                                  static_cast<__nv_bfloat16*>(V), kept_idx_out, reinterpret_cast<int*>(dev_status), st);
  if (e != cudaSuccess) {
    message(err_msg, err_len, cudaGetErrorString(e));
    return BKV_ECUDA;
  }
  return BKV_OK;
}
