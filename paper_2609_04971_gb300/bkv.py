"""Python binding of the C ABI in include/bkv.h (argument marshalling only).

Each ``bkv_*`` function has the C function's name and meaning; tensors are
torch tensors whose device pointers are handed to the library, and the CUDA
stream defaults to torch's current stream.  Nothing here computes: every step
of the method runs in libbkv.so, and this module raises if the library cannot
be loaded (there is no other implementation to fall back on).
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import _build

BKV_OK = 0
BKV_EINVAL = -1
BKV_ENOMEM = -2
BKV_ECUDA = -3
BKV_ETIMEOUT = -4
BKV_ESTATE = -5
BKV_EBOUNDS = -6

KERNEL_NAMES = ("fps_init", "update", "qobs", "score", "select_gather", "keep_all", "cfps", "rope_stage")


# bkv_config.flags options (include/bkv.h)
BKV_F_NONE = 0
BKV_F_MEAN_AGG = 1
BKV_F_CONTINUAL_FPS = 2
BKV_F_CAUSAL_WINDOW = 4


class BkvConfig(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int32), ("batch", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("n_beacons", ctypes.c_int32),
        ("window", ctypes.c_int32), ("n_prefix", ctypes.c_int32), ("capacity", ctypes.c_int32),
        ("rope_theta", ctypes.c_double), ("flags", ctypes.c_uint32),
    ]


class BkvError(RuntimeError):
    def __init__(self, code: int, where: str, detail: str = ""):
        self.code = code
        super().__init__(f"{where}: {bkv_strerror(code)} ({code})" + (f": {detail}" if detail else ""))


_lib = None
_lock = threading.Lock()
_P = ctypes.c_void_p


def load_library(path: str | None = None, build: bool = True):
    """Load libbkv.so (building it in-tree first if it is missing or stale).  With the environment
    variable BKV_CHECKED=1 the process uses the bounds-checked flavour libbkv_checked.so instead."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        checked = os.environ.get("BKV_CHECKED") == "1"
        default = _build.LIB_PATH_CHECKED if checked else _build.LIB_PATH
        p = path or (_build.build(checked=checked) if build else default)
        if not os.path.exists(p):
            raise RuntimeError(f"libbkv.so not found at {p}; run __graft_entry__.build()")
        lib = ctypes.CDLL(p)
        sig = {
            "bkv_create": (ctypes.c_int, [ctypes.POINTER(BkvConfig), _P, ctypes.POINTER(_P)]),
            "bkv_destroy": (None, [_P]),
            "bkv_set_stream": (ctypes.c_int, [_P, _P]),
            "bkv_init_beacons": (ctypes.c_int, [_P, _P, ctypes.c_int32]),
            "bkv_update_beacons": (ctypes.c_int, [_P, _P, ctypes.c_int32, _P]),
            "bkv_update_beacons_seq": (ctypes.c_int, [_P, _P, ctypes.c_int32, _P]),
            "bkv_compress": (ctypes.c_int, [_P, _P, _P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, _P, _P,
                                            _P, _P]),
            "bkv_compress_ragged": (ctypes.c_int, [_P, _P, _P, _P, ctypes.c_int32, _P, _P, _P, _P, _P]),
            "bkv_get_state": (ctypes.c_int, [_P, _P, _P, _P]),
            "bkv_set_state": (ctypes.c_int, [_P, _P, _P, _P]),
            "bkv_get_cfps_state": (ctypes.c_int, [_P, _P, _P]),
            "bkv_set_cfps_state": (ctypes.c_int, [_P, _P, _P]),
            "bkv_sync": (ctypes.c_int, [_P]),
            "bkv_selftest_wait_timeout": (ctypes.c_int, [_P, ctypes.c_int64]),
            "bkv_selftest_bounds": (ctypes.c_int, [_P]),
            "bkv_checked_build": (ctypes.c_int, []),
            "bkv_debug_fail_alloc": (ctypes.c_int, [ctypes.c_int32]),
            "bkv_compress_static": (ctypes.c_int, [ctypes.POINTER(BkvConfig), _P, _P, _P, _P, ctypes.c_int32,
                                                   ctypes.c_int32, ctypes.c_int64, _P, _P, _P, _P, _P, _P,
                                                   ctypes.c_char_p, ctypes.c_size_t]),
            "bkv_profile_enable": (ctypes.c_int, [_P, ctypes.c_int]),
            "bkv_profile_read": (ctypes.c_int, [_P, _P, _P, ctypes.c_int32]),
            "bkv_strerror": (ctypes.c_char_p, [ctypes.c_int]),
            "bkv_last_error": (ctypes.c_char_p, [_P]),
            "bkv_version": (ctypes.c_char_p, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        if path is None:
            _lib = lib
        return lib


def _l():
    return _lib if _lib is not None else load_library()


def _ptr(t: torch.Tensor | None, dtype: torch.dtype, name: str, device=None):
    if t is None:
        return None
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _ptr_any(t: torch.Tensor | None, dtype: torch.dtype, name: str):
    """Pointer of a CUDA or host tensor (the state copies take their direction from the pointer)."""
    if t is None:
        return None
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        if not torch.cuda.is_available():
            return ctypes.c_void_p(0)
        stream = torch.cuda.current_stream()
    handle = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
    return ctypes.c_void_p(handle)


def _expect(t: torch.Tensor | None, n: int, name: str) -> None:
    """The C ABI receives bare pointers and trusts the sizes that the shape implies: a tensor of the
    wrong element count is a ValueError here instead of an out-of-bounds access on the device."""
    if t is not None and t.numel() != n:
        raise ValueError(f"{name} has {t.numel()} elements; the configured shape needs {n}")


def _check(rc: int, where: str, ctx=None) -> None:
    if rc != BKV_OK:
        detail = _l().bkv_last_error(ctx).decode() if ctx is not None else ""
        raise BkvError(rc, where, detail)


# ---------------------------------------------------------------- C-ABI mirror
def bkv_version() -> str:
    return _l().bkv_version().decode()


def bkv_strerror(code: int) -> str:
    return _l().bkv_strerror(int(code)).decode()


def bkv_last_error(ctx) -> str:
    return _l().bkv_last_error(ctx).decode()


def bkv_create(cfg: BkvConfig, stream=None) -> ctypes.c_void_p:
    out = ctypes.c_void_p()
    _check(_l().bkv_create(ctypes.byref(cfg), _stream(stream), ctypes.byref(out)), "bkv_create")
    return out


def bkv_destroy(ctx) -> None:
    if ctx:
        _l().bkv_destroy(ctx)


def bkv_set_stream(ctx, stream=None) -> None:
    _check(_l().bkv_set_stream(ctx, _stream(stream)), "bkv_set_stream", ctx)


def bkv_init_beacons(ctx, q_init: torch.Tensor, n_init: int) -> None:
    _check(_l().bkv_init_beacons(ctx, _ptr(q_init, torch.bfloat16, "q_init"), int(n_init)), "bkv_init_beacons", ctx)


def bkv_update_beacons(ctx, q_new: torch.Tensor, n_new: int, assign_out: torch.Tensor | None = None) -> None:
    _check(_l().bkv_update_beacons(ctx, _ptr(q_new, torch.bfloat16, "q_new"), int(n_new),
                                   _ptr(assign_out, torch.int32, "assign_out")), "bkv_update_beacons", ctx)


def bkv_update_beacons_seq(ctx, q_steps: torch.Tensor, n_steps: int, assign_out: torch.Tensor | None = None) -> None:
    _check(_l().bkv_update_beacons_seq(ctx, _ptr(q_steps, torch.bfloat16, "q_steps"), int(n_steps),
                                       _ptr(assign_out, torch.int32, "assign_out")), "bkv_update_beacons_seq", ctx)


def bkv_compress(ctx, K: torch.Tensor, V: torch.Tensor, L: int, budget: int, t_pos: int,
                 q_recent: torch.Tensor | None, recent_pos, kept_idx_out: torch.Tensor,
                 scores_out: torch.Tensor | None = None) -> None:
    pos = (ctypes.c_int64 * max(1, len(recent_pos)))(*[int(p) for p in recent_pos])
    _check(_l().bkv_compress(ctx, _ptr(K, torch.bfloat16, "K"), _ptr(V, torch.bfloat16, "V"), int(L), int(budget),
                             int(t_pos), _ptr(q_recent, torch.bfloat16, "q_recent"), ctypes.cast(pos, _P),
                             _ptr(kept_idx_out, torch.int32, "kept_idx_out"),
                             _ptr(scores_out, torch.float32, "scores_out")), "bkv_compress", ctx)


def bkv_compress_ragged(ctx, K: torch.Tensor, V: torch.Tensor, L: torch.Tensor, budget: int, t_pos, q_recent,
                        recent_pos, kept_idx_out: torch.Tensor, scores_out: torch.Tensor | None = None) -> None:
    """L: int32 device tensor, one cache length per instance; t_pos: one position per batch row;
    recent_pos: one list of window positions per batch row (see include/bkv.h)."""
    tp = (ctypes.c_int64 * max(1, len(t_pos)))(*[int(p) for p in t_pos])
    flat = [int(p) for row in recent_pos for p in row]
    rp = (ctypes.c_int64 * max(1, len(flat)))(*flat)
    _check(_l().bkv_compress_ragged(ctx, _ptr(K, torch.bfloat16, "K"), _ptr(V, torch.bfloat16, "V"),
                                    _ptr(L, torch.int32, "L"), int(budget), ctypes.cast(tp, _P),
                                    _ptr(q_recent, torch.bfloat16, "q_recent"), ctypes.cast(rp, _P),
                                    _ptr(kept_idx_out, torch.int32, "kept_idx_out"),
                                    _ptr(scores_out, torch.float32, "scores_out")), "bkv_compress_ragged", ctx)


def bkv_get_state(ctx, centroids=None, sums=None, counts=None) -> None:
    """Tensors may live on the device or the host; host results are valid after bkv_sync."""
    _check(_l().bkv_get_state(ctx, _ptr_any(centroids, torch.float32, "centroids"),
                              _ptr_any(sums, torch.float64, "sums"), _ptr_any(counts, torch.int64, "counts")),
           "bkv_get_state", ctx)


def bkv_set_state(ctx, centroids, sums, counts) -> None:
    _check(_l().bkv_set_state(ctx, _ptr_any(centroids, torch.float32, "centroids"),
                              _ptr_any(sums, torch.float64, "sums"), _ptr_any(counts, torch.int64, "counts")),
           "bkv_set_state", ctx)


def bkv_get_cfps_state(ctx, buffers=None, sizes=None) -> None:
    _check(_l().bkv_get_cfps_state(ctx, _ptr_any(buffers, torch.bfloat16, "buffers"),
                                   _ptr_any(sizes, torch.int32, "sizes")), "bkv_get_cfps_state", ctx)


def bkv_set_cfps_state(ctx, buffers, sizes) -> None:
    _check(_l().bkv_set_cfps_state(ctx, _ptr_any(buffers, torch.bfloat16, "buffers"),
                                   _ptr_any(sizes, torch.int32, "sizes")), "bkv_set_cfps_state", ctx)


def bkv_sync(ctx) -> None:
    _check(_l().bkv_sync(ctx), "bkv_sync", ctx)


def bkv_selftest_wait_timeout(ctx, limit_ns: int) -> int:
    """Runs one device wait that is meant to expire after limit_ns (see
    include/bkv.h) and returns the status code bkv_sync reports for it
    (BKV_ETIMEOUT when the expiry path works); raises on other errors."""
    rc = _l().bkv_selftest_wait_timeout(ctx, int(limit_ns))
    if rc not in (BKV_OK, BKV_ETIMEOUT):
        _check(rc, "bkv_selftest_wait_timeout", ctx)
    return rc


def bkv_selftest_bounds(ctx) -> int:
    """Runs one checked out-of-range store (see include/bkv.h) and returns the status code bkv_sync
    reports for it: BKV_EBOUNDS in a checked build, BKV_OK otherwise; raises on other errors."""
    rc = _l().bkv_selftest_bounds(ctx)
    if rc not in (BKV_OK, BKV_EBOUNDS):
        _check(rc, "bkv_selftest_bounds", ctx)
    return rc


def bkv_checked_build() -> bool:
    return bool(_l().bkv_checked_build())


def bkv_debug_fail_alloc(nth: int) -> None:
    """Arms (nth > 0) or disarms (0) the allocation-failure hook of bkv_create (include/bkv.h)."""
    _check(_l().bkv_debug_fail_alloc(int(nth)), "bkv_debug_fail_alloc")


def bkv_profile_enable(ctx, on: bool = True) -> None:
    _check(_l().bkv_profile_enable(ctx, int(bool(on))), "bkv_profile_enable", ctx)


def bkv_profile_read(ctx) -> dict:
    """{kernel name: (total ms, launches)} since the previous read (syncs the stream)."""
    n = len(KERNEL_NAMES)
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int64 * n)()
    _check(_l().bkv_profile_read(ctx, ctypes.cast(ms, _P), ctypes.cast(cnt, _P), n), "bkv_profile_read", ctx)
    return {KERNEL_NAMES[k]: (ms[k], cnt[k]) for k in range(n)}


def bkv_compress_static(cfg: BkvConfig, centroids, counts, K, V, L: int, budget: int, t_pos: int, q_recent,
                        recent_pos, kept_idx_out, scores_out=None, dev_status=None, stream=None) -> None:
    """Context-free compress that allocates no device memory (see include/bkv.h).

    For callers that cannot allocate on the device, e.g. an engine whose KV
    page allocator owns all of HBM.  Scratch lives in a fixed 16 MiB array
    inside the library; concurrent calls on different streams race on it.
    Every tensor's element count is checked against the sizes cfg implies
    before any pointer reaches the library."""
    c = cfg
    n_inst = c.n_layers * c.batch * c.n_kv_heads
    if n_inst < 1 or c.head_dim < 1 or c.capacity < 1 or budget < 1 or c.window < 0 or c.n_beacons < 0:
        raise ValueError("cfg must describe at least one instance of head_dim, capacity and budget >= 1")
    _expect(K, n_inst * c.capacity * c.head_dim, "K")
    _expect(V, n_inst * c.capacity * c.head_dim, "V")
    _expect(kept_idx_out, n_inst * int(budget), "kept_idx_out")
    _expect(scores_out, n_inst * c.capacity, "scores_out")
    _expect(q_recent, c.n_layers * c.batch * c.n_q_heads * c.window * c.head_dim, "q_recent")
    _expect(centroids, n_inst * c.n_beacons * c.head_dim, "centroids")
    _expect(counts, n_inst * c.n_beacons, "counts")
    if dev_status is not None and dev_status.numel() < 1:
        raise ValueError("dev_status must hold one int32")
    if recent_pos is None:
        recent_pos = []
    if c.window > 0 and len(recent_pos) != c.window:
        raise ValueError(f"recent_pos has {len(recent_pos)} positions; the window is {c.window}")
    pos = (ctypes.c_int64 * max(1, len(recent_pos)))(*[int(p) for p in recent_pos])
    msg = ctypes.create_string_buffer(256)
    rc = _l().bkv_compress_static(
        ctypes.byref(cfg), _ptr(centroids, torch.float32, "centroids"), _ptr(counts, torch.int64, "counts"),
        _ptr(K, torch.bfloat16, "K"), _ptr(V, torch.bfloat16, "V"), int(L), int(budget), int(t_pos),
        _ptr(q_recent, torch.bfloat16, "q_recent"), ctypes.cast(pos, _P), _ptr(kept_idx_out, torch.int32, "kept"),
        _ptr(scores_out, torch.float32, "scores_out"), _ptr(dev_status, torch.int32, "dev_status"),
        _stream(stream), msg, ctypes.sizeof(msg))
    if rc != BKV_OK:
        raise BkvError(rc, "bkv_compress_static", msg.value.decode())


# ---------------------------------------------------------------- convenience
class BeaconKV:
    """Owns one context for a model shape and allocates outputs with torch.

    Example::
        bk = BeaconKV(n_layers=36, batch=16, n_q_heads=32, n_kv_heads=8, head_dim=128,
                      n_beacons=8, window=8, capacity=4224, rope_theta=1e6)
        bk.init_beacons(q_init)                       # [L, B, Hq, n_init, d] bf16
        bk.update(q_new)                              # [L, B, Hq, n_new, d] bf16
        kept = bk.compress(K, V, L=4224, budget=4096, t_pos=4223, q_recent=q, recent_pos=[...])
    """

    def __init__(self, *, n_layers, batch, n_q_heads, n_kv_heads, head_dim, n_beacons, window, capacity,
                 rope_theta=0.0, n_prefix=0, stream=None, mean_agg=False, continual_fps=False, causal_window=False):
        flags = ((BKV_F_MEAN_AGG if mean_agg else BKV_F_NONE) | (BKV_F_CONTINUAL_FPS if continual_fps else BKV_F_NONE)
                 | (BKV_F_CAUSAL_WINDOW if causal_window else BKV_F_NONE))
        self.cfg = BkvConfig(n_layers, batch, n_q_heads, n_kv_heads, head_dim, n_beacons, window, n_prefix,
                             capacity, float(rope_theta), flags)
        self.ctx = bkv_create(self.cfg, stream)
        self.n_inst = n_layers * batch * n_kv_heads

    @classmethod
    def for_workload(cls, wl, stream=None, capacity=None, mean_agg=False, continual_fps=False,
                     causal_window=False) -> "BeaconKV":
        return cls(n_layers=wl.n_layers, batch=wl.batch, n_q_heads=wl.n_q_heads, n_kv_heads=wl.n_kv_heads,
                   head_dim=wl.head_dim, n_beacons=wl.n_beacons, window=wl.window,
                   capacity=capacity or wl.capacity, rope_theta=wl.rope_theta, n_prefix=wl.n_prefix, stream=stream,
                   mean_agg=mean_agg, continual_fps=continual_fps, causal_window=causal_window)

    def close(self):
        if self.ctx:
            bkv_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001 - interpreter shutdown
            pass

    # The C ABI receives bare pointers and trusts the sizes that the context's shape implies (_expect).
    _expect = staticmethod(_expect)

    def _rows(self, q: torch.Tensor, name: str) -> int:
        """Queries per query head of a [n_layers, batch, n_q_heads, n, head_dim] block."""
        c = self.cfg
        if q.dim() < 2 or q.shape[-1] != c.head_dim:
            raise ValueError(f"{name} must end in [n, head_dim = {c.head_dim}], got {tuple(q.shape)}")
        n = q.shape[-2]
        self._expect(q, c.n_layers * c.batch * c.n_q_heads * n * c.head_dim, name)
        return n

    def init_beacons(self, q_init: torch.Tensor):
        bkv_init_beacons(self.ctx, q_init, self._rows(q_init, "q_init"))

    def update(self, q_new: torch.Tensor, assign_out: torch.Tensor | None = None):
        n_new = self._rows(q_new, "q_new")
        c = self.cfg
        self._expect(assign_out, c.n_layers * c.batch * c.n_q_heads * n_new, "assign_out")
        bkv_update_beacons(self.ctx, q_new, n_new, assign_out)

    def update_seq(self, q_steps: torch.Tensor, assign_out: torch.Tensor | None = None):
        """Decode steps in order: q_steps is [n_steps, n_layers, batch, n_q_heads, head_dim]."""
        c = self.cfg
        per_step = c.n_layers * c.batch * c.n_q_heads
        if q_steps.dim() < 2 or q_steps.shape[-1] != c.head_dim or q_steps.numel() % (per_step * c.head_dim):
            raise ValueError(f"q_steps must be [n_steps, n_layers, batch, n_q_heads, head_dim = {c.head_dim}], "
                             f"got {tuple(q_steps.shape)}")
        n_steps = q_steps.numel() // (per_step * c.head_dim)
        self._expect(assign_out, per_step * n_steps, "assign_out")
        bkv_update_beacons_seq(self.ctx, q_steps, n_steps, assign_out)

    def compress(self, K, V, *, L, budget, t_pos, q_recent, recent_pos, kept_out=None, scores_out=None):
        c = self.cfg
        per_head = c.n_layers * c.batch * c.n_kv_heads
        self._expect(K, per_head * c.capacity * c.head_dim, "K")
        self._expect(V, per_head * c.capacity * c.head_dim, "V")
        self._expect(q_recent, c.n_layers * c.batch * c.n_q_heads * c.window * c.head_dim, "q_recent")
        if len(recent_pos) != c.window:
            raise ValueError(f"recent_pos has {len(recent_pos)} positions; the window is {c.window}")
        self._expect(kept_out, per_head * budget, "kept_out")
        self._expect(scores_out, per_head * c.capacity, "scores_out")
        if kept_out is None:
            kept_out = torch.empty(c.n_layers, c.batch, c.n_kv_heads, budget, dtype=torch.int32, device=K.device)
        bkv_compress(self.ctx, K, V, L, budget, t_pos, q_recent, recent_pos, kept_out, scores_out)
        return kept_out

    def compress_ragged(self, K, V, *, L, budget, t_pos, q_recent, recent_pos, kept_out=None, scores_out=None):
        """Per-instance cache lengths: L is an int32 CUDA tensor [n_layers, batch, n_kv_heads]; t_pos and
        recent_pos hold one position (one list of window positions) per batch row."""
        c = self.cfg
        per_head = c.n_layers * c.batch * c.n_kv_heads
        self._expect(K, per_head * c.capacity * c.head_dim, "K")
        self._expect(V, per_head * c.capacity * c.head_dim, "V")
        self._expect(L, per_head, "L")
        self._expect(q_recent, c.n_layers * c.batch * c.n_q_heads * c.window * c.head_dim, "q_recent")
        if len(t_pos) != c.batch:
            raise ValueError(f"t_pos has {len(t_pos)} positions; the batch is {c.batch}")
        if len(recent_pos) != c.batch or any(len(r) != c.window for r in recent_pos):
            raise ValueError(f"recent_pos must hold {c.batch} lists of {c.window} positions")
        self._expect(kept_out, per_head * budget, "kept_out")
        self._expect(scores_out, per_head * c.capacity, "scores_out")
        if kept_out is None:
            kept_out = torch.empty(c.n_layers, c.batch, c.n_kv_heads, budget, dtype=torch.int32, device=K.device)
        bkv_compress_ragged(self.ctx, K, V, L, budget, t_pos, q_recent, recent_pos, kept_out, scores_out)
        return kept_out

    def state(self):
        c = self.cfg
        dev = torch.device("cuda", torch.cuda.current_device())
        cent = torch.empty(self.n_inst, c.n_beacons, c.head_dim, dtype=torch.float32, device=dev)
        sums = torch.empty(self.n_inst, c.n_beacons, c.head_dim, dtype=torch.float64, device=dev)
        counts = torch.empty(self.n_inst, c.n_beacons, dtype=torch.int64, device=dev)
        bkv_get_state(self.ctx, cent, sums, counts)
        return cent, sums, counts

    def set_state(self, cent, sums, counts):
        c = self.cfg
        self._expect(cent, self.n_inst * c.n_beacons * c.head_dim, "centroids")
        self._expect(sums, self.n_inst * c.n_beacons * c.head_dim, "sums")
        self._expect(counts, self.n_inst * c.n_beacons, "counts")
        bkv_set_state(self.ctx, cent, sums, counts)

    def cfps_state(self):
        """Continual FPS buffers: (bf16 [L, B, Hq, n_beacons + window, d], int32 sizes [L, B, Hq])."""
        c = self.cfg
        dev = torch.device("cuda", torch.cuda.current_device())
        buf = torch.empty(c.n_layers, c.batch, c.n_q_heads, c.n_beacons + c.window, c.head_dim, dtype=torch.bfloat16,
                          device=dev)
        sizes = torch.empty(c.n_layers, c.batch, c.n_q_heads, dtype=torch.int32, device=dev)
        bkv_get_cfps_state(self.ctx, buf, sizes)
        return buf, sizes

    def set_cfps_state(self, buf, sizes):
        c = self.cfg
        heads = c.n_layers * c.batch * c.n_q_heads
        self._expect(buf, heads * (c.n_beacons + c.window) * c.head_dim, "buffers")
        self._expect(sizes, heads, "sizes")
        bkv_set_cfps_state(self.ctx, buf, sizes)

    def sync(self):
        bkv_sync(self.ctx)
