"""Host-side checks of the C ABI that need no GPU: the library builds, loads and
exports every function include/bkv.h declares; configuration validation and
error strings behave as documented; the workload byte / FLOP accounting is
consistent."""
import ctypes
import os
import re

import pytest

from paper_2609_04971_gb300 import _build, bkv
from paper_2609_04971_gb300.workloads import LLAMA_8B, QWEN3_14B, QWEN3_4B, TINY, n_obs_padded

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "bkv.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(bkv_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    return bkv.load_library()


def test_header_declares_the_api():
    names = _declared()
    for n in ("bkv_create", "bkv_destroy", "bkv_init_beacons", "bkv_update_beacons", "bkv_compress",
              "bkv_get_state", "bkv_set_state", "bkv_sync", "bkv_strerror"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    raw = ctypes.CDLL(_build.LIB_PATH)
    missing = [n for n in _declared() if not hasattr(raw, n)]
    assert not missing, f"declared but not exported: {missing}"


def test_binding_mirrors_every_declared_symbol():
    missing = [n for n in _declared() if not hasattr(bkv, n)]
    assert not missing, f"no Python binding for: {missing}"


def test_strerror_and_version(lib):
    assert bkv.bkv_strerror(0) == "ok"
    assert "invalid" in bkv.bkv_strerror(-1)
    assert bkv.bkv_strerror(-99) == "unknown error"
    assert "sm_103a" in bkv.bkv_version()


@pytest.mark.parametrize("field,value", [
    ("n_kv_heads", 3), ("head_dim", 96), ("n_beacons", 33), ("window", -1), ("window", 65),
    ("capacity", 0), ("capacity", 40000), ("rope_theta", -1.0), ("flags", 8), ("flags", 0x80000000), ("n_layers", 0),
    ("n_prefix", -2)])
def test_create_rejects_bad_config_before_touching_the_gpu(lib, field, value):
    cfg = bkv.BkvConfig(1, 1, 4, 2, 64, 4, 8, 0, 1088, 1e4, 0)
    setattr(cfg, field, value)
    out = ctypes.c_void_p()
    assert lib.bkv_create(ctypes.byref(cfg), None, ctypes.byref(out)) == bkv.BKV_EINVAL
    assert not out.value


@pytest.mark.parametrize("n_beacons,window,n_q_heads", [(0, 8, 4), (8, 0, 4), (20, 13, 4), (16, 16, 16)])
def test_create_rejects_bad_continual_fps_config(lib, n_beacons, window, n_q_heads):
    """Continual FPS needs n_beacons >= 1, window >= 1, n_beacons + window <= 32 and
    G * (n_beacons + window) <= 128 (here G = n_q_heads / 2)."""
    cfg = bkv.BkvConfig(1, 1, n_q_heads, 2, 64, n_beacons, window, 0, 1088, 1e4, bkv.BKV_F_CONTINUAL_FPS)
    out = ctypes.c_void_p()
    assert lib.bkv_create(ctypes.byref(cfg), None, ctypes.byref(out)) == bkv.BKV_EINVAL
    assert not out.value


def test_create_rejects_too_many_scoring_queries(lib):
    cfg = bkv.BkvConfig(1, 1, 64, 4, 128, 8, 8, 0, 1024, 1e4, 0)   # 16 * 8 + 8 = 136 > 128
    out = ctypes.c_void_p()
    assert lib.bkv_create(ctypes.byref(cfg), None, ctypes.byref(out)) == bkv.BKV_EINVAL


def test_null_arguments(lib):
    assert lib.bkv_create(None, None, None) == bkv.BKV_EINVAL
    assert lib.bkv_sync(None) == bkv.BKV_EINVAL
    assert lib.bkv_compress(None, None, None, 1, 1, 0, None, None, None, None) == bkv.BKV_EINVAL
    lib.bkv_destroy(None)
    assert lib.bkv_last_error(None) == b""


def test_byte_accounting_matches_closed_form():
    wl = QWEN3_4B
    per_inst = 4224 * 128 * 2 + 4096 * 128 * 2 * 4 + 4 * 8 * 128 * 2 + 4096 * 4
    assert wl.compress_bytes() == per_inst * 36 * 16 * 8
    assert abs(wl.step_bytes() / 1e9 - 25.06) < 0.02
    assert wl.n_obs == 40 and n_obs_padded(wl.n_obs) == 48
    assert LLAMA_8B.n_obs == 48 and QWEN3_14B.n_obs == 56 and TINY.n_obs == 20
    assert n_obs_padded(QWEN3_14B.n_obs) == 64 and n_obs_padded(TINY.n_obs) == 32


def test_selftest_rejects_null_context(lib):
    assert lib.bkv_selftest_wait_timeout(None, 1_000_000) == bkv.BKV_EINVAL


def test_binding_rejects_tensors_of_the_wrong_size(lib):
    """The C ABI takes bare pointers and trusts the sizes the context's shape implies, so the Python
    binding checks every tensor's element count first: a wrong size is a ValueError before any call
    reaches the library (checked here on a context object with no device context behind it); a right
    size gets as far as the device-pointer check, which rejects these CPU tensors."""
    import torch
    wl = TINY
    bk = bkv.BeaconKV.__new__(bkv.BeaconKV)
    bk.cfg = bkv.BkvConfig(wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.n_beacons,
                           wl.window, 0, wl.capacity, wl.rope_theta, 0)
    bk.ctx = None
    bk.n_inst = wl.n_inst
    nl, B, Hq, Hkv, d, W, cap = wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.window, wl.capacity
    bf = dict(dtype=torch.bfloat16)
    q = torch.zeros(nl, B, Hq, 3, d, **bf)
    K = torch.zeros(nl, B, Hkv, cap, d, **bf)
    qr = torch.zeros(nl, B, Hq, W, d, **bf)
    kept = torch.zeros(nl, B, Hkv, wl.budget, dtype=torch.int32)
    pos = dict(L=wl.L, budget=wl.budget, t_pos=wl.L - 1, recent_pos=list(range(wl.L - W, wl.L)))
    bad = [
        lambda: bk.update(torch.zeros(nl, B, Hq - 1, 3, d, **bf)),                       # a head short
        lambda: bk.update(torch.zeros(nl, B, Hq, 3, d // 2, **bf)),                      # wrong head_dim
        lambda: bk.update(q, torch.zeros(nl, B, Hq, 2, dtype=torch.int32)),              # assign_out too small
        lambda: bk.init_beacons(torch.zeros(nl, B, Hq * 3 * d, **bf)),                   # no row axis
        lambda: bk.compress(K[..., :-1, :], K, q_recent=qr, kept_out=kept, **pos),       # K short of capacity
        lambda: bk.compress(K, K, q_recent=qr[..., :-1, :], kept_out=kept, **pos),      # window short
        lambda: bk.compress(K, K, q_recent=qr, kept_out=kept[..., :-1], **pos),          # kept_out too small
        lambda: bk.compress(K, K, q_recent=qr, kept_out=kept, scores_out=torch.zeros(nl, B, Hkv, cap - 1), **pos),
        lambda: bk.compress(K, K, q_recent=qr, kept_out=kept, **dict(pos, recent_pos=[0])),
        lambda: bk.set_state(torch.zeros(wl.n_inst, wl.n_beacons, d), torch.zeros(wl.n_inst, wl.n_beacons, d - 1),
                             torch.zeros(wl.n_inst, wl.n_beacons, dtype=torch.int64)),
    ]
    for i, call in enumerate(bad):
        with pytest.raises(ValueError):
            call()
    for call in (lambda: bk.update(q), lambda: bk.init_beacons(q),
                 lambda: bk.compress(K, K, q_recent=qr, kept_out=kept, **pos)):
        with pytest.raises(TypeError, match="CUDA tensor"):
            call()


def test_static_compress_rejects_bad_arguments_before_any_cuda_call(lib):
    """bkv_compress_static validates its configuration, pointers, sizes and scratch budget on the host
    and returns BKV_EINVAL with a reason before it enqueues anything.  The pointers below are never
    dereferenced: every case fails validation first."""
    raw = ctypes.CDLL(_build.LIB_PATH)
    fn = raw.bkv_compress_static
    fn.restype = ctypes.c_int
    wl = TINY
    P = ctypes.c_void_p
    dev_a, dev_b, dev_c = P(0x10000), P(0x20000), P(0x30000)   # 16-byte aligned stand-ins, never touched

    def cfg(**kw):
        base = dict(n_layers=wl.n_layers, batch=wl.batch, n_q_heads=wl.n_q_heads, n_kv_heads=wl.n_kv_heads,
                    head_dim=wl.head_dim, n_beacons=wl.n_beacons, window=wl.window, n_prefix=0,
                    capacity=wl.capacity, rope_theta=wl.rope_theta, flags=0)
        base.update(kw)
        return bkv.BkvConfig(*base.values())

    pos = (ctypes.c_int64 * wl.window)(*range(wl.L - wl.window, wl.L))

    def call(c, K=dev_a, V=dev_b, kept=dev_c, L=wl.L, budget=wl.budget, q_recent=dev_a, recent=pos,
             centroids=dev_b, counts=dev_c):
        msg = ctypes.create_string_buffer(200)
        rc = fn(None if c is None else ctypes.byref(c), centroids, counts, K, V, ctypes.c_int32(L),
                ctypes.c_int32(budget), ctypes.c_int64(wl.L - 1), q_recent, recent, kept, None, None, None, msg,
                ctypes.c_size_t(ctypes.sizeof(msg)))
        return rc, msg.value.decode()

    cases = [
        (dict(c=None), "cfg is NULL"),
        (dict(c=cfg(head_dim=96)), "head_dim"),
        (dict(c=cfg(flags=bkv.BKV_F_CONTINUAL_FPS)), "flags"),
        (dict(c=cfg(n_q_heads=3)), "head"),
        (dict(c=cfg(), K=None), "non-NULL"),
        (dict(c=cfg(), V=P(0x20008)), "aligned"),
        (dict(c=cfg(), L=wl.capacity + 1), "L must be"),
        (dict(c=cfg(), budget=wl.window - 1), "budget"),
        (dict(c=cfg(n_layers=64, capacity=32768), L=32768), "scratch"),
        (dict(c=cfg(), q_recent=None), "q_recent"),
        (dict(c=cfg(), recent=None), "recent_pos"),
        (dict(c=cfg(), centroids=None), "centroids"),
    ]
    for kw, why in cases:
        rc, msg = call(**kw)
        assert rc == bkv.BKV_EINVAL and why in msg, (kw, rc, msg)


def test_static_binding_rejects_tensors_of_the_wrong_size():
    """bkv_compress_static has no context, so its binding checks every tensor against the sizes cfg
    implies (and the length of recent_pos against the window) before a pointer reaches the library:
    a wrong size is a ValueError; right sizes reach the device-pointer check, which rejects these CPU
    tensors."""
    import torch
    wl = TINY
    nl, B, Hq, Hkv, d, W, cap, nb = (wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.window,
                                     wl.capacity, wl.n_beacons)
    cfg = bkv.BkvConfig(nl, B, Hq, Hkv, d, nb, W, 0, cap, wl.rope_theta, 0)
    bf = dict(dtype=torch.bfloat16)
    K = torch.zeros(nl, B, Hkv, cap, d, **bf)
    qr = torch.zeros(nl, B, Hq, W, d, **bf)
    kept = torch.zeros(nl, B, Hkv, wl.budget, dtype=torch.int32)
    sc = torch.zeros(nl, B, Hkv, cap)
    cent = torch.zeros(wl.n_inst, nb, d)
    cnt = torch.zeros(wl.n_inst, nb, dtype=torch.int64)
    pos = list(range(wl.L - W, wl.L))
    good = dict(centroids=cent, counts=cnt, K=K, V=K, q_recent=qr, recent_pos=pos, kept_idx_out=kept,
                scores_out=sc)

    def call(**over):
        a = dict(good, **over)
        bkv.bkv_compress_static(cfg, a["centroids"], a["counts"], a["K"], a["V"], wl.L, wl.budget, wl.L - 1,
                                a["q_recent"], a["recent_pos"], a["kept_idx_out"], a["scores_out"])

    bad = [dict(K=K[..., :-1, :].contiguous()), dict(V=torch.zeros(nl, B, Hkv, cap, d // 2, **bf)),
           dict(q_recent=qr[..., :-1, :].contiguous()), dict(kept_idx_out=kept[..., :-1].contiguous()),
           dict(scores_out=sc[..., :-1].contiguous()), dict(centroids=cent[:-1]), dict(counts=cnt[:, :-1]),
           dict(recent_pos=pos[:-1]), dict(recent_pos=None)]
    for over in bad:
        with pytest.raises(ValueError):
            call(**over)
    with pytest.raises(TypeError, match="CUDA tensor"):
        call()


def test_allocation_failure_hook_reports_enomem(lib):
    """bkv_debug_fail_alloc(1) makes bkv_create's first allocation fail before anything is allocated:
    the call returns BKV_ENOMEM with *out NULL, and the hook then disarms itself (the next create fails
    otherwise on a machine without a GPU, or succeeds on one).  Negative arguments are rejected."""
    cfg = bkv.BkvConfig(1, 1, 4, 2, 64, 4, 8, 0, 1088, 1e4, 0)
    out = ctypes.c_void_p()
    assert lib.bkv_debug_fail_alloc(-1) == bkv.BKV_EINVAL
    try:
        assert lib.bkv_debug_fail_alloc(1) == bkv.BKV_OK
        assert lib.bkv_create(ctypes.byref(cfg), None, ctypes.byref(out)) == bkv.BKV_ENOMEM
        assert not out.value
        rc = lib.bkv_create(ctypes.byref(cfg), None, ctypes.byref(out))
        assert rc != bkv.BKV_ENOMEM
        if rc == bkv.BKV_OK:
            lib.bkv_destroy(out)
    finally:
        lib.bkv_debug_fail_alloc(0)


def test_checked_flavour_builds_and_exports_the_same_symbols(lib):
    """The BKV_CHECKED flavour (device-side bounds checks compiled in) builds from the same sources,
    exports every declared symbol and says which flavour it is."""
    path = _build.build(checked=True)
    assert path == _build.LIB_PATH_CHECKED != _build.LIB_PATH
    raw = ctypes.CDLL(path)
    missing = [n for n in _declared() if not hasattr(raw, n)]
    assert not missing, f"declared but not exported by the checked flavour: {missing}"
    assert raw.bkv_checked_build() == 1
    assert lib.bkv_checked_build() == 0
    assert "bounds" in bkv.bkv_strerror(bkv.BKV_EBOUNDS)
