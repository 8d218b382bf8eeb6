"""Python marshalling for the fp64 CPU oracle in ``bkv_oracle.c``.

TEST INFRASTRUCTURE ONLY: tests/, ``__graft_entry__.smoke()`` and bench.py's
CPU-baseline / reference leg are the only callers.  The product library never
imports this module, and this module imports nothing from the product package.

Arrays are numpy; bf16 data travels as ``uint16`` bit patterns.  Each function
wraps one C function and states the paper passage it restates (see the C file
for the step-by-step definition).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bkv_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-fopenmp"]


def build(force: bool = False, src: str = _SRC, out: str = _LIB_PATH) -> str:
    """Compile the oracle with gcc (fp contraction off) and return the .so path."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, src, "-lm"])
    os.replace(tmp, out)
    return out


_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_D = ctypes.c_double

_SIGS = {
    "bkvo_bf16_to_f64": (_D, [ctypes.c_uint16]),
    "bkvo_f32_to_bf16": (ctypes.c_uint16, [ctypes.c_float]),
    "bkvo_round_scoring": (_D, [_D]),
    "bkvo_cosine": (_D, [_P, _P, _I]),
    "bkvo_fps": (_I, [_P, _I, _I, _I, _P, _P]),
    "bkvo_init_beacons": (_I, [_P, _I, _I, _I, _P, _P, _P, _P, _P]),
    "bkvo_update": (None, [_P, _I, _I, _I, _P, _P, _P, _P, _P, _P]),
    "bkvo_rope": (None, [_P, _I, _I64, _D, _P]),
    "bkvo_build_qobs": (_I, [_P, _P, _I, _P, _I, _I, _P, _I64, _I, _D, _P, _P]),
    "bkvo_score": (None, [_P, _P, _I, _P, _I, _I, _P]),
    "bkvo_score_agg": (None, [_P, _P, _I, _P, _I, _I, _I, _P]),
    "bkvo_score_mask": (None, [_P, _P, _P, _I, _P, _P, _I, _I, _I, _P]),
    "bkvo_fps_adopt": (_I, [_P, _I, _I, _I, _P, _P, _P, _P, _P, _P]),
    "bkvo_cfps_update": (_I, [_P, _P, _I, _I, _P, _I, _I, _P, _P, _P, _P, _P, _P, _I]),
    "bkvo_select": (_I, [_P, _I, _I, _I, _I, _P, _P]),
    "bkvo_gather": (None, [_P, _P, _P, _I, _I]),
    "bkvo_step_many": (_I, [_P, _I, _I, _I, _I, _I, _I, _I, _P, _I, _P, _P, _I64, _D, _I, _I,
                            _P, _P, _P, _P, _P, _P, _P]),
}


def load(path: str | None = None):
    """Load (building first if needed) the oracle library; returns the ctypes handle."""
    global _lib
    with _lock:
        if path is not None:
            lib = ctypes.CDLL(path)
        elif _lib is not None:
            return _lib
        else:
            lib = ctypes.CDLL(build())
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        if path is None:
            _lib = lib
        return lib


def _c(a: np.ndarray, dtype) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dtype)


def _p(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


# ---------------------------------------------------------------- bf16 helpers
def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    b = _c(bits, np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def f32_to_bf16(x, lib=None) -> int:
    """Round one binary32 value to bf16 (nearest even); returns the bit pattern."""
    return int((lib or load()).bkvo_f32_to_bf16(float(np.float32(x))))


def round_scoring(x: float, lib=None) -> float:
    """fp64 -> fp32 -> bf16 rounding applied to every scoring query."""
    return float((lib or load()).bkvo_round_scoring(float(x)))


def cosine(a: np.ndarray, b: np.ndarray, lib=None) -> float:
    a = _c(a, np.float64)
    b = _c(b, np.float64)
    return float((lib or load()).bkvo_cosine(_p(a), _p(b), a.shape[-1]))


# ---------------------------------------------------------------- method steps
def fps(q_bits: np.ndarray, m: int, lib=None):
    """Algorithm 1 (Appendix D.1).  q_bits: uint16 [N, d].  Returns (picks, gaps)."""
    q = _c(q_bits, np.uint16)
    n, d = q.shape
    picks = np.full(max(m, 1), -1, np.int32)
    gaps = np.zeros(max(m, 1), np.float64)
    got = (lib or load()).bkvo_fps(_p(q), n, d, m, _p(picks), _p(gaps))
    return picks[:got].copy(), gaps[:got].copy()


def fps_adopt(q_bits: np.ndarray, m: int, forced: np.ndarray | None = None, lib=None):
    """Algorithm 1 in fp64 where forced[k] >= 0 dictates the k-th pick (a choice another implementation
    made at a near-tie; test harness only).  Returns (picks, gaps, alts, margins, vals): the runner-up
    distance and row of each step's argmin, how far the row taken lies above the minimum, and the value
    each step minimises per row ([m, N], +inf for rows already taken).  Raises ValueError for a forced
    row that is out of range or already taken."""
    q = _c(q_bits, np.uint16)
    n, d = q.shape
    k = max(m, 1)
    f = None if forced is None else _c(np.asarray(forced).reshape(-1)[:k], np.int32)
    if f is not None and f.shape[0] < k:
        f = np.concatenate([f, np.full(k - f.shape[0], -1, np.int32)])
    picks = np.full(k, -1, np.int32)
    gaps = np.zeros(k, np.float64)
    alts = np.full(k, -1, np.int32)
    margins = np.zeros(k, np.float64)
    vals = np.zeros((k, max(n, 1)), np.float64)
    got = (lib or load()).bkvo_fps_adopt(_p(q), n, d, m, _p(f), _p(picks), _p(gaps), _p(alts), _p(margins),
                                         _p(vals))
    if got < 0:
        raise ValueError("a forced FPS pick is out of range or already taken")
    return picks[:got].copy(), gaps[:got].copy(), alts[:got].copy(), margins[:got].copy(), vals[:got, :n].copy()


def cfps_events(size: int, b_min: int, b_max: int, n_new: int) -> int:
    """Compressions of a Continual FPS buffer of `size` rows over n_new arrivals."""
    n = 0
    for _ in range(n_new):
        size += 1
        if size >= b_max:
            size, n = b_min, n + 1
    return n


def cfps_update(buf_bits: np.ndarray, size: int, b_min: int, b_max: int, q_new_bits: np.ndarray, lib=None,
                forced: np.ndarray | None = None) -> dict:
    """Continual FPS (Eq. 9) of one query head: append each new query; at b_max queries
    compress the buffer to its fp64 FPS selection of b_min.  buf_bits: uint16 [>= size, d].
    forced: None or [events, b_min] dictated picks (-1 = the argmin; test harness only).
    Returns dict(buf uint16 [b_max, d] with rows [0, size) in use, size, and per compression
    picks / gaps / alts / margins [events, b_min] and vals [events, b_min, b_max])."""
    d = q_new_bits.shape[-1]
    buf = np.zeros((b_max, d), np.uint16)
    buf[:size] = buf_bits[:size]
    q = _c(q_new_bits.reshape(-1, d), np.uint16)
    n_new = q.shape[0]
    cap = cfps_events(size, b_min, b_max, n_new)
    w = max(b_min, 1)
    shape = (max(cap, 1), w)
    ev_p = np.full(shape, -1, np.int32)
    ev_g = np.zeros(shape, np.float64)
    ev_a = np.full(shape, -1, np.int32)
    ev_m = np.zeros(shape, np.float64)
    ev_v = np.zeros(shape + (b_max,), np.float64)
    f = None
    if forced is not None:
        f = np.full(shape, -1, np.int32)
        fa = np.asarray(forced, np.int32).reshape(-1, w)[:shape[0]]
        f[:fa.shape[0]] = fa
    sz = np.array([size], np.int32)
    n_ev = (lib or load()).bkvo_cfps_update(_p(buf), _p(sz), b_min, b_max, _p(q), n_new, d, _p(f), _p(ev_p),
                                            _p(ev_g), _p(ev_a), _p(ev_m), _p(ev_v), shape[0])
    if n_ev < 0:
        raise ValueError("a forced FPS pick is out of range or already taken")
    return dict(buf=buf, size=int(sz[0]), picks=ev_p[:n_ev].copy(), gaps=ev_g[:n_ev].copy(),
                alts=ev_a[:n_ev].copy(), margins=ev_m[:n_ev].copy(), vals=ev_v[:n_ev].copy())


def init_beacons(q_bits: np.ndarray, nb: int, lib=None):
    """FPS seeding of one group's beacons (Appendix D.2 prefill).

    Returns dict(cent fp32 [nb,d], sums fp64 [nb,d], counts int64 [nb], picks, gaps).
    """
    q = _c(q_bits, np.uint16)
    n, d = q.shape
    cent = np.zeros((nb, d), np.float32)
    sums = np.zeros((nb, d), np.float64)
    counts = np.zeros(nb, np.int64)
    picks = np.full(max(nb, 1), -1, np.int32)
    gaps = np.zeros(max(nb, 1), np.float64)
    got = (lib or load()).bkvo_init_beacons(_p(q), n, d, nb, _p(cent), _p(sums), _p(counts), _p(picks), _p(gaps))
    if got < 0:
        raise ValueError("init_beacons needs at least nb queries")
    return dict(cent=cent, sums=sums, counts=counts, picks=picks[:got].copy(), gaps=gaps[:got].copy())


def update(q_bits: np.ndarray, state: dict, override: np.ndarray | None = None, lib=None):
    """Nearest-beacon assignment + running-mean update of one group, in place on ``state``.

    Returns (assign int32 [nq], margin fp64 [nq]) describing the oracle's own argmax.
    """
    q = _c(q_bits, np.uint16)
    nq, d = q.shape
    for k, dt in (("cent", np.float32), ("sums", np.float64), ("counts", np.int64)):
        if state[k].dtype != dt or not state[k].flags.c_contiguous:
            state[k] = _c(state[k], dt)
    nb = state["counts"].shape[0]
    ov = None if override is None else _c(override, np.int32)
    assign = np.zeros(max(nq, 1), np.int32)
    margin = np.zeros(max(nq, 1), np.float64)
    (lib or load()).bkvo_update(_p(q), nq, d, nb, _p(state["cent"]), _p(state["sums"]), _p(state["counts"]),
                                _p(ov), _p(assign), _p(margin))
    return assign[:nq].copy(), margin[:nq].copy()


def rope(x: np.ndarray, pos: int, theta: float, lib=None) -> np.ndarray:
    """Rotate-half rotary embedding of one fp64 vector (no rounding)."""
    x = _c(x, np.float64)
    y = np.zeros_like(x)
    (lib or load()).bkvo_rope(_p(x), x.shape[0], int(pos), float(theta), _p(y))
    return y


def build_qobs(cent, counts, q_recent_bits, recent_pos, t_pos: int, theta: float, lib=None):
    """Q_obs of one group (Section 4.3): recent rows (h*W+w) then beacons.

    Returns (qobs fp64 [M, d] holding bf16-rounded values, valid int32 [M]).
    """
    cent = _c(cent, np.float32)
    counts = _c(counts, np.int64)
    qr = _c(q_recent_bits, np.uint16)
    g, w, d = qr.shape
    nb = counts.shape[0]
    pos = _c(recent_pos, np.int64)
    m = g * w + nb
    qobs = np.zeros((max(m, 1), d), np.float64)
    valid = np.zeros(max(m, 1), np.int32)
    (lib or load()).bkvo_build_qobs(_p(cent), _p(counts), nb, _p(qr), g, w, _p(pos), int(t_pos), d,
                                    float(theta), _p(qobs), _p(valid))
    return qobs[:m].copy(), valid[:m].copy()


def score(qobs: np.ndarray, valid: np.ndarray, k_bits: np.ndarray, lib=None, mean: bool = False,
          qpos: np.ndarray | None = None, kpos: np.ndarray | None = None) -> np.ndarray:
    """Eq. 4 softmax weights, max (or, with mean=True, mean) over the group's valid queries
    (Eq. 6, Section 4.3).  With positions (qpos per query row, kpos per key), key j enters
    query q's softmax only if kpos[j] <= qpos[q] (causal mask)."""
    qo = _c(qobs, np.float64)
    va = _c(valid, np.int32)
    k = _c(k_bits, np.uint16)
    L, d = k.shape
    out = np.zeros(max(L, 1), np.float64)
    if qpos is None:
        (lib or load()).bkvo_score_agg(_p(qo), _p(va), qo.shape[0], _p(k), L, d, int(bool(mean)), _p(out))
    else:
        qp = _c(qpos, np.int64)
        kp = _c(kpos, np.int64)
        assert qp.shape[0] == qo.shape[0] and kp.shape[0] == L
        (lib or load()).bkvo_score_mask(_p(qo), _p(va), _p(qp), qo.shape[0], _p(k), _p(kp), L, d, int(bool(mean)),
                                        _p(out))
    return out[:L].copy()


def causal_positions(G: int, W: int, nb: int, recent_pos, t_pos: int, L: int):
    """Positions for the causal mask inside the recent window (a reading: the paper leaves
    AttnWeight's mask open).  Q_obs row h*W + w (recent slot w of head h) sits at recent_pos[w],
    beacon rows at the current step t_pos; window key j (L - W <= j < L) at t_pos - (L - 1 - j);
    older keys come before every position.  Returns (qpos int64 [G*W + nb], kpos int64 [L])."""
    rp = np.asarray(recent_pos, np.int64)
    qpos = np.concatenate([np.tile(rp[:W], G), np.full(nb, int(t_pos), np.int64)])
    kpos = np.full(L, np.iinfo(np.int64).min, np.int64)
    w0 = max(L - W, 0)
    kpos[w0:] = int(t_pos) - (L - 1 - np.arange(w0, L, dtype=np.int64))
    return qpos, kpos


def select(score_: np.ndarray, budget: int, window: int, n_prefix: int, lib=None):
    """Keep set + TopK + sort (Eq. 7, Algorithm 2).  Returns (kept int32, boundary[2])."""
    s = _c(score_, np.float64)
    L = s.shape[0]
    kept = np.zeros(max(min(L, budget), 1), np.int32)
    bd = np.zeros(2, np.float64)
    n = (lib or load()).bkvo_select(_p(s), L, budget, window, n_prefix, _p(kept), _p(bd))
    if n < 0:
        raise ValueError("budget smaller than n_prefix + window")
    return kept[:n].copy(), bd.copy()


def gather(k_bits: np.ndarray, v_bits: np.ndarray, kept: np.ndarray, lib=None) -> None:
    """Eq. 8 compaction, in place on two uint16 [rows, d] arrays."""
    assert k_bits.dtype == np.uint16 and k_bits.flags.c_contiguous
    assert v_bits.dtype == np.uint16 and v_bits.flags.c_contiguous
    kp = _c(kept, np.int32)
    (lib or load()).bkvo_gather(_p(k_bits), _p(v_bits), _p(kp), kp.shape[0], k_bits.shape[-1])


def step_many(inst, *, G, d, nb, W, n_prefix, cap, q_new, n_new, q_recent, recent_pos, t_pos, theta, L,
              budget, K, V, cent, sums, counts, kept, score_out=None, lib=None) -> int:
    """Update + compress for the listed instances, OpenMP-parallel (CPU baseline).

    All arrays are full-size, C-contiguous and modified in place as the C driver
    documents.  Returns the number of threads used.
    """
    ins = _c(inst, np.int64)
    pos = _c(recent_pos, np.int64)
    for a, dt in ((q_new, np.uint16), (q_recent, np.uint16), (K, np.uint16), (V, np.uint16), (cent, np.float32),
                  (sums, np.float64), (counts, np.int64), (kept, np.int32)):
        assert a.dtype == dt and a.flags.c_contiguous, (a.dtype, dt)
    if score_out is not None:
        assert score_out.dtype == np.float64 and score_out.flags.c_contiguous
    return int((lib or load()).bkvo_step_many(
        _p(ins), ins.shape[0], G, d, nb, W, n_prefix, cap, _p(q_new), n_new, _p(q_recent), _p(pos), int(t_pos),
        float(theta), L, budget, _p(K), _p(V), _p(cent), _p(sums), _p(counts), _p(kept), _p(score_out)))
