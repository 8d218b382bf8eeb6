"""Pins of the oracle's Continual FPS (Section 4.2, Eq. 9; Algorithm 1 in fp32).

Independent routes: the fp64 Algorithm 1 of bkvo_fps (itself pinned by brute
force in test_oracle_beacons.py) away from near-ties, a numpy fp64 brute-force
simulation of the fill-and-compress buffer, closed forms (an orthonormal basis,
a zero query, the buffer before it first fills, the size cycle) and invariants.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O

# fp32 cosine error bound: a 128-term fused dot product plus a division, relative
# to |a| |b|, stays below d * 2^-24 = 8e-6 for d = 128
FP32_GAP = 1e-4


def _bits(x: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _clustered(rng, n, d, k=4, sigma=0.3):
    centres = rng.standard_normal((k, d))
    lab = rng.integers(0, k, n)
    return _bits(centres[lab] + sigma * rng.standard_normal((n, d)))


@pytest.mark.parametrize("seed", range(8))
def test_fps32_agrees_with_fp64_away_from_ties(olib, seed):
    rng = np.random.default_rng(100 + seed)
    n = int(rng.integers(5, 41))
    d = int(rng.choice([16, 64, 128]))
    m = int(rng.integers(1, n + 1))
    q = _clustered(rng, n, d)
    p64, g64 = O.fps(q, m, olib)
    p32, g32 = O.fps32(q, m, olib)
    assert len(p32) == len(p64) == m
    first = np.flatnonzero(p32 != p64)
    if first.size:  # a disagreement is only allowed after an fp64 near-tie
        assert g64[first[0]] < FP32_GAP, f"pick {first[0]} differs with fp64 gap {g64[first[0]]:.2e}"
    else:
        np.testing.assert_allclose(g32, g64, atol=FP32_GAP)


def test_fps32_orthonormal_basis_takes_indices_in_order(olib):
    d = 16
    q = _bits(np.eye(d))
    picks, gaps = O.fps32(q, d, olib)
    np.testing.assert_array_equal(picks, np.arange(d))   # every cosine exact: all ties, lowest index
    np.testing.assert_array_equal(gaps[:-1], 0.0)
    assert gaps[-1] == np.inf                             # no runner-up for the last pick


def test_fps32_zero_query_has_zero_similarity(olib):
    rng = np.random.default_rng(7)
    x = np.abs(rng.standard_normal((6, 8))) + 0.1     # positive rows: pairwise cosines > 0
    x[3] = 0.0
    picks, _ = O.fps32(_bits(x), 2, olib)
    assert picks[0] == 3                              # average similarity 0 is the smallest


def _fps64_numpy(x: np.ndarray, m: int):
    n = len(x)
    nrm = np.sqrt((x * x).sum(1))
    c = (x @ x.T) / np.outer(nrm, nrm)
    p = int(np.argmin(c.mean(1)))
    sel = [p]
    S = c[:, p].copy()
    while len(sel) < min(m, n):
        S2 = S.copy()
        S2[sel] = np.inf
        r = int(np.argmin(S2))
        sel.append(r)
        S = np.maximum(S, c[:, r])
    return sel


def test_cfps_buffer_matches_fp64_brute_force_simulation(olib):
    rng = np.random.default_rng(11)
    d, b_min, b_max = 32, 4, 10
    q = _clustered(rng, 57, d, k=6, sigma=0.5)
    buf, size, picks, gaps = O.cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q, olib)
    assert (gaps > FP32_GAP).all(), "choose a seed without near-ties"
    x = O.bf16_to_f64(q)
    cur = []
    for row in x:
        cur.append(row)
        if len(cur) >= b_max:
            sel = _fps64_numpy(np.array(cur), b_min)
            cur = [cur[i] for i in sel]
    assert size == len(cur)
    np.testing.assert_array_equal(O.bf16_to_f64(buf[:size]), np.array(cur))


def test_cfps_closed_forms(olib):
    rng = np.random.default_rng(12)
    d, b_min, b_max = 16, 3, 7
    q = _clustered(rng, 40, d)
    # before the buffer first fills it is the queries in arrival order
    buf, size, picks, _ = O.cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q[:6], olib)
    assert size == 6 and len(picks) == 0
    np.testing.assert_array_equal(buf[:6], q[:6])
    # size cycle: from s0, every (b_max - b_min) arrivals after the first fill compress once
    for s0, n in [(0, 40), (3, 4), (5, 1), (6, 1), (3, 17)]:
        start = q[:s0]
        buf, size, picks, _ = O.cfps_update(start, s0, b_min, b_max, q[s0:s0 + n], olib)
        s, ev = s0, 0
        for _ in range(n):
            s += 1
            if s >= b_max:
                s, ev = b_min, ev + 1
        assert (size, len(picks)) == (s, ev)
        # every kept row is one of the rows that entered the buffer
        seen = {r.tobytes() for r in np.vstack([start, q[s0:s0 + n]])}
        assert all(r.tobytes() in seen for r in buf[:size])
        # every compression picks b_min distinct buffer positions
        for p in picks:
            assert len(set(p.tolist())) == b_min and p.min() >= 0 and p.max() < b_max
