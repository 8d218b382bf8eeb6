"""Pins of the oracle's Continual FPS (Section 4.2, Eq. 9; Algorithm 1 in fp64)
and of the parity harness's near-tie rule for FPS decisions taken in fp32.

Independent routes: the fp64 Algorithm 1 of bkvo_fps (itself pinned by brute
force in test_oracle_beacons.py), numpy fp64 brute-force FPS with dictated
picks, a numpy fp64 simulation of the fill-and-compress buffer, closed forms (an
orthonormal basis, a zero query, the buffer before it first fills, the size
cycle), fp32 cosines computed by numpy against the tie bound, and numpy FPS
variants that break near-ties the other way (accepted) or depart beyond the
bound (rejected).
"""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from tests import parity as P


def _bits(x: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _clustered(rng, n, d, k=4, sigma=0.3):
    centres = rng.standard_normal((k, d))
    lab = rng.integers(0, k, n)
    return _bits(centres[lab] + sigma * rng.standard_normal((n, d)))


def _cos64(x: np.ndarray) -> np.ndarray:
    nrm = np.sqrt((x * x).sum(1))
    den = np.outer(nrm, nrm)
    with np.errstate(invalid="ignore", divide="ignore"):
        c = (x @ x.T) / den
    c[den == 0] = 0.0
    return c


def _fps_numpy(x: np.ndarray, m: int, choose=None):
    """Algorithm 1 on fp64 rows with numpy; choose(step, values, candidates) picks the row (default: the
    argmin, ties to the lowest index).  Returns (picks, values of the rows taken minus the minimum)."""
    n = len(x)
    c = _cos64(x)
    val = c.mean(1)
    sel, margins = [], []
    S = None
    for k in range(min(m, n)):
        cand = [j for j in range(n) if j not in sel]
        v = val if k == 0 else S
        r = min(cand, key=lambda j: (v[j], j)) if choose is None else choose(k, v, cand)
        margins.append(v[r] - min(v[j] for j in cand))
        sel.append(r)
        S = c[:, r].copy() if k == 0 else np.maximum(S, c[:, r])
    return sel, margins


# ---------------------------------------------------------------- Algorithm 1 with adoption
@pytest.mark.parametrize("seed", range(6))
def test_fps_adopt_without_forcing_is_fps_and_numpy(olib, seed):
    rng = np.random.default_rng(200 + seed)
    n, d = int(rng.integers(4, 33)), int(rng.choice([16, 64, 128]))
    m = int(rng.integers(1, n + 1))
    q = _clustered(rng, n, d)
    p, g = O.fps(q, m, olib)
    pa, ga, alts, margins, _ = O.fps_adopt(q, m, None, olib)
    np.testing.assert_array_equal(pa, p)
    np.testing.assert_array_equal(ga, g)
    assert np.all(margins == 0.0)
    want, _ = _fps_numpy(O.bf16_to_f64(q), m)
    if np.all(g > 1e-9):  # numpy's fp64 cosines round differently: compare away from fp64 ties
        np.testing.assert_array_equal(pa, want)
    # the runner-up reported at each step is the second-smallest candidate
    for k in range(len(pa) - 1):
        assert alts[k] != pa[k] and (alts[k] >= 0) == np.isfinite(g[k])


@pytest.mark.parametrize("seed", range(6))
def test_fps_adopt_continues_from_a_dictated_pick(olib, seed):
    """Dictating step k's row (here: the runner-up, or any unpicked row) gives the farthest-point sequence
    that numpy's Algorithm 1 takes after the same choice, and reports how far that row lies above the
    minimum."""
    rng = np.random.default_rng(300 + seed)
    n, d = int(rng.integers(6, 25)), 32
    m = int(rng.integers(3, n + 1))
    q = _clustered(rng, n, d)
    x = O.bf16_to_f64(q)
    p, g, alts, _, _ = O.fps_adopt(q, m, None, olib)
    k = int(rng.integers(0, m))
    target = int(alts[k]) if alts[k] >= 0 else int(rng.choice([j for j in range(n) if j not in p[:k]]))
    forced = np.full(m, -1, np.int32)
    forced[k] = target
    pf, gf, _, mf, vf = O.fps_adopt(q, m, forced, olib)
    want, wm = _fps_numpy(x, m, choose=lambda s, v, cand: target if s == k else min(cand, key=lambda j: (v[j], j)))
    assert pf[k] == target
    np.testing.assert_array_equal(pf[:k], p[:k])
    np.testing.assert_allclose(mf, wm, rtol=0, atol=1e-12)
    # the reported candidate values: +inf for rows taken before the step, the minimum at the argmin
    for s in range(len(pf)):
        assert np.all(np.isinf(vf[s][pf[:s]])) and np.isfinite(vf[s][pf[s]])
        np.testing.assert_allclose(vf[s][pf[s]] - vf[s].min(), mf[s], atol=0)
    if np.all(gf > 1e-9):
        np.testing.assert_array_equal(pf, want)


def test_fps_adopt_rejects_invalid_dictated_rows(olib):
    rng = np.random.default_rng(9)
    q = _clustered(rng, 8, 16)
    p, _, _, _, _ = O.fps_adopt(q, 4, None, olib)
    with pytest.raises(ValueError):
        O.fps_adopt(q, 4, np.array([-1, p[0], -1, -1]), olib)   # already picked
    with pytest.raises(ValueError):
        O.fps_adopt(q, 4, np.array([8, -1, -1, -1]), olib)      # out of range


def test_fps_orthonormal_basis_takes_indices_in_order(olib):
    d = 16
    q = _bits(np.eye(d))
    picks, gaps, alts, _, vals = O.fps_adopt(q, d, None, olib)
    np.testing.assert_array_equal(picks, np.arange(d))   # every cosine exact: all ties, lowest index
    np.testing.assert_array_equal(gaps[:-1], 0.0)
    np.testing.assert_array_equal(alts[:-1], np.arange(1, d))
    assert gaps[-1] == np.inf and alts[-1] == -1          # no runner-up for the last pick
    np.testing.assert_array_equal(vals[1:][np.isfinite(vals[1:])], 0.0)  # after the first pick: cosines 0


def test_fps_zero_query_has_zero_similarity(olib):
    rng = np.random.default_rng(7)
    x = np.abs(rng.standard_normal((6, 8))) + 0.1     # positive rows: pairwise cosines > 0
    x[3] = 0.0
    picks, _ = O.fps(_bits(x), 2, olib)
    assert picks[0] == 3                              # average similarity 0 is the smallest


# ---------------------------------------------------------------- the fill-and-compress buffer
def test_cfps_buffer_matches_fp64_brute_force_simulation(olib):
    rng = np.random.default_rng(11)
    d, b_min, b_max = 32, 4, 10
    q = _clustered(rng, 57, d, k=6, sigma=0.5)
    r = O.cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q, olib)
    assert (r["gaps"] > 1e-9).all(), "choose a seed without fp64 near-ties"
    x = O.bf16_to_f64(q)
    cur = []
    for row in x:
        cur.append(row)
        if len(cur) >= b_max:
            sel, _ = _fps_numpy(np.array(cur), b_min)
            cur = [cur[i] for i in sel]
    assert r["size"] == len(cur)
    np.testing.assert_array_equal(O.bf16_to_f64(r["buf"][:r["size"]]), np.array(cur))


def test_cfps_closed_forms(olib):
    rng = np.random.default_rng(12)
    d, b_min, b_max = 16, 3, 7
    q = _clustered(rng, 40, d)
    # before the buffer first fills it is the queries in arrival order
    r = O.cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q[:6], olib)
    assert r["size"] == 6 and len(r["picks"]) == 0
    np.testing.assert_array_equal(r["buf"][:6], q[:6])
    # size cycle: from s0, every (b_max - b_min) arrivals after the first fill compress once
    for s0, n in [(0, 40), (3, 4), (5, 1), (6, 1), (3, 17)]:
        start = q[:s0]
        r = O.cfps_update(start, s0, b_min, b_max, q[s0:s0 + n], olib)
        s, ev = s0, 0
        for _ in range(n):
            s += 1
            if s >= b_max:
                s, ev = b_min, ev + 1
        assert (r["size"], len(r["picks"])) == (s, ev) and O.cfps_events(s0, b_min, b_max, n) == ev
        # every kept row is one of the rows that entered the buffer
        seen = {row.tobytes() for row in np.vstack([start, q[s0:s0 + n]])}
        assert all(row.tobytes() in seen for row in r["buf"][:r["size"]])
        # every compression picks b_min distinct buffer positions
        for p in r["picks"]:
            assert len(set(p.tolist())) == b_min and p.min() >= 0 and p.max() < b_max


# ---------------------------------------------------------------- the near-tie rule of the parity harness
@pytest.mark.parametrize("d", [64, 128])
def test_fp32_cosines_stay_within_the_tie_bound(d):
    """numpy's fp32 cosines (fp32 dot products, fp32 norms and division) differ from the fp64 cosines of
    the same bf16 rows by less than the per-cosine bound (2d + 4) 2^-24 that cfps_tie_bound doubles."""
    rng = np.random.default_rng(d)
    x = O.bf16_to_f64(_clustered(rng, 256, d, k=8, sigma=0.2))
    x32 = x.astype(np.float32)
    n32 = np.sqrt((x32 * x32).sum(1, dtype=np.float32))
    c32 = (x32 @ x32.T) / np.outer(n32, n32).astype(np.float32)
    err = np.abs(c32.astype(np.float64) - _cos64(x)).max()
    assert err <= (2 * d + 4) * 2.0 ** -24
    assert P.cfps_tie_bound(d, 32) == 2.0 * (2 * d + 37) * 2.0 ** -24


def _tied_rows(rng, n, d):
    """Rows with many exact cosine ties: small integer vectors, some repeated."""
    x = rng.integers(-2, 3, size=(n, d)).astype(np.float64)
    for i in range(0, n, 3):
        x[(i + 1) % n] = x[i] * 2.0                     # same direction: cosine ties with everything
    x[np.abs(x).sum(1) == 0, 0] = 1.0
    return x


@pytest.mark.parametrize("seed", range(4))
def test_harness_accepts_a_buffer_that_breaks_near_ties_the_other_way(olib, seed):
    """A numpy Continual FPS whose decisions prefer, among candidates within a quarter of the tie bound of
    the minimum, the highest row (the opposite of the oracle's rule) produces a buffer that the harness
    finds among its near-tie branches, with a departure counted."""
    rng = np.random.default_rng(500 + seed)
    d, b_min, b_max = 16, 4, 10
    x = _tied_rows(rng, 40, d)
    q = _bits(x)
    tau = P.cfps_tie_bound(d, b_max)

    def other_way(k, v, cand):
        lo = min(v[j] for j in cand)
        return max(j for j in cand if v[j] - lo <= tau / 4)

    cur = []
    for row in q:
        cur.append(row)
        if len(cur) >= b_max:
            sel, _ = _fps_numpy(O.bf16_to_f64(np.array(cur)), b_min, choose=other_way)
            cur = [cur[i] for i in sel]
    gpu = np.zeros((b_max, d), np.uint16)
    gpu[:len(cur)] = np.array(cur)
    ties = P.match_cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q, gpu, len(cur), olib, tag="other way")
    assert ties > 0
    # and a single FPS over tied rows: the other-way picks are one of the branches
    rows = q[:12]
    sel, _ = _fps_numpy(O.bf16_to_f64(rows), 6, choose=other_way)
    picks, t = P.match_fps(rows, 6, rows[sel], olib, tag="other way fps")
    assert list(picks) == sel and t > 0


def test_harness_rejects_a_departure_beyond_the_tie_bound(olib):
    """A buffer from a numpy Continual FPS that once takes the runner-up where it lies farther than the tie
    bound above the minimum is rejected."""
    rng = np.random.default_rng(13)
    d, b_min, b_max = 32, 4, 10
    q = _clustered(rng, 10, d, k=6, sigma=0.5)       # one compression
    tau = P.cfps_tie_bound(d, b_max)
    r = O.cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q, olib)
    k = int(np.argmax(r["gaps"][0][:-1] > 10 * tau))   # a step with a clear gap
    assert r["gaps"][0][k] > 10 * tau

    def wrong(s, v, cand):
        order = sorted(cand, key=lambda j: (v[j], j))
        return order[1] if s == k else order[0]

    sel, margins = _fps_numpy(O.bf16_to_f64(q), b_min, choose=wrong)
    assert margins[k] > tau
    gpu = np.zeros((b_max, d), np.uint16)
    gpu[:b_min] = q[sel]
    with pytest.raises(AssertionError):
        P.match_cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q, gpu, b_min, olib, tag="wrong")
    # the fp64 sequence itself passes with no departure
    assert P.match_cfps_update(np.zeros((0, d), np.uint16), 0, b_min, b_max, q, r["buf"], r["size"], olib) == 0
