"""Pins of the oracle's beacon maintenance: FPS (Algorithm 1), FPS seeding, and the
nearest-beacon running-mean update.

Independent routes used here: a max-min brute force over scipy's cosine
distance matrix for FPS, orthonormal-basis closed forms, numpy means recomputed
from the reported assignment, and permutation invariance.
"""
import numpy as np
import pytest
import torch
from scipy.spatial.distance import cdist

from oracle import oracle as O


def _bits(x: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _cos_matrix(x: np.ndarray) -> np.ndarray:
    return 1.0 - cdist(x, x, metric="cosine")


def _fps_brute(x: np.ndarray, m: int):
    """FPS by its max-min characterisation: every pick after the first minimises
    the largest cosine to the already-picked set (recomputed from scratch)."""
    C = _cos_matrix(x)
    picks = [int(np.argmin(C.mean(axis=1)))]
    while len(picks) < m:
        rest = [j for j in range(len(x)) if j not in picks]
        worst = [C[j, picks].max() for j in rest]
        picks.append(rest[int(np.argmin(worst))])
    return picks


# ------------------------------------------------------------------ FPS
def test_fps_orthonormal_basis_ties_go_to_lowest_index(olib):
    d = 8
    x = np.eye(d)[:6] * np.array([1, 2, 3, 4, 5, 6])[:, None]  # scaling does not change cosines
    picks, gaps = O.fps(_bits(x), 4, olib)
    np.testing.assert_array_equal(picks, [0, 1, 2, 3])
    assert gaps[0] == 0.0 and gaps[1] == 0.0  # every choice was a tie


def test_fps_outlier_first(olib):
    rng = np.random.default_rng(10)
    base = rng.standard_normal(16)
    x = base + 0.05 * rng.standard_normal((7, 16))
    x = np.vstack([x[:3], -base, x[3:]])  # the outlier sits at row 3
    picks, _ = O.fps(_bits(x), 2, olib)
    assert picks[0] == 3


@pytest.mark.parametrize("seed", range(6))
def test_fps_matches_maxmin_brute_force(olib, seed):
    rng = np.random.default_rng(100 + seed)
    n, d, m = int(rng.integers(5, 12)), int(rng.integers(2, 9)), 0
    m = int(rng.integers(1, n + 1))
    x = rng.standard_normal((n, d)) * rng.uniform(0.1, 5, (n, 1))
    bits = _bits(x)
    picks, gaps = O.fps(bits, m, olib)
    want = _fps_brute(O.bf16_to_f64(bits), m)
    if np.all(gaps > 1e-12):
        np.testing.assert_array_equal(picks, want)
    assert len(set(picks.tolist())) == len(picks)


def test_fps_selected_similarity_is_non_decreasing(olib):
    rng = np.random.default_rng(11)
    x = rng.standard_normal((40, 16))
    picks, _ = O.fps(_bits(x), 12, olib)
    C = _cos_matrix(O.bf16_to_f64(_bits(x)))
    s = [C[picks[k], picks[:k]].max() for k in range(1, len(picks))]
    assert all(b >= a - 1e-12 for a, b in zip(s, s[1:]))


def test_fps_permutation_equivariant(olib):
    rng = np.random.default_rng(12)
    x = rng.standard_normal((20, 8))
    bits = _bits(x)
    picks, gaps = O.fps(bits, 6, olib)
    assert np.all(gaps > 1e-9)
    perm = rng.permutation(20)
    picks_p, _ = O.fps(bits[perm], 6, olib)
    np.testing.assert_array_equal(perm[picks_p], picks)


def test_fps_m_larger_than_n(olib):
    x = np.eye(4)
    picks, _ = O.fps(_bits(x), 10, olib)
    assert sorted(picks.tolist()) == [0, 1, 2, 3]


def test_init_beacons_seeds(olib):
    rng = np.random.default_rng(13)
    bits = _bits(rng.standard_normal((12, 8)))
    st = O.init_beacons(bits, 3, olib)
    picks, _ = O.fps(bits, 3, olib)
    np.testing.assert_array_equal(st["picks"], picks)
    np.testing.assert_array_equal(st["counts"], [1, 1, 1])
    np.testing.assert_array_equal(st["sums"], O.bf16_to_f64(bits[picks]))
    np.testing.assert_array_equal(st["cent"], O.bf16_to_f64(bits[picks]).astype(np.float32))
    with pytest.raises(ValueError):
        O.init_beacons(bits[:2], 3, olib)


# ------------------------------------------------------------------ update
def _state(cent, counts=None):
    cent = np.asarray(cent, np.float32)
    counts = np.ones(len(cent), np.int64) if counts is None else np.asarray(counts, np.int64)
    return dict(cent=cent.copy(), sums=cent.astype(np.float64) * counts[:, None], counts=counts.copy())


def test_update_single_beacon_is_global_mean(olib):
    rng = np.random.default_rng(20)
    seed = _bits(rng.standard_normal((1, 16)))
    st = O.init_beacons(seed, 1, olib)
    allq = [O.bf16_to_f64(seed)]
    for _ in range(3):
        q = _bits(rng.standard_normal((9, 16)))
        assign, _ = O.update(q, st, lib=olib)
        np.testing.assert_array_equal(assign, 0)
        allq.append(O.bf16_to_f64(q))
    allq = np.vstack(allq)
    assert st["counts"][0] == len(allq)
    np.testing.assert_allclose(st["sums"][0], allq.sum(axis=0), rtol=0, atol=1e-12)
    np.testing.assert_array_equal(st["cent"][0], (allq.sum(axis=0) / len(allq)).astype(np.float32))


def test_update_planted_assignment_uses_cosine_not_dot(olib):
    e = np.eye(4)
    # beacon 0 is long but points along e0; beacon 1 is short and points along e1
    st = _state([100.0 * e[0], 0.5 * e[1], 0.5 * e[2]])
    q = _bits(np.array([e[1] + 0.3 * e[0], e[0], 2 * e[2] - 0.1 * e[1], e[1] * 7]))
    assign, margin = O.update(q, st, lib=olib)
    np.testing.assert_array_equal(assign, [1, 0, 2, 1])
    assert np.all(margin > 0)


def test_update_centroid_is_mean_of_assigned(olib):
    rng = np.random.default_rng(21)
    d, nb = 16, 4
    st = _state(rng.standard_normal((nb, d)))
    prior_sums, prior_counts = st["sums"].copy(), st["counts"].copy()
    prior_cent = st["cent"].astype(np.float64)
    q = _bits(rng.standard_normal((50, d)))
    assign, _ = O.update(q, st, lib=olib)
    x = O.bf16_to_f64(q)
    C = 1.0 - cdist(x, prior_cent, "cosine")
    np.testing.assert_array_equal(assign, C.argmax(axis=1))  # call-start centroids decide
    for b in range(nb):
        m = assign == b
        assert st["counts"][b] == prior_counts[b] + m.sum()
        tot = prior_sums[b] + x[m].sum(axis=0)
        np.testing.assert_allclose(st["sums"][b], tot, rtol=0, atol=1e-12)
        np.testing.assert_array_equal(st["cent"][b], (st["sums"][b] / st["counts"][b]).astype(np.float32))


def test_update_permutation_invariant(olib):
    rng = np.random.default_rng(22)
    d, nb = 16, 5
    st0 = _state(rng.standard_normal((nb, d)))
    q = _bits(rng.standard_normal((40, d)))
    st1 = {k: v.copy() for k, v in st0.items()}
    st2 = {k: v.copy() for k, v in st0.items()}
    a1, _ = O.update(q, st1, lib=olib)
    perm = rng.permutation(40)
    a2, _ = O.update(q[perm], st2, lib=olib)
    np.testing.assert_array_equal(a2, a1[perm])
    for k in st1:
        np.testing.assert_array_equal(st1[k], st2[k])


def test_update_zero_query_and_empty_beacon(olib):
    e = np.eye(4)
    st = _state([e[0], e[1]], counts=[1, 0])
    q = _bits(np.array([np.zeros(4), e[1], e[0]]))
    assign, margin = O.update(q, st, lib=olib)
    np.testing.assert_array_equal(assign, [-1, 0, 0])   # count-0 beacon never qualifies
    assert np.isinf(margin[0]) and np.isinf(margin[1])
    assert st["counts"].tolist() == [3, 0]


def test_update_ties_go_to_lowest_beacon(olib):
    e = np.eye(4)
    st = _state([e[0] + e[1], e[0] + e[1], e[2]])
    assign, margin = O.update(_bits(np.array([e[0] + e[1]])), st, lib=olib)
    assert assign[0] == 0 and margin[0] == 0.0


def test_update_override_drives_accumulation(olib):
    e = np.eye(4)
    st = _state([e[0], e[1]])
    q = _bits(np.array([e[0], e[0]]))
    assign, _ = O.update(q, st, override=np.array([1, 1], np.int32), lib=olib)
    np.testing.assert_array_equal(assign, [0, 0])        # still reports its own argmax
    assert st["counts"].tolist() == [1, 3]
    np.testing.assert_allclose(st["sums"][1], 2 * e[0] + e[1])
