"""Pins of the oracle's scoring (Eq. 4, Eq. 6 max and mean forms, group aggregation), selection (Eq. 7 and
the keep set of Algorithm 2) and compaction (Eq. 8).

Independent routes: scipy.special.softmax, numpy lexsort, numpy fancy indexing,
closed forms (identical keys, a single query, two-key logistic), invariants
(window kept, exact budget, ordering, key-shift invariance, duplicated and
invalid queries, causal masks with nothing masked) and a hand-computed worked case stored under tests/golden/.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.special import softmax

from oracle import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bits(x: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _rand_case(rng, M, L, d):
    q = O.bf16_to_f64(_bits(rng.standard_normal((M, d)) * 1.5))
    k = _bits(rng.standard_normal((L, d)))
    return q, k


# ------------------------------------------------------------------ score
@pytest.mark.parametrize("M,L,d", [(1, 7, 4), (3, 50, 8), (6, 129, 16), (5, 300, 64)])
def test_score_matches_scipy_softmax_max(olib, M, L, d):
    rng = np.random.default_rng(M * 1000 + L)
    q, k = _rand_case(rng, M, L, d)
    got = O.score(q, np.ones(M, np.int32), k, olib)
    want = softmax(q @ O.bf16_to_f64(k).T / math.sqrt(d), axis=1).max(axis=0)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=0)


def test_score_identical_keys_is_uniform(olib):
    rng = np.random.default_rng(30)
    L, d = 37, 8
    k = np.tile(_bits(rng.standard_normal((1, d))), (L, 1))
    q, _ = _rand_case(rng, 4, 1, d)
    got = O.score(q, np.ones(4, np.int32), k, olib)
    np.testing.assert_allclose(got, 1.0 / L, rtol=1e-13)


def test_score_single_query_sums_to_one_and_ranks_by_dot(olib):
    rng = np.random.default_rng(31)
    q, k = _rand_case(rng, 1, 200, 16)
    s = O.score(q, np.ones(1, np.int32), k, olib)
    assert s.sum() == pytest.approx(1.0, rel=1e-12)
    dots = q[0] @ O.bf16_to_f64(k).T
    np.testing.assert_array_equal(np.argsort(-s, kind="stable"), np.argsort(-dots, kind="stable"))


def test_score_two_key_logistic_closed_form(olib):
    d = 4
    a = 3.0
    q = np.array([[2.0, 0, 0, 0]])             # q . k / sqrt(4) = k_0
    k = _bits(np.array([[a, 0, 0, 0], [0, 5, 0, 0]]))
    s = O.score(q, np.ones(1, np.int32), k, olib)
    assert s[0] == pytest.approx(1.0 / (1.0 + math.exp(-a)), rel=1e-14)
    assert s[1] == pytest.approx(1.0 / (1.0 + math.exp(a)), rel=1e-14)


def test_score_duplicate_and_invalid_queries(olib):
    rng = np.random.default_rng(32)
    q, k = _rand_case(rng, 4, 90, 8)
    base = O.score(q, np.ones(4, np.int32), k, olib)
    dup = O.score(np.vstack([q, q[1:3]]), np.ones(6, np.int32), k, olib)
    np.testing.assert_array_equal(dup, base)
    loud = np.vstack([q, 50.0 * np.ones((1, 8))])
    inv = O.score(loud, np.array([1, 1, 1, 1, 0], np.int32), k, olib)
    np.testing.assert_array_equal(inv, base)
    none = O.score(q, np.zeros(4, np.int32), k, olib)
    np.testing.assert_array_equal(none, 0.0)


def test_score_key_shift_invariance(olib):
    """Adding one vector mu to every key shifts each query's logits by a constant,
    which the softmax removes (exact-arithmetic property, fp64 keys)."""
    rng = np.random.default_rng(33)
    d, L = 8, 64
    k = rng.integers(-8, 8, (L, d)).astype(np.float64) / 4.0      # exact in bf16
    mu = np.array([0.5, -1.0, 0.25, 2.0, 0.0, -0.75, 1.0, 0.5])
    q = rng.integers(-4, 4, (3, d)).astype(np.float64) / 2.0
    s1 = O.score(q, np.ones(3, np.int32), _bits(k), olib)
    s2 = O.score(q, np.ones(3, np.int32), _bits(k + mu), olib)
    np.testing.assert_allclose(s1, s2, rtol=1e-12)


def test_score_permutation_of_queries(olib):
    rng = np.random.default_rng(34)
    q, k = _rand_case(rng, 7, 120, 16)
    perm = rng.permutation(7)
    a = O.score(q, np.ones(7, np.int32), k, olib)
    b = O.score(q[perm], np.ones(7, np.int32), k, olib)
    np.testing.assert_array_equal(a, b)


# ------------------------------------------------------------------ score, mean form of Eq. 6
@pytest.mark.parametrize("M,L,d", [(1, 9, 4), (4, 77, 8), (7, 260, 32)])
def test_score_mean_matches_scipy_softmax_mean(olib, M, L, d):
    rng = np.random.default_rng(7 * M + L)
    q, k = _rand_case(rng, M, L, d)
    valid = np.ones(M, np.int32)
    valid[M // 2] = 0 if M > 1 else 1
    got = O.score(q, valid, k, olib, mean=True)
    w = softmax(q @ O.bf16_to_f64(k).T / math.sqrt(d), axis=1)
    want = w[valid.astype(bool)].mean(axis=0)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=0)


def test_score_mean_closed_forms_and_bounds(olib):
    rng = np.random.default_rng(35)
    q, k = _rand_case(rng, 5, 140, 16)
    one = np.array([0, 0, 1, 0, 0], np.int32)
    # one valid query: mean == max == that query's softmax row, which sums to one
    m1 = O.score(q, one, k, olib, mean=True)
    np.testing.assert_array_equal(m1, O.score(q, one, k, olib))
    assert m1.sum() == pytest.approx(1.0, rel=1e-12)
    # every query's row sums to one, so the mean does too; and the mean never exceeds the max
    allv = np.ones(5, np.int32)
    mean = O.score(q, allv, k, olib, mean=True)
    assert mean.sum() == pytest.approx(1.0, rel=1e-12)
    assert np.all(mean <= O.score(q, allv, k, olib) * (1 + 1e-15))
    # identical keys: every weight is 1 / L
    kk = np.tile(k[:1], (33, 1))
    np.testing.assert_allclose(O.score(q, allv, kk, olib, mean=True), 1.0 / 33, rtol=1e-13)
    # no valid query: all zero
    np.testing.assert_array_equal(O.score(q, np.zeros(5, np.int32), k, olib, mean=True), 0.0)


def test_score_mean_duplicated_query_weights(olib):
    """Duplicating a query counts it twice in the mean (unlike the max)."""
    rng = np.random.default_rng(36)
    q, k = _rand_case(rng, 2, 60, 8)
    w = softmax(q @ O.bf16_to_f64(k).T / math.sqrt(8), axis=1)
    got = O.score(np.vstack([q, q[:1]]), np.ones(3, np.int32), k, olib, mean=True)
    np.testing.assert_allclose(got, (2 * w[0] + w[1]) / 3, rtol=1e-12)


# ------------------------------------------------------------------ causal mask inside the window
@pytest.mark.parametrize("mean", [False, True])
@pytest.mark.parametrize("M,L,d", [(6, 40, 8), (9, 130, 16)])
def test_score_causal_matches_scipy_softmax_over_visible_keys(olib, mean, M, L, d):
    """Each valid query's softmax runs over the keys at or before its position only (scipy over
    the visible logits); masked weights are 0 and still count in the mean."""
    rng = np.random.default_rng(11 * M + L + mean)
    q, k = _rand_case(rng, M, L, d)
    valid = np.ones(M, np.int32)
    valid[1] = 0
    kpos = np.sort(rng.integers(0, 3 * L, L)).astype(np.int64)
    qpos = rng.integers(kpos[0], kpos[-1] + 2, M).astype(np.int64)
    got = O.score(q, valid, k, olib, mean=mean, qpos=qpos, kpos=kpos)
    lg = q @ O.bf16_to_f64(k).T / math.sqrt(d)
    w = np.zeros((M, L))
    for i in range(M):
        vis = kpos <= qpos[i]
        if vis.any():
            w[i, vis] = softmax(lg[i, vis])
    rows = w[valid.astype(bool)]
    want = rows.mean(axis=0) if mean else rows.max(axis=0)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=0)


def test_score_causal_closed_forms(olib):
    """Keys at positions 0, 1, 2.  A query at position 0 sees only key 0 (weight 1); a zero query at
    position 2 sees all three (weights 1/3).  Max: [1, 1/3, 1/3]; mean: [2/3, 1/6, 1/6]."""
    d = 8
    q = np.zeros((2, d))
    q[0] = O.bf16_to_f64(_bits(np.linspace(-2.0, 3.0, d)))
    k = _bits(np.random.default_rng(3).standard_normal((3, d)))
    qpos, kpos = np.array([0, 2], np.int64), np.array([0, 1, 2], np.int64)
    v = np.ones(2, np.int32)
    np.testing.assert_allclose(O.score(q, v, k, olib, qpos=qpos, kpos=kpos), [1.0, 1 / 3, 1 / 3], rtol=1e-14)
    np.testing.assert_allclose(O.score(q, v, k, olib, mean=True, qpos=qpos, kpos=kpos), [2 / 3, 1 / 6, 1 / 6],
                               rtol=1e-14)


def test_score_causal_without_masked_pairs_is_unmasked_and_positions_follow_the_window(olib):
    """Every query at or after every key: bit-equal to the unmasked score.  causal_positions puts recent
    slot w at recent_pos[w], beacons at t and window key j at t - (L - 1 - j)."""
    rng = np.random.default_rng(5)
    q, k = _rand_case(rng, 7, 90, 16)
    v = np.ones(7, np.int32)
    kpos = np.arange(90, dtype=np.int64)
    qpos = np.full(7, 89, np.int64) + rng.integers(0, 3, 7)
    for mean in (False, True):
        np.testing.assert_array_equal(O.score(q, v, k, olib, mean=mean, qpos=qpos, kpos=kpos),
                                      O.score(q, v, k, olib, mean=mean))
    qp, kp = O.causal_positions(G=2, W=3, nb=1, recent_pos=[97, 98, 99], t_pos=99, L=10)
    np.testing.assert_array_equal(qp, [97, 98, 99, 97, 98, 99, 99])
    assert np.all(kp[:7] < 0) and list(kp[7:]) == [97, 98, 99]


# ------------------------------------------------------------------ select
def _select_lexsort(score, budget, W, npre):
    L = len(score)
    if L <= budget:
        return np.arange(L)
    keep = list(range(npre)) + list(range(L - W, L))
    cand = np.arange(npre, L - W)
    order = np.lexsort((cand, -score[cand]))          # score desc, index asc
    top = cand[order[: budget - len(keep)]]
    return np.sort(np.concatenate([keep, top]).astype(np.int64))


@pytest.mark.parametrize("L,budget,W,npre", [(50, 20, 4, 0), (130, 100, 8, 3), (64, 12, 12, 0),
                                             (40, 40, 4, 0), (30, 60, 4, 1), (200, 9, 8, 1)])
def test_select_matches_lexsort_and_invariants(olib, L, budget, W, npre):
    rng = np.random.default_rng(L + budget)
    score = rng.random(L)
    score[rng.integers(0, L, 5)] = 0.5                 # some exact ties
    kept, bd = O.select(score, budget, W, npre, olib)
    np.testing.assert_array_equal(kept, _select_lexsort(score, budget, W, npre))
    assert len(kept) == min(L, budget)
    assert np.all(np.diff(kept) > 0)
    if L > budget:
        assert set(range(L - W, L)) <= set(kept.tolist())
        assert set(range(npre)) <= set(kept.tolist())
        cand = np.setdiff1d(np.arange(npre, L - W), [])
        taken = np.intersect1d(kept, cand)
        left = np.setdiff1d(cand, kept)
        if len(taken) and len(left):
            assert score[taken].min() >= score[left].max()
            assert bd[0] == score[taken].min() and bd[1] == score[left].max()


def test_select_all_ties_take_lowest_indices(olib):
    kept, _ = O.select(np.full(20, 0.25), 8, 3, 0, olib)
    np.testing.assert_array_equal(kept, [0, 1, 2, 3, 4, 17, 18, 19])


def test_select_budget_below_keep_set_is_rejected(olib):
    with pytest.raises(ValueError):
        O.select(np.ones(30), 5, 4, 2, olib)


# ------------------------------------------------------------------ gather
def test_gather_is_row_indexing(olib):
    rng = np.random.default_rng(40)
    K = rng.integers(0, 65535, (30, 8), dtype=np.uint16)
    V = rng.integers(0, 65535, (30, 8), dtype=np.uint16)
    kept = np.sort(rng.choice(30, 12, replace=False)).astype(np.int32)
    K2, V2 = K.copy(), V.copy()
    O.gather(K2, V2, kept, olib)
    np.testing.assert_array_equal(K2[:12], K[kept])
    np.testing.assert_array_equal(V2[:12], V[kept])
    np.testing.assert_array_equal(K2[12:], K[12:])
    np.testing.assert_array_equal(V2[12:], V[12:])


# ------------------------------------------------------------------ worked case
def test_golden_worked_case(olib):
    """Hand-computed case (tests/golden/worked_case.json): one query, no rotation,
    logits 0, 1, 2, 0, -1 give softmax weights proportional to 1, e, e^2, 1, e^-1."""
    with open(os.path.join(GOLDEN, "worked_case.json")) as f:
        g = json.load(f)
    d = g["head_dim"]
    q_recent = _bits(np.array(g["q_recent"], np.float64).reshape(1, 1, d))
    k = _bits(np.array(g["K"], np.float64))
    qobs, valid = O.build_qobs(np.zeros((0, d), np.float32), np.zeros(0, np.int64), q_recent,
                               np.array([g["t_pos"]], np.int64), g["t_pos"], 0.0, olib)
    s = O.score(qobs, valid, k, olib)
    np.testing.assert_allclose(s, g["score"], rtol=1e-15)
    kept, _ = O.select(s, g["budget"], g["window"], 0, olib)
    np.testing.assert_array_equal(kept, g["kept"])


# ------------------------------------------------------------------ whole-step driver
def test_step_many_equals_per_instance_calls_and_is_thread_independent(olib, monkeypatch):
    rng = np.random.default_rng(50)
    n_inst, G, d, nb, W, L, budget, n_new, cap = 5, 2, 16, 3, 4, 70, 50, 6, 72
    theta, t_pos = 10000.0, 69
    q_new = _bits(rng.standard_normal((n_inst, G, n_new, d)) * 4)
    q_recent = _bits(rng.standard_normal((n_inst, G, W, d)) * 4)
    K = _bits(rng.standard_normal((n_inst, cap, d)))
    V = _bits(rng.standard_normal((n_inst, cap, d)))
    pos = np.arange(t_pos - W + 1, t_pos + 1)
    states = [O.init_beacons(_bits(rng.standard_normal((G * 8, d))), nb, olib) for _ in range(n_inst)]
    cent = np.stack([s["cent"] for s in states])
    sums = np.stack([s["sums"] for s in states])
    counts = np.stack([s["counts"] for s in states])

    # per-instance reference through the individual functions
    Kr, Vr = K.copy(), V.copy()
    kept_r = np.zeros((n_inst, budget), np.int32)
    for e in range(n_inst):
        st = {k: v.copy() for k, v in states[e].items()}
        O.update(q_new[e].reshape(G * n_new, d), st, lib=olib)
        qo, va = O.build_qobs(st["cent"], st["counts"], q_recent[e], pos, t_pos, theta, olib)
        s = O.score(qo, va, Kr[e, :L], olib)
        kp, _ = O.select(s, budget, W, 0, olib)
        kk, vv = Kr[e].copy(), Vr[e].copy()
        O.gather(kk, vv, kp, olib)
        Kr[e], Vr[e] = kk, vv
        kept_r[e] = kp
        states[e] = st

    outs = []
    for inst_order in (np.arange(n_inst), np.array([3, 0, 4, 1, 2])):
        K2, V2 = K.copy(), V.copy()
        c2, s2, n2 = cent.copy(), sums.copy(), counts.copy()
        kept = np.zeros((n_inst, budget), np.int32)
        threads = O.step_many(inst_order, G=G, d=d, nb=nb, W=W, n_prefix=0, cap=cap, q_new=q_new, n_new=n_new,
                              q_recent=q_recent, recent_pos=pos, t_pos=t_pos, theta=theta, L=L, budget=budget,
                              K=K2, V=V2, cent=c2, sums=s2, counts=n2, kept=kept, lib=olib)
        assert threads >= 1
        outs.append((K2, V2, kept, c2))
    for K2, V2, kept, c2 in outs:
        np.testing.assert_array_equal(kept, kept_r)
        np.testing.assert_array_equal(K2, Kr)
        np.testing.assert_array_equal(V2, Vr)
        np.testing.assert_array_equal(c2, np.stack([s["cent"] for s in states]))
