"""Parity harness: the CUDA path (through the C ABI) against the fp64 oracle.

Tolerances:
  * FPS seeds and beacon assignments: identical, except where the oracle's own
    decision was a tie (runner-up within 1e-12), where either choice is valid;
  * beacon state after an update: counts exact, sums within 1e-12 relative,
    centroids within 1e-5 relative to |c| (absolute when |c| < 1);
  * scores: within 1e-3 relative of the oracle's fp64 scores, plus 2^-126
    absolute (fp32 holds no smaller normal value: scores below it cannot keep a
    relative precision);
  * kept index sets: identical except for candidates whose oracle score is
    within 1e-5 relative of the oracle's boundary score (the score of the last
    candidate it took); the GPU set must still hold exactly `budget` rows,
    be strictly ascending and contain the keep set;
  * compacted K / V: byte-identical to the pre-compress rows the GPU kept, in
    every instance, and rows [budget, capacity) of every instance byte-unchanged
    (checked on the device for all instances, sampled or not); score entries
    at or past L untouched;
  * Continual FPS buffers, beacons and merges (Eq. 9, Algorithm 1 in fp64):
    the GPU takes its FPS decisions from fp32 similarities, so at a step
    where the oracle's fp64 runner-up lies within cfps_tie_bound(d, n) of the
    minimum either row is a valid pick; the harness searches those branches
    (the oracle adopting the other row and continuing from it) and the GPU's
    rows must equal one of them exactly.  The departures are counted as ties.
The compress comparison feeds both sides the same inputs, including the
beacon state the GPU produced (after that state passed its own check).
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

from oracle import oracle as O
from paper_2609_04971_gb300 import synth
from paper_2609_04971_gb300.bkv import BeaconKV
from paper_2609_04971_gb300.workloads import Workload

SCORE_RTOL = 1e-3
SCORE_ATOL = 2.0 ** -126
TIE_RTOL = 1e-5
CENT_TOL = 1e-5
ASSIGN_TIE = 1e-12
BRANCH_LIMIT = 256


def cfps_tie_bound(d: int, n: int) -> float:
    """Largest fp64 gap at which an FPS decision taken from fp32 similarities may differ from the fp64 one.
    An fp32 cosine - a d-term fp32 dot product divided by the product of two fp32 norms, each the square
    root of a d-term fp32 dot product - is within (2d + 4) 2^-24 of the exact cosine (a d-term sum has
    relative error at most d 2^-24 of the sum of magnitudes, bounded by |a| |b|; each norm adds half of
    that plus one rounding, the product and the division one each); the first pick's average of n such
    cosines adds (n + 1) 2^-24 (the fp32 sum and the division).  Two candidates' order can flip only when
    their exact values are within twice the larger of these errors."""
    return 2.0 * (2 * d + 4 + n + 1) * 2.0 ** -24


def search_branches(run, tau: float, limit: int = BRANCH_LIMIT):
    """Every outcome of a sequence of FPS decisions that an implementation deciding from similarities
    within tau / 2 of the fp64 ones may reach: run(forced) evaluates the sequence with forced[k] >= 0
    dictating decision k (-1: the fp64 argmin) and returns (result, picks, vals) with vals[k] the values
    decision k minimises over the candidate rows (+inf for rows no longer candidates).  At every
    undictated decision each other row within tau of the minimum is tried too, the oracle continuing from
    it.  Yields (result, number of departures from the argmin)."""
    _, picks, _ = run(None)
    n = len(picks)
    stack = [np.full(n, -1, np.int32)]
    seen = 0
    while stack:
        forced = stack.pop()
        res, picks, vals = run(forced)
        taken = forced >= 0
        for k in np.flatnonzero(taken):
            assert vals[k][forced[k]] - vals[k].min() <= tau, "a dictated pick lies beyond the tie bound"
        yield res, int(taken.sum())
        seen += 1
        assert seen <= limit, f"more than {limit} near-tie branches"
        last = int(np.flatnonzero(taken).max()) if taken.any() else -1
        for k in range(last + 1, n):
            lo = vals[k].min()
            for j in np.flatnonzero(vals[k] - lo <= tau):
                if j != picks[k]:
                    f = forced.copy()
                    f[k] = j
                    stack.append(f)


def fps_branches(rows: np.ndarray, m: int, lib, d: int | None = None):
    """The pick sequences of fp64 FPS over `rows` (uint16 [N, d]) that fp32 decisions may produce."""
    d = rows.shape[-1] if d is None else d
    tau = cfps_tie_bound(d, rows.shape[0])

    def run(forced):
        picks, _, _, _, vals = O.fps_adopt(rows, m, forced, lib)
        return picks, picks, vals

    return search_branches(run, tau)


def match_fps(rows: np.ndarray, m: int, gpu_rows: np.ndarray, lib, tag: str = "") -> tuple:
    """The FPS branch (over rows) whose selected rows, in pick order, equal gpu_rows.  Returns (picks, ties)."""
    for picks, ties in fps_branches(rows, m, lib):
        if len(picks) == len(gpu_rows) and np.array_equal(rows[picks], gpu_rows):
            return picks, ties
    picks, gaps = O.fps(rows, m, lib)
    raise AssertionError(f"{tag}: no fp64 FPS branch gives the GPU's rows (fp64 picks {picks.tolist()}, "
                         f"gaps {np.array2string(gaps, precision=2)})")


def match_cfps_update(buf: np.ndarray, size: int, b_min: int, b_max: int, q_new: np.ndarray, gpu_buf: np.ndarray,
                      gpu_size: int, lib, tag: str = "") -> int:
    """A Continual FPS update of one head (Eq. 9, fp64 Algorithm 1) from the buffer the GPU started from:
    the GPU's buffer after the call must equal the oracle's on one near-tie branch.  Returns the ties."""
    d = q_new.shape[-1]
    tau = cfps_tie_bound(d, b_max)
    n_ev = O.cfps_events(int(size), b_min, b_max, q_new.shape[0])

    def run(forced):
        r = O.cfps_update(buf, int(size), b_min, b_max, q_new, lib,
                          forced=None if forced is None or forced.size == 0 else forced.reshape(n_ev, b_min))
        k = n_ev * b_min
        return (r["size"], r["buf"]), r["picks"].reshape(-1)[:k], r["vals"].reshape(-1, b_max)[:k]

    first = None
    for (sz, want), ties in search_branches(run, tau):
        first = (sz, want) if first is None else first
        if sz == gpu_size and np.array_equal(gpu_buf[:sz], want[:sz]):
            return ties
    sz, want = first
    assert gpu_size == sz, f"{tag}: buffer size {gpu_size} vs {sz}"
    bad = [i for i in range(sz) if not np.array_equal(gpu_buf[i], want[i])]
    raise AssertionError(f"{tag}: buffer rows {bad} differ from every fp64 near-tie branch")


@dataclasses.dataclass
class GpuRun:
    wl: Workload
    inputs: dict
    cent0: np.ndarray
    sums0: np.ndarray
    counts0: np.ndarray
    assign: np.ndarray
    cent1: np.ndarray
    sums1: np.ndarray
    counts1: np.ndarray
    kept: np.ndarray
    scores: np.ndarray | None
    K_before: np.ndarray   # uint16 bits [n_inst, cap, d] (host copy, sampled instances only)
    V_before: np.ndarray
    K_after: np.ndarray
    V_after: np.ndarray
    sample: np.ndarray     # instance ids copied to the host
    mean_agg: bool = False  # Eq. 6 mean form instead of the max
    causal: bool = False    # causal mask inside the recent window
    canary: dict = dataclasses.field(default_factory=dict)  # whole-buffer checks made on the device


def device_canaries(K0: torch.Tensor, V0: torch.Tensor, K1: torch.Tensor, V1: torch.Tensor, kept: torch.Tensor,
                    scores: torch.Tensor | None, L: int, budget: int) -> dict:
    """Whole-buffer checks of one compress on the device, every instance: rows [0, budget) are the
    pre-compress rows at the kept indices (all rows untouched when L <= budget), rows [budget, capacity)
    are byte-unchanged, and score entries at or past L keep the -1 they were filled with."""
    n_inst, cap, d = K0.shape[0] * K0.shape[1] * K0.shape[2], K0.shape[3], K0.shape[4]
    k0, v0 = K0.reshape(n_inst, cap, d), V0.reshape(n_inst, cap, d)
    k1, v1 = K1.reshape(n_inst, cap, d), V1.reshape(n_inst, cap, d)
    out = {}
    if L <= budget:
        out["untouched"] = bool(torch.equal(k1, k0) and torch.equal(v1, v0))
    else:
        idx = kept.reshape(n_inst, budget).long().clamp(0, cap - 1)
        g = idx[:, :, None].expand(n_inst, budget, d)
        out["gathered"] = bool(torch.equal(k1[:, :budget].view(torch.int16), k0.gather(1, g).view(torch.int16)) and
                               torch.equal(v1[:, :budget].view(torch.int16), v0.gather(1, g).view(torch.int16)))
        out["tail_unchanged"] = bool(torch.equal(k1[:, budget:].view(torch.int16), k0[:, budget:].view(torch.int16))
                                     and torch.equal(v1[:, budget:].view(torch.int16), v0[:, budget:].view(torch.int16)))
    if scores is not None:
        out["scores_past_L"] = bool((scores.reshape(n_inst, cap)[:, L:] == -1.0).all())
    return out


def _inst_rows(t: torch.Tensor, wl: Workload) -> torch.Tensor:
    """[layers, batch, heads, n, d] -> [n_inst, G * n, d] (group-major), query tensors only."""
    nl, B, Hq, n, d = t.shape
    return t.reshape(nl * B * wl.n_kv_heads, wl.group * n, d)


def run_gpu(wl: Workload, seed: int = 0, sample=None, with_scores: bool = True, inputs: dict | None = None,
            L: int | None = None, budget: int | None = None, mean_agg: bool = False, causal: bool = False) -> GpuRun:
    dev = torch.device("cuda")
    inp = inputs or synth.step_inputs(wl, seed, dev)
    L = wl.L if L is None else L
    budget = wl.budget if budget is None else budget
    n_inst = wl.n_inst
    sample = np.arange(n_inst) if sample is None else np.asarray(sample)
    sidx = torch.as_tensor(sample, device=dev)

    bk = BeaconKV.for_workload(wl, mean_agg=mean_agg, causal_window=causal)
    try:
        bk.init_beacons(inp["q_init"])
        c0, s0, n0 = [x.cpu().numpy() for x in bk.state()]
        assign = torch.full((wl.n_layers, wl.batch, wl.n_q_heads, wl.n_new), -7, dtype=torch.int32, device=dev)
        bk.update(inp["q_new"], assign)
        c1, s1, n1 = [x.cpu().numpy() for x in bk.state()]
        K, V = inp["K"], inp["V"]
        Kf = K.view(n_inst, wl.capacity, wl.head_dim)
        Vf = V.view(n_inst, wl.capacity, wl.head_dim)
        K_before = Kf.index_select(0, sidx).view(torch.int16).cpu().numpy().view(np.uint16)
        V_before = Vf.index_select(0, sidx).view(torch.int16).cpu().numpy().view(np.uint16)
        scores = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads, wl.capacity), -1.0, device=dev) \
            if with_scores else None
        K0, V0 = K.clone(), V.clone()
        kept = bk.compress(K, V, L=L, budget=budget, t_pos=inp["t_pos"], q_recent=inp["q_recent"],
                           recent_pos=inp["recent_pos"], scores_out=scores)
        bk.sync()
        canary = device_canaries(K0, V0, K, V, kept, scores, L, budget)
        del K0, V0
        K_after = Kf.index_select(0, sidx).view(torch.int16).cpu().numpy().view(np.uint16)
        V_after = Vf.index_select(0, sidx).view(torch.int16).cpu().numpy().view(np.uint16)
    finally:
        bk.close()
    return GpuRun(wl=wl, inputs=inp, cent0=c0, sums0=s0, counts0=n0,
                  assign=assign.view(n_inst, -1).cpu().numpy(), cent1=c1, sums1=s1, counts1=n1,
                  kept=kept.view(n_inst, -1).cpu().numpy(),
                  scores=None if scores is None else scores.view(n_inst, -1).cpu().numpy(),
                  K_before=K_before, V_before=V_before, K_after=K_after, V_after=V_after, sample=sample,
                  mean_agg=mean_agg, causal=causal, canary=canary)


@dataclasses.dataclass
class Report:
    instances: int = 0
    fps_ties: int = 0
    assign_ties: int = 0
    max_cent_err: float = 0.0
    max_score_rel: float = 0.0
    boundary_swaps: int = 0

    def merge(self, o: "Report"):
        self.instances += o.instances
        self.fps_ties += o.fps_ties
        self.assign_ties += o.assign_ties
        self.max_cent_err = max(self.max_cent_err, o.max_cent_err)
        self.max_score_rel = max(self.max_score_rel, o.max_score_rel)
        self.boundary_swaps += o.boundary_swaps


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def logit_tie_rtol(qobs: np.ndarray, valid: np.ndarray, K: np.ndarray) -> float:
    """Score margin (relative) below which fp32 scoring may order two keys either way, for inputs whose
    logits are far from unit spread: the fp32 sum of d exact bf16 products has error at most d 2^-24 of
    the sum of the products' magnitudes, times 1/sqrt(d) on the natural-log scale; the base-2 logits, the
    log-sum-exp and the log-scores are held in fp32 (2^-24 of each magnitude, the log-sum-exp also
    of log2 L).  Twice their sum, never below the default 1e-5."""
    d = K.shape[-1]
    q = np.abs(qobs[valid.astype(bool)])
    if q.size == 0:
        return TIE_RTOL
    k = O.bf16_to_f64(K)
    mag = (q @ np.abs(k).T).max()
    dots = (qobs[valid.astype(bool)] @ k.T) / np.sqrt(d) * np.log2(np.e)
    y_abs = np.abs(dots).max()
    spread = dots.max() - dots.min()
    err_nat = (d + 2) * 2.0 ** -24 * mag / np.sqrt(d)
    err_log2 = 2.0 ** -24 * (3 * y_abs + spread + 2 * np.log2(K.shape[0]))
    return max(TIE_RTOL, 2.0 * (err_nat + np.log(2.0) * err_log2))


def check_instance(run: GpuRun, k: int, L: int | None = None, budget: int | None = None, lib=None,
                   tie_rtol=None) -> Report:
    """Checks sampled instance number k (position in run.sample) against the oracle."""
    wl = run.wl
    lib = lib or O.load()
    e = int(run.sample[k])
    L = wl.L if L is None else L
    budget = wl.budget if budget is None else budget
    G, d, nb, W = wl.group, wl.head_dim, wl.n_beacons, wl.window
    rep = Report(instances=1)
    inp = run.inputs

    q_init = _bits(_inst_rows(inp["q_init"], wl)[e])
    q_new = _bits(_inst_rows(inp["q_new"], wl)[e])
    q_recent = _bits(inp["q_recent"].reshape(wl.n_inst, G, W, d)[e]) if W > 0 else np.zeros((G, 0, d), np.uint16)

    # ---- FPS seeding
    if nb > 0:
        st = O.init_beacons(q_init, nb, lib)
        if not np.array_equal(st["cent"], run.cent0[e]):
            # which query did the GPU pick at each slot?
            x = O.bf16_to_f64(q_init).astype(np.float32)
            gpu_picks = [int(np.flatnonzero((x == run.cent0[e][s]).all(axis=1))[0]) for s in range(nb)]
            first = next(s for s in range(nb) if gpu_picks[s] != st["picks"][s])
            assert st["gaps"][first] < ASSIGN_TIE, \
                f"instance {e}: FPS pick {first} differs (gpu {gpu_picks[first]}, oracle {st['picks'][first]}, " \
                f"gap {st['gaps'][first]:.3e})"
            rep.fps_ties += 1
        else:
            np.testing.assert_array_equal(run.sums0[e], st["sums"])
            np.testing.assert_array_equal(run.counts0[e], st["counts"])
        # ---- update, from the GPU's seed state
        pre = dict(cent=run.cent0[e].copy(), sums=run.sums0[e].copy(), counts=run.counts0[e].copy())
        post = dict(cent=run.cent1[e], sums=run.sums1[e], counts=run.counts1[e])
        ties, cerr = check_update(q_new, pre, run.assign[e], post, lib, tag=f"instance {e}")
        rep.assign_ties += ties
        rep.max_cent_err = cerr

    # ---- compress, on the GPU's beacon state
    rel, swaps = check_compress(wl, run.cent1[e], run.counts1[e], q_recent, inp["recent_pos"], inp["t_pos"],
                                run.K_before[k], run.V_before[k], run.K_after[k], run.V_after[k], run.kept[e],
                                None if run.scores is None else run.scores[e], L, budget, lib, tag=f"instance {e}",
                                mean=run.mean_agg, causal=run.causal, tie_rtol=tie_rtol)
    rep.max_score_rel = rel
    rep.boundary_swaps += swaps
    return rep


def check_run(run: GpuRun, L=None, budget=None, tie_rtol=None) -> Report:
    """Every sampled instance against the oracle.  tie_rtol: the kept-set tie margin (default 1e-5), or
    "fp32-bound" for logit_tie_rtol of each instance's own scoring queries and keys."""
    bad = [k for k, ok in run.canary.items() if not ok]
    assert not bad, f"whole-buffer checks failed on the device: {bad}"
    rep = Report()
    lib = O.load()
    for k in range(len(run.sample)):
        rep.merge(check_instance(run, k, L=L, budget=budget, lib=lib, tie_rtol=tie_rtol))
    return rep


def check_update(q_new: np.ndarray, pre: dict, assign_g: np.ndarray, post: dict, lib, tag: str = "") -> tuple:
    """One beacon update of one instance from state `pre` (fp32 centroids, fp64 sums, int64 counts):
    the GPU's assignments must equal the oracle's except at oracle ties (runner-up within 1e-12), and
    the GPU's state `post` must equal the oracle's state after the GPU's own assignments.
    Returns (ties, centroid error)."""
    st = {kk: v.copy() for kk, v in pre.items()}
    a_o, margin = O.update(q_new, st, lib=lib)
    diff = np.flatnonzero(a_o != assign_g)
    ties = 0
    if diff.size:
        bad = diff[margin[diff] >= ASSIGN_TIE]
        assert bad.size == 0, f"{tag}: {bad.size} assignments differ beyond ties, e.g. query " \
                              f"{bad[0]}: gpu {assign_g[bad[0]]} oracle {a_o[bad[0]]} margin {margin[bad[0]]:.3e}"
        ties = diff.size
        st = {kk: v.copy() for kk, v in pre.items()}
        O.update(q_new, st, override=assign_g, lib=lib)
    np.testing.assert_array_equal(post["counts"], st["counts"], err_msg=f"{tag}: counts")
    np.testing.assert_allclose(post["sums"], st["sums"], rtol=1e-12, atol=1e-12, err_msg=f"{tag}: sums")
    ref = st["cent"].astype(np.float64)
    scale = np.maximum(np.linalg.norm(ref, axis=1, keepdims=True), 1.0)
    cerr = float(np.max(np.abs(post["cent"].astype(np.float64) - ref) / scale)) if ref.size else 0.0
    assert cerr <= CENT_TOL, f"{tag}: centroid error {cerr:.3e}"
    return ties, cerr


def check_compress(wl: Workload, cent: np.ndarray, counts: np.ndarray, q_recent: np.ndarray, recent_pos, t_pos: int,
                   K0: np.ndarray, V0: np.ndarray, K1: np.ndarray, V1: np.ndarray, kept_g: np.ndarray,
                   scores_g: np.ndarray | None, L: int, budget: int, lib, tag: str = "", mean: bool = False,
                   causal: bool = False, tie_rtol: float | None = None) -> tuple:
    """One compress of one instance on the beacon state (cent, counts): scores within 1e-3 (plus 2^-126),
    the kept set equal up to boundary ties (oracle margin below tie_rtol, by default 1e-5), K / V rows
    byte-equal to the kept pre-compress rows.  K0 / V0 and K1 / V1 are the instance's uint16 rows before
    and after; `causal` applies the mask inside the recent window.
    Returns (max score rel err, boundary swaps)."""
    tie = TIE_RTOL if tie_rtol is None else tie_rtol
    W = wl.window
    if L <= budget:
        np.testing.assert_array_equal(kept_g[:L], np.arange(L))
        assert np.all(kept_g[L:] == -1)
        np.testing.assert_array_equal(K1, K0)
        return 0.0, 0
    qobs, valid = O.build_qobs(cent, counts, q_recent, np.asarray(recent_pos, np.int64), t_pos, wl.rope_theta, lib)
    if isinstance(tie, str):
        tie = logit_tie_rtol(qobs, valid, K0[:L])
    if causal and W > 0:
        qpos, kpos = O.causal_positions(q_recent.shape[0], W, counts.shape[0], recent_pos, t_pos, L)
        s_o = O.score(qobs, valid, K0[:L], lib, mean=mean, qpos=qpos, kpos=kpos)
    else:
        s_o = O.score(qobs, valid, K0[:L], lib, mean=mean)
    rel_max = 0.0
    if scores_g is not None:
        s_g = scores_g[:L].astype(np.float64)
        err = np.abs(s_g - s_o)
        over = err - (SCORE_RTOL * s_o + SCORE_ATOL)
        assert over.max() <= 0, f"{tag}: score error {err[over.argmax()]:.3e} at key {int(over.argmax())} " \
                                f"(oracle {s_o[over.argmax()]:.3e})"
        normal = s_o >= 2.0 ** -126
        rel_max = float((err[normal] / s_o[normal]).max()) if normal.any() else 0.0
    kept_o, bd = O.select(s_o, budget, W, wl.n_prefix, lib)
    assert kept_g.shape[0] == budget
    assert np.all(np.diff(kept_g) > 0), f"{tag}: kept indices not strictly ascending"
    keep_set = set(range(wl.n_prefix)) | set(range(L - W, L))
    assert keep_set <= set(kept_g.tolist()), f"{tag}: keep set not retained"
    assert kept_g.min() >= 0 and kept_g.max() < L
    sym = set(kept_g.tolist()) ^ set(kept_o.tolist())
    swaps = 0
    if sym:
        b = bd[0]
        for j in sym:
            assert j not in keep_set
            assert abs(s_o[j] - b) <= tie * b, \
                f"{tag}: key {j} kept by only one side with margin {abs(s_o[j] - b) / b:.3e} (> {tie:.1e})"
        swaps = len(sym) // 2
    np.testing.assert_array_equal(K1[:budget], K0[kept_g], err_msg=f"{tag}: K compaction")
    np.testing.assert_array_equal(V1[:budget], V0[kept_g], err_msg=f"{tag}: V compaction")
    return rel_max, swaps


def check_cfps_compress(wl: Workload, b_min: int, buf: np.ndarray, size: np.ndarray, q_rec: np.ndarray, recent_pos,
                        t_pos: int, K0, V0, K1, V1, kept_g, scores_g, L: int, budget: int, buf_after: np.ndarray,
                        size_after: np.ndarray, lib, tag: str = "", mean: bool = False, causal: bool = False) -> tuple:
    """One compress of one instance in the Continual FPS mode.  buf / size: the G buffers of the
    instance's query heads before the compress (uint16 [G, b_max, d], int [G]); q_rec: their window
    queries (uint16 [G, W, d]); buf_after / size_after: the GPU's buffers after it.  The beacons are
    the fp64 FPS selection (Algorithm 1) of min(b_min, size) rows of each buffer; after an eviction each
    buffer must be the FPS selection of b_min rows of (its beacons, then its window queries).  Both FPS
    steps take their near-tie branches (search_branches): a head's beacons are the branch whose merge
    gives the GPU's buffer, and the compress is checked with those beacons.
    Returns (max score rel err, boundary swaps, FPS ties)."""
    G, d = buf.shape[0], buf.shape[-1]
    cent = np.zeros((G * b_min, d), np.float32)
    counts = np.zeros(G * b_min, np.int64)
    ties = 0
    for g in range(G):
        rows = buf[g, :size[g]]
        chosen = None
        for picks, t_b in fps_branches(rows, b_min, lib):
            beacons = rows[picks]
            if L <= budget:  # no eviction, no merge: the buffer is unchanged, the beacons are not used
                want = rows
                ok = size_after[g] == len(want) and np.array_equal(buf_after[g, :len(want)], want)
                chosen = (beacons, t_b) if ok else chosen
                break
            cand = np.vstack([beacons, q_rec[g]])
            if size_after[g] != min(b_min, len(cand)):
                continue
            for mp, t_m in fps_branches(cand, b_min, lib):
                if np.array_equal(buf_after[g, :len(mp)], cand[mp]):
                    chosen = (beacons, t_b + t_m)
                    break
            if chosen is not None:
                break
        assert chosen is not None, f"{tag} head {g}: no fp64 FPS branch of the beacons and merge gives the " \
                                   f"GPU's buffer after the compress (size {size_after[g]})"
        beacons, t = chosen
        ties += t
        cent[g * b_min:g * b_min + len(beacons)] = O.bf16_to_f64(beacons)
        counts[g * b_min:g * b_min + len(beacons)] = 1
    rel, swaps = check_compress(wl, cent, counts, q_rec, recent_pos, t_pos, K0, V0, K1, V1, kept_g, scores_g, L,
                                budget, lib, tag=tag, mean=mean, causal=causal)
    return rel, swaps, ties


def smoke_decode_steps(wl: Workload, steps: int, seed: int) -> str:
    """A few decode steps (one query per query head each) on the GPU: one bkv_update_beacons call per
    step, each checked against the oracle from the state the GPU carried forward, and the same steps in
    one bkv_update_beacons_seq call, whose state and assignments must be bit-identical."""
    import torch
    from paper_2609_04971_gb300 import bkv, synth
    lib = O.load()
    dev = torch.device("cuda")
    q_init = synth.queries(wl, seed, "q_init", wl.n_init, dev)
    q = synth.queries(wl, seed, "q_decode", steps, dev)                 # [layers, batch, Hq, steps, d]
    q_steps = q.permute(3, 0, 1, 2, 4).contiguous()                    # [steps, layers, batch, Hq, d]
    per_step = wl.n_layers * wl.batch * wl.n_q_heads
    outs, ties = [], 0
    for seq in (False, True):
        bk = bkv.BeaconKV.for_workload(wl)
        try:
            bk.init_beacons(q_init)
            assign = torch.empty(steps, per_step, dtype=torch.int32, device=dev)
            if seq:
                bk.update_seq(q_steps, assign)
            else:
                state = [x.cpu().numpy() for x in bk.state()]
                for t in range(steps):
                    bk.update(q_steps[t].unsqueeze(-2), assign[t])
                    new = [x.cpu().numpy() for x in bk.state()]
                    qb = synth.to_bits(q_steps[t]).reshape(wl.n_inst, wl.group, wl.head_dim)
                    a_g = assign[t].view(wl.n_inst, wl.group).cpu().numpy()
                    for e in range(wl.n_inst):
                        pre = dict(cent=state[0][e].copy(), sums=state[1][e].copy(), counts=state[2][e].copy())
                        post = dict(cent=new[0][e], sums=new[1][e], counts=new[2][e])
                        ties += check_update(qb[e], pre, a_g[e], post, lib, tag=f"decode step {t} instance {e}")[0]
                    state = new
            bk.sync()
            c, sm, n = bk.state()
            outs.append((assign.cpu(), c.cpu().view(torch.int32), sm.cpu().view(torch.int64), n.cpu()))
        finally:
            bk.close()
    for x, y in zip(*outs):
        assert torch.equal(x, y), "bkv_update_beacons_seq differs from one bkv_update_beacons call per step"
    return f"{steps} steps x {wl.n_inst} instances, oracle ties {ties}, seq call bit-identical"
