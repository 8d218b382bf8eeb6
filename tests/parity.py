"""Parity harness: the CUDA path (through the C ABI) against the fp64 oracle.

Tolerances:
  * FPS seeds and beacon assignments: identical, except where the oracle's own
    decision was a tie (runner-up within 1e-12), where either choice is valid;
  * beacon state after an update: counts exact, sums within 1e-12 relative,
    centroids within 1e-5 relative to |c| (absolute when |c| < 1);
  * scores: within 1e-3 relative of the oracle's fp64 scores;
  * kept index sets: identical except for candidates whose oracle score is
    within 1e-5 relative of the oracle's boundary score (the score of the last
    candidate it took); the GPU set must still hold exactly `budget` rows,
    be strictly ascending and contain the keep set;
  * compacted K / V: byte-identical to the pre-compress rows the GPU kept.
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
TIE_RTOL = 1e-5
CENT_TOL = 1e-5
ASSIGN_TIE = 1e-12


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
        kept = bk.compress(K, V, L=L, budget=budget, t_pos=inp["t_pos"], q_recent=inp["q_recent"],
                           recent_pos=inp["recent_pos"], scores_out=scores)
        bk.sync()
        K_after = Kf.index_select(0, sidx).view(torch.int16).cpu().numpy().view(np.uint16)
        V_after = Vf.index_select(0, sidx).view(torch.int16).cpu().numpy().view(np.uint16)
    finally:
        bk.close()
    return GpuRun(wl=wl, inputs=inp, cent0=c0, sums0=s0, counts0=n0,
                  assign=assign.view(n_inst, -1).cpu().numpy(), cent1=c1, sums1=s1, counts1=n1,
                  kept=kept.view(n_inst, -1).cpu().numpy(),
                  scores=None if scores is None else scores.view(n_inst, -1).cpu().numpy(),
                  K_before=K_before, V_before=V_before, K_after=K_after, V_after=V_after, sample=sample,
                  mean_agg=mean_agg, causal=causal)


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


def check_instance(run: GpuRun, k: int, L: int | None = None, budget: int | None = None, lib=None) -> Report:
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
                                mean=run.mean_agg, causal=run.causal)
    rep.max_score_rel = rel
    rep.boundary_swaps += swaps
    return rep


def check_run(run: GpuRun, L=None, budget=None) -> Report:
    rep = Report()
    lib = O.load()
    for k in range(len(run.sample)):
        rep.merge(check_instance(run, k, L=L, budget=budget, lib=lib))
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
                   causal: bool = False) -> tuple:
    """One compress of one instance on the beacon state (cent, counts): scores within 1e-3, the kept set
    equal up to boundary ties, K / V rows byte-equal to the kept pre-compress rows.  K0 / V0 and K1 / V1
    are the instance's uint16 rows before and after; `causal` applies the mask inside the recent window.
    Returns (max score rel err, boundary swaps)."""
    W = wl.window
    if L <= budget:
        np.testing.assert_array_equal(kept_g[:L], np.arange(L))
        assert np.all(kept_g[L:] == -1)
        np.testing.assert_array_equal(K1, K0)
        return 0.0, 0
    qobs, valid = O.build_qobs(cent, counts, q_recent, np.asarray(recent_pos, np.int64), t_pos, wl.rope_theta, lib)
    if causal and W > 0:
        qpos, kpos = O.causal_positions(q_recent.shape[0], W, counts.shape[0], recent_pos, t_pos, L)
        s_o = O.score(qobs, valid, K0[:L], lib, mean=mean, qpos=qpos, kpos=kpos)
    else:
        s_o = O.score(qobs, valid, K0[:L], lib, mean=mean)
    rel_max = 0.0
    if scores_g is not None:
        s_g = scores_g[:L].astype(np.float64)
        rel = np.abs(s_g - s_o) / np.maximum(s_o, 1e-300)
        rel_max = float(rel.max())
        assert rel_max <= SCORE_RTOL, f"{tag}: score rel err {rel_max:.3e} at key {int(rel.argmax())}"
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
            assert abs(s_o[j] - b) <= TIE_RTOL * b, \
                f"{tag}: key {j} kept by only one side with margin {abs(s_o[j] - b) / b:.3e} (> 1e-5)"
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
    the fp32 FPS selection of min(b_min, size) rows of each buffer; after an eviction each buffer must
    be the FPS selection of b_min rows of (its beacons, then its window queries).
    Returns (max score rel err, boundary swaps)."""
    G, d = buf.shape[0], buf.shape[-1]
    cent = np.zeros((G * b_min, d), np.float32)
    counts = np.zeros(G * b_min, np.int64)
    beacons = []
    for g in range(G):
        picks, _ = O.fps32(buf[g, :size[g]], b_min, lib)
        rows = buf[g][picks]
        beacons.append(rows)
        cent[g * b_min:g * b_min + len(picks)] = O.bf16_to_f64(rows)
        counts[g * b_min:g * b_min + len(picks)] = 1
    rel, swaps = check_compress(wl, cent, counts, q_rec, recent_pos, t_pos, K0, V0, K1, V1, kept_g, scores_g, L,
                                budget, lib, tag=tag, mean=mean, causal=causal)
    for g in range(G):
        if L > budget:
            cand = np.vstack([beacons[g], q_rec[g]])
            picks, _ = O.fps32(cand, b_min, lib)
            want = cand[picks]
        else:
            want = buf[g, :size[g]]
        assert size_after[g] == len(want), f"{tag} head {g}: buffer size {size_after[g]} vs {len(want)}"
        np.testing.assert_array_equal(buf_after[g, :len(want)], want, err_msg=f"{tag} head {g}: buffer after merge")
    return rel, swaps
