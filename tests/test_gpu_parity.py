"""CUDA path (through the C ABI) against the fp64 oracle, element by element.

Sizes span several 128-key tiles and ragged tails; the full-size workloads run
in the launch configuration bench.py times and are checked on sampled
instances.  Tolerances are stated in tests/parity.py.
"""
import numpy as np
import pytest
import torch

from paper_2609_04971_gb300 import synth
from paper_2609_04971_gb300.workloads import LLAMA_8B, QWEN3_14B, QWEN3_4B, QWEN3_8B_TRACE, TINY

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from tests import parity as P


def _run(wl, seed=0, sample=None, **kw):
    run = P.run_gpu(wl, seed=seed, sample=sample, **kw)
    rep = P.check_run(run, L=kw.get("L"), budget=kw.get("budget"))
    print(f"{wl.name}: {rep}")
    return run, rep


def test_tiny_workload_all_instances():
    _run(TINY)


@pytest.mark.parametrize("wl", [
    QWEN3_4B.scaled(name="qwen3_4b_1L_b2", n_layers=1, batch=2),
    LLAMA_8B.scaled(name="llama_8b_1L_b2", n_layers=1, batch=2),
    QWEN3_14B.scaled(name="qwen3_14b_1L_b1", n_layers=1, batch=1),
], ids=lambda w: w.name)
def test_reduced_batch_full_length(wl):
    _run(wl)


@pytest.mark.parametrize("L,budget", [(1000, 700), (100, 50), (129, 128), (300, 17), (640, 639)])
def test_ragged_lengths(L, budget):
    wl = QWEN3_4B.scaled(name=f"ragged_L{L}_B{budget}", n_layers=1, batch=1, L=L, budget=budget)
    _run(wl, seed=L)


def test_head_dim_64_ragged():
    wl = TINY.scaled(name="d64_L777", L=777, budget=400, n_layers=2, batch=3)
    _run(wl, seed=3)


def test_prefix_kept():
    wl = QWEN3_4B.scaled(name="prefix4", n_layers=1, batch=1, L=600, budget=300, n_prefix=4)
    _run(wl, seed=5)


def test_recent_only_no_beacons():
    wl = QWEN3_4B.scaled(name="nb0", n_layers=1, batch=2, L=500, budget=260, n_beacons=0)
    _run(wl, seed=6)


def test_beacons_only_no_window():
    wl = LLAMA_8B.scaled(name="w0", n_layers=1, batch=1, L=400, budget=200, window=0)
    _run(wl, seed=7)


def test_budget_equals_keep_set():
    wl = QWEN3_4B.scaled(name="ksel0", n_layers=1, batch=1, L=300, budget=8)
    _run(wl, seed=8)


def test_no_eviction_when_cache_fits():
    wl = QWEN3_4B.scaled(name="fits", n_layers=1, batch=1, L=256, budget=300)
    _run(wl, seed=9)


def test_no_rotation_and_max_queries():
    # G * W + nb = 8 * 12 + 32 = 128 scoring queries (the maximum), theta = 0
    wl = QWEN3_4B.scaled(name="m128", n_layers=1, batch=1, n_q_heads=64, n_kv_heads=8, window=12, n_beacons=32,
                         L=700, budget=500, rope_theta=0.0, n_init=64, n_clusters=32)
    _run(wl, seed=10)


@pytest.mark.parametrize("wl", [
    # 128 scoring queries, 40 tiles: two score launches of 64 queries, each resident in tensor memory
    QWEN3_4B.scaled(name="long_m128_L5000", n_layers=1, batch=1, n_q_heads=64, n_kv_heads=8, window=12,
                    n_beacons=32, L=5000, budget=3000, n_init=64, n_clusters=32),
    # 128 scoring queries, 235 tiles: both launches stream tiles past the resident ones
    QWEN3_4B.scaled(name="long_m128_L30000", n_layers=1, batch=1, n_q_heads=64, n_kv_heads=8, window=12,
                    n_beacons=32, L=30000, budget=20000, n_init=64, n_clusters=32),
    # 48 scoring queries, 157 tiles: resident tiles plus streaming tiles in every CTA
    QWEN3_4B.scaled(name="long_L20000", n_layers=1, batch=1, L=20000, budget=12000),
], ids=lambda w: w.name)
def test_long_cache_streaming_tiles(wl):
    _run(wl, seed=13)


def test_identical_keys_tie_everywhere():
    """All keys equal: every score is 1/L, the kept set is the lowest-index
    candidates plus the window (ties go to the lower index)."""
    wl = QWEN3_4B.scaled(name="flat", n_layers=1, batch=1, L=400, budget=100)
    dev = torch.device("cuda")
    from paper_2609_04971_gb300 import synth
    inp = synth.step_inputs(wl, 11, dev)
    inp["K"][:] = inp["K"][:, :, :, :1, :]
    run = P.run_gpu(wl, inputs=inp)
    want = np.concatenate([np.arange(92), np.arange(392, 400)])
    for e in range(wl.n_inst):
        np.testing.assert_array_equal(run.kept[e], want)
        np.testing.assert_allclose(run.scores[e][:400], 1.0 / 400, rtol=1e-5)


@pytest.mark.parametrize("wl", [QWEN3_4B, LLAMA_8B, QWEN3_14B], ids=lambda w: w.name)
def test_full_size_sampled(wl):
    rng = np.random.default_rng(0)
    sample = np.unique(np.concatenate([[0, wl.n_inst - 1], rng.choice(wl.n_inst, 6, replace=False)]))
    run, rep = _run(wl, sample=sample)
    # every instance, not only the sampled ones: budget, order, keep set
    kept = run.kept
    assert kept.shape == (wl.n_inst, wl.budget)
    assert np.all(np.diff(kept, axis=1) > 0)
    assert np.all(kept[:, -wl.window:] == np.arange(wl.L - wl.window, wl.L))
    assert run.counts1.sum(axis=1).min() == wl.group * (wl.n_init * 0 + wl.n_new) + wl.n_beacons


# ---------------------------------------------------------------- a few queries per instance (decode steps)
@pytest.mark.parametrize("wl", [
    QWEN3_4B.scaled(name="few_n1", n_layers=1, batch=2, n_new=1),   # 4 rows per instance: one decode step
    QWEN3_4B.scaled(name="few_n3", n_layers=1, batch=2, n_new=3),   # 12 rows
    QWEN3_4B.scaled(name="few_n8", n_layers=1, batch=2, n_new=8),   # 32 rows: the largest few-query call
    QWEN3_4B.scaled(name="few_n9", n_layers=1, batch=2, n_new=9),   # 36 rows: the batched kernel
    TINY.scaled(name="few_d64_n4", n_new=4),                        # head_dim 64, 8 rows
    QWEN3_14B.scaled(name="few_g5_n1", n_layers=1, batch=2, n_new=1),  # GQA group 5: 5 rows, 16 beacons
    QWEN3_4B.scaled(name="few_g8_nb32_n4", n_layers=1, batch=1, n_q_heads=64, n_kv_heads=8, window=12, n_beacons=32,
                    L=700, budget=500, n_init=64, n_clusters=32, n_new=4),   # 32 rows, 32 beacons
    QWEN3_4B.scaled(name="qwen3_4b_decode_step", n_new=1),          # all 4608 instances, sampled
    QWEN3_8B_TRACE.scaled(name="qwen3_8b_trace_decode_step"),       # the long trace's step: 16 beacons, 4608
], ids=lambda w: w.name)
def test_few_queries_per_instance(wl):
    sample = None
    if wl.n_inst > 64:
        rng = np.random.default_rng(1)
        sample = np.unique(np.concatenate([[0, wl.n_inst - 1], rng.choice(wl.n_inst, 6, replace=False)]))
    _run(wl, seed=wl.n_new + 30, sample=sample)


def test_few_queries_with_zero_queries():
    """Zero queries stay unassigned (-1) and add nothing, in the few-query kernel."""
    wl = QWEN3_4B.scaled(name="few_zero", n_layers=1, batch=1, n_new=2)
    from paper_2609_04971_gb300 import synth
    inp = synth.step_inputs(wl, 33, torch.device("cuda"))
    inp["q_new"][:, :, ::3, 1, :] = 0
    run, _ = _run(wl, inputs=inp)
    assert (run.assign == -1).sum() > 0


def test_deterministic_across_runs():
    wl = QWEN3_4B.scaled(name="det", n_layers=1, batch=2, L=900, budget=500)
    a = P.run_gpu(wl, seed=12)
    b = P.run_gpu(wl, seed=12)
    np.testing.assert_array_equal(a.kept, b.kept)
    np.testing.assert_array_equal(a.scores, b.scores)
    np.testing.assert_array_equal(a.cent1, b.cent1)
    np.testing.assert_array_equal(a.K_after, b.K_after)


def test_stream_switch_matches_one_stream():
    """Calls split across two streams by bkv_set_stream give the results of one stream: the switch orders
    the new stream after the work already enqueued on the old one."""
    from paper_2609_04971_gb300 import bkv
    wl = QWEN3_4B.scaled(name="switch", n_layers=2, batch=2)
    dev = torch.device("cuda")
    inp = synth.step_inputs(wl, 31, dev)
    outs = []
    for switch in (False, True):
        K, V = inp["K"].clone(), inp["V"].clone()
        s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        torch.cuda.synchronize()
        bk = bkv.BeaconKV.for_workload(wl, stream=s1)
        try:
            with torch.cuda.stream(s1):
                bk.init_beacons(inp["q_init"])
                bk.update(inp["q_new"])
            if switch:
                bkv.bkv_set_stream(bk.ctx, s2)
            with torch.cuda.stream(s2 if switch else s1):
                kept = bk.compress(K, V, L=wl.L, budget=wl.budget, t_pos=inp["t_pos"], q_recent=inp["q_recent"],
                                   recent_pos=inp["recent_pos"])
                state = bk.state()
            bk.sync()
            torch.cuda.synchronize()
            outs.append([kept.cpu(), K.cpu(), V.cpu()] + [t.cpu() for t in state])
        finally:
            bk.close()
    for a, b in zip(*outs):
        assert torch.equal(a, b)


# ---------------------------------------------------------------- causal mask inside the window (BKV_F_CAUSAL_WINDOW)
def _shift_positions(inp, W, t_pos, recent_pos):
    inp = dict(inp)
    inp["t_pos"] = int(t_pos)
    inp["recent_pos"] = [int(p) for p in recent_pos][:W]
    return inp


@pytest.mark.parametrize("mean", [False, True], ids=["max", "mean"])
@pytest.mark.parametrize("wl,seed", [
    (TINY.scaled(name="causal_tiny"), 41),
    (QWEN3_4B.scaled(name="causal_qwen3_4b_1L_b2", n_layers=1, batch=2), 42),
    (QWEN3_4B.scaled(name="causal_ragged_L300_B40_w16", n_layers=1, batch=1, L=300, budget=40, window=16), 43),
    (QWEN3_4B.scaled(name="causal_long_L20000", n_layers=1, batch=1, L=20000, budget=9000), 44),
    (QWEN3_4B.scaled(name="causal_nb0", n_layers=1, batch=1, L=500, budget=260, n_beacons=0), 45),
    (QWEN3_4B.scaled(name="causal_m128", n_layers=1, batch=1, n_q_heads=64, n_kv_heads=8, window=12, n_beacons=32,
                     L=900, budget=600, n_init=64, n_clusters=32), 47),
], ids=lambda x: getattr(x, "name", str(x)))
def test_causal_window(wl, seed, mean):
    _run(wl, seed=seed, mean_agg=mean, causal=True)


@pytest.mark.parametrize("case", ["decode_after_evictions", "sparse_recent_positions"])
def test_causal_window_positions(case):
    """Positions that are not the last L rows: a decode step long after earlier evictions (t = 9000 with
    640 cached rows), and recent queries at scattered earlier positions (some see no window row, one
    sees them all)."""
    wl = QWEN3_4B.scaled(name=f"causal_{case}", n_layers=1, batch=1, L=640, budget=300, window=8)
    inp = synth.step_inputs(wl, 46, torch.device("cuda"))
    if case == "decode_after_evictions":
        inp = _shift_positions(inp, 8, 9000, range(8993, 9001))
    else:
        inp = _shift_positions(inp, 8, 9000, [100, 8990, 8994, 8995, 8996, 8998, 9000, 9000])
    _run(wl, seed=46, inputs=inp, causal=True)


# ---------------------------------------------------------------- Eq. 6 mean form (BKV_F_MEAN_AGG)
@pytest.mark.parametrize("wl,seed", [
    (TINY.scaled(name="mean_tiny"), 11),
    (QWEN3_4B.scaled(name="mean_qwen3_4b_1L_b2", n_layers=1, batch=2), 12),
    (QWEN3_4B.scaled(name="mean_ragged_L300_B17", n_layers=1, batch=1, L=300, budget=17), 13),
    (QWEN3_4B.scaled(name="mean_long_L20000", n_layers=1, batch=1, L=20000, budget=9000), 14),
    (LLAMA_8B.scaled(name="mean_w0", n_layers=1, batch=1, L=400, budget=200, window=0), 15),
    (QWEN3_4B.scaled(name="mean_m128", n_layers=1, batch=1, n_q_heads=64, n_kv_heads=8, window=12, n_beacons=32,
                     L=900, budget=600, n_init=64, n_clusters=32), 16),
    (QWEN3_4B.scaled(name="mean_m80", n_layers=1, batch=1, window=16, L=700, budget=300), 17),
], ids=lambda x: getattr(x, "name", str(x)))
def test_mean_aggregation(wl, seed):
    _run(wl, seed=seed, mean_agg=True)
