"""Continual FPS beacons (BKV_F_CONTINUAL_FPS) through the C ABI against the oracle.

Every query head is checked: the FPS seeding (fp64 similarities; picks equal up
to ties below 1e-12), the fill-and-compress buffer after a call of many new
queries, the compress on the resulting beacons (scores, kept set, compacted
rows, as in tests/parity.py) and the post-eviction merge.  The buffer, beacon
and merge FPS steps are compared with Algorithm 1 in fp64: the kernels decide
from fp32 similarities, so where the fp64 runner-up lies within
tests/parity.cfps_tie_bound of the minimum either row is accepted and the
oracle continues from the GPU's choice (tests/parity.search_branches).
"""
import numpy as np
import pytest
import torch

from paper_2609_04971_gb300.workloads import QWEN3_4B, TINY

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from oracle import oracle as O
    from paper_2609_04971_gb300 import synth
    from paper_2609_04971_gb300.bkv import BeaconKV
    from tests import parity as P


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _heads(t: torch.Tensor, d: int) -> np.ndarray:
    """[L, B, Hq, n, d] bf16 -> uint16 [heads, n, d]."""
    return _bits(t).reshape(-1, t.shape[-2], d)


def _run_cfps(wl, seed, b_min, L=None, budget=None, n_new=None, mean_agg=False, causal=False, sample=None):
    """One init + update + compress; every instance is checked, or only the instances in `sample` (the
    others still on their sizes and kept sets)."""
    dev = torch.device("cuda")
    inp = synth.step_inputs(wl, seed, dev)
    L = wl.L if L is None else L
    budget = wl.budget if budget is None else budget
    d, G, W = wl.head_dim, wl.group, wl.window
    b_max = b_min + W
    lib = O.load()
    q_new_t = inp["q_new"] if n_new is None else inp["q_new"][..., :n_new, :].contiguous()
    bk = BeaconKV(n_layers=wl.n_layers, batch=wl.batch, n_q_heads=wl.n_q_heads, n_kv_heads=wl.n_kv_heads, head_dim=d,
                  n_beacons=b_min, window=W, capacity=wl.capacity, rope_theta=wl.rope_theta, n_prefix=wl.n_prefix,
                  continual_fps=True, mean_agg=mean_agg, causal_window=causal)
    try:
        bk.init_beacons(inp["q_init"])
        buf0, size0 = [x.cpu() for x in bk.cfps_state()]
        bk.update(q_new_t)
        buf1, size1 = [x.cpu() for x in bk.cfps_state()]
        K, V = inp["K"], inp["V"]
        n_inst = wl.n_inst
        insts = np.arange(n_inst) if sample is None else np.asarray(sample)
        sel = torch.as_tensor(insts, device=dev)

        def rows(t):  # the checked instances' cache rows, [len(insts), capacity, d] uint16
            return _bits(t.view(n_inst, wl.capacity, d).index_select(0, sel))

        Kb, Vb = rows(K), rows(V)
        scores = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads, wl.capacity), -1.0, device=dev)
        kept = bk.compress(K, V, L=L, budget=budget, t_pos=inp["t_pos"], q_recent=inp["q_recent"],
                           recent_pos=inp["recent_pos"], scores_out=scores)
        buf2, size2 = [x.cpu() for x in bk.cfps_state()]
        bk.sync()
        K1, V1 = rows(K), rows(V)
    finally:
        bk.close()

    q_init = _heads(inp["q_init"], d)
    q_new = _heads(q_new_t, d)
    q_rec = _heads(inp["q_recent"], d)
    buf0 = buf0.view(torch.int16).numpy().view(np.uint16).reshape(-1, b_max, d)
    buf1 = buf1.view(torch.int16).numpy().view(np.uint16).reshape(-1, b_max, d)
    buf2 = buf2.view(torch.int16).numpy().view(np.uint16).reshape(-1, b_max, d)
    size0, size1, size2 = (x.numpy().reshape(-1) for x in (size0, size1, size2))
    heads = (insts[:, None] * G + np.arange(G)[None, :]).reshape(-1)
    fps_ties = buf_ties = 0
    for h in heads:
        # ---- seeding: fp64 FPS of the head's prompt queries
        picks, gaps = O.fps(q_init[h], b_min, lib)
        assert size0[h] == b_min
        if not np.array_equal(buf0[h, :b_min], q_init[h][picks]):
            first = next(k for k in range(b_min) if not np.array_equal(buf0[h, k], q_init[h][picks[k]]))
            assert gaps[first] < P.ASSIGN_TIE, f"head {h}: seed pick {first} differs, fp64 gap {gaps[first]:.2e}"
            fps_ties += 1
        # ---- update from the GPU's seed: fp64 Eq. 9 up to near-ties of the fp32 decisions
        buf_ties += P.match_cfps_update(buf0[h], int(size0[h]), b_min, b_max, q_new[h], buf1[h], int(size1[h]), lib,
                                        tag=f"head {h}: buffer after update")

    # every head: the sizes of a head depend only on the call's lengths
    assert np.all(size0 == b_min)
    assert np.all(size1 == size1[heads[0]]) and np.all(size2 == size2[heads[0]])

    rel_max, swaps, cmp_ties = 0.0, 0, 0
    kept_h = kept.view(n_inst, budget).cpu().numpy()
    s_h = scores.view(n_inst, wl.capacity).cpu().numpy()
    if L > budget:  # every instance: ascending, the recent window kept
        assert np.all(np.diff(kept_h, axis=1) > 0)
        assert np.all(kept_h[:, budget - W:] == np.arange(L - W, L))
    for i, e in enumerate(insts):
        hs = slice(e * G, (e + 1) * G)
        r, sw, t = P.check_cfps_compress(wl, b_min, buf1[hs], size1[hs], q_rec[hs], inp["recent_pos"],
                                         inp["t_pos"], Kb[i], Vb[i], K1[i], V1[i], kept_h[e], s_h[e], L, budget,
                                         buf2[hs], size2[hs], lib, tag=f"instance {e}", mean=mean_agg, causal=causal)
        rel_max, swaps, cmp_ties = max(rel_max, r), swaps + sw, cmp_ties + t
    print(f"{wl.name}: {len(heads)} heads checked, seed ties {fps_ties}, buffer ties {buf_ties}, "
          f"beacon/merge ties {cmp_ties}, max score rel err {rel_max:.2e}, swaps {swaps}")


@pytest.mark.parametrize("wl,b_min,seed", [
    (TINY.scaled(name="cfps_tiny_d64"), 4, 21),
    (QWEN3_4B.scaled(name="cfps_qwen3_4b_1L_b1_nb8", n_layers=1, batch=1), 8, 22),
    (QWEN3_4B.scaled(name="cfps_qwen3_4b_1L_b1_nb16_w16", n_layers=1, batch=1, window=16), 16, 23),
], ids=lambda x: getattr(x, "name", str(x)))
def test_continual_fps_step(wl, b_min, seed):
    _run_cfps(wl, seed, b_min)


def test_continual_fps_full_size_sampled():
    """The Qwen3-4B step that the benchmark times in this mode (36 layers, batch 16, 8 beacons + 8 window
    queries per query head, 128 new queries per head): eight sampled instances checked in full."""
    wl = QWEN3_4B.scaled(n_beacons=8, name="qwen3_4b_cfps8")
    rng = np.random.default_rng(1)
    sample = np.unique(np.concatenate([[0, wl.n_inst - 1], rng.choice(wl.n_inst, 6, replace=False)]))
    _run_cfps(wl, 30, 8, sample=sample)


def test_continual_fps_short_call_and_no_eviction():
    """A call too short to fill the buffer (no FPS), then a compress with L <= budget (no merge)."""
    wl = QWEN3_4B.scaled(name="cfps_short_fits", n_layers=1, batch=1, L=256, budget=300)
    _run_cfps(wl, 24, 8, n_new=3)


def test_continual_fps_ragged_cache():
    wl = QWEN3_4B.scaled(name="cfps_ragged_L1000_B700", n_layers=1, batch=2, L=1000, budget=700)
    _run_cfps(wl, 25, 8)


def test_continual_fps_with_mean_aggregation():
    wl = QWEN3_4B.scaled(name="cfps_mean_1L_b1", n_layers=1, batch=1, L=900, budget=500)
    _run_cfps(wl, 26, 8, mean_agg=True)


def test_continual_fps_with_causal_window():
    wl = QWEN3_4B.scaled(name="cfps_causal_1L_b1", n_layers=1, batch=1, L=900, budget=500)
    _run_cfps(wl, 28, 8, causal=True)


def test_continual_fps_all_options_at_128_queries():
    """16 beacons + 16 window queries per head (the paper's buffer sizes): 128 scoring queries per group, so
    two score launches folded into one score, with the mean form and the causal mask."""
    wl = QWEN3_4B.scaled(name="cfps_nb16_w16_mean_causal", n_layers=1, batch=1, window=16, L=1200, budget=700)
    _run_cfps(wl, 29, 16, mean_agg=True, causal=True)


def test_continual_fps_state_round_trip():
    """bkv_set_cfps_state restores buffers that bkv_get_cfps_state saved: an update from the restored
    state gives the same buffers as from the original."""
    wl = QWEN3_4B.scaled(name="cfps_state", n_layers=1, batch=1)
    dev = torch.device("cuda")
    inp = synth.step_inputs(wl, 27, dev)
    kw = dict(n_layers=1, batch=1, n_q_heads=wl.n_q_heads, n_kv_heads=wl.n_kv_heads, head_dim=wl.head_dim,
              n_beacons=8, window=wl.window, capacity=wl.capacity, rope_theta=wl.rope_theta, continual_fps=True)
    a, b = BeaconKV(**kw), BeaconKV(**kw)
    try:
        a.init_beacons(inp["q_init"])
        a.update(inp["q_new"][..., :37, :].contiguous())
        buf, sizes = a.cfps_state()
        b.set_cfps_state(buf, sizes)
        rest = inp["q_new"][..., 37:, :].contiguous()
        a.update(rest)
        b.update(rest)
        (ba, sa), (bb, sb) = a.cfps_state(), b.cfps_state()
        torch.cuda.synchronize()
        assert torch.equal(sa, sb)
        for h in range(sa.numel()):
            n = int(sa.view(-1)[h])
            assert torch.equal(ba.view(-1, ba.shape[-2], ba.shape[-1])[h, :n], bb.view(-1, bb.shape[-2], bb.shape[-1])[h, :n])
        with pytest.raises(Exception):
            a.state()      # no centroid state in this mode
    finally:
        a.close()
        b.close()
