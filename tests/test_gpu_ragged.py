"""bkv_compress_ragged: a cache length per instance and positions per batch row, through the C ABI,
against the fp64 oracle instance by instance (tests/parity.check_compress with the instance's own L,
t_pos and recent positions).

The lengths mix instances left untouched (L <= budget), instances one row above the budget, a few
tiles, a full cache, and (in the long case) caches that stream tiles past the tensor-memory ring;
they differ per layer as well as per batch row.  Every instance is checked: kept indices, scores,
compacted rows, rows past the budget unchanged, untouched instances byte-identical.  Forms: max,
mean, causal window, Continual FPS beacons; and a length outside 1..capacity (reported by bkv_sync,
that instance untouched, the others compressed).
"""
import numpy as np
import pytest
import torch

from paper_2609_04971_gb300.workloads import QWEN3_4B

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from oracle import oracle as O
    from paper_2609_04971_gb300 import bkv, synth
    from tests import parity as P


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _lengths(wl, budget, cap, seed, long_rows=()):
    """Per-instance lengths [layers, batch, kv]: per batch row a base length, varied per layer."""
    rng = np.random.default_rng(seed)
    nl, B, Hkv = wl.n_layers, wl.batch, wl.n_kv_heads
    base = [cap, budget, budget + 1, max(1, budget // 2), budget + 130, cap - 37][:B]
    while len(base) < B:
        base.append(int(rng.integers(budget + 1, cap + 1)))
    for b in long_rows:
        base[b] = cap
    L = np.zeros((nl, B, Hkv), np.int32)
    for l in range(nl):
        for b in range(B):
            jitter = 0 if l == 0 else int(rng.integers(-20, 21))
            L[l, b, :] = min(cap, max(1, base[b] + jitter))
    return L


def _run_ragged(wl, budget, seed, mean=False, causal=False, cfps_beacons=0, bad=None):
    dev = torch.device("cuda")
    lib = O.load()
    cap = wl.capacity
    inp = synth.step_inputs(wl, seed, dev)
    n_inst, G, W, d = wl.n_inst, wl.group, wl.window, wl.head_dim
    Ls = _lengths(wl, budget, cap, seed)
    if bad is not None:
        Ls.reshape(-1)[bad] = cap + 5
    # positions per batch row: row b's newest token is at t_b, its window the W steps before
    t_rows = [int(Ls[0, b, 0]) - 1 + 1000 * b for b in range(wl.batch)]
    rp_rows = [[t - W + 1 + w for w in range(W)] for t in t_rows]
    if causal:  # one row with scattered recent positions (some see no window row)
        rp_rows[0] = [t_rows[0] - 5000, t_rows[0] - 3] + rp_rows[0][2:]
    L_dev = torch.as_tensor(Ls, device=dev)
    kw = dict(mean_agg=mean, causal_window=causal)
    if cfps_beacons:
        bk = bkv.BeaconKV(n_layers=wl.n_layers, batch=wl.batch, n_q_heads=wl.n_q_heads, n_kv_heads=wl.n_kv_heads,
                          head_dim=d, n_beacons=cfps_beacons, window=W, capacity=cap, rope_theta=wl.rope_theta,
                          continual_fps=True, **kw)
    else:
        bk = bkv.BeaconKV.for_workload(wl, **kw)
    try:
        bk.init_beacons(inp["q_init"])
        bk.update(inp["q_new"])
        if cfps_beacons:
            buf, size = bk.cfps_state()
            buf, size = _bits(buf).reshape(-1, cfps_beacons + W, d), size.cpu().numpy().reshape(-1)
        else:
            cent, _, counts = [x.cpu().numpy() for x in bk.state()]
        K0, V0 = _bits(inp["K"]).reshape(n_inst, cap, d), _bits(inp["V"]).reshape(n_inst, cap, d)
        scores = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads, cap), -1.0, device=dev)
        kept = bk.compress_ragged(inp["K"], inp["V"], L=L_dev, budget=budget, t_pos=t_rows,
                                  q_recent=inp["q_recent"], recent_pos=rp_rows, scores_out=scores)
        if bad is not None:
            with pytest.raises(bkv.BkvError) as ei:
                bk.sync()
            assert ei.value.code == bkv.BKV_EINVAL and "length" in str(ei.value)
        bk.sync()
        if cfps_beacons:
            buf2, size2 = bk.cfps_state()
            buf2, size2 = _bits(buf2).reshape(-1, cfps_beacons + W, d), size2.cpu().numpy().reshape(-1)
    finally:
        bk.close()
    K1, V1 = _bits(inp["K"]).reshape(n_inst, cap, d), _bits(inp["V"]).reshape(n_inst, cap, d)
    kept = kept.view(n_inst, budget).cpu().numpy()
    s_g = scores.view(n_inst, cap).cpu().numpy()
    q_rec = _bits(inp["q_recent"]).reshape(n_inst, G, W, d)
    Lf = Ls.reshape(-1)
    rel_max, swaps, ties, n_evicted = 0.0, 0, 0, 0
    for e in range(n_inst):
        b = (e // wl.n_kv_heads) % wl.batch
        L = int(Lf[e])
        tag = f"instance {e} (L = {L}, batch row {b})"
        if not (1 <= L <= cap):  # rejected length: untouched, kept all -1
            assert np.all(kept[e] == -1), tag
            np.testing.assert_array_equal(K1[e], K0[e], err_msg=tag)
            np.testing.assert_array_equal(V1[e], V0[e], err_msg=tag)
            continue
        if L > budget:
            n_evicted += 1
            # rows past the budget, and past L, are byte-unchanged
            np.testing.assert_array_equal(K1[e, budget:], K0[e, budget:], err_msg=tag)
            np.testing.assert_array_equal(V1[e, budget:], V0[e, budget:], err_msg=tag)
            assert np.all(s_g[e, L:] == -1.0), tag
        else:
            np.testing.assert_array_equal(V1[e], V0[e], err_msg=tag)
            assert np.all(s_g[e] == -1.0), tag
        if cfps_beacons:
            hs = slice(e * G, (e + 1) * G)
            r, sw, t = P.check_cfps_compress(wl, cfps_beacons, buf[hs], size[hs], q_rec[e], rp_rows[b], t_rows[b],
                                             K0[e], V0[e], K1[e], V1[e], kept[e], s_g[e], L, budget, buf2[hs],
                                             size2[hs], lib, tag=tag, mean=mean, causal=causal)
            ties += t
        else:
            r, sw = P.check_compress(wl, cent[e], counts[e], q_rec[e], rp_rows[b], t_rows[b], K0[e], V0[e], K1[e],
                                     V1[e], kept[e], s_g[e], L, budget, lib, tag=tag, mean=mean, causal=causal)
        rel_max, swaps = max(rel_max, r), swaps + sw
    assert n_evicted > 0 and n_evicted < n_inst
    print(f"{wl.name}: {n_inst} instances, {n_evicted} compressed, max score rel err {rel_max:.2e}, "
          f"boundary swaps {swaps}, FPS ties {ties}")


RAGGED = QWEN3_4B.scaled(name="ragged_2L_b6_cap1200", n_layers=2, batch=6, L=1200, budget=300)


@pytest.mark.parametrize("form", ["max", "mean", "causal", "causal_mean"])
def test_ragged_lengths_per_instance(form):
    _run_ragged(RAGGED, 300, seed=81, mean="mean" in form, causal="causal" in form)


def test_ragged_long_caches_stream_tiles():
    """Capacity 20000: the plan is made for the longest cache, so the long instances stream tiles past
    the tensor-memory ring while the short ones own a few tiles per CTA or none."""
    wl = QWEN3_4B.scaled(name="ragged_1L_b3_cap20000", n_layers=1, batch=3, L=20000, budget=5000)
    _run_ragged(wl, 5000, seed=82)


def test_ragged_with_continual_fps():
    _run_ragged(RAGGED, 300, seed=83, cfps_beacons=8)


def test_ragged_rejects_a_length_outside_the_capacity():
    _run_ragged(RAGGED, 300, seed=84, bad=[5, 40])


def test_ragged_equals_uniform_compress_when_every_length_is_equal():
    """With one length for every instance and one position set for every batch row, the ragged entry
    point computes what bkv_compress computes: identical kept indices, scores and K / V bytes."""
    wl = QWEN3_4B.scaled(name="ragged_uniform_1L_b2", n_layers=1, batch=2, L=1000, budget=700)
    dev = torch.device("cuda")
    inp = synth.step_inputs(wl, 85, dev)
    outs = []
    for ragged in (False, True):
        K, V = inp["K"].clone(), inp["V"].clone()
        bk = bkv.BeaconKV.for_workload(wl)
        try:
            bk.init_beacons(inp["q_init"])
            bk.update(inp["q_new"])
            sc = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads, wl.capacity), -1.0, device=dev)
            if ragged:
                L = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads), wl.L, dtype=torch.int32, device=dev)
                kept = bk.compress_ragged(K, V, L=L, budget=wl.budget, t_pos=[inp["t_pos"]] * wl.batch,
                                          q_recent=inp["q_recent"], recent_pos=[inp["recent_pos"]] * wl.batch,
                                          scores_out=sc)
            else:
                kept = bk.compress(K, V, L=wl.L, budget=wl.budget, t_pos=inp["t_pos"], q_recent=inp["q_recent"],
                                   recent_pos=inp["recent_pos"], scores_out=sc)
            bk.sync()
        finally:
            bk.close()
        outs.append((kept.cpu(), sc.cpu(), K.cpu(), V.cpu()))
    for a, b in zip(*outs):
        assert torch.equal(a, b)
