"""Algorithm 2's phase machine on a decode trace, Continual FPS beacons, through the C ABI.

A shortened long-decode workload (one layer, one batch row, 8 KV heads, 4 query
heads per KV head, drifting query clusters) after a 128-token prompt, at two
B_max -> B_min settings (320 -> 256, and 320 -> 280 = 7/8 B_max with 4 leading
rows always kept):

  * while the cache holds at most B_max - window rows, each step's query of
    every head joins that head's buffer (bkv_update_beacons, n_new = 1;
    the buffer is compressed by FPS whenever it fills, Eq. 9);
  * the next `window` steps' queries are kept aside with their positions as
    the recent queries (the beacons are frozen: the buffers no longer change);
  * when the cache reaches B_max rows it is compressed to B_min rows
    (bkv_compress with the frozen beacons and the recent queries), and each
    buffer becomes the FPS selection of its beacons and recent queries.

Every update is checked against the oracle's fp64 buffer (Eq. 9, Algorithm 1)
up to near-ties of the kernels' fp32 decisions (tests/parity.search_branches),
and every compress as in tests/parity.py, always from the state the GPU
carried forward.
"""
import numpy as np
import pytest
import torch

from paper_2609_04971_gb300.workloads import QWEN3_8B_TRACE

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from oracle import oracle as O
    from paper_2609_04971_gb300 import synth
    from paper_2609_04971_gb300.bkv import BeaconKV
    from tests import parity as P


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("steps,b_min,kv_min,kv_grow,n_prefix", [
    (420, 8, 256, 64, 0),
    (420, 8, 280, 40, 4),  # B_min = 7/8 B_max (Section 4.1), with 4 leading rows always kept
])
def test_algorithm2_trace_every_step(steps, b_min, kv_min, kv_grow, n_prefix):
    kv_max = kv_min + kv_grow
    wl = QWEN3_8B_TRACE.scaled(name="trace_cfps_1L_b1", n_layers=1, batch=1, L=kv_max, budget=kv_min,
                               trace_steps=steps, n_prefix=n_prefix)
    dev = torch.device("cuda")
    lib = O.load()
    G, d, W, Hq = wl.group, wl.head_dim, wl.window, wl.n_q_heads
    b_max = b_min + W
    n_inst = wl.n_inst
    gen = synth.TraceGen(wl, seed=31, device=dev)
    q_init, k0, v0 = gen.prefill()
    K = torch.zeros(wl.n_layers, wl.batch, wl.n_kv_heads, kv_max, d, dtype=torch.bfloat16, device=dev)
    V = torch.zeros_like(K)
    L = wl.prefill
    K[:, :, :, :L] = k0
    V[:, :, :, :L] = v0
    pos = L                       # absolute position of the next token
    recent, recent_pos = [], []

    bk = BeaconKV(n_layers=wl.n_layers, batch=wl.batch, n_q_heads=Hq, n_kv_heads=wl.n_kv_heads, head_dim=d,
                  n_beacons=b_min, window=W, capacity=kv_max, rope_theta=wl.rope_theta, n_prefix=wl.n_prefix,
                  continual_fps=True)

    def state():
        buf, sizes = bk.cfps_state()
        return _bits(buf).reshape(-1, b_max, d), sizes.cpu().numpy().reshape(-1)

    updates = compresses = swaps = ties = 0
    worst = 0.0
    try:
        bk.init_beacons(q_init)
        buf, size = state()
        for step in range(steps):
            q = gen.step_queries()                                   # [1, 1, Hq, 1, d]
            k, v = gen.kv_rows(1)
            K[:, :, :, L] = k[:, :, :, 0]
            V[:, :, :, L] = v[:, :, :, 0]
            L += 1
            if L <= kv_max - W:                                      # observation phase
                bk.update(q)
                nbuf, nsize = state()
                qh = _bits(q).reshape(-1, 1, d)                     # [heads, 1, d]
                for h in range(qh.shape[0]):
                    ties += P.match_cfps_update(buf[h], int(size[h]), b_min, b_max, qh[h], nbuf[h], int(nsize[h]),
                                                lib, tag=f"step {step} head {h}")
                buf, size = nbuf, nsize
                updates += 1
            else:                                                    # recent phase (beacons frozen)
                recent.append(q[:, :, :, 0])
                recent_pos.append(pos)
            if L == kv_max:                                          # compress to kv_min rows
                q_recent = torch.stack(recent, dim=3)                # [1, 1, Hq, W, d]
                K0 = _bits(K).reshape(n_inst, kv_max, d)
                V0 = _bits(V).reshape(n_inst, kv_max, d)
                scores = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads, kv_max), -1.0, device=dev)
                kept = bk.compress(K, V, L=L, budget=kv_min, t_pos=pos, q_recent=q_recent, recent_pos=list(recent_pos),
                                   scores_out=scores)
                bk.sync()
                nbuf, nsize = state()
                K1 = _bits(K).reshape(n_inst, kv_max, d)
                V1 = _bits(V).reshape(n_inst, kv_max, d)
                kept_h = kept.view(n_inst, kv_min).cpu().numpy()
                s_h = scores.view(n_inst, kv_max).cpu().numpy()
                qr = _bits(q_recent).reshape(-1, W, d)
                for e in range(n_inst):
                    hs = slice(e * G, (e + 1) * G)
                    r, sw, t = P.check_cfps_compress(wl, b_min, buf[hs], size[hs], qr[hs], recent_pos, pos, K0[e],
                                                     V0[e], K1[e], V1[e], kept_h[e], s_h[e], L, kv_min, nbuf[hs],
                                                     nsize[hs], lib, tag=f"step {step} instance {e}")
                    worst, swaps, ties = max(worst, r), swaps + sw, ties + t
                buf, size = nbuf, nsize
                L = kv_min
                recent, recent_pos = [], []
                compresses += 1
            pos += 1
    finally:
        bk.close()
    print(f"trace (Algorithm 2, Continual FPS): {steps} steps, {updates} updates, {compresses} compresses, "
          f"worst score rel err {worst:.2e}, boundary swaps {swaps}, FPS near-tie departures {ties}")
    first = kv_max - wl.prefill                                      # steps until the first compress
    assert compresses == 1 + (steps - first) // kv_grow
