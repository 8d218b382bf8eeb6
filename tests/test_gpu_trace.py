"""Decode trace through the C ABI against the fp64 oracle at every step.

A shortened version of the long-trace workload (one layer, one batch row, 8 KV
heads, 4 query heads per KV head, 16 beacons, drifting query clusters): after
a 128-token prompt, every decode step adds one pre-RoPE query per query head
(one beacon update with n_new = 1, four queries per instance) and one K / V
row; whenever the cache reaches budget + 64 rows it is compressed to the
budget.  Every update is checked (assignments up to oracle ties, counts, sums,
centroids) and every compress (scores, kept set, compacted rows), each from
the state the GPU carried forward.
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


@pytest.mark.parametrize("steps,budget", [(400, 256)])
def test_decode_trace_every_step(steps, budget):
    grow = 64
    wl = QWEN3_8B_TRACE.scaled(name="trace_1L_b1", n_layers=1, batch=1, L=budget + grow, budget=budget,
                               trace_steps=steps)
    dev = torch.device("cuda")
    lib = O.load()
    n_inst, G, d, W, Hq = wl.n_inst, wl.group, wl.head_dim, wl.window, wl.n_q_heads
    gen = synth.TraceGen(wl, seed=21, device=dev)
    q_init, k0, v0 = gen.prefill()
    cap = wl.capacity
    K = torch.zeros(wl.n_layers, wl.batch, wl.n_kv_heads, cap, d, dtype=torch.bfloat16, device=dev)
    V = torch.zeros_like(K)
    L = wl.prefill
    K[:, :, :, :L] = k0
    V[:, :, :, :L] = v0
    pos = L                      # absolute position of the next token
    hist, hist_pos = [], []      # recent decode queries per query head and their positions

    bk = BeaconKV.for_workload(wl)
    ties = swaps = compresses = 0
    worst_cent = worst_score = 0.0
    try:
        bk.init_beacons(q_init)
        state = [x.cpu().numpy() for x in bk.state()]
        assign = torch.empty(wl.n_layers, wl.batch, Hq, 1, dtype=torch.int32, device=dev)
        for step in range(steps):
            q = gen.step_queries()                           # [1, 1, Hq, 1, d]
            bk.update(q, assign)
            new_state = [x.cpu().numpy() for x in bk.state()]
            qb = _bits(q).reshape(n_inst, G, d)              # group-major rows of each instance
            a_g = assign.view(n_inst, G).cpu().numpy()
            for e in range(n_inst):
                pre = dict(cent=state[0][e].copy(), sums=state[1][e].copy(), counts=state[2][e].copy())
                post = dict(cent=new_state[0][e], sums=new_state[1][e], counts=new_state[2][e])
                t, c = P.check_update(qb[e], pre, a_g[e], post, lib, tag=f"step {step} instance {e}")
                ties += t
                worst_cent = max(worst_cent, c)
            state = new_state

            k, v = gen.kv_rows(1)
            K[:, :, :, L] = k[:, :, :, 0]
            V[:, :, :, L] = v[:, :, :, 0]
            L += 1
            hist.append(q[:, :, :, 0])
            hist_pos.append(pos)
            pos += 1
            hist, hist_pos = hist[-W:], hist_pos[-W:]

            if L == budget + grow:
                q_recent = torch.stack(hist, dim=3)          # [1, 1, Hq, W, d]
                K0 = _bits(K.view(n_inst, cap, d))
                V0 = _bits(V.view(n_inst, cap, d))
                scores = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads, cap), -1.0, device=dev)
                kept = bk.compress(K, V, L=L, budget=budget, t_pos=pos - 1, q_recent=q_recent,
                                   recent_pos=list(hist_pos), scores_out=scores)
                bk.sync()
                K1 = _bits(K.view(n_inst, cap, d))
                V1 = _bits(V.view(n_inst, cap, d))
                kept_h = kept.view(n_inst, budget).cpu().numpy()
                s_h = scores.view(n_inst, cap).cpu().numpy()
                qr = _bits(q_recent).reshape(n_inst, G, W, d)
                for e in range(n_inst):
                    r, sw = P.check_compress(wl, state[0][e], state[2][e], qr[e], hist_pos, pos - 1, K0[e], V0[e],
                                             K1[e], V1[e], kept_h[e], s_h[e], L, budget, lib,
                                             tag=f"step {step} instance {e}")
                    worst_score = max(worst_score, r)
                    swaps += sw
                compresses += 1
                L = budget
    finally:
        bk.close()
    print(f"trace: {steps} steps, {compresses} compresses, assignment ties {ties}, worst centroid error "
          f"{worst_cent:.2e}, worst score rel err {worst_score:.2e}, boundary swaps {swaps}")
    assert compresses == (steps - (budget + grow - wl.prefill)) // grow + 1
