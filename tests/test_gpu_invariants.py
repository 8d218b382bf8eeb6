"""The compress path on inputs far from unit logit spread, and the invariants the
method promises, through the C ABI against the fp64 oracle.

Large logit ranges (Eq. 4 over all L keys; Eq. 6 max and mean forms; the causal
mask inside the window), at a cache length whose tiles stream past the
tensor-memory ring (L = 20000):
  * every key scaled by 24: logits of standard deviation ~24, base-2 spread far
    beyond 64 (the score kernel's running sums move their reference);
  * a key planted late in the cache with a logit near +60 for one recent query,
    after a planted +20 key earlier (the reference moves twice, in a later
    CTA's share of the keys than the first);
  * 3000 rows anti-aligned with the mean direction of the recent queries, at
    logits near -400 for the queries along it (weights far below the smallest
    normal fp32 value; queries nearly orthogonal to it see moderate logits).
Scores are compared within 1e-3 relative plus 2^-126 absolute (fp32 holds no
smaller normal value).  For the scaled keys the kept-set tie margin is derived
from the fp32 error bound of the logits (tests/parity.logit_tie_rtol): the
default 1e-5 is below what fp32 scoring can resolve there.

Permutation invariance (the running mean and the max-form score do not depend
on the order of the query set): permuting the new queries within a call and
the query heads within each group leaves the beacon state, the scores, the
kept sets and the compacted rows bit-identical, and permutes the assignments.
"""
import math

import numpy as np
import pytest
import torch

from paper_2609_04971_gb300.workloads import QWEN3_4B

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from oracle import oracle as O
    from paper_2609_04971_gb300 import synth
    from tests import parity as P

LONG = QWEN3_4B.scaled(name="logits_L20000", n_layers=1, batch=1, L=20000, budget=9000)


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _recent_rows(wl, inp, e: int) -> np.ndarray:
    """The rotated, bf16-rounded recent scoring queries of instance e (fp64 [G * W, d]), from the oracle."""
    G, W, d = wl.group, wl.window, wl.head_dim
    qr = _bits(inp["q_recent"].reshape(wl.n_inst, G, W, d)[e])
    qobs, _ = O.build_qobs(np.zeros((0, d), np.float32), np.zeros(0, np.int64), qr,
                           np.asarray(inp["recent_pos"], np.int64), inp["t_pos"], wl.rope_theta)
    return qobs


def _large_logit_inputs(case: str, seed: int):
    wl = LONG
    dev = torch.device("cuda")
    inp = synth.step_inputs(wl, seed, dev)
    K = inp["K"].view(wl.n_inst, wl.capacity, wl.head_dim)
    d = wl.head_dim
    if case == "keys_x24":
        K.copy_((K.float() * 24.0).to(torch.bfloat16))
    elif case == "late_spike_60":
        for e in range(wl.n_inst):
            q = _recent_rows(wl, inp, e)
            for row, logit, target in ((1000, 20.0, q[0]), (wl.L - 100, 60.0, q[0]), (wl.L - 2000, 45.0, q[5])):
                k = logit * math.sqrt(d) * target / float(target @ target)
                K[e, row] = torch.as_tensor(k, dtype=torch.float32, device=dev).to(torch.bfloat16)
    elif case == "negative_rows":
        g = torch.Generator(device=dev)
        g.manual_seed(seed + 1)
        for e in range(wl.n_inst):
            q = _recent_rows(wl, inp, e)
            u = q.mean(0)
            u = u / np.linalg.norm(u)
            beta = 400.0 * math.sqrt(d) / float(np.linalg.norm(q, axis=1).mean())
            k = torch.as_tensor(-beta * u, dtype=torch.float32, device=dev)
            K[e, 5000:8000] = (k[None, :] + 0.1 * torch.randn(3000, d, device=dev, generator=g)).to(torch.bfloat16)
    else:
        raise ValueError(case)
    return wl, inp


@pytest.mark.parametrize("form", ["max", "mean", "causal"])
@pytest.mark.parametrize("case", ["keys_x24", "late_spike_60", "negative_rows"])
def test_large_logit_ranges(case, form):
    wl, inp = _large_logit_inputs(case, seed=71)
    run = P.run_gpu(wl, inputs=inp, mean_agg=form == "mean", causal=form == "causal")
    rep = P.check_run(run, tie_rtol="fp32-bound" if case == "keys_x24" else None)
    print(f"{case}/{form}: {rep}")


def test_permutation_invariance():
    wl = QWEN3_4B.scaled(name="perm_1L_b2_L3000", n_layers=1, batch=2, L=3000, budget=2000)
    dev = torch.device("cuda")
    base = synth.step_inputs(wl, 62, dev)
    G, n, d = wl.group, wl.n_new, wl.head_dim
    g = torch.Generator().manual_seed(5)
    row_perm = torch.randperm(n, generator=g).to(dev)
    head_perm = torch.randperm(G, generator=g).to(dev)

    def heads(t):  # [nl, B, Hq, m, d] -> [nl, B, Hkv, G, m, d]
        return t.view(wl.n_layers, wl.batch, wl.n_kv_heads, G, t.shape[-2], d)

    perm = dict(base)
    perm["q_new"] = heads(base["q_new"])[:, :, :, head_perm][..., row_perm, :].reshape(base["q_new"].shape)
    perm["q_recent"] = heads(base["q_recent"])[:, :, :, head_perm].reshape(base["q_recent"].shape).contiguous()
    perm["q_new"] = perm["q_new"].contiguous()
    runs = []
    for inp in (base, perm):
        inp = dict(inp, K=base["K"].clone(), V=base["V"].clone())
        runs.append(P.run_gpu(wl, inputs=inp))
    a, b = runs
    for name in ("cent1", "sums1", "counts1", "kept", "scores", "K_after", "V_after"):
        np.testing.assert_array_equal(getattr(a, name), getattr(b, name), err_msg=name)
    # assignments: query (h', r') of the permuted call is query (head_perm[h'], row_perm[r']) of the original
    ia = a.assign.reshape(wl.n_inst, G, n)
    ib = b.assign.reshape(wl.n_inst, G, n)
    np.testing.assert_array_equal(ib, ia[:, head_perm.cpu()][:, :, row_perm.cpu()])
    print(f"permutation: {P.check_run(a)}")
