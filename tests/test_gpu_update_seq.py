"""bkv_update_beacons_seq: a run of decode steps in one call against one bkv_update_beacons call per
step (n_new = 1), through the C ABI.  The two must agree bit for bit: every assignment, every
centroid, running sum and count.  The per-step calls are themselves checked against the fp64 oracle
at every step of a decode trace (test_gpu_trace.py), so this equality carries that parity over.

Shapes: the long-trace shape (head_dim 128, 4 query heads and 16 beacons per KV head, drifting
clusters); head_dim 64 with 4 beacons and 8 query heads; 32 query heads and 32 beacons (one instance
per warp's full shared-memory state); one query head per KV head; more instances than the persistent
grid holds at once; states with duplicate beacons, empty slots and a zero centroid, and queries equal
to centroids (exact ties, exact re-decisions); zero queries; the step-by-step forms (Continual FPS,
more than 32 query heads per KV head, no beacons).
"""
import pytest
import torch

from paper_2609_04971_gb300.workloads import QWEN3_8B_TRACE

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from paper_2609_04971_gb300 import bkv, synth


def _steps(wl, n_steps, seed, zero_frac=0.0):
    """[n_steps, layers, batch, q_heads, d] decode queries from the drifting trace generator; a
    fraction of them set to zero (skipped by the update)."""
    gen = synth.TraceGen(wl, seed=seed, device=torch.device("cuda"))
    q_init, _, _ = gen.prefill()
    q = torch.stack([gen.step_queries()[:, :, :, 0] for _ in range(n_steps)])
    if zero_frac > 0.0:
        g = torch.Generator(device="cuda").manual_seed(seed + 1)
        z = torch.rand(q.shape[:-1], generator=g, device="cuda") < zero_frac
        q[z] = 0
    return q_init, q.contiguous()


def _ctx(wl, **kw):
    return bkv.BeaconKV(n_layers=wl.n_layers, batch=wl.batch, n_q_heads=wl.n_q_heads, n_kv_heads=wl.n_kv_heads,
                        head_dim=wl.head_dim, n_beacons=wl.n_beacons, window=wl.window, capacity=wl.capacity,
                        rope_theta=wl.rope_theta, **kw)


def _snapshot(bk, cfps):
    if cfps:
        return [t.cpu() for t in bk.cfps_state()]
    c, s, n = bk.state()
    return [c.cpu().view(torch.int32), s.cpu().view(torch.int64), n.cpu()]


def _compare(wl, q_steps, q_init=None, state=None, cfps=False, with_assign=True, chunks=None):
    """Per-step calls and seq calls (in chunks of the given step counts) from the same start."""
    n_steps = q_steps.shape[0]
    per_step = wl.n_layers * wl.batch * wl.n_q_heads
    outs = []
    for seq in (False, True):
        bk = _ctx(wl, continual_fps=cfps)
        try:
            if state is not None:
                bk.set_state(*state)
            else:
                bk.init_beacons(q_init)
            assign = torch.full((n_steps, per_step), -7, dtype=torch.int32, device="cuda")
            if seq:
                t = 0
                for n in chunks or [n_steps]:
                    bk.update_seq(q_steps[t:t + n], assign[t:t + n] if with_assign else None)
                    t += n
                assert t == n_steps
            else:
                for t in range(n_steps):
                    bk.update(q_steps[t].unsqueeze(-2), assign[t] if with_assign else None)
            bk.sync()
            outs.append((assign.cpu(), _snapshot(bk, cfps)))
        finally:
            bk.close()
    (a0, s0), (a1, s1) = outs
    assert torch.equal(a0, a1), "assignments differ"
    for x, y, name in zip(s0, s1, ("centroids", "sums", "counts")):
        assert torch.equal(x, y), f"{name} differ"
    return a0


TRACE = QWEN3_8B_TRACE.scaled(name="trace_2L_b3", n_layers=2, batch=3)


def test_seq_equals_per_step_trace_shape():
    q_init, q = _steps(TRACE, 150, seed=31)
    a = _compare(TRACE, q, q_init)
    assert (a >= 0).all()  # every query assigned (no zero queries here)


def test_seq_in_chunks_and_without_assignments():
    q_init, q = _steps(TRACE, 64, seed=32, zero_frac=0.05)
    _compare(TRACE, q, q_init, chunks=[1, 17, 30, 16])
    _compare(TRACE, q, q_init, chunks=[1] * 64)
    _compare(TRACE, q, q_init, with_assign=False)


@pytest.mark.parametrize("shape", ["d64_g8_nb4", "d128_g32_nb32", "d64_g1_nb8", "d128_g2_nb3", "d128_g5_nb16",
                                   "d64_g5_nb2", "d128_g16_nb16"])
def test_seq_equals_per_step_shapes(shape):
    kw = {
        "d64_g8_nb4": dict(head_dim=64, n_q_heads=16, n_kv_heads=2, n_beacons=4, n_clusters=4),
        "d128_g32_nb32": dict(head_dim=128, n_q_heads=64, n_kv_heads=2, n_beacons=32, n_clusters=24, window=2),
        "d64_g1_nb8": dict(head_dim=64, n_q_heads=8, n_kv_heads=8, n_beacons=8, n_clusters=8),
        "d128_g2_nb3": dict(head_dim=128, n_q_heads=8, n_kv_heads=4, n_beacons=3, n_clusters=3),
        "d128_g5_nb16": dict(head_dim=128, n_q_heads=40, n_kv_heads=8, n_beacons=16, n_clusters=16),  # Qwen3-14B
        "d64_g5_nb2": dict(head_dim=64, n_q_heads=10, n_kv_heads=2, n_beacons=2, n_clusters=2),
        "d128_g16_nb16": dict(head_dim=128, n_q_heads=32, n_kv_heads=2, n_beacons=16, n_clusters=16, window=4),
    }[shape]
    wl = QWEN3_8B_TRACE.scaled(name=shape, n_layers=2, batch=2, **kw)
    q_init, q = _steps(wl, 45, seed=33, zero_frac=0.1)
    a = _compare(wl, q, q_init)
    assert (a == -1).any() and (a >= 0).any()


def test_seq_more_instances_than_resident_warps():
    """2560 instances: the persistent warps take several instances each, reusing their shared memory."""
    wl = QWEN3_8B_TRACE.scaled(name="many", n_layers=4, batch=40, n_q_heads=32, n_kv_heads=16, head_dim=64,
                               n_beacons=8, n_clusters=8)
    q_init, q = _steps(wl, 6, seed=34)
    _compare(wl, q, q_init)


def test_seq_duplicate_beacons_and_exact_ties():
    """Duplicate centroids (exact ties: the lower beacon wins), empty slots, a zero centroid with a
    count, and queries equal to centroids or to their negatives: the exact re-decision path at most
    steps."""
    wl = QWEN3_8B_TRACE.scaled(name="ties", n_layers=1, batch=2, n_q_heads=16, n_kv_heads=4, n_beacons=8,
                               n_clusters=4)
    n_inst, nb, d, G = wl.n_inst, wl.n_beacons, wl.head_dim, wl.group
    g = torch.Generator().manual_seed(35)
    base = torch.randn(n_inst, 4, d, generator=g).to(torch.bfloat16).float()
    cent = torch.cat([base, base[:, :2], torch.zeros(n_inst, 2, d)], dim=1)  # beacons 4, 5 duplicate 0, 1
    counts = torch.tensor([3, 1, 2, 5, 4, 2, 0, 7], dtype=torch.int64).repeat(n_inst, 1)  # 6 empty, 7 zero
    sums = cent.double() * counts.unsqueeze(-1).double()
    state = (cent.cuda(), sums.cuda(), counts.cuda())
    steps = 40
    pick = torch.randint(0, 8, (steps, n_inst, G), generator=g)
    sign = torch.where(torch.rand(steps, n_inst, G, generator=g) < 0.2, -1.0, 1.0)
    q = torch.stack([torch.stack([cent[e, pick[t, e]] for e in range(n_inst)]) for t in range(steps)])
    q = (q * sign.unsqueeze(-1)).to(torch.bfloat16)
    q = q.view(steps, wl.n_layers, wl.batch, wl.n_q_heads, d).cuda().contiguous()
    a = _compare(wl, q, state=state)
    assert (a >= 0).any()


@pytest.mark.parametrize("form", ["continual_fps", "g40", "no_beacons"])
def test_seq_step_by_step_forms(form):
    if form == "continual_fps":
        wl = TRACE.scaled(name="cfps", n_beacons=8)
        q_init, q = _steps(wl, 30, seed=36)
        a = _compare(wl, q, q_init, cfps=True)
        assert (a == -1).all()
    elif form == "g40":
        wl = TRACE.scaled(name="g40", n_q_heads=80, n_kv_heads=2, n_clusters=8, window=2, n_init=64)
        q_init, q = _steps(wl, 12, seed=37)
        _compare(wl, q, q_init)
    else:
        wl = TRACE.scaled(name="nb0", n_beacons=0)
        q = torch.randn(5, wl.n_layers, wl.batch, wl.n_q_heads, wl.head_dim, device="cuda").to(torch.bfloat16)
        bk = _ctx(wl)
        try:
            assign = torch.zeros(5, wl.n_layers * wl.batch * wl.n_q_heads, dtype=torch.int32, device="cuda")
            bk.update_seq(q, assign)
            bk.sync()
            assert (assign == -1).all()
        finally:
            bk.close()


def test_seq_rejects_bad_arguments():
    bk = _ctx(TRACE)
    try:
        q = torch.zeros(3, TRACE.n_layers, TRACE.batch, TRACE.n_q_heads, TRACE.head_dim, dtype=torch.bfloat16,
                        device="cuda")
        with pytest.raises(bkv.BkvError) as ei:  # no beacon state yet
            bk.update_seq(q)
        assert ei.value.code == bkv.BKV_ESTATE
        with pytest.raises(ValueError):
            bk.update_seq(q[..., :64].contiguous())
        with pytest.raises(bkv.BkvError) as ei:
            bkv.bkv_update_beacons_seq(bk.ctx, q, -1)
        assert ei.value.code == bkv.BKV_EINVAL
        bkv.bkv_update_beacons_seq(bk.ctx, q, 0)  # no-op, even before any state
    finally:
        bk.close()


def _large_state(wl, seed, base, spread):
    """Sums far from zero (|s| around `base`, on the 2^-40 grid), counts in the thousands, centroids
    fp32(s / n): the running sums cross 2^13, 2^14, ... (the double's grid coarsens) over the steps."""
    n_inst, nb, d = wl.n_inst, wl.n_beacons, wl.head_dim
    g = torch.Generator().manual_seed(seed)
    counts = torch.randint(2000, 6000, (n_inst, nb), generator=g, dtype=torch.int64)
    sign = torch.where(torch.rand(n_inst, nb, d, generator=g) < 0.5, -1.0, 1.0).double()
    mag = base + spread * torch.rand(n_inst, nb, d, generator=g, dtype=torch.float64)
    sums = torch.round(sign * mag * 2.0 ** 20) / 2.0 ** 20  # multiples of 2^-20
    cent = (sums / counts.unsqueeze(-1).double()).float()
    return cent, sums, counts


@pytest.mark.parametrize("case", ["cross_2p13", "near_binades", "past_2p18"])
def test_seq_large_running_sums(case):
    """Running sums past 2^13, where fold_sum rounds every step's total to the double's grid: the seq
    kernel's exact parts must round alike; sums starting just below powers of two (the binade read
    exactly); sums that reach 2^18 (the warp's columns go to fp64 form mid-call)."""
    wl = QWEN3_8B_TRACE.scaled(name="large", n_layers=1, batch=2, n_q_heads=16, n_kv_heads=4, n_beacons=8,
                               n_clusters=8)
    base, spread = {"cross_2p13": (7000.0, 3000.0), "near_binades": (0.0, 0.0),
                    "past_2p18": (260000.0, 3000.0)}[case]
    cent, sums, counts = _large_state(wl, 40, base, spread)
    if case == "near_binades":  # each element a few 2^-20 steps below 2^k, k = 13 .. 17
        g = torch.Generator().manual_seed(41)
        k = torch.randint(13, 18, sums.shape, generator=g)
        below = torch.randint(1, 64, sums.shape, generator=g).double() * 2.0 ** -20
        sgn = torch.where(torch.rand(sums.shape, generator=g) < 0.5, -1.0, 1.0).double()
        sums = sgn * (2.0 ** k.double() - below)
        cent = (sums / counts.unsqueeze(-1).double()).float()
    steps = 60
    n_inst, G, d = wl.n_inst, wl.group, wl.head_dim
    g = torch.Generator().manual_seed(42)
    pick = torch.randint(0, wl.n_beacons, (steps, n_inst, G), generator=g)
    direction = torch.sign(cent)  # queries along the centroids' signs: the sums keep growing in magnitude
    q = torch.stack([torch.stack([direction[e, pick[t, e]] for e in range(n_inst)]) for t in range(steps)])
    scale = 2.0 ** -10 if case == "near_binades" else 3.0
    noise = torch.randn(q.shape, generator=g) * (0.25 * scale)
    q = (q * scale + noise).to(torch.bfloat16)
    q = q.view(steps, wl.n_layers, wl.batch, wl.n_q_heads, d).cuda().contiguous()
    a = _compare(wl, q, state=(cent.cuda(), sums.cuda(), counts.cuda()))
    assert (a >= 0).all()


def test_seq_and_per_step_calls_against_the_oracle():
    """Every per-step call checked against the fp64 oracle from the GPU's carried state, and the seq call
    bit-identical to them (the check __graft_entry__.smoke() runs)."""
    from paper_2609_04971_gb300.workloads import TINY
    from tests import parity as P
    P.smoke_decode_steps(TINY, steps=12, seed=3)
    P.smoke_decode_steps(QWEN3_8B_TRACE.scaled(name="trace_1L_b2", n_layers=1, batch=2), steps=20, seed=4)
