"""Device-side failure reporting without a device fault: a bounded wait that
nothing completes expires, the kernel records it in the error word and
returns, bkv_sync reports BKV_ETIMEOUT once, and the context keeps working."""
import pytest
import torch

from paper_2609_04971_gb300 import bkv
from paper_2609_04971_gb300.workloads import TINY

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from tests import parity as P


def test_expired_wait_reports_timeout_then_context_recovers():
    bk = bkv.BeaconKV.for_workload(TINY)
    try:
        assert bkv.bkv_selftest_wait_timeout(bk.ctx, 20_000_000) == bkv.BKV_ETIMEOUT   # 20 ms limit
        bkv.bkv_sync(bk.ctx)                                       # the error word was cleared
        assert bkv.bkv_selftest_wait_timeout(bk.ctx, 1_000_000) == bkv.BKV_ETIMEOUT    # and can expire again
        with pytest.raises(bkv.BkvError):
            bkv.bkv_selftest_wait_timeout(bk.ctx, 10)              # limit below 1 us is rejected
    finally:
        bk.close()
    # the device and the library still compute correct results afterwards
    run = P.run_gpu(TINY)
    P.check_run(run)


def test_rejected_arguments_leave_everything_untouched():
    """Argument errors of bkv_update_beacons and bkv_compress are caught on the host before any work is
    enqueued: each call raises with its documented code, and K, V, the kept-index output and the beacon
    state are unchanged afterwards; an update of zero queries is a no-op."""
    from paper_2609_04971_gb300 import synth
    wl = TINY
    dev = torch.device("cuda")
    inp = synth.step_inputs(wl, 3, dev)
    K, V = inp["K"], inp["V"]
    kept = torch.full((wl.n_layers, wl.batch, wl.n_kv_heads, wl.budget), -7, dtype=torch.int32, device=dev)
    pos = dict(t_pos=inp["t_pos"], recent_pos=inp["recent_pos"])

    def code_of(fn):
        with pytest.raises(bkv.BkvError) as ei:
            fn()
        return ei.value.code

    bk = bkv.BeaconKV.for_workload(wl)
    try:
        # before bkv_init_beacons: no beacon state yet
        assert code_of(lambda: bkv.bkv_update_beacons(bk.ctx, inp["q_new"], wl.n_new)) == bkv.BKV_ESTATE
        assert code_of(lambda: bkv.bkv_compress(bk.ctx, K, V, wl.L, wl.budget, q_recent=inp["q_recent"],
                                                kept_idx_out=kept, **pos)) == bkv.BKV_ESTATE
        bk.init_beacons(inp["q_init"])
        state0 = [t.clone() for t in bk.state()]
        K0, V0 = K.clone(), V.clone()
        q_odd = inp["q_new"].view(-1)[1:]  # 2 bytes past a 16-byte boundary
        K_odd = K.view(-1)[1:]
        assert code_of(lambda: bkv.bkv_update_beacons(bk.ctx, inp["q_new"], -1)) == bkv.BKV_EINVAL
        assert code_of(lambda: bkv.bkv_update_beacons(bk.ctx, q_odd, wl.n_new)) == bkv.BKV_EINVAL
        bkv.bkv_update_beacons(bk.ctx, inp["q_new"], 0)  # no queries: nothing to do
        for L, budget, k, q in [(0, wl.budget, K, inp["q_recent"]),                 # empty cache
                                (wl.capacity + 1, wl.budget, K, inp["q_recent"]),   # past the capacity
                                (wl.L, wl.window - 1, K, inp["q_recent"]),          # budget below the window
                                (wl.L, wl.budget, K_odd, inp["q_recent"]),          # misaligned K
                                (wl.L, wl.budget, K, None)]:                        # window queries missing
            assert code_of(lambda: bkv.bkv_compress(bk.ctx, k, V, L, budget, q_recent=q, kept_idx_out=kept,
                                                    **pos)) == bkv.BKV_EINVAL, (L, budget)
        bk.sync()
        assert torch.equal(K, K0) and torch.equal(V, V0)
        assert bool((kept == -7).all())
        for a, b in zip(bk.state(), state0):
            assert torch.equal(a, b)
        # the context still works: a valid step keeps the budget with the window
        bk.update(inp["q_new"])
        bk.compress(K, V, L=wl.L, budget=wl.budget, q_recent=inp["q_recent"], kept_out=kept, **pos)
        bk.sync()
        k_h = kept.view(-1, wl.budget).cpu()
        assert bool((k_h[:, 1:] > k_h[:, :-1]).all())
        assert bool((k_h[:, -wl.window:] == torch.arange(wl.L - wl.window, wl.L, dtype=torch.int32)).all())
    finally:
        bk.close()


def test_state_round_trip_through_host_memory():
    """bkv_get_state / bkv_set_state take host buffers as well as device ones: a state saved to pageable
    and pinned host tensors and restored into a second context gives, after the same update, the same
    state as the original context."""
    from paper_2609_04971_gb300 import bkv, synth
    from paper_2609_04971_gb300.workloads import QWEN3_4B
    wl = QWEN3_4B.scaled(name="state_host", n_layers=1, batch=2)
    dev = torch.device("cuda")
    inp = synth.step_inputs(wl, 57, dev)
    a, b = bkv.BeaconKV.for_workload(wl), bkv.BeaconKV.for_workload(wl)
    try:
        a.init_beacons(inp["q_init"])
        a.update(inp["q_new"][..., :64, :].contiguous())
        shape = (wl.n_inst, wl.n_beacons)
        host = [torch.empty(shape + (wl.head_dim,), dtype=torch.float32),
                torch.empty(shape + (wl.head_dim,), dtype=torch.float64, pin_memory=True),
                torch.empty(shape, dtype=torch.int64)]
        bkv.bkv_get_state(a.ctx, *host)
        a.sync()
        dev_state = a.state()
        torch.cuda.synchronize()
        for h, d in zip(host, dev_state):
            assert torch.equal(h, d.cpu())
        bkv.bkv_set_state(b.ctx, *host)
        rest = inp["q_new"][..., 64:, :].contiguous()
        a.update(rest)
        b.update(rest)
        for x, y in zip(a.state(), b.state()):
            assert torch.equal(x, y)
    finally:
        a.close()
        b.close()
