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
