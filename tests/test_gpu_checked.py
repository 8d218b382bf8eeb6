"""Diagnostics without a device fault: the device-side bounds checks of the BKV_CHECKED flavour and
the allocation-failure path of bkv_create.

- The checked flavour (libbkv_checked.so, built on first use) runs the parity suites of the
  per-instance-length compress, the Continual FPS mode and the error paths with no check firing: a
  check that fired would make bkv_sync raise BKV_EBOUNDS.  Its self-test makes one checked store
  one past the logical end of an array twice that long and must report BKV_EBOUNDS; the default
  flavour has no checks and reports BKV_OK for the same store.
- bkv_create with its n-th allocation failing (bkv_debug_fail_alloc) returns BKV_ENOMEM for every n
  up to its allocation count, leaves *out NULL and releases what it had allocated: the device's free
  memory is the same after all those failures."""
import ctypes
import os
import subprocess
import sys

import pytest
import torch

from paper_2609_04971_gb300 import bkv
from paper_2609_04971_gb300.workloads import TINY

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_default_flavour_has_no_checks():
    assert not bkv.bkv_checked_build()
    bk = bkv.BeaconKV.for_workload(TINY)
    try:
        assert bkv.bkv_selftest_bounds(bk.ctx) == bkv.BKV_OK
        bkv.bkv_sync(bk.ctx)
    finally:
        bk.close()


_CHECKED_SELFTEST = """
from paper_2609_04971_gb300 import bkv
from paper_2609_04971_gb300.workloads import TINY
assert bkv.bkv_checked_build()
bk = bkv.BeaconKV.for_workload(TINY)
assert bkv.bkv_selftest_bounds(bk.ctx) == bkv.BKV_EBOUNDS
bkv.bkv_sync(bk.ctx)                                      # the error word was cleared
assert bkv.bkv_selftest_bounds(bk.ctx) == bkv.BKV_EBOUNDS  # and reports again
bk.close()
print("checked selftest ok")
"""


def _checked_env():
    env = dict(os.environ, BKV_CHECKED="1")
    env["PYTHONPATH"] = ROOT + os.pathsep + env.get("PYTHONPATH", "")
    return env


def test_checked_flavour_selftest_reports_ebounds():
    r = subprocess.run([sys.executable, "-c", _CHECKED_SELFTEST], cwd=ROOT, env=_checked_env(),
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "checked selftest ok" in r.stdout


def test_checked_flavour_parity_suites_run_clean():
    """The same parity tests, in a process that loads the checked flavour: every compress, update
    and Continual FPS call syncs without BKV_EBOUNDS and still matches the oracle."""
    tests = ["tests/test_gpu_ragged.py", "tests/test_gpu_errors.py",
             "tests/test_gpu_parity.py::test_tiny_workload_all_instances",
             "tests/test_gpu_parity.py::test_ragged_lengths", "tests/test_gpu_parity.py::test_prefix_kept",
             "tests/test_gpu_parity.py::test_identical_keys_tie_everywhere",
             "tests/test_gpu_parity.py::test_few_queries_per_instance",
             "tests/test_gpu_cfps.py::test_continual_fps_step", "tests/test_gpu_cfps.py::test_continual_fps_ragged_cache",
             "tests/test_zz_no_alloc.py"]
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", *tests], cwd=ROOT,
                       env=_checked_env(), capture_output=True, text=True, timeout=1500)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]


def test_allocation_failure_at_each_allocation_of_create():
    # 64 instances x 32768 rows: the score scratch alone is 8 MB, so a buffer left behind by a
    # failed create would show in the device's free memory after a few dozen failures
    cfg = bkv.BkvConfig(8, 2, 16, 4, 128, 16, 8, 0, 32768, 1e6, 0)
    lib = bkv.load_library()
    out = ctypes.c_void_p()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert lib.bkv_create(ctypes.byref(cfg), stream, ctypes.byref(out)) == bkv.BKV_OK
    lib.bkv_destroy(out)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    failures = 0
    try:
        for nth in range(1, 200):
            lib.bkv_debug_fail_alloc(nth)
            out = ctypes.c_void_p()
            rc = lib.bkv_create(ctypes.byref(cfg), stream, ctypes.byref(out))
            if rc == bkv.BKV_OK:  # nth is past the last allocation: the hook did not fire
                lib.bkv_destroy(out)
                break
            assert rc == bkv.BKV_ENOMEM, (nth, rc)
            assert not out.value
            failures += 1
    finally:
        lib.bkv_debug_fail_alloc(0)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert failures >= 13, failures  # the device buffers plus the pinned staging ring
    assert abs(free1 - free0) < 4 << 20, (free0, free1)
    # and a context made afterwards works
    from tests import parity as P
    P.check_run(P.run_gpu(TINY))
