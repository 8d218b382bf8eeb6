"""The beacon update's integer fold of a call's exact sum into the fp64 running sum, against the fp64
addition it replaces (tests/cuda/fold_check.cu, built with nvcc for sm_103a and run on the GPU):
bit-identical wherever that addition is exact before its one rounding, within one ulp where it rounds
twice, and identical on the values that keep the fp64 route."""
import os
import shutil
import subprocess
import tempfile

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2609_04971_gb300", "csrc")


def test_integer_fold_matches_fp64_addition():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    with tempfile.TemporaryDirectory() as tmp:
        exe = os.path.join(tmp, "fold_check")
        subprocess.check_call([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-I", CSRC,
                               "-o", exe, os.path.join(HERE, "cuda", "fold_check.cu")])
        out = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    print(out.stdout)
    assert out.returncode == 0, out.stdout + out.stderr
