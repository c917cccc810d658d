"""The bounds-checked build (libbdcommit_checks.so, -DBD_CHECKS) on the GPU:
the same parity cases through it report no index outside its buffer (the
device status word stays clear) and still match the oracle. It stands in
for a memory checker, which is not available on this GPU pool.

The cases run in a child process that loads the checked library through
BD_LIBRARY, so this process keeps the normal build."""

import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CASES = [
    # bf16 head, one and several token groups, K tail; mask token in the last tile; degenerate windows
    "tests/test_gpu_parity.py::test_small_tensor_core",
    "tests/test_gpu_parity.py::test_mask_token_suppressed",
    "tests/test_gpu_parity.py::test_nothing_masked",
    "tests/test_gpu_parity.py::test_everything_masked_and_every_block_eligible",
    # heads decoded in the kernel (f16 rows) and W8A8 (E4M3 rows)
    "tests/test_gpu_nvfp4.py::test_small",
    "tests/test_gpu_w8a8.py::test_w8a8_small",
]


def test_parity_cases_through_the_bounds_checked_build():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sys.path.insert(0, ROOT)
    from paper_2609_33887_gb300 import build as bld

    path = bld.build(checks=True)
    env = dict(os.environ, BD_LIBRARY=path)
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider"] + CASES,
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
    assert " passed" in r.stdout
