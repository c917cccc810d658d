"""Failure detection of the kernels' bounded waits, without a fault: a wait on a
barrier nothing completes runs out (about 1 s), the kernel records the timeout
and returns, the host reads BD_ERR_TIMEOUT once, and the context keeps working."""

import time

import numpy as np
import pytest
import torch

from tests.helpers import oracle_on_workload
from tests.parity import compare
from workloads import B8X2X32_BF16, generate, scaled

pytestmark = pytest.mark.gpu

bdc = pytest.importorskip("paper_2609_33887_gb300")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    yield


def test_bounded_wait_reports_timeout_and_context_survives():
    from paper_2609_33887_gb300 import bdcommit as B

    assert B.bd_get_device_status() == 0
    t0 = time.time()
    assert B.bd_selftest_timeout() == 0
    assert B.bd_get_device_status() == B.BD_ERR_TIMEOUT
    waited = time.time() - t0
    assert 0.9 < waited < 10.0, waited
    assert B.bd_get_device_status() == 0  # read once, then cleared
    # the context still runs the commit step correctly
    wl = generate(scaled(B8X2X32_BF16, n_seq=2, n_slots=2, d=256, V=1000))
    g = wl.to("cuda")
    tokens, conf, commit, _ = bdc.commit_step(g.hidden, g.weight, g.pos_masked, g.block_flags, 2, 2, 32, wl.tau)
    torch.cuda.synchronize()
    assert B.bd_get_device_status() == 0
    out = {"tokens": tokens.cpu().numpy(), "conf": conf.cpu().numpy(),
           "commit": commit.cpu().numpy().view(np.uint32)}
    rep = compare(out, oracle_on_workload(wl), wl.tau, "bf16", 32, 2)
    assert rep.ok(), rep.failures
