"""The commit step's per-threshold counts as Redline's cost input, on the GPU.

Several forwards of the commit step (bd_commit_step with out_counts) give, per
accept threshold, the tokens committed per forward and per sequence
(bd_redline_tpf); Redline then deploys the threshold with the best TPF among
the valid ones. The GPU counts must match the oracle's up to the positions the
commit-step tolerance exempts, and the deployment must match the oracle's run
on the oracle's own counts.
"""

import numpy as np
import pytest
import torch

from oracle import redline_oracle as RO
from tests.helpers import oracle_on_workload
from tests.parity import compare
from workloads import B8X2X32_BF16, generate, scaled
from workloads.redline_inputs import outcome_matrix

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


def test_tpf_from_commit_counts_feeds_redline():
    from paper_2609_33887_gb300 import redline as N

    taus = (0.5, 0.7, 0.8, 0.9, 0.95, 0.99)
    gpu_steps, ref_steps, exempt = [], [], 0
    for step in range(4):
        cfg = scaled(B8X2X32_BF16, n_seq=8, n_slots=4, d=200, V=3000, tau=taus, seed=100 + step)
        wl = generate(cfg)
        g = wl.to("cuda")
        tokens, conf, commit, counts = bdc.commit_step(
            g.hidden, g.weight, g.pos_masked, g.block_flags, cfg.n_seq, cfg.n_slots, cfg.block_len, wl.tau,
            mask_token_id=wl.mask_token_id, counts=True)
        torch.cuda.synchronize()
        assert bdc.bd_get_device_status() == 0
        out = {"tokens": tokens.cpu().numpy(), "conf": conf.cpu().numpy(),
               "commit": commit.cpu().numpy().view(np.uint32), "counts": counts.cpu().numpy()}
        ref = oracle_on_workload(wl)
        rep = compare(out, ref, wl.tau, cfg.weight_dtype, cfg.block_len, cfg.n_slots)
        assert rep.ok(), rep.failures
        exempt += rep.commit_mismatch_exempt
        gpu_steps.append(out["counts"].sum(axis=0))
        ref_steps.append(ref["counts"].sum(axis=0))
    gpu_counts = np.stack(gpu_steps).astype(np.int32)   # [steps, T], summed over sequences
    ref_counts = np.stack(ref_steps).astype(np.int64)
    assert np.all(np.abs(gpu_counts.sum(0) - ref_counts.sum(0)) <= exempt)

    n_seq = 8
    tpf = N.bd_redline_tpf(gpu_counts, n_seq)
    tpf_exact = RO.tpf_from_counts(gpu_counts.tolist(), n_seq)
    assert all(abs(a - float(b)) <= 1e-15 * max(1.0, float(b)) for a, b in zip(tpf, tpf_exact))
    assert all(a >= b for a, b in zip(tpf, tpf[1:]))  # a lower threshold never commits less

    # a synthetic calibration record over the thresholds: the strictest one is
    # the reference, looser thresholds carry larger joint risks
    risks = [0.09, 0.07, 0.05, 0.03, 0.01, 0.0]
    outcomes = outcome_matrix(1012, risks, ref=5, ref_acc=0.8, seed=7)
    V = N.bd_redline_violations(outcomes, 5)
    tpf_ref = [float(x) for x in RO.tpf_from_counts(ref_counts.tolist(), n_seq)]
    for alpha in (0.05, 0.08, 0.10, 0.15):
        got = N.bd_redline_select(V, tpf, 1012, alpha, 5)
        want = RO.redline(list(V), tpf_ref, 1012, alpha, 0.10, 5)
        assert list(got["valid"]) == want["valid"]
        assert got["deployed"] == want["deployed"], (alpha, tpf, tpf_ref)
