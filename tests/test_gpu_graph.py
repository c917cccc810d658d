"""The commit step captured into a CUDA graph (caller-provided workspace):
replays give the eager outputs, and the LM-head events recorded inside the
capture time the kernel on every replay."""

import numpy as np
import pytest
import torch

from workloads import B8X2X32_BF16, generate, scaled

pytestmark = pytest.mark.gpu

bdc = pytest.importorskip("paper_2609_33887_gb300")
B = bdc.bdcommit


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    yield


def test_graph_replay_matches_eager_and_times_the_lmhead():
    cfg = scaled(B8X2X32_BF16, n_seq=4, n_slots=2, d=512, V=5000)
    wl = generate(cfg).to("cuda")
    P = cfg.P
    args = (wl.hidden, wl.weight, None, wl.pos_masked, wl.block_flags, cfg.n_seq, cfg.n_slots, cfg.block_len, -1,
            cfg.tau)
    ws = torch.empty(B.bd_workspace_size(*args), dtype=torch.uint8, device="cuda")

    def outs():
        return (torch.empty(P, dtype=torch.int32, device="cuda"), torch.empty(P, device="cuda"),
                torch.empty(P, dtype=torch.int32, device="cuda"))

    eager = outs()
    assert B.bd_commit_step_ex(*args, *eager, workspace=ws) == 0
    torch.cuda.synchronize()

    got = outs()
    ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    s = torch.cuda.current_stream()
    ev[0].record(s)
    ev[1].record(s)  # create the handles before capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        rc = B.bd_commit_step_ex(*args, *got, workspace=ws, stream=torch.cuda.current_stream(), lmhead_events=ev)
    assert rc == 0
    for _ in range(3):
        for t in got:
            t.fill_(-5)
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(got[0], eager[0]) and torch.equal(got[2], eager[2])
        assert torch.equal(got[1], eager[1])
        assert ev[0].elapsed_time(ev[1]) > 0
    assert B.bd_get_device_status() == 0
