"""bd_commit_step_static, the entry point that allocates nothing.

Some callers cannot allocate device memory: code running inside an allocator
or memory-pool callback, a process whose device memory a framework's caching
allocator already owns, or a serving loop that cannot take cudaMalloc's
implicit synchronisation. For them the library runs the commit step in a
fixed 32 MiB device array it owns from load time. These tests call that
entry point through the C ABI and check it against bd_commit_step_ex, within
the tolerances of the parity tests, on two calls in a row (the array keeps
the previous call's contents). This file sorts last so that a run that stops
at its first failure has already run every other test.
"""

import numpy as np
import pytest
import torch

from tests.helpers import oracle_on_workload
from tests.parity import compare
from workloads import B256X8X64_E4M3, B64X4X64_BF16, B8X2X32_BF16, generate, scaled, TINY_F32

pytestmark = pytest.mark.gpu

bdc = pytest.importorskip("paper_2609_33887_gb300")
B = bdc.bdcommit

CONF_TOL = 2e-3  # bf16 / f32 confidence tolerance of the parity tests


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    yield


def _outputs(P, dev):
    return (torch.full((P,), -7, dtype=torch.int32, device=dev), torch.full((P,), -7.0, device=dev),
            torch.full((P,), -7, dtype=torch.int32, device=dev))


def _run(wl, static):
    cfg = wl.cfg
    g = wl.to("cuda")
    tok, conf, com = _outputs(cfg.P, g.hidden.device)
    args = (g.hidden, g.weight, g.weight_scale, g.pos_masked, g.block_flags, cfg.n_seq, cfg.n_slots,
            cfg.block_len, cfg.mask_token_id, cfg.tau, tok, conf, com)
    rc = B.bd_commit_step_static(*args) if static else B.bd_commit_step_ex(*args)
    assert rc == B.BD_OK, B.bd_status_string(rc)
    torch.cuda.synchronize()
    if static:
        st = B.bd_static_device_status(None)
        assert st == B.BD_OK, B.bd_status_string(st)
    return tok.cpu().numpy(), conf.cpu().numpy(), com.cpu().numpy().view(np.uint32)


@pytest.mark.parametrize("cfg", [B8X2X32_BF16, TINY_F32, scaled(B256X8X64_E4M3, n_seq=4, n_slots=4, d=512, V=5000)],
                         ids=["b8x2x32_bf16", "tiny_f32", "e4m3_small"])
def test_static_matches_the_allocating_entry_point_twice(cfg):
    wl = generate(cfg)
    ref_tok, ref_conf, ref_com = _run(wl, static=False)
    for _ in range(2):
        tok, conf, com = _run(wl, static=True)
        assert np.array_equal(tok, ref_tok)
        assert np.abs(conf.astype(np.float64) - ref_conf).max() <= CONF_TOL
        assert np.array_equal(com, ref_com)
    assert (ref_tok >= 0).sum() > 0


@pytest.mark.parametrize("share", ["0", "1"])
def test_static_with_spill_pairs_beside_clusters(share, monkeypatch):
    # the LM head as two launches (clusters of two pairs, sharing head tiles
    # or token rows, and the spill pairs) inside the fixed array
    monkeypatch.setenv("BD_PAIR_MC", "2")
    monkeypatch.setenv("BD_PAIR_SPILL", "1")
    monkeypatch.setenv("BD_SPILL_PCT", "50")
    monkeypatch.setenv("BD_PAIR_SHARE", share)
    wl = generate(scaled(B8X2X32_BF16, n_seq=4, d=256, V=3000, name="b4x2x32_v3000"))
    ref_tok, ref_conf, ref_com = _run(wl, static=False)
    tok, conf, com = _run(wl, static=True)
    assert np.array_equal(tok, ref_tok)
    assert np.abs(conf.astype(np.float64) - ref_conf).max() <= CONF_TOL
    assert np.array_equal(com, ref_com)
    assert (ref_tok >= 0).sum() > 0


def test_static_rejects_windows_beyond_its_array():
    # the 64 x 4 x 64, d = 4096 window needs far more than 32 MiB of workspace;
    # the call is refused before anything is queued
    cfg = scaled(B64X4X64_BF16, V=1024, name="too_large")
    P = cfg.P
    dev = torch.device("cuda")
    h = torch.zeros((P, cfg.d), dtype=torch.bfloat16, device=dev)
    w = torch.zeros((cfg.V, cfg.d), dtype=torch.bfloat16, device=dev)
    pm = torch.ones(P, dtype=torch.uint8, device=dev)
    bf = torch.ones(cfg.n_blocks, dtype=torch.uint8, device=dev)
    tok, conf, com = _outputs(P, dev)
    assert B.bd_workspace_size(h, w, None, pm, bf, cfg.n_seq, cfg.n_slots, cfg.block_len, -1, cfg.tau) > 32 << 20
    rc = B.bd_commit_step_static(h, w, None, pm, bf, cfg.n_seq, cfg.n_slots, cfg.block_len, -1, cfg.tau,
                                 tok, conf, com)
    assert rc == B.BD_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert int(tok[0]) == -7  # nothing was written


def test_static_matches_the_oracle():
    # the static path against the float64 oracle directly (not only against
    # the allocating entry point), at the parity tests' tolerances
    wl = generate(B8X2X32_BF16)
    tok, conf, com = _run(wl, static=True)
    ref = oracle_on_workload(wl)
    rep = compare({"tokens": tok, "conf": conf, "commit": com}, ref, wl.tau, wl.cfg.weight_dtype,
                  wl.cfg.block_len, wl.cfg.n_slots)
    assert rep.ok(), rep.failures
    assert rep.n_live > 250


def test_static_calls_allocate_no_device_memory():
    # Every buffer the calls use exists before the first measurement; the
    # first static call has loaded the library's module (its 32 MiB array is
    # part of the module), so any later change of the device's free memory
    # would be an allocation by the call itself.
    wl = generate(scaled(B8X2X32_BF16, n_seq=4, name="b4x2x32"))
    cfg = wl.cfg
    g = wl.to("cuda")
    tok, conf, com = _outputs(cfg.P, g.hidden.device)
    args = (g.hidden, g.weight, g.weight_scale, g.pos_masked, g.block_flags, cfg.n_seq, cfg.n_slots,
            cfg.block_len, cfg.mask_token_id, cfg.tau, tok, conf, com)
    assert B.bd_commit_step_static(*args) == B.BD_OK
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        assert B.bd_commit_step_static(*args) == B.BD_OK
    assert B.bd_static_device_status(None) == B.BD_OK
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


def test_static_status_reports_a_timeout_once():
    # the bounded-wait self-test aimed at the static array's status word: the
    # next read reports the timeout and clears it, and the next static call
    # runs normally and reads clean
    assert B.bd_static_selftest_timeout(None) == B.BD_OK
    assert B.bd_static_device_status(None) == B.BD_ERR_TIMEOUT
    assert B.bd_static_device_status(None) == B.BD_OK
    # the allocating path's status word is a different word: untouched
    assert B.bd_get_device_status(None) == B.BD_OK
    wl = generate(scaled(B8X2X32_BF16, n_seq=2, name="b2x2x32"))
    tok, _, _ = _run(wl, static=True)
    assert (tok >= 0).sum() > 0
