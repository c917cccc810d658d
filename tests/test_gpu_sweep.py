"""The commit sweep on the GPU (bd_commit_sweep) against the sweep oracle.

Integer work, so everything is compared exactly: the window's tokens, masks
and flags after the update, the committed and resolved counts, the cache
output of every committed block, and the cache entries it must not touch.
"""

import numpy as np
import pytest
import torch

from oracle import sweep_oracle as SO
from tests.helpers import oracle_on_workload
from tests.parity import compare
from workloads import B8X2X32_BF16, generate, scaled
from workloads.sweep_inputs import random_step, random_window

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


def dev(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a).view(dtype)).cuda()


def gpu_sweep(state, win, st, sc, k, options):
    tok_d, pm_d, fl_d = state
    cache, ncom, nres = bdc.commit_sweep(tok_d, pm_d, fl_d, win.n_seq, win.n_slots, win.block_len,
                                         dev(st.astype(np.int32), np.int32), dev(sc.astype(np.uint32), np.int32),
                                         k, mask_token_id=win.mask_token_id, options=options)
    torch.cuda.synchronize()
    return cache.cpu().numpy(), ncom.cpu().numpy(), nres.cpu().numpy()


def assert_same(state, cache, ncom, nres, ref, n_seq, B, L, seqs=None):
    tok, pm, fl = (t.cpu().numpy() for t in state)
    seqs = range(n_seq) if seqs is None else seqs
    for s in seqs:
        w = slice(s * B * L, (s + 1) * B * L)
        assert np.array_equal(tok[w], ref["tokens"][w]), s
        assert np.array_equal(pm[w], ref["pos_masked"][w]), s
        assert np.array_equal(fl[s * B:(s + 1) * B], ref["block_flags"][s * B:(s + 1) * B]), s
        assert ncom[s] == ref["n_committed"][s] and nres[s] == ref["n_resolved"][s], s
        c = int(ncom[s])
        assert np.array_equal(cache[w][:c * L].reshape(c, L), ref["cache"][s]), s
        assert np.all(cache[w][c * L:] == -1), s  # entries past the committed blocks are untouched


SHAPES = [(8, 2, 32, 4), (32, 4, 32, 8), (64, 4, 64, 16), (256, 8, 64, 16), (5, 4, 7, 3), (2, 64, 4, 32),
          (1, 1, 1, 1), (3, 64, 64, 5)]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
@pytest.mark.parametrize("options", [0, 1, 2, 3])
def test_sweep_parity(shape, options):
    n_seq, B, L, T = shape
    for seed in range(3):
        win = random_window(n_seq, B, L, seed=seed, irregular=seed == 1, mask_token_id=-1 if seed == 2 else 156895)
        st, sc = random_step(win, T, seed=seed)
        k = (seed * 7) % T
        ref = SO.commit_sweep(win.tokens, win.pos_masked, win.block_flags, st, sc, k, n_seq, B, L,
                              win.mask_token_id, options)
        state = (dev(win.tokens, np.int32), dev(win.pos_masked, np.uint8), dev(win.block_flags, np.uint8))
        cache, ncom, nres = gpu_sweep(state, win, st, sc, k, options)
        assert_same(state, cache, ncom, nres, ref, n_seq, B, L)


def test_multi_step_decode_keeps_parity_and_the_invariant():
    """40 decode steps, the window carried on the device and in the oracle; after
    every sweep both agree and no block is active, complete and preceded only by
    committed blocks."""
    n_seq, B, L, T = 16, 4, 32, 8
    win = random_window(n_seq, B, L, seed=5)
    state = (dev(win.tokens, np.int32), dev(win.pos_masked, np.uint8), dev(win.block_flags, np.uint8))
    opts = SO.SWEEP_ADMIT | SO.SWEEP_ELIGIBLE_OLDEST
    chains = 0
    for step in range(40):
        st, sc = random_step(win, T, seed=900 + step, full_frac=0.25)
        k = step % T
        ref = SO.commit_sweep(win.tokens, win.pos_masked, win.block_flags, st, sc, k, n_seq, B, L,
                              win.mask_token_id, opts)
        cache, ncom, nres = gpu_sweep(state, win, st, sc, k, opts)
        assert_same(state, cache, ncom, nres, ref, n_seq, B, L)
        pm, fl = state[1].cpu().numpy(), state[2].cpu().numpy()
        assert SO.exact_committable_uncommitted(pm, fl, n_seq, B, L) == 0
        chains += int((ncom >= 2).sum())
        win.tokens, win.pos_masked, win.block_flags = ref["tokens"], ref["pos_masked"], ref["block_flags"]
    assert chains > 0


def test_errors_and_empty_window():
    z = torch.zeros(8, dtype=torch.int32, device="cuda")
    m = torch.zeros(8, dtype=torch.uint8, device="cuda")
    f = torch.zeros(2, dtype=torch.uint8, device="cuda")
    with pytest.raises(bdc.BdError):
        bdc.commit_sweep(z, m, f, 1, 2, 4, z, z, 32)
    with pytest.raises(bdc.BdError):
        bdc.commit_sweep(z, m, f, 1, 2, 4, z, z, 0, options=8)
    cache, ncom, nres = bdc.commit_sweep(z, m, f, 0, 2, 4, z, z, 0)
    assert ncom.numel() == 0


def test_decode_loop_commit_step_then_sweep():
    """Eight forwards of a decode loop: the commit step on the device window's
    masks, then the sweep at the deployed threshold, against the oracle's commit
    step and sweep on the oracle's own window. If a commit decision at the
    deployed threshold falls inside the commit step's tolerance, the two windows
    may legitimately part: the sequences concerned are left out of that step's
    comparison and the loop ends there."""
    # 8-position blocks so that blocks complete within a few forwards
    cfg = scaled(B8X2X32_BF16, n_seq=8, n_slots=4, block_len=8, d=200, V=3000, tau=(0.5, 0.7, 0.9, 0.95))
    wl0 = generate(cfg)
    n_seq, B, L = cfg.n_seq, cfg.n_slots, cfg.block_len
    k = 1  # deploy tau = 0.7
    opts = SO.SWEEP_ADMIT | SO.SWEEP_ELIGIBLE_OLDEST
    P = n_seq * B * L
    tokens0 = np.where(wl0.pos_masked.numpy() != 0, -1, 7).astype(np.int32)
    ref_state = {"tokens": tokens0, "pos_masked": wl0.pos_masked.numpy().copy(),
                 "block_flags": wl0.block_flags.numpy().copy()}
    state = (dev(tokens0, np.int32), dev(ref_state["pos_masked"], np.uint8), dev(ref_state["block_flags"], np.uint8))
    weight = wl0.weight.cuda()
    gen = torch.Generator().manual_seed(77)
    steps_done, committed = 0, 0
    for step in range(8):
        hidden = wl0.hidden[torch.randperm(P, generator=gen)].contiguous()
        wl = generate(cfg)
        wl.hidden = hidden
        wl.pos_masked = torch.from_numpy(ref_state["pos_masked"].copy())
        wl.block_flags = torch.from_numpy(ref_state["block_flags"].copy())
        ref_commit = oracle_on_workload(wl)
        tok_g, conf_g, com_g, _ = bdc.commit_step(hidden.cuda(), weight, state[1], state[2], n_seq, B, L, cfg.tau,
                                                  mask_token_id=cfg.mask_token_id)
        torch.cuda.synchronize()
        gpu_out = {"tokens": tok_g.cpu().numpy(), "conf": conf_g.cpu().numpy(),
                   "commit": com_g.cpu().numpy().view(np.uint32)}
        rep = compare(gpu_out, ref_commit, cfg.tau, cfg.weight_dtype, L, B)
        assert rep.ok(), rep.failures
        bit_g = (gpu_out["commit"] >> k) & 1
        bit_r = (ref_commit["commit"].astype(np.uint32) >> k) & 1
        tok_diff = (gpu_out["tokens"] != ref_commit["tokens"]) & (bit_r == 1)
        parted = [s for s in range(n_seq) if np.any(bit_g[s * B * L:(s + 1) * B * L] != bit_r[s * B * L:(s + 1) * B * L])
                  or np.any(tok_diff[s * B * L:(s + 1) * B * L])]
        cache, ncom, nres = bdc.commit_sweep(state[0], state[1], state[2], n_seq, B, L, tok_g, com_g, k,
                                             mask_token_id=cfg.mask_token_id, options=opts)
        torch.cuda.synchronize()
        ref = SO.commit_sweep(ref_state["tokens"], ref_state["pos_masked"], ref_state["block_flags"],
                              ref_commit["tokens"].astype(np.int32), ref_commit["commit"].astype(np.uint32), k,
                              n_seq, B, L, cfg.mask_token_id, opts)
        assert_same(state, cache.cpu().numpy(), ncom.cpu().numpy(), nres.cpu().numpy(), ref, n_seq, B, L,
                    seqs=[s for s in range(n_seq) if s not in parted])
        assert SO.exact_committable_uncommitted(state[1].cpu().numpy(), state[2].cpu().numpy(), n_seq, B, L) == 0
        steps_done += 1
        committed += int(ncom.sum())
        ref_state = ref
        if parted:
            break
    assert steps_done >= 3 and committed > 0
