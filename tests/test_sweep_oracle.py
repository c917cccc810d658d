"""Pins of the commit-sweep oracle (no GPU).

* hand-derived cases (tests/golden/sweep_cases.json), each with its passage;
* an independent whole-array formulation of the same update on seeded
  windows: the number committed is the length of the leading run of active,
  complete blocks after resolution (the proposition's "exhaustive within a
  step" and the in-order condition together), the cache holds exactly those
  blocks, the window is the rest shifted left and refilled;
* the maximal-exact-commit invariant over simulated decodes: after every
  sweep no block is active, complete and preceded only by committed blocks;
  resolved tokens are conserved; chains of blocks commit in one step.
"""

from __future__ import annotations

import json
import os

import numpy as np
import pytest

from oracle import sweep_oracle as S
from workloads.sweep_inputs import random_step, random_window

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "sweep_cases.json")
with open(GOLDEN) as fh:
    CASES = json.load(fh)["cases"]


@pytest.mark.parametrize("c", CASES, ids=lambda c: c["name"])
def test_golden_cases(c):
    r = S.commit_sweep(np.array(c["window_tokens"]), np.array(c["pos_masked"]), np.array(c["block_flags"]),
                       np.array(c["step_tokens"]), np.array(c["step_commit"], dtype=np.uint32), c["tau_index"],
                       1, c["n_slots"], c["block_len"], c["mask_token_id"], c["options"])
    e = c["expect"]
    assert r["tokens"].tolist() == e["tokens"]
    assert r["pos_masked"].tolist() == e["pos_masked"]
    assert r["block_flags"].tolist() == e["block_flags"]
    assert r["n_resolved"].tolist() == e["n_resolved"]
    assert r["n_committed"].tolist() == e["n_committed"]
    assert [x.tolist() for x in r["cache"]] == e["cache"]


def vectorised_update(win, step_tokens, step_commit, k, options):
    """The same update written over whole arrays, independently of the oracle's loops."""
    S_, B, L = win.n_seq, win.n_slots, win.block_len
    act = (win.block_flags & 1).astype(bool).reshape(S_, B)
    live = win.pos_masked.reshape(S_, B, L).astype(bool) & act[:, :, None]
    hit = live & (((step_commit.reshape(S_, B, L) >> np.uint32(k)) & 1) == 1)
    tok = np.where(hit, step_tokens.reshape(S_, B, L), win.tokens.reshape(S_, B, L))
    msk = win.pos_masked.reshape(S_, B, L).astype(bool) & ~hit
    good = act & ~msk.any(axis=2)                    # active and complete
    run = np.cumprod(good, axis=1).sum(axis=1)       # leading run length per sequence
    fill = win.mask_token_id if win.mask_token_id >= 0 else -1
    new_tok = np.full((S_, B, L), fill, dtype=np.int32)
    new_msk = np.ones((S_, B, L), dtype=np.uint8)
    new_flg = np.full((S_, B), 1 if options & S.SWEEP_ADMIT else 0, dtype=np.uint8)
    flg = win.block_flags.reshape(S_, B)
    for s in range(S_):
        c = run[s]
        new_tok[s, :B - c] = tok[s, c:]
        new_msk[s, :B - c] = msk[s, c:]
        new_flg[s, :B - c] = flg[s, c:]
    if options & S.SWEEP_ELIGIBLE_OLDEST:
        new_flg &= np.uint8(0xFD)
        a = (new_flg & 1).astype(bool)
        first = np.where(a.any(axis=1), a.argmax(axis=1), -1)
        for s in range(S_):
            if first[s] >= 0:
                new_flg[s, first[s]] |= 2
    cache = [tok[s, :run[s]] for s in range(S_)]
    return (new_tok.ravel(), new_msk.ravel(), new_flg.ravel(), hit.sum(axis=(1, 2)).astype(np.int32),
            run.astype(np.int32), cache)


@pytest.mark.parametrize("shape", [(8, 2, 32), (4, 4, 32), (3, 8, 64), (5, 4, 7), (2, 32, 4), (1, 1, 16)])
@pytest.mark.parametrize("options", [0, 1, 2, 3])
def test_against_whole_array_formulation(shape, options):
    n_seq, B, L = shape
    for seed in range(4):
        win = random_window(n_seq, B, L, seed=seed, irregular=seed % 2 == 1,
                            mask_token_id=-1 if seed == 3 else 156895)
        T = 1 + seed * 5
        st, sc = random_step(win, T, seed=seed)
        k = seed % T
        r = S.commit_sweep(win.tokens, win.pos_masked, win.block_flags, st, sc, k, n_seq, B, L,
                           win.mask_token_id, options)
        tok, msk, flg, nres, ncom, cache = vectorised_update(win, st, sc, k, options)
        assert np.array_equal(r["tokens"], tok)
        assert np.array_equal(r["pos_masked"], msk)
        assert np.array_equal(r["block_flags"], flg)
        assert np.array_equal(r["n_resolved"], nres)
        assert np.array_equal(r["n_committed"], ncom)
        assert all(np.array_equal(a, b) for a, b in zip(r["cache"], cache))


def test_invariant_over_simulated_decodes():
    """Many decode steps of windows shaped like the workloads (in-order admission,
    oldest block eligible): zero exact-committable-but-uncommitted blocks after
    every sweep, committed blocks never hold a masked position, every resolved
    token is either in the cache or still in the window, and chains commit."""
    multi = 0
    for n_seq, B, L, T in ((8, 2, 32, 4), (4, 4, 32, 8), (2, 8, 16, 16)):
        win = random_window(n_seq, B, L, seed=B)
        resolved_total = np.zeros(n_seq, dtype=np.int64)
        cached_total = np.zeros(n_seq, dtype=np.int64)
        unmasked0 = (win.pos_masked.reshape(n_seq, -1) == 0).sum(axis=1) - \
            ((win.pos_masked.reshape(n_seq, B, L) == 0) & ((win.block_flags.reshape(n_seq, B) & 1) == 0)[:, :, None]
             ).sum(axis=(1, 2))
        for step in range(120):
            st, sc = random_step(win, T, seed=1000 * B + step, full_frac=0.2)
            r = S.commit_sweep(win.tokens, win.pos_masked, win.block_flags, st, sc, step % T, n_seq, B, L,
                               win.mask_token_id, S.SWEEP_ADMIT | S.SWEEP_ELIGIBLE_OLDEST)
            assert S.exact_committable_uncommitted(r["pos_masked"], r["block_flags"], n_seq, B, L) == 0
            for s in range(n_seq):
                blocks = r["cache"][s]
                assert blocks.shape == (r["n_committed"][s], L)
                assert not np.any(blocks == (win.mask_token_id if win.mask_token_id >= 0 else -1))
                cached_total[s] += blocks.size
                multi += r["n_committed"][s] >= 2
            resolved_total += r["n_resolved"]
            win.tokens, win.pos_masked, win.block_flags = r["tokens"], r["pos_masked"], r["block_flags"]
            in_window = ((win.pos_masked.reshape(n_seq, B, L) == 0) &
                         ((win.block_flags.reshape(n_seq, B) & 1) == 1)[:, :, None]).sum(axis=(1, 2))
            assert np.array_equal(cached_total + in_window, resolved_total + unmasked0)
    assert multi > 0  # chains of ready blocks committed in one step occurred


def test_exact_committable_predicate():
    pm = np.array([0, 0, 1, 1], dtype=np.uint8)
    assert S.exact_committable_uncommitted(pm, np.array([1, 1], np.uint8), 1, 2, 2) == 1
    assert S.exact_committable_uncommitted(pm, np.array([0, 1], np.uint8), 1, 2, 2) == 0
    pm = np.array([1, 0, 0, 0], dtype=np.uint8)
    assert S.exact_committable_uncommitted(pm, np.array([1, 1], np.uint8), 1, 2, 2) == 0  # in-order wait
