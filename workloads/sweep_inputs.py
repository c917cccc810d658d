"""Seeded synthetic inputs for the commit sweep (block-buffer update).

Holds no step of the sweep. A window is n_seq sequences of n_slots block
slots of block_len positions (position p = (s * n_slots + b) * block_len + j),
shaped like the paper's engine windows: a prefix of active blocks per
sequence (the rest placeholders), masked fractions that fall with a block's
age, the oldest active block fallback-eligible. A step input is what the
commit step hands the sweep: a token per position and commit bits nested
over an ascending threshold grid (a position committed at threshold k is
committed at every lower one), with some blocks resolved in full so that
complete blocks and chains of them occur, and junk bits on positions the
sweep must ignore (unmasked positions, placeholder slots).
"""

from __future__ import annotations

from dataclasses import dataclass

import numpy as np

ACTIVE = 1
FALLBACK_ELIGIBLE = 2


@dataclass
class Window:
    tokens: np.ndarray       # int32 [P]
    pos_masked: np.ndarray   # uint8 [P]
    block_flags: np.ndarray  # uint8 [S * B]
    n_seq: int
    n_slots: int
    block_len: int
    mask_token_id: int


def random_window(n_seq: int, n_slots: int, block_len: int, *, V: int = 151936, mask_token_id: int = 156895,
                  seed: int = 0, irregular: bool = False) -> Window:
    rng = np.random.default_rng(seed)
    B, L = n_slots, block_len
    P = n_seq * B * L
    tokens = rng.integers(0, V, size=P, dtype=np.int64).astype(np.int32)
    pos_masked = np.zeros(P, dtype=np.uint8)
    flags = np.zeros(n_seq * B, dtype=np.uint8)
    for s in range(n_seq):
        n_active = int(rng.integers(0, B + 1))
        for b in range(B):
            base = (s * B + b) * L
            if b < n_active or (irregular and rng.random() < 0.2):
                flags[s * B + b] = ACTIVE
                # older blocks are further along: expected masked fraction grows with b
                frac = min(1.0, max(0.0, rng.normal((b + 1) / (B + 1), 0.25)))
                if rng.random() < 0.25:
                    frac = 0.0  # already complete
                pos_masked[base:base + L] = (rng.random(L) < frac).astype(np.uint8)
            else:
                pos_masked[base:base + L] = 1  # placeholders are mask-filled
        act = np.flatnonzero(flags[s * B:(s + 1) * B] & ACTIVE)
        if act.size:
            flags[s * B + act[0]] |= FALLBACK_ELIGIBLE
    tokens[pos_masked != 0] = mask_token_id if mask_token_id >= 0 else -1
    return Window(tokens, pos_masked, flags, n_seq, B, L, mask_token_id)


def random_step(win: Window, T: int, *, V: int = 151936, seed: int = 0, full_frac: float = 0.3,
                junk: bool = True):
    """(step_tokens int32 [P], step_commit uint32 [P]) for one commit step over `win`."""
    rng = np.random.default_rng(seed + 104729)
    B, L = win.n_slots, win.block_len
    P = win.tokens.size
    step_tokens = rng.integers(0, V, size=P, dtype=np.int64).astype(np.int32)
    level = rng.integers(0, T + 1, size=P)  # committed at thresholds 0 .. level-1
    for blk in range(win.n_seq * B):
        if rng.random() < full_frac:
            level[blk * L:(blk + 1) * L] = T  # every masked position of the block resolves
    bits = ((np.uint64(1) << level.astype(np.uint64)) - np.uint64(1)).astype(np.uint32)
    live = (win.pos_masked != 0) & (np.repeat(win.block_flags & ACTIVE, L) != 0)
    if junk:
        noise = rng.integers(0, 1 << min(T, 31), size=P, dtype=np.int64).astype(np.uint32)
        step_commit = np.where(live, bits, noise)
    else:
        step_commit = np.where(live, bits, np.uint32(0))
    return step_tokens, step_commit.astype(np.uint32)
