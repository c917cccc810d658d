"""Oracle of the commit sweep and block-buffer update (test infrastructure).

Plain restatement, block by block in Python, of the state update that follows
the commit step in every decode step. Only the tests, the smoke check and the
CPU-baseline leg of the benchmark use it; the library (bd_commit_sweep) shares
no code with it.

Passages followed:
  * Engine appendix (slot states): each request keeps a fixed number of block
    slots; a slot holds a placeholder, an active block, a committed block on
    its way to the cache, or a cached block; the accept rule decides which
    positions of an active block are resolved in a step, and the commit sweep
    commits resolved blocks in order.
  * Maximal-exact-commit appendix, proof part (1): the sweep visits the buffer
    from left to right and commits a block exactly when it is active,
    complete (no masked position), commit-ready and its predecessor is
    committed; a block committed in this pass satisfies its successor's
    predecessor condition in the same pass, so chains commit in one step;
    committed blocks form a prefix that leaves the buffer, shifting the rest.
  * Same appendix, part (2): under the default commit semantics (no sampler
    state map) every complete active block is commit-ready.
  * Same appendix, statement and validation: afterwards no block is active,
    complete and preceded only by committed blocks (zero exact-committable
    but uncommitted blocks); `exact_committable_uncommitted` counts them.

Inputs and outputs use the library's layout: position p = (s * B + b) * L + j;
block_flags bit 0 = active, bit 1 = fallback-eligible; step_commit bit k set
when the commit step committed the position at threshold k.
"""

from __future__ import annotations

from typing import Dict, List

import numpy as np

ACTIVE = 1
FALLBACK_ELIGIBLE = 2

SWEEP_ADMIT = 1             # vacated slots come back as admitted, all-masked blocks
SWEEP_ELIGIBLE_OLDEST = 2   # after the sweep, only the oldest active block is fallback-eligible


def commit_sweep(window_tokens: np.ndarray, pos_masked: np.ndarray, block_flags: np.ndarray,
                 step_tokens: np.ndarray, step_commit: np.ndarray, tau_index: int,
                 n_seq: int, n_slots: int, block_len: int, mask_token_id: int, options: int = 0) -> Dict:
    """One decode step's state update at threshold index tau_index.

    Returns new copies of the window (tokens, pos_masked, block_flags) and, per
    sequence, the number of positions resolved, the number of blocks committed
    and their tokens in commit order ("cache": list of [n_committed, L] arrays).
    """
    B, L = n_slots, block_len
    tok = np.array(window_tokens, dtype=np.int32).copy()
    msk = np.array(pos_masked, dtype=np.uint8).copy()
    flg = np.array(block_flags, dtype=np.uint8).copy()
    fill = np.int32(mask_token_id if mask_token_id >= 0 else -1)
    n_resolved = np.zeros(n_seq, dtype=np.int32)
    n_committed = np.zeros(n_seq, dtype=np.int32)
    cache: List[np.ndarray] = []

    for s in range(n_seq):
        # the accept rule's decisions at the deployed threshold resolve positions of active blocks
        for b in range(B):
            if not flg[s * B + b] & ACTIVE:
                continue
            for j in range(L):
                p = (s * B + b) * L + j
                if msk[p] and (int(step_commit[p]) >> tau_index) & 1:
                    tok[p] = step_tokens[p]
                    msk[p] = 0
                    n_resolved[s] += 1

        # the sweep, left to right
        state = ["active" if flg[s * B + b] & ACTIVE else "placeholder" for b in range(B)]
        for b in range(B):
            complete = not any(msk[(s * B + b) * L + j] for j in range(L))
            ready = complete  # default semantics: complete implies commit-ready
            pred_committed = b == 0 or state[b - 1] == "committed"
            if state[b] == "active" and complete and ready and pred_committed:
                state[b] = "committed"

        # committed blocks go to the cache in buffer order (under in-order commit
        # they are a prefix); the remaining blocks keep their order and move to
        # the front; the vacated slots at the end are refilled
        kept = [b for b in range(B) if state[b] != "committed"]
        gone = [b for b in range(B) if state[b] == "committed"]
        n_committed[s] = len(gone)
        cache.append(np.array([tok[(s * B + b) * L:(s * B + b + 1) * L] for b in gone],
                              dtype=np.int32).reshape(len(gone), L))
        old_tok = tok[s * B * L:(s + 1) * B * L].copy()
        old_msk = msk[s * B * L:(s + 1) * B * L].copy()
        old_flg = flg[s * B:(s + 1) * B].copy()
        for b in range(B):
            dst = slice((s * B + b) * L, (s * B + b + 1) * L)
            if b < len(kept):
                src = kept[b]
                tok[dst] = old_tok[src * L:(src + 1) * L]
                msk[dst] = old_msk[src * L:(src + 1) * L]
                flg[s * B + b] = old_flg[src]
            else:
                tok[dst] = fill
                msk[dst] = 1
                flg[s * B + b] = ACTIVE if options & SWEEP_ADMIT else 0

        if options & SWEEP_ELIGIBLE_OLDEST:
            first = True
            for b in range(B):
                f = int(flg[s * B + b]) & ~FALLBACK_ELIGIBLE
                if first and f & ACTIVE:
                    f |= FALLBACK_ELIGIBLE
                    first = False
                flg[s * B + b] = f

    return {"tokens": tok, "pos_masked": msk, "block_flags": flg, "n_resolved": n_resolved,
            "n_committed": n_committed, "cache": cache}


def exact_committable_uncommitted(pos_masked: np.ndarray, block_flags: np.ndarray, n_seq: int, n_slots: int,
                                  block_len: int) -> int:
    """Blocks that are active, complete and have no uncommitted predecessor in
    the window (the validation predicate; it ignores commit readiness). Every
    block still in the window is uncommitted, so only a first slot can count."""
    B, L = n_slots, block_len
    count = 0
    for s in range(n_seq):
        for b in range(B):
            active = bool(block_flags[s * B + b] & ACTIVE)
            complete = not any(pos_masked[(s * B + b) * L + j] for j in range(L))
            no_uncommitted_pred = b == 0  # every earlier slot holds an uncommitted block
            if active and complete and no_uncommitted_pred:
                count += 1
    return count
