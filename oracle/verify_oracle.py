"""Oracle of speculative-decoding verification (test infrastructure).

Plain float64 restatement of the acceptance rules the paper tests for
speculative decoding. Only the tests, the smoke check and the CPU-baseline leg
of the benchmark use it; the library (bd_verify_step) shares no code with it.

Passages followed:
  * Typical-acceptance appendix: a draft token x is accepted when the
    target's probability of it exceeds min(eps, a * exp(-H)), H the entropy
    of the target's next-token distribution, with a = sqrt(eps); lower eps
    accepts more.
  * Lossless-reference appendix: the reference accepts x only when it equals
    the target's argmax (greedy verification).
  * Joint-risk-against-net-accuracy appendix: the measure is accepted tokens
    for each target forward; a request accepts the longest prefix of its
    draft tokens that pass, and the target forward adds one token of its own.

The target distribution is the full softmax of the LM head's logits
(p_v = exp(l_v - M) / sum_u exp(l_u - M)); the entropy is the definition
H = -sum_v p_v log p_v over the entries with p_v > 0.
"""

from __future__ import annotations

import math
from typing import Dict, Optional, Sequence

import numpy as np

from .commit_oracle import hidden_f64, lm_head_logits

LOSSLESS_BIT = 31


def row_stats(logits: np.ndarray):
    """(argmax token (lowest index on ties), probabilities, entropy, top-2 gap) of one row."""
    l = np.asarray(logits, dtype=np.float64)
    M = float(np.max(l))
    token = int(np.flatnonzero(l == M)[0])
    e = np.exp(l - M)
    p = e / np.sum(e)
    nz = p[p > 0]
    H = float(-np.sum(nz * np.log(nz)))
    others = np.delete(l, token)
    gap = float(M - np.max(others)) if others.size else math.inf
    return token, p, H, gap


def accepts(p_x: float, H: float, eps: float) -> bool:
    """Typical acceptance: p(x) > min(eps, sqrt(eps) * exp(-H))."""
    return p_x > min(eps, math.sqrt(eps) * math.exp(-H))


def verify_step(hidden_raw: np.ndarray, hidden_dtype: str, w_raw: np.ndarray, w_dtype: str,
                w_scale: Optional[np.ndarray], draft: Sequence[int], n_req: int, n_draft: int,
                eps: Sequence[float], eps_f32: bool = True) -> Dict[str, np.ndarray]:
    """Verification of n_req requests of n_draft draft tokens each.

    Row q * (n_draft + 1) + i of the hidden states holds the target's state
    whose next-token distribution verifies draft token i of request q
    (draft[q * n_draft + i]); the last row of a request gives its bonus token.
    Returns per row: tokens (argmax), p_draft (target probability of the draft
    token, 0 on bonus rows), entropy, accept (bit k: accepted at eps[k]; bit
    31: lossless, the draft equals the argmax), gap (top-2 logit gap); per
    request: accepted[q, k] = length of the accepted prefix at eps[k], column
    len(eps) for the lossless rule.
    """
    R = n_req * (n_draft + 1)
    E = len(eps)
    eps_v = [float(np.float32(e)) if eps_f32 else float(e) for e in eps]
    h = hidden_f64(hidden_raw, hidden_dtype)
    logits = lm_head_logits(h, w_raw, w_dtype, w_scale)
    tokens = np.zeros(R, dtype=np.int64)
    p_draft = np.zeros(R, dtype=np.float64)
    entropy = np.zeros(R, dtype=np.float64)
    gap = np.zeros(R, dtype=np.float64)
    accept = np.zeros(R, dtype=np.uint32)
    for q in range(n_req):
        for i in range(n_draft + 1):
            r = q * (n_draft + 1) + i
            tok, p, H, gp = row_stats(logits[r])
            tokens[r], entropy[r], gap[r] = tok, H, gp
            if i == n_draft:
                continue  # the bonus row verifies nothing
            x = int(draft[q * n_draft + i])
            p_draft[r] = p[x]
            bits = 0
            for k, e in enumerate(eps_v):
                if accepts(p[x], H, e):
                    bits |= 1 << k
            if x == tok:
                bits |= 1 << LOSSLESS_BIT
            accept[r] = bits
    accepted = np.zeros((n_req, E + 1), dtype=np.int64)
    for q in range(n_req):
        for k in range(E + 1):
            bit = LOSSLESS_BIT if k == E else k
            n = 0
            while n < n_draft and (int(accept[q * (n_draft + 1) + n]) >> bit) & 1:
                n += 1
            accepted[q, k] = n
    return {"tokens": tokens, "p_draft": p_draft, "entropy": entropy, "accept": accept, "gap": gap,
            "accepted": accepted, "eps": np.array(eps_v)}


def tokens_per_forward(accepted: np.ndarray) -> np.ndarray:
    """Accepted tokens for each target forward, per setting: accepted prefix + the target's own token."""
    return accepted.mean(axis=0) + 1.0
