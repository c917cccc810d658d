"""CPU oracles: float64 for the block-diffusion commit step and for
speculative verification, exact rationals for the Redline selection, plain
loops for the commit sweep.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its ``cpu_baseline`` leg and its ``--impl reference`` arm) may
import this package. The CUDA library and its Python binding never import it,
and it imports nothing from them: the two share no code.

Parity status: every function here is pinned by ``tests/test_oracle_pins.py``
(closed forms, a 50-digit brute force, invariants, a logsumexp cross-check and
hand-derived commit-rule cases). The only reading that no paper number can pin
is which blocks may take the top-1 fallback: that is an input (the caller's
``block_flags``), not a computation of the oracle. ``redline_oracle`` is
pinned by ``tests/test_redline_oracle.py`` (every p-value, valid mark and
deployment of the paper's appendix grid tables, the calibration-size table,
brute-force enumeration, closed-testing identities and an exact family-wise
error). ``sweep_oracle`` is pinned by ``tests/test_sweep_oracle.py``
(hand-derived cases, an independent whole-array formulation, and the
maximal-exact-commit invariant over simulated decodes). ``verify_oracle`` is
pinned by ``tests/test_verify_oracle.py`` (closed forms, a 50-digit brute
force, a hand-derived case for both branches of the rule, the nesting in eps,
and the paper's lossless tokens per forward from its draft agreement).
"""

from . import redline_oracle, sweep_oracle, verify_oracle
from .commit_oracle import (
    ACTIVE,
    FALLBACK_ELIGIBLE,
    commit_block,
    commit_step,
    decode_bf16,
    decode_e4m3,
    lm_head_logits,
    row_confidence,
    weights_f64,
)

__all__ = [
    "ACTIVE",
    "FALLBACK_ELIGIBLE",
    "commit_block",
    "commit_step",
    "decode_bf16",
    "decode_e4m3",
    "lm_head_logits",
    "redline_oracle",
    "sweep_oracle",
    "verify_oracle",
    "row_confidence",
    "weights_f64",
]
