"""Seeded synthetic calibration outcomes for the Redline selection.

Shared by the oracle tests and the native-path tests; holds no step of the
selection itself (no counting, no p-value, no test). Shapes follow the grids
the paper reports: n calibration prompts in {420, 500, 512, 542, 664, 1012}
and grids of m in {6, 7, 8, 16, 25, 50} configurations, one of them the
reference.

An outcome matrix is uint8 [n, m], prompt-major: entry (i, lam) is 1 when
configuration lam answers prompt i correctly. Configuration lam has a target
joint risk R[lam] = Pr[reference correct and lam wrong]: the reference is
correct with probability `ref_acc`, and given that, lam is wrong with
probability R[lam] / ref_acc. With `shared=True` one uniform per prompt decides
every configuration (the positively dependent draw of the paper's Monte Carlo
check); otherwise each configuration draws its own. On prompts the reference
gets wrong, lam is right with probability `gain`.
"""

from __future__ import annotations

from dataclasses import dataclass
from typing import List, Sequence

import numpy as np

PAPER_GRID_SHAPES = [(1012, 7), (542, 8), (1012, 8), (664, 8), (512, 8), (420, 8), (500, 16), (1012, 50)]


def outcome_matrix(n: int, risks: Sequence[float], ref: int, *, ref_acc: float = 0.85, gain: float = 0.05,
                   shared: bool = True, seed: int = 0) -> np.ndarray:
    m = len(risks)
    if not 0 <= ref < m:
        raise ValueError("reference index out of range")
    if any(r < 0 or r > ref_acc for r in risks):
        raise ValueError("each joint risk must lie in [0, ref_acc]")
    rng = np.random.default_rng(seed)
    ref_ok = rng.random(n) < ref_acc
    if shared:
        u = np.repeat(rng.random((n, 1)), m, axis=1)
    else:
        u = rng.random((n, m))
    g = rng.random((n, m))
    cond = np.asarray(risks, dtype=np.float64) / ref_acc
    out = np.where(ref_ok[:, None], u >= cond[None, :], g < gain).astype(np.uint8)
    out[:, ref] = ref_ok.astype(np.uint8)
    return out


def losses_matrix(n: int, risks: Sequence[float], *, shared: bool, seed: int) -> np.ndarray:
    """Outcomes whose reference column is always correct, so that the joint loss
    of (i, lam) is 1 exactly when u < R[lam]: the paper's Monte Carlo draw.
    Column 0 is the reference (risk 0); columns 1.. carry `risks`."""
    return outcome_matrix(n, [0.0] + list(risks), 0, ref_acc=1.0, gain=0.0, shared=shared, seed=seed)


@dataclass
class Grid:
    outcomes: np.ndarray  # uint8 [n, m]
    cost: np.ndarray      # float64 [m], TPF-like (higher is better)
    ref: int
    risks: List[float]


def random_grid(n: int, m: int, *, seed: int, risk_hi: float = 0.18, shared: bool = True) -> Grid:
    """A grid like the paper's block-diffusion grids: a reference of TPF 2.5-5.5,
    configurations of TPF 0.6x-1.8x the reference's, joint risks up to risk_hi."""
    rng = np.random.default_rng(seed + 7919)
    ref = int(rng.integers(0, m))
    ref_tpf = float(rng.uniform(2.5, 5.5))
    cost = ref_tpf * rng.uniform(0.6, 1.8, size=m)
    cost[ref] = ref_tpf
    risks = list(rng.uniform(0.0, risk_hi, size=m))
    risks[ref] = 0.0
    out = outcome_matrix(n, risks, ref, ref_acc=float(rng.uniform(0.6, 0.95)), shared=shared, seed=seed)
    return Grid(out, cost.astype(np.float64), ref, risks)
