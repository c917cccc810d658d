"""Oracle of the Redline selection (test infrastructure).

Plain, slow, exact restatement of how the paper turns calibration outcomes
into a deployed serving configuration. Only the tests, the smoke check and the
CPU-baseline leg of the benchmark use this module; the product path
(libbdcommit's bd_redline_* entry points) shares no code with it.

Arithmetic is exact: probabilities are `fractions.Fraction`s and every
decision (p <= threshold) is taken on exact rationals. Floats given as alpha,
delta or R are converted with `Fraction(x)`, i.e. at their exact binary value,
so the oracle and the native path decide on the same numbers.

Passages followed:
  * Eq. 1 (Sec. 3.1) and the setup appendix: the joint loss of prompt i is 1
    exactly when the reference answers it correctly and configuration lambda
    does not; V_lambda counts those prompts.
  * Sec. 3.2 step (ii) and the exact-binomial appendix:
    p_lambda = Pr[Bin(n, alpha) <= V_lambda], testing H0: R(lambda) > alpha.
  * Sec. 3.2 step (iii) and the Holm appendix: sort the p-values, reject while
    p_(i) <= delta / (m - i + 1), stop at the first failure.
  * Holm appendix: Bonferroni (p <= delta / m) as the conservative floor.
  * Fixed-sequence appendix: walk a data-independent order, test each at the
    full delta, stop at the first failure.
  * Sec. 3.2 step (iv) and the deployment appendix: deploy the valid
    configuration with the best cost (highest TPF, or least memory); the
    reference when nothing is valid.
  * Error-levels appendix: the smallest budget with a gain is the smallest
    budget of a grid at which a configuration cheaper than the reference is
    deployed.
  * Calibration-size table: the largest violation count that passes at a
    level, and the power of the exact test at a true risk R.
"""

from __future__ import annotations

import math
from fractions import Fraction
from typing import Dict, List, Optional, Sequence

HOLM = "holm"
BONFERRONI = "bonferroni"
FIXED_SEQUENCE = "fixed_sequence"
PROCEDURES = (HOLM, BONFERRONI, FIXED_SEQUENCE)


def as_fraction(x) -> Fraction:
    """Exact rational of a float (its binary value), a decimal string or a Fraction."""
    if isinstance(x, Fraction):
        return x
    if isinstance(x, str):
        return Fraction(x)
    if isinstance(x, int):
        return Fraction(x)
    return Fraction(float(x))


# --------------------------------------------------------------------------
# Step (ii): violation counts and the exact binomial p-value
# --------------------------------------------------------------------------
def joint_violations(outcomes: Sequence[Sequence[int]], ref: int) -> List[int]:
    """V_lambda from a prompt x configuration matrix of 0/1 correctness (Eq. 1).

    outcomes[i][lam] = 1 when configuration lam answers prompt i correctly.
    A prompt counts against lam when the reference column is 1 and lam's is 0.
    """
    m = len(outcomes[0]) if len(outcomes) else 0
    V = [0] * m
    for row in outcomes:
        if row[ref]:
            for lam in range(m):
                if not row[lam]:
                    V[lam] += 1
    return V


def binom_cdf(k: int, n: int, alpha) -> Fraction:
    """Pr[Bin(n, alpha) <= k] = sum_{j=0}^{k} C(n, j) alpha^j (1 - alpha)^(n - j), exactly."""
    a = as_fraction(alpha)
    if k < 0:
        return Fraction(0)
    total = Fraction(0)
    for j in range(0, min(k, n) + 1):
        total += math.comb(n, j) * a**j * (1 - a) ** (n - j)
    return total


def _scaled_terms(n: int, a: Fraction):
    """Yield C(n, j) a^j (1 - a)^(n - j) * den^n for j = 0..n as exact integers,
    where a = num / den. Consecutive terms follow the ratio
    C(n, j+1) / C(n, j) * num / (den - num) = (n - j) num / ((j + 1)(den - num))."""
    num, den = a.numerator, a.denominator
    q = den - num
    if q == 0:  # a = 1: all mass at j = n
        for j in range(n + 1):
            yield den**n if j == n else 0
        return
    t = q**n
    for j in range(n + 1):
        yield t
        if j < n:
            t = t * (n - j) * num // ((j + 1) * q)


def binom_cdf_sum(k: int, n: int, alpha) -> Fraction:
    """The same sum as binom_cdf, accumulated over the exact integer terms of
    _scaled_terms and normalised once (fast for large n and any alpha)."""
    a = as_fraction(alpha)
    if k < 0:
        return Fraction(0)
    acc = 0
    for j, t in enumerate(_scaled_terms(n, a)):
        if j > k:
            break
        acc += t
    return Fraction(acc, a.denominator**n)


def binom_cdf_table(n: int, alpha, k_max: int) -> List[Fraction]:
    """[Pr[Bin(n, alpha) <= k] for k = 0..k_max], accumulated once over the terms."""
    a = as_fraction(alpha)
    den_n = a.denominator**n
    out = []
    acc = 0
    for j, t in enumerate(_scaled_terms(n, a)):
        if j > k_max:
            break
        acc += t
        out.append(Fraction(acc, den_n))
    out.extend([Fraction(1)] * (k_max + 1 - len(out)))
    return out


def p_value(V: int, n: int, alpha) -> Fraction:
    """p = Pr_{Bin(n, alpha)}[S <= V] for H0: R > alpha (exact-binomial appendix)."""
    return binom_cdf_sum(V, n, alpha)


def p_values(V: Sequence[int], n: int, alpha) -> List[Fraction]:
    return [p_value(v, n, alpha) for v in V]


# --------------------------------------------------------------------------
# Step (iii): the multiple-testing procedures
# --------------------------------------------------------------------------
def holm(p: Sequence[Fraction], delta) -> List[bool]:
    """Holm step-down at family-wise level delta (Sec. 3.2 (iii), Holm appendix)."""
    d = as_fraction(delta)
    m = len(p)
    order = sorted(range(m), key=lambda i: p[i])
    valid = [False] * m
    for rank, i in enumerate(order, start=1):
        if p[i] <= d / (m - rank + 1):
            valid[i] = True
        else:
            break
    return valid


def bonferroni(p: Sequence[Fraction], delta) -> List[bool]:
    """Each hypothesis at delta / m (Holm appendix: the conservative floor)."""
    d = as_fraction(delta)
    m = len(p)
    return [pi <= d / m for pi in p]


def fixed_sequence(p: Sequence[Fraction], order: Sequence[int], delta) -> List[bool]:
    """Walk `order` testing each at the full delta; stop at the first failure."""
    d = as_fraction(delta)
    valid = [False] * len(p)
    for i in order:
        if p[i] <= d:
            valid[i] = True
        else:
            break
    return valid


def test(p: Sequence[Fraction], delta, procedure: str = HOLM, order: Optional[Sequence[int]] = None) -> List[bool]:
    if procedure == HOLM:
        return holm(p, delta)
    if procedure == BONFERRONI:
        return bonferroni(p, delta)
    if procedure == FIXED_SEQUENCE:
        if order is None:
            raise ValueError("fixed-sequence testing needs an order")
        return fixed_sequence(p, order, delta)
    raise ValueError(f"unknown procedure {procedure!r}")


# --------------------------------------------------------------------------
# Step (iv): deployment
# --------------------------------------------------------------------------
def better(a: float, b: float, higher_is_better: bool) -> bool:
    return a > b if higher_is_better else a < b


def deploy(valid: Sequence[bool], cost: Sequence[float], ref: int, higher_is_better: bool = True) -> int:
    """The valid configuration with the best cost; ties go to the lowest index;
    the reference when nothing is valid."""
    best = -1
    for i, ok in enumerate(valid):
        if ok and (best < 0 or better(cost[i], cost[best], higher_is_better)):
            best = i
    return ref if best < 0 else best


def redline(V: Sequence[int], cost: Sequence[float], n: int, alpha, delta, ref: int,
            procedure: str = HOLM, order: Optional[Sequence[int]] = None,
            higher_is_better: bool = True) -> Dict:
    """Steps (ii)-(iv) on one grid at one budget."""
    p = p_values(V, n, alpha)
    valid = test(p, delta, procedure, order)
    return {"p": p, "valid": valid, "deployed": deploy(valid, cost, ref, higher_is_better)}


def sweep(V: Sequence[int], cost: Sequence[float], n: int, alphas: Sequence, delta, ref: int,
          procedure: str = HOLM, order: Optional[Sequence[int]] = None,
          higher_is_better: bool = True) -> Dict:
    """Redline at every budget of `alphas`; `first_gain` is the index of the
    smallest budget whose deployed configuration beats the reference's cost
    (-1 if none): the smallest budget with a gain."""
    deployed, n_valid = [], []
    first_gain = -1
    for j, a in enumerate(alphas):
        r = redline(V, cost, n, a, delta, ref, procedure, order, higher_is_better)
        deployed.append(r["deployed"])
        n_valid.append(sum(r["valid"]))
        if first_gain < 0 and better(cost[r["deployed"]], cost[ref], higher_is_better):
            first_gain = j
    return {"deployed": deployed, "n_valid": n_valid, "first_gain": first_gain}


# --------------------------------------------------------------------------
# Calibration size
# --------------------------------------------------------------------------
def critical_count(n: int, alpha, level) -> int:
    """Largest V with Pr[Bin(n, alpha) <= V] <= level; -1 if even V = 0 fails."""
    a = as_fraction(alpha)
    lv = as_fraction(level)
    bound = lv * a.denominator**n  # compare sum of scaled terms against level * den^n
    acc = 0
    c = -1
    for j, t in enumerate(_scaled_terms(n, a)):
        acc += t
        if acc <= bound:
            c = j
        else:
            break
    return c


def power(n: int, R, alpha, level) -> Fraction:
    """Probability that a configuration of true risk R passes a test at `level`:
    Pr[Bin(n, R) <= critical_count(n, alpha, level)]."""
    c = critical_count(n, alpha, level)
    return binom_cdf_sum(c, n, R) if c >= 0 else Fraction(0)


# --------------------------------------------------------------------------
# Cost input from the commit step
# --------------------------------------------------------------------------
def tpf_from_counts(counts: Sequence[Sequence[int]], n_seq: int) -> List[Fraction]:
    """Tokens committed per forward per sequence for each accept threshold:
    counts[s][t] is the number of positions that forward s committed at
    threshold t over n_seq sequences."""
    S = len(counts)
    T = len(counts[0]) if S else 0
    return [sum(Fraction(counts[s][t]) for s in range(S)) / (S * n_seq) if S and n_seq else Fraction(0)
            for t in range(T)]
