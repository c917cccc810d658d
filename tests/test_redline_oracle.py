"""Pins of the Redline oracle against what the paper prints and what the
mathematics fixes (no GPU).

* every p-value, Holm-valid mark and deployed configuration of the appendix
  grid tables (tests/golden/redline_grids.json);
* the deployed gains and the smallest budgets with a gain of the table of
  deployments at three budgets (Sec. 5);
* single p-values printed in the text: the Holm-against-Bonferroni passage,
  the error-levels appendix and the 50-configuration grid appendix;
* the calibration-size table, parts (a) and (b);
* the binomial CDF against brute-force enumeration and closed forms;
* Holm and fixed sequence against their closed-testing forms;
* family-wise error of the paper's Monte Carlo setting, exactly and simulated.
"""

from __future__ import annotations

import itertools
import json
import math
import os
from decimal import ROUND_HALF_UP, Decimal
from fractions import Fraction as F

import numpy as np
import pytest

from oracle import redline_oracle as R
from tests.redline_helpers import exact_holm_fwer_nested
from workloads.redline_inputs import losses_matrix, outcome_matrix

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "redline_grids.json")
with open(GOLDEN) as fh:
    GRIDS = json.load(fh)
DELTA = F(GRIDS["delta"])
BUDGETS = [F(b) for b in GRIDS["budgets"]]


def grid(name):
    return next(g for g in GRIDS["grids"] if g["grid"] == name)


def printed_match(p: F, s: str) -> bool:
    """p rounds to the printed string: '0.019' to its decimals, '3e-14' or
    '8.5e-4' to its significant digits."""
    if "e" in s:
        mant, exp = s.split("e")
        unit = F(1, 10 ** (len(mant.split(".")[1]) if "." in mant else 0))
        scale = F(10) ** int(exp)
        return (F(mant) - unit / 2) * scale <= p < (F(mant) + unit / 2) * scale
    dec = len(s.split(".")[1])
    return abs(p - F(s)) <= F(1, 2 * 10**dec)


# --------------------------------------------------------------------------
# the appendix grid tables
# --------------------------------------------------------------------------
@pytest.mark.parametrize("g", GRIDS["grids"], ids=lambda g: g["grid"])
def test_grid_table(g):
    V = [c["k"] for c in g["configs"]]
    cost = [c["tpf"] for c in g["configs"]]
    for c in g["configs"]:
        assert printed_match(F(c["k"], g["n"]), c["rhat"]), c
    assert V[g["reference"]] == 0
    for b, alpha in enumerate(BUDGETS):
        r = R.redline(V, cost, g["n"], alpha, DELTA, g["reference"])
        for c, p, ok in zip(g["configs"], r["p"], r["valid"]):
            assert printed_match(p, c["p"][b]), (g["grid"], float(alpha), c["name"], float(p), c["p"][b])
            assert ok == c["valid"][b], (g["grid"], float(alpha), c["name"])
        assert r["deployed"] == g["deployed"][b], (g["grid"], float(alpha))


UNLOCK = {  # grid: (gain % at alpha 0.10, 0.15, 0.20; smallest budget with a gain)
    "LLaDA2 math": ((37.5, 37.5, 37.5), F("0.07")),
    "LLaDA2 code": ((0.0, 33.7, 42.4), F("0.11")),
    "SDAR math": ((13.1, 36.6, 36.6), F("0.10")),
    "SDAR code": ((0.0, 25.7, 59.7), F("0.11")),
}


@pytest.mark.parametrize("name", list(UNLOCK))
def test_unlock_table(name):
    """Deployed TPF gains at three budgets and alpha_min (Sec. 5, table of
    deployments), recomputed from the grid tables on the fine budget grid.
    The printed TPFs carry three decimals, so a gain may differ by 0.1 point."""
    g = grid(name)
    V = [c["k"] for c in g["configs"]]
    cost = [c["tpf"] for c in g["configs"]]
    gains, amin = UNLOCK[name]
    for alpha, want in zip((F("0.10"), F("0.15"), F("0.20")), gains):
        d = R.redline(V, cost, g["n"], alpha, DELTA, g["reference"])["deployed"]
        got = 100 * (cost[d] / cost[g["reference"]] - 1)
        assert abs(got - want) <= 0.1 + 1e-9, (alpha, got, want)
    fine = [F(i, 100) for i in range(1, 31)]
    s = R.sweep(V, cost, g["n"], fine, DELTA, g["reference"])
    assert fine[s["first_gain"]] == amin


def test_holm_against_bonferroni_passage():
    """LLaDA2 math at alpha = 0.07: acc90/semi90 (54/1012) has p = 0.0190,
    above Bonferroni's 0.1/7 = 0.0143 and under Holm's 0.025 at its rank 4;
    Holm deploys it (TPF 5.17, +17.4 %), Bonferroni acc95/semi70 (4.57, +3.9 %)."""
    g = grid("LLaDA2 math")
    V = [c["k"] for c in g["configs"]]
    cost = [c["tpf"] for c in g["configs"]]
    names = [c["name"] for c in g["configs"]]
    alpha = F("0.07")
    p = R.p_values(V, g["n"], alpha)
    i = names.index("acc90/semi90")
    assert printed_match(p[i], "0.0190")
    assert p[i] > DELTA / 7 and printed_match(DELTA / 7, "0.0143")
    rank = sorted(range(len(p)), key=lambda j: p[j]).index(i) + 1
    assert rank == 4 and DELTA / (len(p) - rank + 1) == F("0.025")
    holm = R.redline(V, cost, g["n"], alpha, DELTA, g["reference"], R.HOLM)
    bonf = R.redline(V, cost, g["n"], alpha, DELTA, g["reference"], R.BONFERRONI)
    assert names[holm["deployed"]] == "acc90/semi90"
    assert names[bonf["deployed"]] == "acc95/semi70"
    ref = cost[g["reference"]]
    assert round(100 * (cost[holm["deployed"]] / ref - 1), 1) == 17.4
    assert round(100 * (cost[bonf["deployed"]] / ref - 1), 1) == 3.9
    # Holm's valid set contains Bonferroni's (Holm appendix)
    assert all(h or not b for h, b in zip(holm["valid"], bonf["valid"]))


def test_error_levels_across_grids():
    """SDAR math at alpha = 0.10 with delta = 0.10 / 4: the deployed
    acc90/semi90 keeps p = 8.5e-4 under Holm's 0.025 / 6 at its rank."""
    g = grid("SDAR math")
    V = [c["k"] for c in g["configs"]]
    cost = [c["tpf"] for c in g["configs"]]
    names = [c["name"] for c in g["configs"]]
    r = R.redline(V, cost, g["n"], F("0.10"), DELTA / 4, g["reference"])
    i = names.index("acc90/semi90")
    assert r["deployed"] == i
    assert printed_match(r["p"][i], "8.5e-4")
    rank = sorted(range(len(V)), key=lambda j: r["p"][j]).index(i) + 1
    assert (DELTA / 4) / (len(V) - rank + 1) == F("0.025") / 6


def test_delta_sensitivity():
    """The math deployments at alpha = 0.10 do not move for delta in {0.10, 0.05, 0.01}."""
    for name, want in (("LLaDA2 math", "acc85/semi70"), ("SDAR math", "acc90/semi90")):
        g = grid(name)
        V = [c["k"] for c in g["configs"]]
        cost = [c["tpf"] for c in g["configs"]]
        for delta in (F("0.10"), F("0.05"), F("0.01")):
            d = R.redline(V, cost, g["n"], F("0.10"), delta, g["reference"])["deployed"]
            assert g["configs"][d]["name"] == want


def test_printed_scalar_pvalues():
    """p-values quoted in the text and small tables."""
    cases = [
        (73, 1012, "0.10", "0.001"),    # LLaDA2 math grid, acc85/semi70
        (54, 1012, "0.07", "0.0190"),   # Holm against Bonferroni passage
        (72, 1012, "0.10", "8.5e-4"),   # error levels across grids
        (73, 500, "0.20", "0.001"),     # distilled acc85/semi70 on MATH-500
        (74, 1012, "0.10", "0.0018"),   # 50-configuration grid at alpha = 0.10
    ]
    for k, n, a, s in cases:
        assert printed_match(R.p_value(k, n, F(a)), s), (k, n, a, s)
    # the 50-configuration passage: Bonferroni's delta / 50 and Holm's 0.0056 at rank 33
    assert F("0.0018") < DELTA / 50 == F("0.002")
    assert printed_match(DELTA / (50 - 33 + 1), "0.0056")


# --------------------------------------------------------------------------
# calibration size
# --------------------------------------------------------------------------
def half_up(x: F, places: int) -> Decimal:
    return (Decimal(x.numerator) / Decimal(x.denominator)).quantize(Decimal(1).scaleb(-places), ROUND_HALF_UP)


SAMPLESIZE_B = {  # n: largest passing R-hat (%) at delta/8, delta/50, delta (alpha = 0.10)
    542: ("7.0", "6.3", "8.1"),
    664: ("7.4", "6.6", "8.4"),
    1012: ("7.8", "7.3", "8.7"),
    2000: ("8.5", "8.1", "9.1"),
    5000: ("9.0", "8.8", "9.4"),
}


@pytest.mark.parametrize("n", list(SAMPLESIZE_B))
def test_samplesize_margin(n):
    """Calibration-size table (b): the largest empirical risk that passes at
    alpha = 0.10, i.e. 100 * c / n for the critical count c, rounded half up."""
    for level, want in zip((DELTA / 8, DELTA / 50, DELTA), SAMPLESIZE_B[n]):
        c = R.critical_count(n, F("0.10"), level)
        assert str(half_up(100 * F(c, n), 1)) == want, (n, float(level), c)
        # c is the boundary: c passes, c + 1 does not
        assert R.binom_cdf(c, n, F("0.10")) <= level < R.binom_cdf(c + 1, n, F("0.10"))


SAMPLESIZE_A = [  # alpha, true R, prompts for power 0.8 at m = 8, 16, 50
    ("0.02", "0.01", (1623, 1828, 2274)),
    ("0.05", "0.04", (4320, 5048, 6217)),
    ("0.05", "0.03", (1008, 1189, 1444)),
    ("0.10", "0.09", (8407, 9842, 12179)),
    ("0.10", "0.08", (2066, 2406, 2966)),
]


@pytest.mark.parametrize("row", SAMPLESIZE_A, ids=lambda r: f"a{r[0]}_R{r[1]}")
def test_samplesize_power(row):
    """Calibration-size table (a): from the printed n on, a configuration of
    true risk R passes Holm's first step delta / m with probability >= 0.8; at
    n - 1 it does not (the last failure of the sawtooth)."""
    a, r, ns = row
    for m, n0 in zip((8, 16, 50), ns):
        lv = DELTA / m
        assert R.power(n0, F(r), F(a), lv) >= F("0.8"), (a, r, m, n0)
        assert R.power(n0 - 1, F(r), F(a), lv) < F("0.8"), (a, r, m, n0)


# --------------------------------------------------------------------------
# the binomial CDF itself
# --------------------------------------------------------------------------
def test_cdf_brute_force():
    """Pr[S <= k] by enumerating all 2^n loss vectors of n Bernoulli(alpha) prompts."""
    for n in (0, 1, 2, 5, 9):
        for a in (F(1, 10), F(1, 3), F(7, 8)):
            probs = [F(0)] * (n + 1)
            for x in itertools.product((0, 1), repeat=n):
                s = sum(x)
                probs[s] += a**s * (1 - a) ** (n - s)
            for k in range(-1, n + 2):
                want = sum(probs[: max(0, min(k, n) + 1)], F(0))
                assert R.binom_cdf(k, n, a) == want


def test_cdf_closed_forms():
    for n in (1, 10, 100, 400):
        for a in (F(1, 20), F(1, 10), F(1, 2), F(9, 10)):
            assert R.binom_cdf(n, n, a) == 1
            assert R.binom_cdf(0, n, a) == (1 - a) ** n
            assert R.binom_cdf(n - 1, n, a) == 1 - a**n
    for n in (7, 40, 120):
        for k in range(0, n):
            # symmetry: S ~ Bin(n, a) <=> n - S ~ Bin(n, 1 - a)
            assert R.binom_cdf(k, n, F(3, 10)) == 1 - R.binom_cdf(n - k - 1, n, F(7, 10))
    # the stochastic ordering behind super-uniformity: p decreases as the risk grows
    for k in (0, 30, 73):
        ps = [R.binom_cdf(k, 1012, F(j, 100)) for j in range(1, 30)]
        assert all(x > y for x, y in zip(ps, ps[1:]))
    # the reference row of every grid: V = 0 gives (1 - alpha)^n, printed 3e-23 at n = 1012, alpha = 0.05
    assert printed_match(R.p_value(0, 1012, F("0.05")), "3e-23")
    # table, integer-term sum and critical count agree with the direct sum
    tab = R.binom_cdf_table(300, F("0.07"), 320)
    assert tab == [R.binom_cdf(k, 300, F("0.07")) for k in range(321)]
    for a in (F(0), F(1), F(0.3), F("0.07")):
        assert all(R.binom_cdf_sum(k, 60, a) == R.binom_cdf(k, 60, a) for k in range(-1, 62))
    for lv in (F(1, 1000), F(1, 80), F(1, 10), F(1, 2)):
        c = R.critical_count(300, F("0.07"), lv)
        assert all((t <= lv) == (k <= c) for k, t in enumerate(tab))


def test_cdf_degenerate():
    assert R.binom_cdf(-1, 10, F(1, 2)) == 0
    assert R.binom_cdf(0, 0, F(1, 2)) == 1
    assert R.binom_cdf(3, 10, F(0)) == 1
    assert R.binom_cdf(9, 10, F(1)) == 0 and R.binom_cdf(10, 10, F(1)) == 1
    assert R.critical_count(10, F(1, 2), F(1, 10**6)) == -1
    assert R.power(10, F(1, 10), F(1, 2), F(1, 10**6)) == 0


# --------------------------------------------------------------------------
# the procedures against their closed-testing forms
# --------------------------------------------------------------------------
def closed_testing(p, delta, local):
    """Reject H_i iff every intersection hypothesis containing i is rejected by `local`."""
    m = len(p)
    out = []
    for i in range(m):
        ok = True
        for size in range(1, m + 1):
            for S in itertools.combinations(range(m), size):
                if i in S and not local(S):
                    ok = False
                    break
            if not ok:
                break
        out.append(ok)
    return out


def test_holm_is_closed_bonferroni():
    """Holm equals closed testing with Bonferroni local tests (min_S p <= delta / |S|)."""
    rng = np.random.default_rng(5)
    for _ in range(300):
        m = int(rng.integers(1, 7))
        p = [F(int(x), 1000) for x in rng.integers(0, 120, size=m)]
        delta = F(1, 10)
        want = closed_testing(p, delta, lambda S: min(p[j] for j in S) <= delta / len(S))
        assert R.holm(p, delta) == want


def test_fixed_sequence_is_closed_testing():
    """Fixed sequence equals closed testing whose local test of H_S checks the
    first hypothesis of S in the walk order at the full delta."""
    rng = np.random.default_rng(6)
    for _ in range(300):
        m = int(rng.integers(1, 7))
        p = [F(int(x), 1000) for x in rng.integers(0, 200, size=m)]
        order = [int(v) for v in rng.permutation(m)]
        pos = {v: j for j, v in enumerate(order)}
        delta = F(1, 10)
        want = closed_testing(p, delta, lambda S: p[min(S, key=lambda j: pos[j])] <= delta)
        assert R.fixed_sequence(p, order, delta) == want


def test_bonferroni_inside_holm_and_deploy_rules():
    rng = np.random.default_rng(7)
    for _ in range(200):
        m = int(rng.integers(1, 12))
        p = [F(int(x), 10000) for x in rng.integers(0, 400, size=m)]
        h, b = R.holm(p, F(1, 10)), R.bonferroni(p, F(1, 10))
        assert all(hh or not bb for hh, bb in zip(h, b))
    # nothing valid: the reference; ties: the lowest index; memory: the least
    assert R.deploy([False, False, False], [3.0, 5.0, 4.0], ref=1) == 1
    assert R.deploy([True, True, True], [5.0, 5.0, 4.0], ref=2) == 0
    assert R.deploy([True, True, False], [16.0, 5.6, 3.2], ref=0, higher_is_better=False) == 1


def test_joint_violations():
    """V counts prompts the reference answers and the configuration does not (Eq. 1);
    prompts the reference misses never count, whatever the configuration does."""
    out = [
        [1, 1, 0, 0],
        [1, 0, 1, 0],
        [0, 1, 0, 1],
        [1, 1, 1, 1],
        [0, 0, 0, 0],
    ]
    assert R.joint_violations(out, 0) == [0, 1, 1, 2]
    assert R.joint_violations(out, 1) == [1, 0, 2, 1]
    rng = np.random.default_rng(3)
    M = rng.integers(0, 2, size=(200, 6))
    for ref in range(6):
        V = R.joint_violations(M.tolist(), ref)
        assert V == [int(np.sum((M[:, ref] == 1) & (M[:, j] == 0))) for j in range(6)]


def test_generator_hits_target_risks():
    """Seeded outcomes carry the intended joint risks (sanity of the test inputs)."""
    risks = [0.0, 0.02, 0.07, 0.12]
    out = outcome_matrix(20000, risks, 0, ref_acc=0.8, shared=False, seed=11)
    V = R.joint_violations(out.tolist(), 0)
    assert V[0] == 0
    for v, r in zip(V[1:], risks[1:]):
        assert abs(v / 20000 - r) < 5 * math.sqrt(r * (1 - r) / 20000)


def test_tpf_from_counts():
    counts = [[10, 6, 2], [8, 8, 2], [12, 4, 2]]
    assert R.tpf_from_counts(counts, 2) == [F(30, 6), F(18, 6), F(6, 6)]


# --------------------------------------------------------------------------
# family-wise error (validity appendix, synthetic Monte Carlo)
# --------------------------------------------------------------------------
def test_montecarlo_fwer_paper_setting():
    """Five configurations of true risk {0.01, 0.02, 0.07, 0.07, 0.07}, alpha =
    0.05, n = 800, shared uniform: the exact FWER of Holm is far below delta
    (1.6e-5; the paper's 4,000 simulated trials saw one rejection, 0.0003), and
    a 4,000-trial simulation sees at most a handful."""
    risks = [F("0.01"), F("0.02"), F("0.07"), F("0.07"), F("0.07")]
    exact = exact_holm_fwer_nested(800, F("0.05"), DELTA, risks)
    assert 1e-5 < exact < 3e-5
    tab = R.binom_cdf_table(800, F("0.05"), 800)
    bad = 0
    for t in range(4000):
        L = losses_matrix(800, [float(r) for r in risks], shared=True, seed=t)
        V = R.joint_violations(L.tolist(), 0)[1:]
        valid = R.holm([tab[v] for v in V], DELTA)
        bad += any(valid[j] for j in (2, 3, 4))
    assert bad <= 3


def test_montecarlo_fwer_near_boundary():
    """Nulls just above the budget make errors frequent enough to measure:
    true risks {0.02, 0.055, 0.055} at alpha = 0.05, n = 400, delta = 0.10.
    The simulated FWER matches the exact nested-count value within 4 standard
    errors and both stay under delta."""
    risks = [F("0.02"), F("0.055"), F("0.055")]
    n, alpha = 400, F("0.05")
    exact = exact_holm_fwer_nested(n, alpha, DELTA, risks)
    assert 0.005 < exact < float(DELTA)
    tab = R.binom_cdf_table(n, alpha, n)
    trials, bad = 3000, 0
    for t in range(trials):
        L = losses_matrix(n, [float(r) for r in risks], shared=True, seed=100000 + t)
        V = R.joint_violations(L.tolist(), 0)[1:]
        valid = R.holm([tab[v] for v in V], DELTA)
        bad += valid[1] or valid[2]
    se = math.sqrt(exact * (1 - exact) / trials)
    assert abs(bad / trials - exact) < 4 * se + 1e-12, (bad / trials, exact)
