"""Parity of the native Redline entry points (include/redline.h, host code of
libbdcommit, called through the C ABI) with the exact oracle. No GPU.

Tolerances. The native p-value is one binomial probability by Loader's
saddle-point expansion times a ratio recurrence over the shorter tail, in
double precision: relative error a few hundred ulps at worst, so p-values
must agree within 1e-12 relative (plus 2e-16 absolute for values near 1).
Counts (violations, critical counts, calibration sizes) and decisions are
compared exactly; a decision may differ only where the exact p-value lies
within 1e-10 relative of its threshold, and the cases below are checked to
stay clear of that.
"""

from __future__ import annotations

import ctypes
import json
import math
import os
import random
import shutil
from fractions import Fraction as F

import numpy as np
import pytest

from oracle import redline_oracle as R
from paper_2609_33887_gb300 import bdcommit as B
from paper_2609_33887_gb300 import redline as N
from tests.redline_helpers import exact_holm_fwer_nested
from workloads.redline_inputs import PAPER_GRID_SHAPES, losses_matrix, random_grid

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "redline_grids.json")
with open(GOLDEN) as fh:
    GRIDS = json.load(fh)
BUDGETS = [float(b) for b in GRIDS["budgets"]]
FINE = [i / 100 for i in range(1, 31)]
REL = 1e-12


@pytest.fixture(scope="module", autouse=True)
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no CUDA toolkit")
    import __graft_entry__

    __graft_entry__.build()
    return B.load_library()


def close(got: float, exact: F) -> bool:
    e = float(exact)
    return abs(got - e) <= REL * e + 2e-16


def near_threshold(p: F, thresholds) -> bool:
    return any(t > 0 and abs(p - t) <= F(1, 10**10) * t for t in thresholds)


def all_thresholds(m: int, delta: float):
    d = F(delta)
    return [d / k for k in range(1, m + 1)]


def status_of(fn, *a, **k) -> int:
    with pytest.raises(B.BdError) as e:
        fn(*a, **k)
    return e.value.status


# --------------------------------------------------------------------------
# the binomial CDF
# --------------------------------------------------------------------------
def test_binom_cdf_against_exact():
    rng = random.Random(1)
    for _ in range(250):
        n = rng.choice([1, 2, 5, 17, 100, 420, 512, 542, 664, 800, 1012, 2000])
        a = rng.choice([0.01, 0.02, 0.05, 0.07, 0.1, 0.15, 0.2, 0.5, 0.9, rng.random()])
        if rng.random() < 0.4:
            k = rng.randint(0, n)
        else:
            k = max(0, min(n, int(n * a + rng.gauss(0, 3) * math.sqrt(n * a * (1 - a)))))
        assert close(N.bd_binom_cdf(k, n, a), R.binom_cdf_sum(k, n, F(a))), (k, n, a)
    # large n at decimal budgets. The oracle takes the decimal itself: the
    # double's relative error (<= 2^-53) moves p by under 1e-13 relative here.
    for n, a in ((5000, "0.1"), (12179, "0.1"), (20000, "0.05"), (50000, "0.02")):
        af = float(a)
        for z in (-6, -3, -1, 0, 1, 3):
            k = int(n * af + z * math.sqrt(n * af * (1 - af)))
            assert close(N.bd_binom_cdf(k, n, af), R.binom_cdf_sum(k, n, F(a))), (k, n, a)


def test_binom_cdf_edges():
    assert N.bd_binom_cdf(-1, 10, 0.3) == 0.0
    assert N.bd_binom_cdf(10, 10, 0.3) == 1.0 and N.bd_binom_cdf(99, 10, 0.3) == 1.0
    assert N.bd_binom_cdf(0, 0, 0.3) == 1.0
    assert N.bd_binom_cdf(3, 10, 0.0) == 1.0
    assert N.bd_binom_cdf(9, 10, 1.0) == 0.0
    assert close(N.bd_binom_cdf(0, 1012, 0.05), (1 - F(0.05)) ** 1012)
    assert close(N.bd_binom_cdf(9, 10, 0.5), 1 - F(1, 2) ** 10)
    for bad in (-0.1, 1.1, float("nan")):
        assert status_of(N.bd_binom_cdf, 1, 10, bad) == -10
    assert status_of(N.bd_binom_cdf, 1, -1, 0.5) == -2


# --------------------------------------------------------------------------
# the paper's grids
# --------------------------------------------------------------------------
@pytest.mark.parametrize("g", GRIDS["grids"], ids=lambda g: g["grid"])
def test_grid_tables_native(g):
    V = [c["k"] for c in g["configs"]]
    cost = [c["tpf"] for c in g["configs"]]
    for b, alpha in enumerate(BUDGETS):
        got = N.bd_redline_select(V, cost, g["n"], alpha, g["reference"], delta=0.10)
        want = R.redline(V, cost, g["n"], alpha, 0.10, g["reference"])
        for x, e in zip(got["p"], want["p"]):
            assert close(x, e)
        assert list(got["valid"]) == want["valid"] == [c["valid"][b] for c in g["configs"]]
        assert got["deployed"] == want["deployed"] == g["deployed"][b]
    for proc in ("holm", "bonferroni"):
        got = N.bd_redline_sweep(V, cost, g["n"], FINE, g["reference"], delta=0.10, procedure=proc)
        want = R.sweep(V, cost, g["n"], FINE, 0.10, g["reference"], procedure=proc)
        assert list(got["deployed"]) == want["deployed"]
        assert list(got["n_valid"]) == want["n_valid"]
        assert got["first_gain"] == want["first_gain"]


def test_unlock_smallest_budgets_native():
    want = {"LLaDA2 math": 0.07, "LLaDA2 code": 0.11, "SDAR math": 0.10, "SDAR code": 0.11}
    for g in GRIDS["grids"]:
        if g["grid"] in want:
            V = [c["k"] for c in g["configs"]]
            cost = [c["tpf"] for c in g["configs"]]
            s = N.bd_redline_sweep(V, cost, g["n"], FINE, g["reference"])
            assert FINE[s["first_gain"]] == want[g["grid"]]


# --------------------------------------------------------------------------
# seeded grids shaped like the paper's
# --------------------------------------------------------------------------
@pytest.mark.parametrize("shape", PAPER_GRID_SHAPES, ids=lambda s: f"n{s[0]}_m{s[1]}")
def test_random_grids_parity(shape):
    n, m = shape
    for seed in range(3):
        gr = random_grid(n, m, seed=1000 * n + 10 * m + seed)
        V = N.bd_redline_violations(gr.outcomes, gr.ref)
        assert list(V) == R.joint_violations(gr.outcomes.tolist(), gr.ref)
        order = [int(x) for x in np.random.default_rng(seed).permutation(m)]
        for alpha in (0.05, 0.08, 0.10, 0.15, 0.20):
            p_exact = R.p_values(list(V), n, alpha)
            assert not any(near_threshold(p, all_thresholds(m, 0.10)) for p in p_exact)
            for proc in ("holm", "bonferroni", "fixed_sequence"):
                o = order if proc == "fixed_sequence" else None
                got = N.bd_redline_select(V, gr.cost, n, alpha, gr.ref, delta=0.10, procedure=proc, order=o)
                valid = R.test(p_exact, 0.10, proc, o)
                assert all(close(x, e) for x, e in zip(got["p"], p_exact))
                assert list(got["valid"]) == valid, (shape, seed, alpha, proc)
                assert got["deployed"] == R.deploy(valid, list(gr.cost), gr.ref)


def test_memory_cost_and_deploy_rules():
    # quantization grids deploy the least memory among the valid configurations
    V = [0, 30, 45, 70]
    mem = [16.0, 8.5, 5.7, 4.2]
    for alpha in (0.05, 0.08, 0.10, 0.15):
        got = N.bd_redline_select(V, mem, 512, alpha, 0, higher_is_better=False)
        want = R.redline(V, mem, 512, alpha, 0.10, 0, higher_is_better=False)
        assert got["deployed"] == want["deployed"]
    assert N.bd_redline_deploy([0, 0, 0], [3.0, 5.0, 4.0], 1) == 1
    assert N.bd_redline_deploy([1, 1, 1], [5.0, 5.0, 4.0], 2) == 0
    assert N.bd_redline_deploy([1, 1, 0], [16.0, 5.6, 3.2], 0, higher_is_better=False) == 1


def test_procedures_direct():
    rng = np.random.default_rng(9)
    for _ in range(300):
        m = int(rng.integers(1, 20))
        p = [F(int(x), 10000) for x in rng.integers(0, 500, size=m)]
        order = [int(x) for x in rng.permutation(m)]
        pf = [float(x) for x in p]
        if any(near_threshold(x, all_thresholds(m, 0.1)) for x in p):
            continue  # an exact tie with a threshold: double rounding may decide either way
        assert list(N.bd_redline_test(pf, 0.1, "holm")) == R.holm(p, 0.1)
        assert list(N.bd_redline_test(pf, 0.1, "bonferroni")) == R.bonferroni(p, 0.1)
        assert list(N.bd_redline_test(pf, 0.1, "fixed_sequence", order)) == R.fixed_sequence(p, order, 0.1)


# --------------------------------------------------------------------------
# calibration size
# --------------------------------------------------------------------------
SAMPLESIZE_B = {542: (7.0, 6.3, 8.1), 664: (7.4, 6.6, 8.4), 1012: (7.8, 7.3, 8.7),
                2000: (8.5, 8.1, 9.1), 5000: (9.0, 8.8, 9.4)}
SAMPLESIZE_A = [(0.02, 0.01, (1623, 1828, 2274)), (0.05, 0.04, (4320, 5048, 6217)),
                (0.05, 0.03, (1008, 1189, 1444)), (0.10, 0.09, (8407, 9842, 12179)),
                (0.10, 0.08, (2066, 2406, 2966))]


def test_samplesize_native():
    """The calibration-size table: (b) from the critical count, rounded half up
    on the exact per-mille; (a) from the prompts-needed scan up to 3 n0."""
    for n, row in SAMPLESIZE_B.items():
        for level, want in zip((0.1 / 8, 0.1 / 50, 0.1), row):
            c = N.bd_redline_critical_count(n, 0.10, level)
            assert c == R.critical_count(n, F(0.10), F(level))
            assert (2000 * c + n) // (2 * n) == round(10 * want)  # floor(1000 c / n + 1/2)
    for a, r, ns in SAMPLESIZE_A:
        for m, n0 in zip((8, 16, 50), ns):
            assert N.bd_redline_min_calibration(r, a, 0.1 / m, 0.8, 3 * n0) == n0, (a, r, m, n0)
            for n in (n0 - 1, n0, n0 + 37):  # the oracle on the decimals, as above
                assert close(N.bd_redline_power(n, r, a, 0.1 / m), R.power(n, F(str(r)), F(str(a)), F(1, 10 * m)))


def test_calibration_edges():
    assert N.bd_redline_critical_count(10, 0.5, 1e-6) == -1
    assert N.bd_redline_critical_count(10, 0.5, 1.0) == 10
    assert N.bd_redline_critical_count(0, 0.5, 0.1) == -1
    assert N.bd_redline_power(10, 0.1, 0.5, 1e-6) == 0.0
    assert N.bd_redline_min_calibration(0.09, 0.10, 0.1 / 8, 0.8, 100) == -1  # not reached by n = 100
    assert N.bd_redline_min_calibration(0.0, 0.10, 0.1, 0.0, 50) == 1
    assert status_of(N.bd_redline_min_calibration, 0.09, 0.10, 0.1, 0.8, 0) == -2
    assert status_of(N.bd_redline_min_calibration, 0.09, 0.10, 0.1, 1.5, 10) == -10
    assert status_of(N.bd_redline_critical_count, -1, 0.1, 0.1) == -2
    assert status_of(N.bd_redline_power, 10, float("nan"), 0.1, 0.1) == -10


# --------------------------------------------------------------------------
# argument errors: a negative status
# --------------------------------------------------------------------------
def test_argument_errors():
    sel = N.bd_redline_select
    assert status_of(sel, [0, 5], [1.0, 2.0], 10, 0.1, 2) == -2          # ref out of range
    assert status_of(sel, [0, 11], [1.0, 2.0], 10, 0.1, 0) == -2         # V > n
    assert status_of(sel, [0, -1], [1.0, 2.0], 10, 0.1, 0) == -2         # V < 0
    assert status_of(sel, [], [], 10, 0.1, 0) == -2                       # m = 0
    assert status_of(sel, [0, 1], [1.0, float("nan")], 10, 0.1, 0) == -10
    assert status_of(sel, [0, 1], [1.0, float("inf")], 10, 0.1, 0) == -10
    assert status_of(sel, [0, 1], [1.0, 2.0], 10, float("nan"), 0) == -10
    assert status_of(sel, [0, 1], [1.0, 2.0], 10, 0.1, 0, delta=0.0) == -10
    assert status_of(sel, [0, 1], [1.0, 2.0], 10, 0.1, 0, delta=1.5) == -10
    assert status_of(sel, [0, 1], [1.0, 2.0], 10, 0.1, 0, procedure=7) == -10
    assert status_of(sel, [0, 1], [1.0, 2.0], 10, 0.1, 0, procedure="fixed_sequence") == -1
    assert status_of(sel, [0, 1], [1.0, 2.0], 10, 0.1, 0, procedure="fixed_sequence", order=[0, 0]) == -10
    assert status_of(sel, [0, 1], [1.0, 2.0], 10, 0.1, 0, procedure="fixed_sequence", order=[0, 2]) == -10
    assert status_of(N.bd_redline_test, [0.1, float("nan")], 0.1) == -10
    assert status_of(N.bd_redline_pvalues, [0, 3], 2, 0.1) == -2
    assert status_of(N.bd_redline_violations, np.ones((4, 3), np.uint8), 3) == -2
    assert status_of(N.bd_redline_sweep, [0, 1], [1.0, 2.0], 10, [0.1, 2.0], 0) == -10
    assert status_of(N.bd_redline_tpf, np.array([[1, -1]], np.int32), 2) == -10
    assert status_of(N.bd_redline_tpf, np.array([[1, 1]], np.int32), 0) == -2
    assert status_of(N.bd_redline_deploy, [1, 0], [1.0, float("nan")], 0) == -10
    lib = B.load_library()
    N._L()
    assert lib.bd_binom_cdf(1, 2, 0.5, None) == -1
    assert lib.bd_redline_select(None, 0.1, None, None, None, None) == -1
    out = ctypes.c_int64(-7)
    assert lib.bd_redline_critical_count(10, 0.1, 0.1, None) == -1
    assert lib.bd_redline_critical_count(-3, 0.1, 0.1, ctypes.byref(out)) == -2 and out.value == -7  # untouched


def test_degenerate_grids():
    # n = 0: every p-value is 1; only delta = 1 with one hypothesis rejects
    got = N.bd_redline_select([0, 0], [1.0, 2.0], 0, 0.1, 0)
    assert list(got["p"]) == [1.0, 1.0] and not got["valid"].any() and got["deployed"] == 0
    got = N.bd_redline_select([0], [1.0], 0, 0.1, 0, delta=1.0)
    assert list(got["valid"]) == [True] and got["deployed"] == 0
    # the reference alone
    got = N.bd_redline_select([0], [4.4], 1012, 0.05, 0)
    assert got["valid"][0] and got["deployed"] == 0
    # no prompts in the outcome matrix
    assert list(N.bd_redline_violations(np.zeros((0, 3), np.uint8), 1)) == [0, 0, 0]
    # alpha at 0 and 1
    assert list(N.bd_redline_pvalues([0, 3], 10, 0.0)) == [1.0, 1.0]
    assert list(N.bd_redline_pvalues([0, 3, 10], 10, 1.0)) == [0.0, 0.0, 1.0]
    # no budgets
    s = N.bd_redline_sweep([0, 1], [1.0, 2.0], 10, [], 0)
    assert s["deployed"].size == 0 and s["first_gain"] == -1


def test_tpf_parity():
    rng = np.random.default_rng(4)
    counts = rng.integers(0, 200, size=(37, 9)).astype(np.int32)
    got = N.bd_redline_tpf(counts, 8)
    want = R.tpf_from_counts(counts.tolist(), 8)
    assert all(abs(g - float(w)) <= 1e-15 * float(w) for g, w in zip(got, want))
    assert list(N.bd_redline_tpf(np.zeros((0, 3), np.int32), 4)) == [0.0, 0.0, 0.0]


# --------------------------------------------------------------------------
# family-wise error through the native path
# --------------------------------------------------------------------------
def test_montecarlo_fwer_native():
    """The synthetic Monte Carlo of the validity appendix (five configurations
    of true risk {0.01, 0.02, 0.07, 0.07, 0.07}, alpha = 0.05, n = 800, 4,000
    trials): Holm on the shared draw, Bonferroni and fixed sequence on
    independent draws. The exact FWERs are 1.6e-5 (Holm, shared draw) and
    about 1.3e-4 (fixed sequence walking in risk order), so a handful of
    errors at most in 4,000 trials."""
    risks = [0.01, 0.02, 0.07, 0.07, 0.07]
    bad = {"holm": 0, "bonferroni": 0, "fixed_sequence": 0}
    for t in range(4000):
        for j, (proc, shared) in enumerate((("holm", True), ("bonferroni", False), ("fixed_sequence", False))):
            L = losses_matrix(800, risks, shared=shared, seed=3 * t + j)
            V = N.bd_redline_violations(L, 0)[1:]
            valid = N.bd_redline_test(N.bd_redline_pvalues(V, 800, 0.05), 0.10, proc,
                                      [0, 1, 2, 3, 4] if proc == "fixed_sequence" else None)
            bad[proc] += bool(valid[2:].any())
    assert bad["holm"] <= 3 and bad["bonferroni"] <= 3 and bad["fixed_sequence"] <= 5, bad


def test_montecarlo_near_boundary_native():
    """Nulls just above the budget (true risks {0.02, 0.055, 0.055}, alpha =
    0.05, n = 400): the simulated FWER of Holm matches the exact nested-count
    value within 4 standard errors, and stays under delta."""
    risks = [F("0.02"), F("0.055"), F("0.055")]
    exact = exact_holm_fwer_nested(400, F("0.05"), F("0.10"), risks)
    trials, bad = 20000, 0
    for t in range(trials):
        L = losses_matrix(400, [float(r) for r in risks], shared=True, seed=500000 + t)
        V = N.bd_redline_violations(L, 0)[1:]
        valid = N.bd_redline_test(N.bd_redline_pvalues(V, 400, 0.05), 0.10, "holm")
        bad += bool(valid[1] or valid[2])
    se = math.sqrt(exact * (1 - exact) / trials)
    assert abs(bad / trials - exact) < 4 * se, (bad / trials, exact)
    assert bad / trials < 0.10
