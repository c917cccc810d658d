"""Pins of the speculative-verification oracle (no GPU).

* closed forms: a uniform target (H = log V, every eps < 1 accepts, eps = 1
  does not, the rule being strict); one planted logit (p and H in closed form);
* a 50-digit brute force of p and H on small random rows;
* properties that follow from the rule: acceptance is nested in eps (a lower
  eps accepts more, as the typical-acceptance appendix says), and the target's
  argmax is always accepted for eps < 1 (e^{-H} <= p_max), so the lossless
  reference accepts a subset;
* the paper's lossless figures under per-token draft agreement a with four
  draft tokens: 1 + sum_{i=1..4} a^i gives 4.14 at a = 0.905 (Llama pair) and
  3.99 at a = 0.887 (Qwen pair), and the oracle on seeded drafts with that
  agreement reproduces the expectation.
"""

from __future__ import annotations

import math

import numpy as np
import pytest

from oracle import verify_oracle as VO
from workloads.rawio import dtype_tag, raw_numpy
from workloads.verify_inputs import generate_verify, SPEC_LLAMA8B, verify_scaled

mpmath = pytest.importorskip("mpmath")


def run(wl):
    c = wl.cfg
    return VO.verify_step(raw_numpy(wl.hidden), dtype_tag(wl.hidden), raw_numpy(wl.weight), dtype_tag(wl.weight),
                          None if wl.weight_scale is None else raw_numpy(wl.weight_scale),
                          wl.draft.numpy(), c.n_req, c.n_draft, c.eps)


def test_uniform_target():
    V = 1000
    tok, p, H, gap = VO.row_stats(np.zeros(V))
    assert tok == 0 and gap == 0.0
    assert abs(H - math.log(V)) < 1e-12 and np.allclose(p, 1.0 / V)
    for eps in (0.8, 0.5, 0.1, 0.02):
        assert VO.accepts(p[17], H, eps)  # sqrt(eps)/V < 1/V
    assert not VO.accepts(p[17], H, 1.0)   # threshold min(1, 1/V) = p: strict inequality
    # a certain target at eps = 1: p = 1, H = 0, threshold min(1, e^0) = 1 exactly, so the strict rule rejects
    tok, p, H, _ = VO.row_stats(np.array([0.0, -np.inf, -np.inf]))
    assert p[0] == 1.0 and H == 0.0 and not VO.accepts(p[0], H, 1.0) and VO.accepts(p[0], H, 0.999)


def test_hand_case_both_branches_of_the_min():
    """p = (0.6, 0.25, 0.15): H = 0.9377 nats, e^{-H} = 0.3915.
    eps = 0.25: threshold min(0.25, 0.5 * 0.3915 = 0.1958) = 0.1958, so the
    draft of probability 0.25 passes and the one of 0.15 does not (with the
    coefficient a = eps instead of sqrt(eps) it would: 0.25 * 0.3915 = 0.0979).
    eps = 0.04: threshold min(0.04, 0.2 * 0.3915 = 0.0783) = 0.04, so 0.15 passes."""
    tok, p, H, _ = VO.row_stats(np.log(np.array([0.6, 0.25, 0.15])))
    assert tok == 0 and abs(H - 0.93770) < 1e-4
    assert VO.accepts(p[1], H, 0.25) and not VO.accepts(p[2], H, 0.25)
    assert VO.accepts(p[2], H, 0.04)
    assert VO.accepts(p[0], H, 0.8) and not VO.accepts(p[2], H, 0.8)


@pytest.mark.parametrize("b", [0.5, 3.0, 9.0, 20.0])
def test_one_planted_logit(b):
    V = 5000
    l = np.zeros(V)
    l[123] = b
    tok, p, H, gap = VO.row_stats(l)
    Z = 1 + (V - 1) * math.exp(-b)
    assert tok == 123 and abs(gap - b) < 1e-12
    assert abs(p[123] - 1 / Z) < 1e-13 and abs(p[0] - math.exp(-b) / Z) < 1e-15
    assert abs(H - (math.log(Z) + (V - 1) * b * math.exp(-b) / Z)) < 1e-10


def test_brute_force_50_digits():
    rng = np.random.default_rng(3)
    mpmath.mp.dps = 50
    for _ in range(200):
        V = int(rng.integers(2, 40))
        l = rng.normal(0, 3, size=V)
        tok, p, H, _ = VO.row_stats(l)
        ls = [mpmath.mpf(float(x)) for x in l]
        Z = mpmath.fsum(mpmath.e ** x for x in ls)
        ps = [mpmath.e ** x / Z for x in ls]
        Hs = -mpmath.fsum(q * mpmath.log(q) for q in ps)
        assert abs(H - float(Hs)) < 1e-12
        assert max(abs(p[i] - float(ps[i])) for i in range(V)) < 1e-14
        assert tok == int(np.argmax(l))


@pytest.fixture(scope="module")
def small():
    cfg = verify_scaled(SPEC_LLAMA8B, n_req=40, n_draft=6, d=96, V=3000, boost_lo=2.0, boost_hi=14.0,
                        agree=0.7, seed=5)
    wl = generate_verify(cfg)
    return wl, run(wl)


def test_nested_and_lossless_inside_typical(small):
    wl, r = small
    c = wl.cfg
    order = np.argsort(r["eps"])[::-1]  # from the strictest eps (largest) to the most lenient
    E = len(c.eps)
    for row in range(c.rows):
        bits = int(r["accept"][row])
        acc = [(bits >> int(k)) & 1 for k in order]
        assert acc == sorted(acc)  # once accepted at some eps, accepted at every smaller eps
        if (bits >> VO.LOSSLESS_BIT) & 1:
            assert all((bits >> k) & 1 for k in range(E) if r["eps"][k] < 1.0)
    # accepted prefixes follow the same nesting
    for q in range(c.n_req):
        lens = r["accepted"][q, order]
        assert list(lens) == sorted(lens)
        assert all(r["accepted"][q, E] <= r["accepted"][q, k] for k in range(E) if r["eps"][k] < 1.0)


def test_structure_of_the_outputs(small):
    wl, r = small
    c = wl.cfg
    D, E = c.n_draft, len(c.eps)
    acc = r["accept"].reshape(c.n_req, D + 1)
    assert np.all(acc[:, D] == 0) and np.all(r["p_draft"].reshape(c.n_req, D + 1)[:, D] == 0)
    for k in range(E + 1):
        bit = VO.LOSSLESS_BIT if k == E else k
        ok = ((acc[:, :D] >> np.uint32(bit)) & 1).astype(bool)
        lead = np.where(ok.all(axis=1), D, np.argmin(ok, axis=1))
        assert np.array_equal(r["accepted"][:, k], lead)
    # the lossless rule: accepted exactly where the draft is the argmax
    d = wl.draft.numpy().reshape(c.n_req, D)
    t = r["tokens"].reshape(c.n_req, D + 1)[:, :D]
    assert np.array_equal(((acc[:, :D] >> np.uint32(31)) & 1).astype(bool), d == t)


def test_paper_lossless_figures_from_agreement():
    """Accepted tokens per target forward under i.i.d. agreement a with four
    drafts: 1 + a + a^2 + a^3 + a^4, printed as 4.14 (a = 0.905) and 3.99 (a = 0.887)."""
    assert round(1 + sum(0.905**i for i in range(1, 5)), 2) == 4.14
    assert round(1 + sum(0.887**i for i in range(1, 5)), 2) == 3.99
    for a in (0.905, 0.887):
        cfg = verify_scaled(SPEC_LLAMA8B, n_req=3000, n_draft=4, d=64, V=256, boost_lo=10.0, boost_hi=18.0,
                            agree=a, eps=(0.1,), hidden_dtype="f32", weight_dtype="f32", seed=21)
        wl = generate_verify(cfg)
        r = run(wl)
        # the planted entries are the argmax: the drafts agree at rate a by construction
        assert np.array_equal(r["tokens"], wl.planted.numpy())
        tpf = VO.tokens_per_forward(r["accepted"])[-1]
        want = 1 + sum(a**i for i in range(1, 5))
        lens = r["accepted"][:, -1]
        se = lens.std() / math.sqrt(lens.size)
        assert abs(tpf - want) < 4 * se, (tpf, want)
