"""Helpers shared by the Redline tests."""

from __future__ import annotations

import math

from oracle import redline_oracle as R


def exact_holm_fwer_nested(n, alpha, delta, risks):
    """FWER of Holm when every configuration's losses come from one shared
    uniform per prompt (risks sorted ascending, one per hypothesis of the
    family). The counts are nested, V_0 <= V_1 <= ..., so the sorted p-values
    follow the risk order, and Holm rejects a hypothesis with R > alpha only
    if it rejects the first of them, at sorted position f: that needs
    V_i <= c_i for every i <= f, with c_i the critical count at
    delta / (m - i). The V_i are prefix sums of multinomial cell counts of the
    uniform over [0, r_0), [r_0, r_1), ..., [r_{f-1}, r_f) and [r_f, 1)."""
    m = len(risks)
    assert list(risks) == sorted(risks)
    tab = R.binom_cdf_table(n, alpha, n)
    crit = [max([v for v in range(n + 1) if tab[v] <= delta / (m - i)], default=-1) for i in range(m)]
    f = next(i for i, r in enumerate(risks) if r > alpha)
    widths = [float(risks[0])] + [float(risks[i] - risks[i - 1]) for i in range(1, f + 1)]
    rest = 1.0 - float(risks[f])
    lg = math.lgamma
    total = 0.0

    def rec(i, used, logp):
        nonlocal total
        if i > f:
            r = n - used
            total += math.exp(lg(n + 1) + logp - lg(r + 1) + r * math.log(rest))
            return
        top = crit[i] - used if widths[i] > 0 else min(0, crit[i] - used)
        for c in range(0, top + 1):
            rec(i + 1, used + c, logp + (c * math.log(widths[i]) if c else 0.0) - lg(c + 1))

    rec(0, 0, 0.0)
    return total
