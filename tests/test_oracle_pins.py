"""Pins of the float64 oracle against things other than itself.

Each test fixes the oracle to a closed form, an exhaustive 50-digit brute
force, a library routine for a special case, a hand-derived case, or an
invariant of the rule, chosen so that a dropped term, a wrong sign, a wrong
index, a transposed operand or a flipped comparison fails at least one test.
"""

import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle.commit_oracle import hidden_f64

HERE = os.path.dirname(os.path.abspath(__file__))


# ---------------------------------------------------------------- formats --

def test_bf16_decode_matches_torch_on_every_pattern():
    codes = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = oracle.decode_bf16(codes)
    ref = torch.from_numpy(codes.view(np.int16).copy()).view(torch.bfloat16).float().double().numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])


def test_e4m3_decode_matches_torch_on_every_code():
    codes = np.arange(256, dtype=np.uint8)
    ours = oracle.decode_e4m3(codes)
    ref = torch.from_numpy(codes.copy()).view(torch.float8_e4m3fn).float().double().numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])


def test_e4m3_spot_values_from_the_format_definition():
    dec = lambda c: float(oracle.decode_e4m3(np.array([c], dtype=np.uint8))[0])
    assert dec(0x38) == 1.0  # exponent field 7 = bias
    assert dec(0xB8) == -1.0
    assert dec(0x7E) == 448.0  # largest finite: 1.75 * 2^8
    assert dec(0x08) == 2.0 ** -6  # smallest normal
    assert dec(0x01) == 2.0 ** -9  # smallest subnormal
    assert dec(0x00) == 0.0
    assert math.isnan(dec(0x7F)) and math.isnan(dec(0xFF))


def test_e4m3_weights_apply_the_row_scale():
    codes = np.array([[0x38, 0x40], [0x38, 0xB8]], dtype=np.uint8)  # 1, 2 / 1, -1
    scale = np.array([0.5, 3.0], dtype=np.float32)
    w = oracle.weights_f64(codes, "e4m3", scale)
    assert np.array_equal(w, np.array([[0.5, 1.0], [3.0, -3.0]]))


def test_e4m3_weights_equal_the_elementwise_decode_times_the_row_scale():
    # every code (NaN codes included) in random rows against the format's
    # decode applied element by element, times the row scale
    rng = np.random.default_rng(3)
    codes = rng.integers(0, 256, size=(300, 77), dtype=np.uint8)
    codes[0, :] = np.arange(77, dtype=np.uint8) + 179  # the top codes, 0xFF (NaN) among them
    scale = rng.uniform(1e-4, 3.0, size=300).astype(np.float32)
    w = oracle.weights_f64(codes, "e4m3", scale)
    ref = oracle.decode_e4m3(codes) * scale.astype(np.float64)[:, None]
    nan = np.isnan(ref)
    assert nan.any() and np.array_equal(np.isnan(w), nan)
    assert np.array_equal(w[~nan], ref[~nan])


# ----------------------------------------------------------- closed forms --

def _planted_head(V, d, v_star, k_star):
    w = np.zeros((V, d), dtype=np.float32)
    w[v_star, k_star] = 1.0
    return w


@pytest.mark.parametrize("b", [0.5, 3.0, 8.25, 20.0, 40.0])
@pytest.mark.parametrize("mask_id", [-1, 0, 36])
def test_single_planted_logit_closed_form(b, mask_id):
    # One head row v* = 11 is e_2 and every other row is zero, and h = b * e_2:
    # logit v* is b and every other logit is 0, so the mask-suppressed softmax
    # gives conf = 1 / (1 + (V' - 1) e^{-b}), V' = V minus the suppressed id.
    V, d, v_star = 37, 5, 11
    w = _planted_head(V, d, v_star, 2)
    h = np.zeros((1, d))
    h[0, 2] = b
    logits = oracle.lm_head_logits(h, w, "f32")
    tok, conf, gap = oracle.row_confidence(logits[0], mask_id)
    Vp = V - (1 if 0 <= mask_id < V else 0)
    expect = 1.0 / (1.0 + (Vp - 1) * math.exp(-b))
    assert tok == v_star
    assert abs(conf - expect) <= 1e-15 * expect
    assert gap == pytest.approx(b, rel=1e-15)


def test_planted_logit_on_the_mask_token_is_suppressed():
    # The planted entry is the mask token itself: it is removed, every other
    # logit is 0, so conf = 1/(V-1) and the token is the lowest other index.
    V, d, v_star = 37, 5, 11
    w = _planted_head(V, d, v_star, 2)
    h = np.array([[0, 0, 30.0, 0, 0]])
    tok, conf, gap = oracle.row_confidence(oracle.lm_head_logits(h, w, "f32")[0], v_star)
    assert tok == 0
    assert conf == pytest.approx(1.0 / (V - 1), rel=1e-15)
    assert gap == 0.0


@pytest.mark.parametrize("mask_id,token", [(-1, 0), (0, 1), (5, 0)])
def test_zero_hidden_gives_uniform_confidence(mask_id, token):
    V, d = 64, 8
    rng = np.random.default_rng(0)
    w = rng.standard_normal((V, d)).astype(np.float32)
    tok, conf, gap = oracle.row_confidence(oracle.lm_head_logits(np.zeros((1, d)), w, "f32")[0], mask_id)
    Vp = V - (1 if mask_id >= 0 else 0)
    assert tok == token
    assert conf == pytest.approx(1.0 / Vp, rel=1e-15)
    assert gap == 0.0


def test_head_orientation_is_vocab_by_hidden():
    # A [V, d] head with distinct rows: the token must be the row most aligned
    # with h. Reading the head as [d, V] (a transposed operand) cannot even run.
    V, d = 9, 4
    w = np.zeros((V, d), dtype=np.float32)
    for v in range(V):
        w[v, v % d] = 1.0 + v  # row v points along axis v % d with length 1 + v
    h = np.array([[0.0, 0.0, 1.0, 0.0]])
    tok, _, _ = oracle.row_confidence(oracle.lm_head_logits(h, w, "f32")[0])
    assert tok == 6  # rows 2 and 6 point along axis 2; row 6 is longer
    with pytest.raises(ValueError):
        oracle.lm_head_logits(h, w.T.copy(), "f32")


# ------------------------------------------------------------ brute force --

def test_brute_force_50_digits_on_small_integer_problems():
    mp = pytest.importorskip("mpmath")
    mp.mp.dps = 50
    rng = np.random.default_rng(1234)
    for trial in range(300):
        V = int(rng.integers(1, 17))
        d = int(rng.integers(1, 9))
        w = rng.integers(-3, 4, size=(V, d)).astype(np.float32)
        h = rng.integers(-3, 4, size=(1, d)).astype(np.float64)
        mask_id = int(rng.integers(-1, V)) if V > 1 else -1
        # exact integer logits, summed term by term
        ex = [sum(int(h[0, k]) * int(w[v, k]) for k in range(d)) for v in range(V)]
        keep = [v for v in range(V) if v != mask_id]
        M = max(ex[v] for v in keep)
        tok_exact = min(v for v in keep if ex[v] == M)
        s = mp.fsum(mp.exp(ex[v] - M) for v in keep)
        conf_exact = 1 / s
        tok, conf, _ = oracle.row_confidence(oracle.lm_head_logits(h, w, "f32")[0], mask_id)
        assert tok == tok_exact, (trial, ex, mask_id)
        assert abs(conf - float(conf_exact)) < 1e-12, trial


def test_logsumexp_cross_check_on_tiny_workload():
    sp = pytest.importorskip("scipy.special")
    from workloads import generate, TINY_F32
    from tests.helpers import raw_numpy

    wl = generate(TINY_F32)
    h = hidden_f64(raw_numpy(wl.hidden), "f32")
    w = raw_numpy(wl.weight).astype(np.float64)
    for p in range(wl.P):
        l = w @ h[p]  # independent: a matrix-vector product, then logsumexp
        conf_lse = math.exp(l.max() - sp.logsumexp(l))
        tok, conf, _ = oracle.row_confidence(oracle.lm_head_logits(h[p:p + 1], raw_numpy(wl.weight), "f32")[0])
        assert tok == int(np.argmax(l))
        assert abs(conf - conf_lse) < 1e-12


# ------------------------------------------------------- commit rule cases --

def _golden_cases():
    with open(os.path.join(HERE, "golden", "commit_rule_cases.json")) as f:
        return json.load(f)["cases"]


@pytest.mark.parametrize("case", _golden_cases(), ids=lambda c: c["name"])
def test_commit_rule_hand_derived(case):
    bits = oracle.commit_block(case["conf"], case["masked"], case["active"], case["eligible"], case["taus"])
    assert [int(b) for b in bits] == case["expected"], case["why"]


# ------------------------------------------------------------- invariants --

def _small_random_step(seed, fallback="oldest", T=6, mask_id=-1, active="all"):
    from workloads import WorkloadConfig, generate
    from tests.helpers import oracle_on_workload

    cfg = WorkloadConfig(name="inv", n_seq=3, n_slots=3, block_len=8, mask_frac=0.5,
                         d=16, V=50, hidden_dtype="f32", weight_dtype="f32",
                         boost="single", boost_frac=0.5, boost_lo=0.0, boost_hi=8.0,
                         tau=tuple(np.linspace(0.0, 1.2, T)), seed=seed,
                         mask_token_id=mask_id, fallback=fallback, active=active)
    wl = generate(cfg)
    return wl, oracle_on_workload(wl)


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("fallback", ["oldest", "all", "none"])
def test_commit_invariants(seed, fallback):
    wl, out = _small_random_step(seed, fallback=fallback, active="first_half" if seed % 2 else "all")
    cfg = wl.cfg
    L = cfg.block_len
    flags = wl.block_flags.numpy()
    masked = wl.pos_masked.numpy().astype(bool)
    active_pos = np.repeat((flags & oracle.ACTIVE) != 0, L)
    elig = np.repeat((flags & oracle.FALLBACK_ELIGIBLE) != 0, L)
    live = masked & active_pos
    conf, commit, tokens = out["conf"], out["commit"], out["tokens"]
    taus = [float(np.float32(t)) for t in wl.tau]
    # confidences lie in (0, 1] exactly where a prediction is made
    assert np.all((conf[live] > 0) & (conf[live] <= 1))
    assert np.all(conf[~live] == 0) and np.all(tokens[~live] == -1)
    assert np.all((tokens[live] >= 0) & (tokens[live] < cfg.V))
    # commits are a subset of masked positions of active blocks
    assert np.all(commit[~live] == 0)
    # tau = 0 commits every such position
    assert taus[0] == 0.0
    assert np.array_equal((commit & 1) != 0, live)
    # tau > 1 leaves only the fallback: one position per eligible block with masks
    top = len(taus) - 1
    assert taus[top] > 1.0
    hit = ((commit >> np.uint32(top)) & 1).reshape(-1, L)
    for blk in range(cfg.n_blocks):
        expect = int(elig[blk * L] and live[blk * L:(blk + 1) * L].any())
        assert int(hit[blk].sum()) == expect
        if expect:
            j = int(np.argmax(hit[blk]))
            cb = conf[blk * L:(blk + 1) * L]
            assert cb[j] == cb[live[blk * L:(blk + 1) * L]].max()
    # commit sets shrink as tau grows
    for k in range(1, len(taus)):
        lo = (commit >> np.uint32(k - 1)) & 1
        hi = (commit >> np.uint32(k)) & 1
        assert np.all(hi <= lo)
    # per-sequence counts are the popcounts of the bits
    for s in range(cfg.n_seq):
        seg = commit[s * cfg.n_slots * L:(s + 1) * cfg.n_slots * L]
        for k in range(len(taus)):
            assert out["counts"][s, k] == int(np.count_nonzero((seg >> np.uint32(k)) & 1))


def test_vocab_permutation_permutes_tokens_only():
    rng = np.random.default_rng(7)
    V, d = 40, 6
    w = rng.standard_normal((V, d)).astype(np.float32)
    h = rng.standard_normal((5, d))
    perm = rng.permutation(V)
    base = oracle.lm_head_logits(h, w, "f32")
    moved = oracle.lm_head_logits(h, w[perm], "f32")
    inv = np.argsort(perm)
    for i in range(h.shape[0]):
        t0, c0, _ = oracle.row_confidence(base[i])
        t1, c1, _ = oracle.row_confidence(moved[i])
        assert inv[t0] == t1
        assert c1 == pytest.approx(c0, rel=1e-13)


def test_sampled_blocks_match_full_evaluation():
    wl, full = _small_random_step(11)
    from tests.helpers import oracle_on_workload

    part = oracle_on_workload(wl, blocks=[1, 4, 7])
    ev = part["evaluated"]
    assert ev.sum() == 3 * wl.cfg.block_len
    for key in ("tokens", "conf", "commit"):
        assert np.array_equal(part[key][ev], full[key][ev])


# ---------------------------------------------------- the merge operator --

def _partial(l, lo):
    """(max, sum of exp(l - max), lowest argmax) of one chunk starting at index lo."""
    m = float(np.max(l))
    if m == -math.inf:
        return (-math.inf, 0.0, 1 << 30)
    return (m, float(np.sum(np.exp(l - m))), lo + int(np.flatnonzero(l == m)[0]))


def _combine(x, y):
    """The merge rule the CUDA kernels apply across CTAs, restated: the larger
    max wins and the other sum is rescaled to it; equal maxima add their sums
    and keep the lower index."""
    (m1, s1, a1), (m2, s2, a2) = x, y
    if m2 > m1:
        return (m2, s2 + (s1 * math.exp(m1 - m2) if m1 > -math.inf else 0.0), a2)
    if m2 == m1:
        return (m1, s1 + s2 if m1 > -math.inf else 0.0, min(a1, a2))
    return (m1, s1 + (s2 * math.exp(m2 - m1) if m2 > -math.inf else 0.0), a1)


@pytest.mark.parametrize("seed", range(6))
def test_chunked_merge_equals_the_single_pass(seed):
    """Splitting the vocabulary into any number of chunks (uneven, some holding
    only the suppressed entry) and merging their partials in any order and
    grouping gives the oracle's single-pass token and confidence: the merge is
    associative and commutative and keeps the lowest index on equal maxima.
    Small integer logits make ties across chunks frequent."""
    rng = np.random.default_rng(seed)
    for _ in range(40):
        V = int(rng.integers(2, 60))
        l = rng.integers(-3, 4, size=V).astype(np.float64)
        mask = int(rng.integers(-1, V))
        token, conf, _ = oracle.commit_oracle.row_confidence(l, mask)
        lm = l.copy()
        if mask >= 0:
            lm[mask] = -np.inf
        k = int(rng.integers(1, V + 1))
        cuts = np.sort(rng.choice(np.arange(1, V), size=min(k - 1, V - 1), replace=False)) if V > 1 else []
        bounds = [0, *[int(c) for c in cuts], V]
        parts = [_partial(lm[a:b], a) for a, b in zip(bounds[:-1], bounds[1:])]
        order = rng.permutation(len(parts))
        # a random binary tree over the shuffled partials
        pool = [parts[i] for i in order]
        while len(pool) > 1:
            i = int(rng.integers(0, len(pool) - 1))
            pool[i:i + 2] = [_combine(pool[i], pool[i + 1])]
        m, s, a = pool[0]
        assert a == token
        assert abs(1.0 / s - conf) < 1e-12
