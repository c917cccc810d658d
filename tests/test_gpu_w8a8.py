"""The W8A8 variant of the precision lever (E4M3 head x E4M3 activations on
the 8-bit tensor path, tcgen05.mma kind::f8f6f4) against the oracle.

Parity: the oracle quantises every hidden row with its own per-row E4M3
quantiser (oracle.quantize_rows_e4m3) and runs the float64 commit step on the
dequantised activations; the kernel must match it within the E4M3 head's
tolerances (the products of two E4M3 values are exact in fp32, so the GPU
differs from the oracle only by fp32 accumulation and softmax rounding).

Deviation: the same step against the oracle on the unquantised bf16
activations, i.e. what the 8-bit activations cost; the bounds asserted here
are the measured deviation with margin, not a parity tolerance.
"""

import numpy as np
import pytest
import torch

from tests.helpers import oracle_on_workload, raw_numpy
from tests.parity import compare
from workloads import B256X8X64_E4M3, B8X2X32_BF16, generate, scaled
from workloads.configs import by_name

pytestmark = pytest.mark.gpu

bdc = pytest.importorskip("paper_2609_33887_gb300")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__

    __graft_entry__.build()
    torch.cuda.set_device(0)
    yield


def run_w8a8(wl, variant=0):
    cfg = wl.cfg
    g = wl.to("cuda")
    tokens, conf, commit, counts = bdc.commit_step(
        g.hidden, g.weight, g.pos_masked, g.block_flags, cfg.n_seq, cfg.n_slots, cfg.block_len, wl.tau,
        weight_scale=g.weight_scale, mask_token_id=wl.mask_token_id, counts=True, variant=variant,
        fp8_activations=True)
    torch.cuda.synchronize()
    st = bdc.bd_get_device_status()
    assert st == 0, bdc.bd_status_string(st)
    return {"tokens": tokens.cpu().numpy(), "conf": conf.cpu().numpy(),
            "commit": commit.cpu().numpy().view(np.uint32), "counts": counts.cpu().numpy()}


def oracle_w8a8(wl, blocks=None):
    """The oracle on the activations the W8A8 head multiplies."""
    import oracle
    from oracle import commit_oracle as C

    cfg = wl.cfg
    h32 = wl.hidden.float().numpy()  # bf16 values, exact in float32
    codes, scale = C.quantize_rows_e4m3(h32)
    hq = C.dequantize_rows_e4m3(codes, scale)
    return oracle.commit_step(hq, "f64", raw_numpy(wl.weight), "e4m3", raw_numpy(wl.weight_scale),
                              raw_numpy(wl.pos_masked), raw_numpy(wl.block_flags), cfg.n_seq, cfg.n_slots,
                              cfg.block_len, wl.mask_token_id, wl.tau, blocks=blocks)


def check(wl, out=None, blocks=None):
    out = run_w8a8(wl) if out is None else out
    ref = oracle_w8a8(wl, blocks=blocks)
    rep = compare(out, ref, wl.tau, "e4m3", wl.cfg.block_len, wl.cfg.n_slots)
    assert rep.ok(), rep.failures
    return out, rep


SMALL = {
    # one token group, ragged last vocabulary tile
    "e4m3_g64": scaled(B256X8X64_E4M3, n_seq=4, n_slots=4, block_len=8, d=512, V=5000),
    # two token groups (257..320 rows), width with a K tail of 80 columns
    "e4m3_g294_ktail": scaled(B8X2X32_BF16, weight_dtype="e4m3", d=336, V=3000, mask_frac=0.6),
    # narrow rows (one partial 128-column stage), mask token in the last tile
    "e4m3_d48_mask": scaled(B256X8X64_E4M3, n_seq=3, n_slots=2, block_len=16, d=48, V=700, mask_token_id=699),
}


@pytest.mark.parametrize("name", sorted(SMALL))
def test_w8a8_small(name):
    _, rep = check(generate(SMALL[name]))
    assert rep.n_live > 0


def test_w8a8_zero_rows():
    """All-zero hidden rows quantise to scale 0: their logits are 0 and the
    confidence is uniform over the live vocabulary."""
    wl = generate(SMALL["e4m3_g64"])
    wl.hidden[::3] = 0
    out, _ = check(wl)
    live = out["tokens"][::3] >= 0
    V_live = wl.cfg.V - (1 if wl.mask_token_id >= 0 else 0)
    assert np.allclose(out["conf"][::3][live], 1.0 / V_live, rtol=1e-3)


def test_w8a8_needs_e4m3_pair_head():
    wl = generate(scaled(B8X2X32_BF16, d=256, V=1000))  # bf16 head
    g = wl.to("cuda")
    c = wl.cfg
    with pytest.raises(bdc.BdError):
        bdc.commit_step(g.hidden, g.weight, g.pos_masked, g.block_flags, c.n_seq, c.n_slots, c.block_len, wl.tau,
                        fp8_activations=True)
    wl = generate(SMALL["e4m3_g64"])
    g = wl.to("cuda")
    c = wl.cfg
    with pytest.raises(bdc.BdError):  # the one-CTA kernel has no W8A8 instantiation
        bdc.commit_step(g.hidden, g.weight, g.pos_masked, g.block_flags, c.n_seq, c.n_slots, c.block_len, wl.tau,
                        weight_scale=g.weight_scale, variant=2, fp8_activations=True)


def test_w8a8_full_window_and_deviation():
    """The bench window with an E4M3 head (8 x 2 x 32, d = 2048, V = 151936):
    parity on every position, then the deviation from the exact oracle on the
    bf16 activations."""
    wl = generate(by_name("b8x2x32_d2048_v151936_e4m3"))
    out, rep = check(wl)
    exact = oracle_on_workload(wl)
    live = exact["tokens"] >= 0
    agree = float(np.mean(out["tokens"][live] == exact["tokens"][live]))
    dconf = float(np.max(np.abs(out["conf"][live] - exact["conf"][live])))
    print(f"W8A8 vs exact: token agreement {agree:.4f}, max |dconf| {dconf:.4f}, live {int(live.sum())}")
    assert agree >= 0.97
    assert dconf <= 0.1


def test_w8a8_row_magnitudes_across_the_bf16_range():
    """Per-row scales from 2^-90 to 2^90 times the generated rows (exact in bf16)."""
    wl = generate(SMALL["e4m3_g294_ktail"])
    exps = (-90, -40, -12, 0, 12, 40, 90)
    k = torch.tensor(exps, dtype=torch.float64)[torch.arange(wl.hidden.shape[0]) % len(exps)]
    wl.hidden = (wl.hidden.double() * torch.exp2(k)[:, None]).to(wl.hidden.dtype)
    _, rep = check(wl)
    assert rep.n_live > 0


def test_w8a8_lossless_rows_match_the_exact_step():
    """Rows the per-row quantiser reproduces exactly (E4M3 values times 2^k,
    largest magnitude 448 * 2^k): the W8A8 step must match the exact oracle on
    the bf16 rows themselves."""
    from oracle import commit_oracle as C

    wl = generate(SMALL["e4m3_g294_ktail"])
    rng = np.random.default_rng(21)
    finite = C.decode_e4m3(np.arange(256))
    finite = finite[np.isfinite(finite)]
    P, d = wl.hidden.shape
    h = rng.choice(finite, size=(P, d)) * 2.0 ** -6
    h[:, 0] = np.where(rng.random(P) < 0.5, 448.0, -448.0) * 2.0 ** -6
    k = rng.integers(-8, 3, size=P).astype(np.float64)
    wl.hidden = torch.from_numpy(h * np.exp2(k)[:, None]).to(torch.bfloat16)
    assert np.array_equal(wl.hidden.double().numpy(), h * np.exp2(k)[:, None])  # exact in bf16
    out = run_w8a8(wl)
    rep = compare(out, oracle_on_workload(wl), wl.tau, "e4m3", wl.cfg.block_len, wl.cfg.n_slots)
    assert rep.ok(), rep.failures
    assert rep.n_live > 0


def test_w8a8_largest_window_sampled_blocks():
    """The largest window (256 x 8 x 64, d = 5120, more than 8192 positions:
    205 token groups of 256, several bands of the plan) with W8A8, on sampled
    whole blocks including those of the first and last compacted rows."""
    wl = generate(B256X8X64_E4M3)
    cfg = wl.cfg
    act = np.repeat((wl.block_flags.numpy() & 1) != 0, cfg.block_len)
    rows = np.flatnonzero((wl.pos_masked.numpy() != 0) & act)
    rng = np.random.default_rng(8)
    blocks = sorted({int(rows[0]) // cfg.block_len, int(rows[-1]) // cfg.block_len,
                     int(rows[len(rows) // 2]) // cfg.block_len}
                    | set(rng.choice(cfg.n_blocks, size=5, replace=False).tolist()))
    _, rep = check(wl, blocks=blocks)
    assert rep.n_live > 0
