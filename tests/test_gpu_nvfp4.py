"""NVFP4 heads (the 4-bit weight lever) on the GPU against the float64 oracle.

The library decodes every E2M1 x E4M3 product exactly (to f16 inside the
commit step's LM head, to bf16 elsewhere) and applies the per-row scale to the
fp32 logit, so the bf16 path's tolerances apply (tokens and commit bits exact
away from near-ties, confidence within 2e-3). The CTA-pair kernel decodes the
codes itself when code and block-scale rows start on 16-byte boundaries
(BD_FUSED_DECODE, default on), and otherwise from a bf16 copy decoded
beforehand; both are checked. In the first case the token rows travel as f16
scaled by a power of two per row, so rows spanning the bf16 exponent range
are checked too.
"""

import numpy as np
import pytest
import torch

from tests.helpers import oracle_on_workload
from tests.parity import compare
from workloads import B8X2X32_BF16, generate, scaled
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


def padded_rows(t, multiple=16):
    """The same rows in a tensor whose row stride is a multiple of `multiple` bytes."""
    ld = (t.shape[1] + multiple - 1) // multiple * multiple
    out = torch.zeros(t.shape[0], ld, dtype=t.dtype, device=t.device)
    out[:, : t.shape[1]] = t
    return out[:, : t.shape[1]]


def run(wl, variant=0, pad_scales=False):
    cfg = wl.cfg
    g = wl.to("cuda")
    scales = padded_rows(g.weight_block_scale) if pad_scales else g.weight_block_scale
    head = bdc.Nvfp4Head(padded_rows(g.weight), scales, cfg.d)
    tokens, conf, commit, counts = bdc.commit_step(
        g.hidden, head, g.pos_masked, g.block_flags, cfg.n_seq, cfg.n_slots, cfg.block_len, wl.tau,
        weight_scale=g.weight_scale, mask_token_id=wl.mask_token_id, counts=True, variant=variant)
    torch.cuda.synchronize()
    assert bdc.bd_get_device_status() == 0
    return {"tokens": tokens.cpu().numpy(), "conf": conf.cpu().numpy(),
            "commit": commit.cpu().numpy().view(np.uint32), "counts": counts.cpu().numpy()}


def check(wl, variant=0, blocks=None, pad_scales=False):
    ref = oracle_on_workload(wl, blocks=blocks)
    rep = compare(run(wl, variant, pad_scales), ref, wl.tau, "nvfp4", wl.cfg.block_len, wl.cfg.n_slots)
    assert rep.ok(), rep.failures
    return rep


SMALL = {
    "r128_d256": scaled(B8X2X32_BF16, n_seq=2, n_slots=2, d=256, V=1000, weight_dtype="nvfp4"),
    # ragged width: a K tail, an odd number of 16-element blocks, padded code rows
    "r1024_d200": scaled(B8X2X32_BF16, n_seq=8, n_slots=4, d=200, V=3000, weight_dtype="nvfp4"),
    "r294_d320": scaled(B8X2X32_BF16, d=320, V=2600, mask_frac=0.6, weight_dtype="nvfp4"),
}


@pytest.mark.parametrize("name", sorted(SMALL))
@pytest.mark.parametrize("variant", [0, 1, 2, 3])
def test_small(name, variant):
    rep = check(generate(SMALL[name]), variant)
    assert rep.n_live > 0


@pytest.mark.parametrize("name", sorted(SMALL))
@pytest.mark.parametrize("fused", [True, False])
def test_pair_fused_and_decoded(name, fused, monkeypatch):
    """The pair kernel decoding the codes in shared memory (16-byte aligned code
    and scale rows, K tails included) and the same kernel on the decoded copy."""
    if not fused:
        monkeypatch.setenv("BD_FUSED_DECODE", "0")
    rep = check(generate(SMALL[name]), variant=3, pad_scales=True)
    assert rep.n_live > 0


def test_pair_fused_mask_token_in_last_tile():
    """The in-kernel decode with a suppressed mask token inside the partial last v-tile."""
    cfg = scaled(B8X2X32_BF16, n_seq=4, n_slots=2, d=256, V=2900, weight_dtype="nvfp4", mask_token_id=2899)
    rep = check(generate(cfg), variant=3, pad_scales=True)
    assert rep.n_live > 0


def test_bench_window_nvfp4_head():
    """The 8 x 2 x 32 window with the 151936 x 2048 head in NVFP4, every masked position."""
    wl = generate(by_name("b8x2x32_d2048_v151936_nvfp4"))
    rep = check(wl)
    assert rep.n_live > 250


def test_verify_with_nvfp4_head():
    from oracle import verify_oracle as VO
    from workloads.generate import quantize_nvfp4
    from workloads.rawio import dtype_tag, raw_numpy
    from workloads.verify_inputs import generate_verify, SPEC_LLAMA8B, verify_scaled

    cfg = verify_scaled(SPEC_LLAMA8B, n_req=12, n_draft=4, d=256, V=2000, weight_dtype="f32", seed=8)
    wl = generate_verify(cfg)
    codes, bs, rs = quantize_nvfp4(wl.weight)
    ref = VO.verify_step(raw_numpy(wl.hidden), dtype_tag(wl.hidden), (codes.numpy(), bs.numpy()), "nvfp4",
                         rs.numpy(), wl.draft.numpy(), cfg.n_req, cfg.n_draft, cfg.eps)
    head = bdc.Nvfp4Head(padded_rows(codes.cuda()), bs.cuda(), cfg.d)
    out = bdc.verify_step(wl.hidden.cuda(), head, wl.draft.cuda(), cfg.n_req, cfg.n_draft, cfg.eps,
                          weight_scale=rs.cuda())
    torch.cuda.synchronize()
    g = {k: v.cpu().numpy() for k, v in out.items()}
    near = ref["gap"] < 1e-3
    assert np.all((g["tokens"] == ref["tokens"]) | near)
    assert np.max(np.abs(g["p_draft"] - ref["p_draft"])) <= 2e-3
    assert np.max(np.abs(g["entropy"] - ref["entropy"])) <= 1e-2


def scale_rows_by_powers_of_two(wl, exps=(-90, -40, -12, 0, 12, 40, 90)):
    """Hidden rows multiplied by 2^k (exact in bf16), k cycling over exps."""
    k = torch.tensor(exps, dtype=torch.float64)[torch.arange(wl.hidden.shape[0]) % len(exps)]
    wl.hidden = (wl.hidden.double() * torch.exp2(k)[:, None]).to(wl.hidden.dtype)
    return wl


@pytest.mark.parametrize("fused", [True, False])
def test_row_magnitudes_across_the_bf16_range(fused, monkeypatch):
    if not fused:
        monkeypatch.setenv("BD_FUSED_DECODE", "0")
    rep = check(scale_rows_by_powers_of_two(generate(SMALL["r294_d320"])), variant=3)
    assert rep.n_live > 0
