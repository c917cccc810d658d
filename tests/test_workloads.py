"""The seeded input generator: shapes, dtypes, reproducibility, planted boosts."""

import numpy as np
import pytest
import torch

from workloads import (ACTIVE, B256X8X64_E4M3, B32X4X32_TIED, B64X4X64_BF16, B8X2X32_BF16, CONFIGS,
    FALLBACK_ELIGIBLE, generate, scaled, TINY_F32)


def test_five_workloads_have_the_stated_shapes():
    shapes = [(c.n_seq, c.n_slots, c.block_len, c.d, c.V, len(c.tau)) for c in CONFIGS]
    assert shapes == [
        (1, 1, 32, 256, 4096, 1),
        (8, 2, 32, 2048, 151936, 4),
        (32, 4, 32, 2048, 157184, 8),
        (64, 4, 64, 4096, 151936, 16),
        (256, 8, 64, 5120, 157184, 16),
    ]
    assert B8X2X32_BF16.tau == (0.7, 0.8, 0.9, 0.95)
    for c in (B32X4X32_TIED, B64X4X64_BF16, B256X8X64_E4M3):
        assert 0.95 in c.tau and list(c.tau) == sorted(c.tau)
    assert B32X4X32_TIED.tau[0] == 0.5 and B32X4X32_TIED.tau[-1] == pytest.approx(0.98)
    assert B64X4X64_BF16.tau[0] == pytest.approx(0.3) and B64X4X64_BF16.tau[-1] == pytest.approx(0.99)


def test_tiny_is_seeded_and_reproducible():
    a = generate(TINY_F32)
    b = generate(TINY_F32)
    assert torch.equal(a.hidden, b.hidden) and torch.equal(a.weight, b.weight)
    assert a.hidden.dtype == torch.float32 and a.weight.shape == (4096, 256)
    assert int(a.pos_masked.sum()) == 32
    assert a.block_flags.tolist() == [ACTIVE | FALLBACK_ELIGIBLE]


def test_tiny_plants_plus_eight_on_half_the_positions():
    wl = generate(TINY_F32)
    h = wl.hidden.double()
    w = wl.weight.double()
    logits = h @ w.T
    # a planted position has one logit about 8 above its N(0, 1) value, so its
    # top-2 gap is large; unplanted positions have the small gaps of the two
    # largest of 4096 normal draws
    top2 = logits.topk(2, dim=1).values
    planted = ((top2[:, 0] - top2[:, 1]) > 1.5).sum().item()
    assert planted == 16


def test_scaled_bf16_and_e4m3_variants():
    c = scaled(B256X8X64_E4M3, n_seq=2, n_slots=2, d=128, V=1000)
    wl = generate(c)
    assert wl.weight.dtype == torch.float8_e4m3fn and wl.weight_scale.shape == (1000,)
    deq = wl.weight.float() * wl.weight_scale[:, None]
    assert torch.all(deq.abs().amax(dim=1) > 0)
    # the largest code of every row is 448 (absmax / 448 scaling)
    assert torch.all(wl.weight.float().abs().amax(dim=1) == 448.0)
    assert wl.hidden.dtype == torch.bfloat16
    flags = wl.block_flags.view(2, 2)
    assert flags[:, 0].tolist() == [ACTIVE | FALLBACK_ELIGIBLE] * 2
    assert flags[:, 1].tolist() == [ACTIVE] * 2


def test_mask_fraction_is_close_to_the_stated_rate():
    c = scaled(B8X2X32_BF16, d=8, V=64)
    wl = generate(c)
    frac = wl.pos_masked.float().mean().item()
    assert abs(frac - 0.6) < 0.07


def test_nvfp4_head_quantisation():
    """The NVFP4 head: per row the largest block scale is 448 (E4M3 max), and the
    decoded head is close to the N(0, 1/d) draw it quantises (4-bit codes with
    16-element blocks: relative RMS error well under 15%)."""
    import math

    import numpy as np
    import torch

    from oracle import commit_oracle as C
    from workloads.generate import quantize_nvfp4

    V, d = 512, 200
    w = torch.randn(V, d, generator=torch.Generator().manual_seed(3)) / math.sqrt(d)
    codes, bs, rs = quantize_nvfp4(w)
    assert codes.shape == (V, 100) and bs.shape == (V, 13) and rs.shape == (V,)
    bsv = C.decode_e4m3(bs.numpy())
    assert np.allclose(bsv.max(axis=1), 448.0)
    deq = C.weights_f64((codes.numpy(), bs.numpy()), "nvfp4", rs.numpy(), d=d)
    err = np.sqrt(np.mean((deq - w.numpy()) ** 2)) / np.sqrt(np.mean(w.numpy() ** 2))
    assert err < 0.15, err
    # odd widths leave the last high nibble empty
    codes, bs, rs = quantize_nvfp4(w[:, :33])
    assert codes.shape == (V, 17) and np.all((codes[:, -1].numpy() >> 4) == 0)
