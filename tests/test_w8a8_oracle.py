"""Pins of the oracle's E4M3 encoder and per-row activation quantisation (the
W8A8 variant of the precision lever), no GPU.

* every finite E4M3 code round-trips through decode and encode;
* values halfway between neighbouring codes go to the even code (round to
  nearest, ties to even), magnitudes above 448 saturate;
* hand-picked values from the format's definition (bias 7, three mantissa
  bits, subnormals of 2^-9);
* the encoder agrees with PyTorch's float8_e4m3fn conversion on in-range values;
* the row quantiser maps each row's largest magnitude to +-448, stays within
  the format's rounding bound, and zero rows stay zero.
"""

import numpy as np
import pytest

from oracle import commit_oracle as C


def finite_codes():
    c = np.arange(256, dtype=np.uint8)
    return c[(c & 0x7F) != 0x7F]


def test_round_trip_every_finite_code():
    c = finite_codes()
    assert np.array_equal(C.encode_e4m3(C.decode_e4m3(c)), c)


def test_ties_go_to_the_even_code():
    grid = C.decode_e4m3(np.arange(0x7F, dtype=np.uint8))
    mid = (grid[:-1] + grid[1:]) / 2
    got = C.encode_e4m3(mid).astype(np.int64)
    lo = np.arange(0x7E)
    expect = np.where(lo % 2 == 0, lo, lo + 1)
    assert np.array_equal(got, expect)
    # just above / below a midpoint picks the nearer neighbour
    assert np.array_equal(C.encode_e4m3(mid * (1 + 1e-9)).astype(np.int64), lo + 1)
    assert np.array_equal(C.encode_e4m3(mid * (1 - 1e-9)).astype(np.int64), lo)


def test_hand_values_and_saturation():
    assert C.encode_e4m3(np.array([1.0]))[0] == 0x38
    assert C.encode_e4m3(np.array([0.0625]))[0] == 0x18   # 2^-4: exponent field 3
    assert C.encode_e4m3(np.array([2.0 ** -9]))[0] == 0x01  # smallest subnormal
    assert C.encode_e4m3(np.array([2.0 ** -10]))[0] == 0x00  # halfway to 0: even code 0
    assert C.encode_e4m3(np.array([1.5 * 2.0 ** -9]))[0] == 0x02  # halfway between 0x01 and 0x02
    assert C.encode_e4m3(np.array([448.0]))[0] == 0x7E
    assert C.encode_e4m3(np.array([449.0, 1e6]))[0] == 0x7E
    assert C.encode_e4m3(np.array([-1e6]))[0] == 0xFE
    assert C.encode_e4m3(np.array([-0.0]))[0] == 0x80


def test_matches_torch_float8_conversion():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("no float8 in this torch")
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.uniform(-448, 448, 20000), rng.normal(0, 1e-2, 20000), rng.normal(0, 3, 20000)])
    ours = C.encode_e4m3(x)
    theirs = torch.from_numpy(x.astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    # float32 rounding of x may move a value across a tie; compare on values exactly representable in float32
    x32 = x.astype(np.float32).astype(np.float64)
    assert np.array_equal(C.encode_e4m3(x32), theirs)
    assert np.mean(ours == theirs) > 0.999


def test_row_quantiser():
    rng = np.random.default_rng(4)
    h = (rng.normal(size=(64, 200)) * rng.uniform(1e-3, 50, size=(64, 1))).astype(np.float32)
    h[5] = 0.0
    h[7, :] = 0.0
    h[7, 3] = -2.5
    codes, scale = C.quantize_rows_e4m3(h)
    deq = C.dequantize_rows_e4m3(codes, scale)
    assert np.all(deq[5] == 0) and scale[5] == 0
    amax_idx = np.argmax(np.abs(h), axis=1)
    rows = np.array([i for i in range(64) if i != 5])
    assert np.all((codes[rows, amax_idx[rows]] & 0x7F) == 0x7E)
    assert codes[7, 3] == 0xFE and np.count_nonzero(codes[7]) == 1
    # rounding bound: relative 2^-4 on normals, absolute half a subnormal step (2^-10) times the scale
    err = np.abs(deq - h)
    bound = np.abs(h) * 2.0 ** -4 + 2.0 ** -10 * scale[:, None].astype(np.float64) + 1e-12
    assert np.all(err <= bound)
    # scale = amax / 448 in float32
    assert np.array_equal(scale[rows], (np.max(np.abs(h[rows]), axis=1) / np.float32(448)).astype(np.float32))


def representable_rows(rng, n, d):
    """Rows that the per-row E4M3 quantiser reproduces exactly: every entry an
    E4M3 value times 2^k_row, and the row's largest magnitude 448 * 2^k_row
    (so inv = 2^-k_row exactly and every code is the entry's own)."""
    finite = C.decode_e4m3(np.arange(256))
    finite = finite[np.isfinite(finite)]
    h = rng.choice(finite, size=(n, d))
    h[:, 0] = np.where(rng.random(n) < 0.5, 448.0, -448.0)
    k = rng.integers(-20, 4, size=n).astype(np.float64)
    return (h * np.exp2(k)[:, None]).astype(np.float32)


def test_quantiser_is_exact_on_representable_rows():
    rng = np.random.default_rng(9)
    h = representable_rows(rng, 40, 96)
    codes, scale = C.quantize_rows_e4m3(h)
    assert np.array_equal(C.dequantize_rows_e4m3(codes, scale), h.astype(np.float64))


def test_w8a8_step_equals_exact_step_on_representable_rows():
    """Where quantisation is lossless, the W8A8 oracle (the step on the
    dequantised rows) is the exact step itself."""
    rng = np.random.default_rng(10)
    L, S, B, d, V = 8, 2, 2, 64, 300
    P = L * S * B
    h = representable_rows(rng, P, d)
    w = rng.normal(size=(V, d)).astype(np.float32)
    pm = (rng.random(P) < 0.7).astype(np.uint8)
    flags = np.array([3, 1, 1, 3], dtype=np.uint8)
    taus = [0.3, 0.6, 0.9]
    exact = C.commit_step(h, "f32", w, "f32", None, pm, flags, B, S, L, -1, taus)
    codes, scale = C.quantize_rows_e4m3(h)
    w8 = C.commit_step(C.dequantize_rows_e4m3(codes, scale), "f64", w, "f32", None, pm, flags, B, S, L, -1, taus)
    for key in ("tokens", "commit", "counts"):
        assert np.array_equal(exact[key], w8[key])
    assert np.array_equal(exact["conf"], w8["conf"])
