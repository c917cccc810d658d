"""Pins of the oracle's NVFP4 decoding (the 4-bit weight lever), no GPU.

* E2M1 codes against the format's table (OCP microscaling formats: magnitudes
  0, 0.5, 1, 1.5, 2, 3, 4, 6; the sign bit is bit 3, so code 8 is -0);
* the element layout (low nibble first, one E4M3 scale per 16 elements, odd
  widths) on hand-written rows;
* that every E2M1 x E4M3 product is exactly a bfloat16, which the library's
  decode to bf16 relies on (brute force over all finite pairs);
* that a head given as NVFP4 and the same head pre-decoded give the same
  commit step.
"""

import numpy as np

from oracle import commit_oracle as C

E2M1_TABLE = [0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0]


def test_e2m1_table():
    v = C.decode_e2m1(np.arange(16))
    assert list(v[:8]) == E2M1_TABLE
    assert list(v[8:]) == [-x for x in E2M1_TABLE]
    assert np.signbit(v[8]) and not np.signbit(v[0])


def test_layout_hand_rows():
    # byte 0x21: element 0 = code 1 (0.5), element 1 = code 2 (1.0); byte 0xF7: 6.0 then -6.0
    codes = np.array([[0x21, 0xF7, 0x0D]], dtype=np.uint8)
    # E4M3 0x38 = 1.0 scales elements 0..15, 0x40 = 2.0 scales elements 16..
    bs = np.array([[0x38]], dtype=np.uint8)
    assert list(C.decode_nvfp4(codes, bs, 5)[0]) == [0.5, 1.0, 6.0, -6.0, -3.0]  # odd width: high nibble unused
    codes = np.zeros((2, 17), dtype=np.uint8)
    codes[:, 8] = 0x32  # elements 16 (code 2 = 1.0) and 17 (code 3 = 1.5)
    codes[1, 0] = 0x07  # row 1, element 0 = 6.0
    bs = np.array([[0x38, 0x40, 0x30], [0x30, 0x38, 0x48]], dtype=np.uint8)  # 1, 2, 0.5 / 0.5, 1, 4
    w = C.decode_nvfp4(codes, bs, 34)
    assert w[0, 16] == 2.0 and w[0, 17] == 3.0 and w[1, 16] == 1.0 and w[1, 17] == 1.5
    assert w[1, 0] == 3.0 and np.count_nonzero(w) == 5
    # a per-row scale multiplies whole rows
    ws = C.weights_f64((codes, bs), "nvfp4", np.array([2.0, -1.0], dtype=np.float32), d=34)
    assert np.array_equal(ws, w * np.array([[2.0], [-1.0]]))


def test_products_are_bfloat16_exact():
    e2 = C.decode_e2m1(np.arange(16))
    e4 = C.decode_e4m3(np.arange(256))
    prod = np.outer(e2, e4[np.isfinite(e4)]).ravel()
    as32 = prod.astype(np.float32)
    assert np.array_equal(as32.astype(np.float64), prod)
    bits = as32.view(np.uint32)
    assert np.all((bits & 0xFFFF) == 0)  # the low 16 bits of the binary32 pattern are zero: a bfloat16


def test_commit_step_same_as_decoded_head():
    rng = np.random.default_rng(1)
    V, d, P = 300, 40, 32
    codes = rng.integers(0, 256, size=(V, d // 2), dtype=np.uint8)
    bs = rng.integers(0x20, 0x48, size=(V, 3), dtype=np.uint8)
    rs = rng.uniform(0.01, 0.1, size=V).astype(np.float32)
    h = rng.normal(size=(P, d)).astype(np.float32)
    pm = np.ones(P, dtype=np.uint8)
    flags = np.array([3], dtype=np.uint8)
    a = C.commit_step(h, "f32", (codes, bs), "nvfp4", rs, pm, flags, 1, 1, P, -1, [0.5, 0.9])
    w64 = C.weights_f64((codes, bs), "nvfp4", rs, d=d)
    b = C.commit_step(h, "f32", w64, "f64", None, pm, flags, 1, 1, P, -1, [0.5, 0.9])
    for k in ("tokens", "commit", "counts"):
        assert np.array_equal(a[k], b[k])
    assert np.array_equal(a["conf"], b["conf"])
