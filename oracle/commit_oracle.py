"""Float64 oracle of the per-forward commit step of a multi-block diffusion engine.

TEST INFRASTRUCTURE (see the package docstring): a plain, slow, obviously
correct restatement of what the paper defines, used only to check the CUDA
library. Every function cites the passage it follows.

What the step computes, in the paper's terms:
  * the engine keeps fixed block slots per request; an *active* block is being
    denoised, and the accept threshold decides which of its positions resolve
    in a step (App. F, opening paragraph);
  * a still-masked position's prediction is read from the mask-suppressed
    softmax that the engine commits from (App. B.1, "Entropy of the deeper
    blocks"): the softmax over the LM-head logits with the mask token removed;
    its argmax is the token and its maximum probability the confidence;
  * a position commits when its confidence is at or above the accept threshold
    (Sec. 3.1 and App. B.1: "at or above the accept threshold of 0.95");
  * when no position of the block clears the threshold, the rule falls back to
    the top-1 token (App. B.2, protocol of the self-distillation targets);
  * each threshold of a grid is one operating point of the serving grid
    (App. F.3), so the rule is applied once per threshold.

Readings where the paper is silent (each also listed in the design notes):
  * ">=" rather than ">" (App. B.1 says "at or above");
  * which blocks may take the fallback is a per-block flag supplied by the
    caller's scheduler (``FALLBACK_ELIGIBLE``), not something the step decides;
  * the fallback commits the one masked position of the block with the highest
    confidence, as its argmax token; ties go to the lowest position;
  * argmax ties go to the lowest vocabulary index;
  * the fallback is evaluated separately for every threshold of the grid;
  * confidence = maximum softmax probability at temperature 1 (greedy decoding,
    App. F.3).
"""

from __future__ import annotations

import math
from typing import Dict, Iterable, List, Optional, Sequence, Tuple

import numpy as np

ACTIVE = 1
FALLBACK_ELIGIBLE = 2


# ---------------------------------------------------------------------------
# Stored formats -> float64 values
# ---------------------------------------------------------------------------

def decode_bf16(raw: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns (uint16) -> float64.

    A bfloat16 value is the upper half of an IEEE-754 binary32 value, so the
    pattern shifted left by 16 bits is that binary32 value exactly.
    """
    raw = np.asarray(raw, dtype=np.uint16)
    return (raw.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def decode_e4m3(raw: np.ndarray) -> np.ndarray:
    """FP8 E4M3 bit patterns (uint8) -> float64, per the OCP 8-bit floating-point
    format: 1 sign bit, 4 exponent bits (bias 7), 3 mantissa bits; exponent
    field 0 encodes subnormals m/8 * 2^-6; no infinities; S.1111.111 is NaN.

    This is the weight format of the FP8 precision lever (App. E.4 lists the
    quantised weight grids; the per-output-channel e4m3 variant is this
    library's instance of that lever).
    """
    raw = np.asarray(raw, dtype=np.uint8).astype(np.int64)
    sign = np.where(raw & 0x80, -1.0, 1.0)
    e = (raw >> 3) & 0xF
    m = (raw & 0x7).astype(np.float64)
    normal = sign * (1.0 + m / 8.0) * np.exp2(e.astype(np.float64) - 7.0)
    sub = sign * (m / 8.0) * 2.0 ** -6
    out = np.where(e == 0, sub, normal)
    out = np.where((e == 15) & ((raw & 0x7) == 7), np.nan, out)
    return out


def encode_e4m3(x: np.ndarray) -> np.ndarray:
    """float64 values -> FP8 E4M3 codes (uint8), rounding to the nearest
    representable value with ties to the even code, magnitudes above the
    largest finite value 448 saturating to 448 (the "satfinite" conversion the
    W8A8 activations go through). The sign is kept, -0 included.

    Written from the format's definition: the non-negative finite codes
    0x00..0x7E are increasing in value (decode_e4m3), so a value's two
    neighbours on that grid are found by bisection."""
    x = np.asarray(x, dtype=np.float64)
    grid = decode_e4m3(np.arange(0x7F, dtype=np.uint8))  # 0x00..0x7E, increasing
    a = np.minimum(np.abs(x), grid[-1])
    hi = np.clip(np.searchsorted(grid, a, side="left"), 0, len(grid) - 1)  # first grid value >= a
    lo = np.maximum(hi - 1, 0)
    d_lo = a - grid[lo]
    d_hi = grid[hi] - a
    take_hi = (d_hi < d_lo) | ((d_hi == d_lo) & (hi % 2 == 0))
    code = np.where(a == grid[hi], hi, np.where(take_hi, hi, lo)).astype(np.uint8)
    return np.where(np.signbit(x), code | 0x80, code).astype(np.uint8)


def quantize_rows_e4m3(h: np.ndarray):
    """Per-row E4M3 quantisation of activations (the W8A8 variant of the
    precision lever): for row i with a = max_k |h[i, k]| (float32),
    inv = fl32(448 / a), codes = encode_e4m3(fl32(h[i, k] * inv)) and the
    row's dequantisation scale fl32(a / 448); an all-zero row gets codes 0 and
    scale 0. Every float32 operation is one correctly rounded IEEE operation,
    so a device implementation that performs the same operations produces the
    same codes. Returns (codes uint8 [n, d], scale float32 [n])."""
    h = np.asarray(h, dtype=np.float32)
    amax = np.max(np.abs(h), axis=1) if h.shape[1] else np.zeros(h.shape[0], np.float32)
    codes = np.zeros(h.shape, dtype=np.uint8)
    scale = np.zeros(h.shape[0], dtype=np.float32)
    nz = amax > 0
    inv = np.zeros_like(amax)
    inv[nz] = np.float32(448.0) / amax[nz]
    y = (h * inv[:, None]).astype(np.float32)
    codes[nz] = encode_e4m3(y[nz].astype(np.float64))
    scale[nz] = amax[nz] / np.float32(448.0)
    return codes, scale


def dequantize_rows_e4m3(codes: np.ndarray, scale: np.ndarray) -> np.ndarray:
    """The float64 activations the W8A8 LM head multiplies: code value times the row scale."""
    return decode_e4m3(codes) * np.asarray(scale, dtype=np.float64)[:, None]


def decode_e2m1(codes: np.ndarray) -> np.ndarray:
    """FP4 E2M1 codes (0..15) -> float64, per the OCP microscaling 4-bit float:
    1 sign bit, 2 exponent bits (bias 1), 1 mantissa bit; exponent field 0
    encodes the subnormal m * 0.5; no infinities or NaN. The magnitudes of
    codes 0..7 are 0, 0.5, 1, 1.5, 2, 3, 4, 6."""
    c = np.asarray(codes, dtype=np.int64) & 0xF
    sign = np.where(c & 0x8, -1.0, 1.0)
    e = (c >> 1) & 0x3
    m = (c & 0x1).astype(np.float64)
    normal = (1.0 + m / 2.0) * np.exp2(e.astype(np.float64) - 1.0)
    return sign * np.where(e == 0, m * 0.5, normal)


def decode_nvfp4(codes: np.ndarray, block_scale: np.ndarray, d: int) -> np.ndarray:
    """NVFP4 rows -> float64 [rows, d] (the 4-bit weight lever).

    Row layout: element k of a row is the E2M1 code in the low nibble of byte
    k // 2 when k is even, the high nibble when k is odd (codes [rows,
    ceil(d / 2)]); each run of 16 elements shares one E4M3 scale, element k
    using block_scale[:, k // 16] (block_scale [rows, ceil(d / 16)]). Value =
    e2m1(code) * e4m3(block scale)."""
    codes = np.asarray(codes, dtype=np.uint8)
    k = np.arange(d)
    byte = codes[:, k // 2].astype(np.int64)
    nib = np.where(k % 2 == 0, byte & 0xF, byte >> 4)
    bs = decode_e4m3(np.asarray(block_scale, dtype=np.uint8)[:, k // 16])
    return decode_e2m1(nib) * bs


def weights_f64(raw, dtype: str, scale: Optional[np.ndarray] = None, d: Optional[int] = None) -> np.ndarray:
    """Stored LM-head rows [rows, d] -> float64 values.

    f32 and bf16 rows are used as stored. e4m3 rows are the stored code times
    the row's (output channel's) float32 scale, i.e. exactly the dequantised
    weights the library is handed, not the matrix before quantisation. nvfp4
    rows are given as the pair (codes, block scales) and need the width d;
    their values are decode_nvfp4 times the optional per-row float32 scale.
    "f64" rows are values already decoded by this function (a caller that
    evaluates many samples of one head decodes it once).
    """
    if dtype == "f64":
        return np.asarray(raw, dtype=np.float64)
    if dtype == "nvfp4":
        codes, bscale = raw
        w = decode_nvfp4(codes, bscale, int(d))
        if scale is not None:
            w = w * np.asarray(scale, dtype=np.float32).astype(np.float64)[:, None]
        return w
    if dtype == "f32":
        return np.asarray(raw, dtype=np.float32).astype(np.float64)
    if dtype == "bf16":
        return decode_bf16(raw)
    if dtype == "e4m3":
        if scale is None:
            raise ValueError("e4m3 weights need a per-row scale")
        # decode_e4m3 of each of the 256 codes, looked up per element: the same
        # values as decoding the matrix element by element, without its
        # full-size temporaries (a 157184 x 5120 head would need ~40 GB)
        table = decode_e4m3(np.arange(256, dtype=np.uint8))
        w = table[np.asarray(raw, dtype=np.uint8)]
        w *= np.asarray(scale, dtype=np.float32).astype(np.float64)[:, None]
        return w
    raise ValueError(dtype)


def hidden_f64(raw: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "f64":  # values already decoded (e.g. the W8A8 variant's dequantised activations)
        return np.asarray(raw, dtype=np.float64)
    if dtype == "f32":
        return np.asarray(raw, dtype=np.float32).astype(np.float64)
    if dtype == "bf16":
        return decode_bf16(raw)
    raise ValueError(dtype)


# ---------------------------------------------------------------------------
# LM head and the mask-suppressed softmax (App. B.1)
# ---------------------------------------------------------------------------

def lm_head_logits(h: np.ndarray, w_raw: np.ndarray, w_dtype: str,
                   w_scale: Optional[np.ndarray] = None, chunk_rows: int = 8192) -> np.ndarray:
    """logits[i, v] = sum_k h[i, k] * w[v, k] in float64, for every vocabulary row v.

    ``h`` is float64 [n, d]; ``w_raw`` is the stored [V, d] head. The head is
    decoded a slice of rows at a time only to bound memory; every logit is one
    full dot product (a library matrix product serves as that step).
    """
    h = np.asarray(h, dtype=np.float64)
    packed = isinstance(w_raw, tuple)  # nvfp4: (codes, block scales)
    V = w_raw[0].shape[0] if packed else w_raw.shape[0]
    out = np.empty((h.shape[0], V), dtype=np.float64)
    for r0 in range(0, V, chunk_rows):
        r1 = min(V, r0 + chunk_rows)
        sc = None if w_scale is None else w_scale[r0:r1]
        rows = tuple(x[r0:r1] for x in w_raw) if packed else w_raw[r0:r1]
        w = weights_f64(rows, w_dtype, sc, d=h.shape[1])
        out[:, r0:r1] = h @ w.T
    return out


def row_confidence(logits: np.ndarray, mask_token_id: int = -1) -> Tuple[int, float, float]:
    """(token, confidence, top-2 gap) of one position (App. B.1).

    The mask token's logit is removed (set to -inf) when an id in [0, V) is
    given. token = lowest index attaining the maximum logit M;
    confidence = max softmax probability = exp(M - M) / sum_v exp(l_v - M)
               = 1 / sum_v exp(l_v - M);
    gap = M minus the largest logit of any other index (used only to exempt
    near-ties from the parity comparison).
    """
    l = np.array(logits, dtype=np.float64, copy=True)
    V = l.shape[0]
    if 0 <= mask_token_id < V:
        l[mask_token_id] = -np.inf
    M = float(np.max(l))
    token = int(np.flatnonzero(l == M)[0])
    s = float(np.sum(np.exp(l - M)))
    conf = 1.0 / s
    others = np.delete(l, token)
    gap = float(M - np.max(others)) if others.size and np.isfinite(np.max(others)) else math.inf
    return token, conf, gap


# ---------------------------------------------------------------------------
# Threshold commit with the per-block top-1 fallback (Sec. 3.1, App. B.1, B.2)
# ---------------------------------------------------------------------------

def commit_block(conf: Sequence[float], masked: Sequence[bool], active: bool, eligible: bool,
                 taus: Sequence[float]) -> np.ndarray:
    """Commit bits of one block: bit k of position j set <=> j commits at taus[k].

    For every threshold tau_k (one operating point each, App. F.3):
      C_k = { masked j : conf[j] >= tau_k }                 (at or above, Sec. 3.1)
      if C_k is empty, the block may take the fallback and it still holds a
      masked position, then C_k = { the masked j of highest confidence,
      lowest j on ties }                                    (top-1 fallback, App. B.2)
    Inactive blocks resolve nothing (App. F: only active blocks are denoised).
    """
    L = len(conf)
    bits = np.zeros(L, dtype=np.uint32)
    if not active:
        return bits
    masked_js = [j for j in range(L) if masked[j]]
    for k, tau in enumerate(taus):
        chosen = [j for j in masked_js if conf[j] >= tau]
        if not chosen and eligible and masked_js:
            best = masked_js[0]
            for j in masked_js[1:]:
                if conf[j] > conf[best]:
                    best = j
            chosen = [best]
        for j in chosen:
            bits[j] |= np.uint32(1) << np.uint32(k)
    return bits


def commit_step(hidden_raw: np.ndarray, hidden_dtype: str,
                w_raw: np.ndarray, w_dtype: str, w_scale: Optional[np.ndarray],
                pos_masked: np.ndarray, block_flags: np.ndarray,
                n_seq: int, n_slots: int, block_len: int,
                mask_token_id: int, taus: Sequence[float],
                blocks: Optional[Iterable[int]] = None,
                taus_f32: bool = True) -> Dict[str, np.ndarray]:
    """The whole commit step over the window, looped per position and per block.

    Inputs are the stored arrays: hidden [P, d] (f32 values or bf16 bit
    patterns), the head [V, d] (f32, bf16 bit patterns or e4m3 codes plus a
    per-row scale), ``pos_masked`` [P] (1 = still masked), ``block_flags``
    [n_seq * n_slots] (bit 0 active, bit 1 may take the fallback), and the
    threshold grid. Position p = (s * n_slots + b) * block_len + j.

    ``blocks`` restricts the evaluation to whole blocks (flat block indices);
    positions of other blocks keep the defaults and ``evaluated`` is False
    there. ``taus_f32`` compares against the thresholds as float32 values, the
    precision they are handed to the library in.

    Returns tokens (int32, -1 where nothing is predicted), conf (float64, 0
    there), commit (uint32 bit masks), gap (float64, nan there), counts
    (int64 [n_seq, T], committed positions per sequence and threshold) and
    evaluated (bool).
    """
    P = n_seq * n_slots * block_len
    n_blocks = n_seq * n_slots
    taus = [float(np.float32(t)) if taus_f32 else float(t) for t in taus]
    T = len(taus)
    pos_masked = np.asarray(pos_masked).reshape(P)
    block_flags = np.asarray(block_flags).reshape(n_blocks)
    blocks = list(range(n_blocks)) if blocks is None else sorted(set(int(b) for b in blocks))

    tokens = np.full(P, -1, dtype=np.int32)
    conf = np.zeros(P, dtype=np.float64)
    commit = np.zeros(P, dtype=np.uint32)
    gap = np.full(P, np.nan, dtype=np.float64)
    counts = np.zeros((n_seq, T), dtype=np.int64)
    evaluated = np.zeros(P, dtype=bool)

    # positions whose prediction is needed: masked positions of active blocks
    need: List[int] = []
    for blk in blocks:
        base = blk * block_len
        evaluated[base:base + block_len] = True
        if block_flags[blk] & ACTIVE:
            need.extend(base + j for j in range(block_len) if pos_masked[base + j])

    if need:
        h = hidden_f64(np.asarray(hidden_raw)[need], hidden_dtype)
        logits = lm_head_logits(h, w_raw, w_dtype, w_scale)
        for i, p in enumerate(need):
            tok, c, g = row_confidence(logits[i], mask_token_id)
            tokens[p] = tok
            conf[p] = c
            gap[p] = g

    for blk in blocks:
        base = blk * block_len
        f = int(block_flags[blk])
        masked = [bool(pos_masked[base + j]) and bool(f & ACTIVE) for j in range(block_len)]
        bits = commit_block(conf[base:base + block_len], masked, bool(f & ACTIVE),
                            bool(f & FALLBACK_ELIGIBLE), taus)
        commit[base:base + block_len] = bits
        s = blk // n_slots
        for k in range(T):
            counts[s, k] += int(np.count_nonzero(bits & (np.uint32(1) << np.uint32(k))))

    return {"tokens": tokens, "conf": conf, "commit": commit, "gap": gap,
            "counts": counts, "evaluated": evaluated}
