"""The five synthetic workloads of the commit step, and down-scaled variants.

Each workload is a window of ``n_seq`` sequences x ``n_slots`` block slots x
``block_len`` positions (the fixed-slot block buffer of App. F), a hidden
state per position, an LM-head weight matrix stored as [V, d] (one row per
vocabulary entry, the K-major layout of an ``nn.Linear`` head), and a grid of
accept thresholds.

Readings where the workload description leaves a detail open:
  * seeds: the Tiny workload uses seed 0; the others use their index (1..4);
  * every slot of the buffer holds an active block (buffer depth = blocks in
    flight), and only the oldest block of each sequence (slot 0) may take the
    top-1 fallback;
  * the 8-value grid spans linspace(0.5, 0.98, 8) and the 16-value grids
    linspace(0.3, 0.99, 16) and linspace(0.5, 0.99, 16); in each, the
    interior value nearest 0.95 is replaced by 0.95 itself, the engine's
    default accept threshold (App. F.3);
  * the near-tied mix of the 2048 x 157184 workload: 30% of positions boost two
    distinct columns by the same b ~ U[2, 10], 30% boost one column by
    b ~ U[2, 10], 40% are left alone.
"""

from __future__ import annotations

import dataclasses
from dataclasses import dataclass
from typing import Tuple

import numpy as np


def _grid(lo: float, hi: float, n: int) -> Tuple[float, ...]:
    vals = [float(v) for v in np.linspace(lo, hi, n)]
    if n > 2:
        interior = list(range(1, n - 1))
        j = min(interior, key=lambda i: abs(vals[i] - 0.95))
        vals[j] = 0.95
    return tuple(vals)


@dataclass(frozen=True)
class WorkloadConfig:
    name: str
    n_seq: int
    n_slots: int
    block_len: int
    mask_frac: float  # >= 1.0 means every position is still masked
    d: int
    V: int
    hidden_dtype: str  # "f32" | "bf16"
    weight_dtype: str  # "f32" | "bf16" | "e4m3" | "nvfp4"
    boost: str  # "fixed_half" | "single" | "tied_mix" | "none"
    boost_frac: float
    boost_lo: float
    boost_hi: float
    tau: Tuple[float, ...]
    seed: int
    mask_token_id: int = -1
    fallback: str = "oldest"  # "oldest" | "all" | "none"
    active: str = "all"  # "all" | "first_half"

    @property
    def P(self) -> int:
        return self.n_seq * self.n_slots * self.block_len

    @property
    def n_blocks(self) -> int:
        return self.n_seq * self.n_slots


# the small case the oracle runs in full (exact fp32 path)
TINY_F32 = WorkloadConfig(
    name="tiny_f32_d256_v4096",
    n_seq=1, n_slots=1, block_len=32, mask_frac=1.0,
    d=256, V=4096, hidden_dtype="f32", weight_dtype="f32",
    boost="fixed_half", boost_frac=0.5, boost_lo=8.0, boost_hi=8.0,
    tau=(0.9,), seed=0,
)
# the bench window: 8 sequences x 2 slots x 32 positions
B8X2X32_BF16 = WorkloadConfig(
    name="b8x2x32_d2048_v151936_bf16",
    n_seq=8, n_slots=2, block_len=32, mask_frac=0.6,
    d=2048, V=151936, hidden_dtype="bf16", weight_dtype="bf16",
    boost="single", boost_frac=0.4, boost_lo=2.0, boost_hi=10.0,
    tau=(0.7, 0.8, 0.9, 0.95), seed=1,
)
# 32 x 4 x 32 with tied top logits
B32X4X32_TIED = WorkloadConfig(
    name="b32x4x32_d2048_v157184_bf16_tied",
    n_seq=32, n_slots=4, block_len=32, mask_frac=0.5,
    d=2048, V=157184, hidden_dtype="bf16", weight_dtype="bf16",
    boost="tied_mix", boost_frac=0.6, boost_lo=2.0, boost_hi=10.0,
    tau=_grid(0.5, 0.98, 8), seed=2,
)
# 64 x 4 x 64, d = 4096
B64X4X64_BF16 = WorkloadConfig(
    name="b64x4x64_d4096_v151936_bf16",
    n_seq=64, n_slots=4, block_len=64, mask_frac=0.5,
    d=4096, V=151936, hidden_dtype="bf16", weight_dtype="bf16",
    boost="single", boost_frac=0.5, boost_lo=0.0, boost_hi=12.0,
    tau=_grid(0.3, 0.99, 16), seed=3,
)
# 256 x 8 x 64 with an FP8 head, d = 5120
B256X8X64_E4M3 = WorkloadConfig(
    name="b256x8x64_d5120_v157184_e4m3",
    n_seq=256, n_slots=8, block_len=64, mask_frac=0.4,
    d=5120, V=157184, hidden_dtype="bf16", weight_dtype="e4m3",
    boost="single", boost_frac=0.5, boost_lo=0.0, boost_hi=12.0,
    tau=_grid(0.5, 0.99, 16), seed=4,
)

CONFIGS = (TINY_F32, B8X2X32_BF16, B32X4X32_TIED, B64X4X64_BF16, B256X8X64_E4M3)


# The precision levers on the bench window (not among the five workloads):
# the b8x2x32 window and head shape with an NVFP4 or an E4M3 head.
EXTRA_CONFIGS = (
    dataclasses.replace(B8X2X32_BF16, name="b8x2x32_d2048_v151936_nvfp4", weight_dtype="nvfp4"),
    # the 8-bit levers on the same window: an E4M3 head (W8A16 and W8A8)
    dataclasses.replace(B8X2X32_BF16, name="b8x2x32_d2048_v151936_e4m3", weight_dtype="e4m3"),
    # a quarter of the largest window (64 of its 256 sequences, the same head): the same LM-head plan
    # regime (clusters of two pairs, several bands) at a size multi-pass profiler captures can hold
    dataclasses.replace(B256X8X64_E4M3, name="b64x8x64_d5120_v157184_e4m3", n_seq=64),
)


def by_name(name: str) -> WorkloadConfig:
    for c in CONFIGS + EXTRA_CONFIGS:
        if c.name == name:
            return c
    raise KeyError(name)


def scaled(cfg: WorkloadConfig, **overrides) -> WorkloadConfig:
    """A copy of ``cfg`` with some fields replaced (down-scaled parity cases)."""
    name = overrides.pop("name", None)
    if name is None:
        parts = [f"{k}={v}" for k, v in sorted(overrides.items())]
        name = cfg.name + "[" + ",".join(parts) + "]"
    return dataclasses.replace(cfg, name=name, **overrides)
