"""Seeded synthetic inputs for speculative-decoding verification (typical
acceptance and its lossless reference).

Holds no step of the verification (no logits, no softmax, no acceptance
rule). A verification batch is n_req requests, each with n_draft draft tokens:
the target forward yields n_draft + 1 rows per request, row
q * (n_draft + 1) + i verifying draft token i of request q (i < n_draft) and
the last row giving the bonus token. Hidden states and the LM head are drawn
as in the commit-step workloads (N(0, 1) states, N(0, 1/d) head rows); every
row then gets one planted boost of size b ~ U[boost_lo, boost_hi] on a random
vocabulary entry c (h += b * w_c / ||w_c||^2, which raises logit c by about
b), and the draft token of a draft row is c with probability `agree`, else a
uniformly drawn other entry. With boosts well above the spread of the other
logits, c is the target's argmax, so `agree` is the per-token agreement
between draft and target that the paper reports (90.5% for the Llama pair,
88.7% for the Qwen pair, four draft tokens).

Workloads follow the paper's two target models: Llama-3.1-8B (d = 4096,
V = 128256) and Qwen2.5-7B (d = 3584, V = 152064); their settings grid is the
paper's eleven epsilons. They stand in for the GSM8K drafts, which are not used.
"""

from __future__ import annotations

import dataclasses
import math
from dataclasses import dataclass
from typing import Optional, Tuple

import torch

from .generate import _add

EPS_GRID = (0.8, 0.7, 0.6, 0.5, 0.45, 0.4, 0.3, 0.2, 0.1, 0.05, 0.02)


@dataclass(frozen=True)
class VerifyConfig:
    name: str
    n_req: int
    n_draft: int
    d: int
    V: int
    hidden_dtype: str  # "bf16" | "f32"
    weight_dtype: str  # "bf16" | "e4m3" | "f32"
    boost_lo: float
    boost_hi: float
    agree: float
    eps: Tuple[float, ...]
    seed: int

    @property
    def rows(self) -> int:
        return self.n_req * (self.n_draft + 1)


# Llama-3.1-8B's LM-head shape, 64 requests x (4 drafts + 1)
SPEC_LLAMA8B = VerifyConfig(
    name="spec_llama8b_r64x5_d4096_v128256_bf16", n_req=64, n_draft=4, d=4096, V=128256,
    hidden_dtype="bf16", weight_dtype="bf16", boost_lo=8.0, boost_hi=18.0, agree=0.905, eps=EPS_GRID, seed=11,
)
# Qwen2.5-7B's LM-head shape, 64 requests x (4 drafts + 1)
SPEC_QWEN7B = VerifyConfig(
    name="spec_qwen7b_r64x5_d3584_v152064_bf16", n_req=64, n_draft=4, d=3584, V=152064,
    hidden_dtype="bf16", weight_dtype="bf16", boost_lo=8.0, boost_hi=18.0, agree=0.887, eps=EPS_GRID, seed=12,
)

VERIFY_CONFIGS = (SPEC_LLAMA8B, SPEC_QWEN7B)


def verify_by_name(name: str) -> VerifyConfig:
    for c in VERIFY_CONFIGS:
        if c.name == name:
            return c
    raise KeyError(name)


def verify_scaled(cfg: VerifyConfig, **overrides) -> VerifyConfig:
    name = overrides.pop("name", None)
    if name is None:
        name = cfg.name + "[" + ",".join(f"{k}={v}" for k, v in sorted(overrides.items())) + "]"
    return dataclasses.replace(cfg, name=name, **overrides)


@dataclass
class VerifyWorkload:
    cfg: VerifyConfig
    hidden: torch.Tensor                  # [rows, d]
    weight: torch.Tensor                  # [V, d]
    weight_scale: Optional[torch.Tensor]  # [V] for e4m3 heads
    draft: torch.Tensor                   # int32 [n_req * n_draft]
    planted: torch.Tensor                 # int64 [rows]: the boosted entry of each row (for input statistics only)

    def to(self, device) -> "VerifyWorkload":
        return VerifyWorkload(self.cfg, self.hidden.to(device), self.weight.to(device),
                              None if self.weight_scale is None else self.weight_scale.to(device),
                              self.draft.to(device), self.planted)


def generate_verify(cfg: VerifyConfig) -> VerifyWorkload:
    g = torch.Generator().manual_seed(cfg.seed)
    R, d, V = cfg.rows, cfg.d, cfg.V
    hidden = torch.randn(R, d, generator=g, dtype=torch.float32)
    weight = torch.randn(V, d, generator=g, dtype=torch.float32).mul_(1.0 / math.sqrt(d))
    scale = None
    if cfg.weight_dtype == "f32":
        stored = weight
    elif cfg.weight_dtype == "bf16":
        stored = weight.to(torch.bfloat16)
    elif cfg.weight_dtype == "e4m3":
        absmax = weight.abs().amax(dim=1)
        scale = (absmax / 448.0).to(torch.float32)
        stored = torch.empty(V, d, dtype=torch.float8_e4m3fn)
        for r0 in range(0, V, 8192):
            r1 = min(V, r0 + 8192)
            stored[r0:r1] = (weight[r0:r1] / scale[r0:r1, None]).to(torch.float8_e4m3fn)
    else:
        raise ValueError(cfg.weight_dtype)
    del weight
    planted = torch.randint(0, V, (R,), generator=g)
    b = cfg.boost_lo + (cfg.boost_hi - cfg.boost_lo) * torch.rand(R, generator=g)
    _add(hidden, stored, scale, torch.arange(R), planted, b)
    # draft tokens: the planted entry with probability `agree`, else another entry
    u = torch.rand(R, generator=g)
    other = torch.randint(0, V - 1, (R,), generator=g)
    other = other + (other >= planted).to(other.dtype)
    tok = torch.where(u < cfg.agree, planted, other)
    rows = torch.arange(R).reshape(cfg.n_req, cfg.n_draft + 1)[:, : cfg.n_draft].reshape(-1)
    draft = tok[rows].to(torch.int32).contiguous()
    hidden = hidden.to(torch.bfloat16 if cfg.hidden_dtype == "bf16" else torch.float32).contiguous()
    return VerifyWorkload(cfg, hidden, stored.contiguous(), scale, draft, planted)
