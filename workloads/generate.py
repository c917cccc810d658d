"""Draw one synthetic commit-step input from a seeded torch CPU generator.

Draw order (fixed, so a seed names one input): the masked-position flags,
then the hidden states, then the LM-head weights, then the planted boosts.

A planted boost of size b on vocabulary entry v at position p moves the
hidden state along that entry's weight row,
    h_p <- h_p + b * w_v / ||w_v||^2      (fp32, then rounded to the stored dtype)
which raises that position's logit for v by about b.  It is part of building
the input only: whatever values end up stored are what both the oracle and
the CUDA library read.
"""

from __future__ import annotations

import hashlib
import math
from dataclasses import dataclass
from typing import Optional, Tuple

import torch

from .configs import WorkloadConfig

ACTIVE = 1  # block_flags bit 0: the slot holds an active block
FALLBACK_ELIGIBLE = 2  # block_flags bit 1: the block may take the top-1 fallback

_TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}


@dataclass
class Workload:
    cfg: WorkloadConfig
    hidden: torch.Tensor  # [P, d], float32 or bfloat16
    weight: torch.Tensor  # [V, d], float32, bfloat16 or float8_e4m3fn; nvfp4: uint8 codes [V, ceil(d/2)]
    weight_scale: Optional[torch.Tensor]  # [V] float32 for e4m3 and nvfp4 weights, else None
    pos_masked: torch.Tensor  # [P] uint8, 1 = still masked
    block_flags: torch.Tensor  # [n_seq * n_slots] uint8
    tau: Tuple[float, ...]
    mask_token_id: int
    weight_block_scale: Optional[torch.Tensor] = None  # nvfp4: uint8 E4M3 codes [V, ceil(d/16)]

    @property
    def P(self) -> int:
        return self.cfg.P

    def digests(self) -> dict:
        """SHA-256 (first 16 hex digits) of each stored input tensor's bytes, so a
        run can record exactly which inputs it used."""
        out = {}
        for name in ("hidden", "weight", "weight_scale", "weight_block_scale", "pos_masked", "block_flags"):
            t = getattr(self, name)
            if t is not None:
                raw = t.detach().to("cpu").contiguous().view(torch.uint8).numpy().tobytes()
                out[name] = hashlib.sha256(raw).hexdigest()[:16]
        return out

    def to(self, device) -> "Workload":
        return Workload(
            cfg=self.cfg,
            hidden=self.hidden.to(device),
            weight=self.weight.to(device),
            weight_scale=None if self.weight_scale is None else self.weight_scale.to(device),
            pos_masked=self.pos_masked.to(device),
            block_flags=self.block_flags.to(device),
            tau=self.tau,
            mask_token_id=self.mask_token_id,
            weight_block_scale=None if self.weight_block_scale is None else self.weight_block_scale.to(device),
        )


def block_flags_for(cfg: WorkloadConfig) -> torch.Tensor:
    flags = torch.zeros(cfg.n_seq, cfg.n_slots, dtype=torch.uint8)
    if cfg.active == "all":
        flags[:, :] = ACTIVE
    elif cfg.active == "first_half":
        flags[:, : max(1, cfg.n_slots // 2)] = ACTIVE
    else:
        raise ValueError(cfg.active)
    if cfg.fallback == "oldest":
        flags[:, 0] |= FALLBACK_ELIGIBLE
    elif cfg.fallback == "all":
        flags |= FALLBACK_ELIGIBLE
    elif cfg.fallback != "none":
        raise ValueError(cfg.fallback)
    # eligibility only means something for active blocks
    flags[(flags & ACTIVE) == 0] = 0
    return flags.reshape(-1).contiguous()


def _realised_rows(weight_stored: torch.Tensor, scale: Optional[torch.Tensor], rows: torch.Tensor) -> torch.Tensor:
    if weight_stored.dtype == torch.float8_e4m3fn:
        # index through the byte view: some torch builds cannot index float8 tensors on the CPU
        w = weight_stored.view(torch.uint8)[rows].view(torch.float8_e4m3fn).float()
    else:
        w = weight_stored[rows].float()
    if scale is not None:
        w = w * scale[rows, None]
    return w


def generate(cfg: WorkloadConfig) -> Workload:
    """Build the seeded input of ``cfg`` on the host (CPU tensors)."""
    g = torch.Generator(device="cpu")
    g.manual_seed(cfg.seed)
    P, d, V = cfg.P, cfg.d, cfg.V

    # 1. masked-position flags
    if cfg.mask_frac >= 1.0:
        pos_masked = torch.ones(P, dtype=torch.uint8)
    elif cfg.mask_frac <= 0.0:
        pos_masked = torch.zeros(P, dtype=torch.uint8)
    else:
        pos_masked = (torch.rand(P, generator=g) < cfg.mask_frac).to(torch.uint8)
    block_flags = block_flags_for(cfg)

    # 2. hidden states, N(0, 1)
    hidden = torch.randn(P, d, generator=g, dtype=torch.float32)

    # 3. LM-head weights, N(0, 1/d), stored [V, d]
    weight = torch.randn(V, d, generator=g, dtype=torch.float32)
    weight.mul_(1.0 / math.sqrt(d))
    scale = None
    if cfg.weight_dtype == "f32":
        stored = weight
    elif cfg.weight_dtype == "bf16":
        stored = weight.to(torch.bfloat16)
    elif cfg.weight_dtype == "e4m3":
        # per-output-channel scale from the row's absolute maximum; 448 is the
        # largest finite e4m3 value; conversion rounds to nearest even
        absmax = weight.abs().amax(dim=1)
        scale = (absmax / 448.0).to(torch.float32)
        stored = torch.empty(V, d, dtype=torch.float8_e4m3fn)
        step = 8192
        for r0 in range(0, V, step):
            r1 = min(V, r0 + step)
            stored[r0:r1] = (weight[r0:r1] / scale[r0:r1, None]).to(torch.float8_e4m3fn)
    elif cfg.weight_dtype == "nvfp4":
        stored, bscale, scale = quantize_nvfp4(weight)
    else:
        raise ValueError(cfg.weight_dtype)

    # 4. planted boosts (along the unquantised rows for a 4-bit head)
    if cfg.boost != "none":
        if cfg.weight_dtype == "nvfp4":
            _plant(cfg, g, hidden, weight, None)
        else:
            _plant(cfg, g, hidden, stored, scale)
    del weight

    hidden = hidden.to(_TORCH_DTYPE[cfg.hidden_dtype]).contiguous()
    return Workload(
        cfg=cfg,
        hidden=hidden,
        weight=stored.contiguous(),
        weight_scale=scale,
        pos_masked=pos_masked,
        block_flags=block_flags,
        tau=tuple(float(t) for t in cfg.tau),
        mask_token_id=cfg.mask_token_id,
        weight_block_scale=bscale if cfg.weight_dtype == "nvfp4" else None,
    )


_E2M1 = torch.tensor([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])


def quantize_nvfp4(weight: torch.Tensor, chunk: int = 4096):
    """[V, d] float32 -> NVFP4 (codes uint8 [V, ceil(d/2)], E4M3 block scales uint8
    [V, ceil(d/16)], row scales float32 [V]). Per row, the row scale makes the
    largest block scale 448 (the largest E4M3 value); a block's scale is its
    absolute maximum / (6 * row scale) rounded to E4M3; each element is
    x / (block scale * row scale) rounded to the nearest E2M1 value, ties to
    the even code. Element k sits in the low nibble of byte k // 2 when k is even."""
    V, d = weight.shape
    nb = (d + 15) // 16
    dp = nb * 16
    codes = torch.zeros(V, (d + 1) // 2, dtype=torch.uint8)
    bscale = torch.zeros(V, nb, dtype=torch.uint8)
    rscale = torch.zeros(V, dtype=torch.float32)
    for r0 in range(0, V, chunk):
        r1 = min(V, r0 + chunk)
        w = torch.zeros(r1 - r0, dp)
        w[:, :d] = weight[r0:r1]
        blk = w.view(r1 - r0, nb, 16)
        amax = blk.abs().amax(dim=2)
        rs = (amax.amax(dim=1) / (6.0 * 448.0)).clamp_min(1e-30)
        bs8 = (amax / (6.0 * rs[:, None])).to(torch.float8_e4m3fn)
        bsv = bs8.float()
        denom = (bsv * rs[:, None]).clamp_min(1e-38)
        q = (blk / denom[:, :, None]).clamp(-6.0, 6.0)
        mag = q.abs().reshape(-1, 1)
        dist = (mag - _E2M1[None, :]).abs() + (torch.arange(8) % 2)[None, :] * 1e-7  # ties to the even code
        idx = dist.argmin(dim=1)
        sign = ((q.reshape(-1) < 0) & (idx > 0)).to(torch.int64)
        code = (idx | (sign << 3)).view(r1 - r0, dp)[:, :d]
        if d % 2:
            code = torch.cat([code, torch.zeros(r1 - r0, 1, dtype=code.dtype)], dim=1)
        codes[r0:r1] = (code[:, 0::2] | (code[:, 1::2] << 4)).to(torch.uint8)
        bscale[r0:r1] = bs8.view(torch.uint8)
        rscale[r0:r1] = rs
    return codes.contiguous(), bscale.contiguous(), rscale.contiguous()


def _plant(cfg, g, hidden, stored, scale):
    P, V = cfg.P, cfg.V
    if cfg.boost == "fixed_half":
        n = int(round(P * cfg.boost_frac))
        pos = torch.randperm(P, generator=g)[:n]
        cols = torch.randint(0, V, (n,), generator=g)
        b = torch.full((n,), float(cfg.boost_lo))
        _add(hidden, stored, scale, pos, cols, b)
        return
    u = torch.rand(P, generator=g)
    b = cfg.boost_lo + (cfg.boost_hi - cfg.boost_lo) * torch.rand(P, generator=g)
    col1 = torch.randint(0, V, (P,), generator=g)
    col2 = torch.randint(0, V - 1, (P,), generator=g)
    col2 = col2 + (col2 >= col1).to(col2.dtype)  # distinct from col1
    if cfg.boost == "single":
        pos = torch.nonzero(u < cfg.boost_frac).reshape(-1)
        _add(hidden, stored, scale, pos, col1[pos], b[pos])
    elif cfg.boost == "tied_mix":
        tied = torch.nonzero(u < 0.3).reshape(-1)
        single = torch.nonzero((u >= 0.3) & (u < 0.6)).reshape(-1)
        _add(hidden, stored, scale, tied, col1[tied], b[tied])
        _add(hidden, stored, scale, tied, col2[tied], b[tied])
        _add(hidden, stored, scale, single, col1[single], b[single])
    else:
        raise ValueError(cfg.boost)


def _add(hidden, stored, scale, pos, cols, b, chunk=4096):
    for i in range(0, pos.numel(), chunk):
        p = pos[i : i + chunk]
        c = cols[i : i + chunk]
        w = _realised_rows(stored, scale, c)
        nrm2 = (w * w).sum(dim=1, keepdim=True)
        hidden[p] += b[i : i + chunk, None] * w / nrm2
