"""Test harness glue: torch tensors -> the raw numpy arrays the oracle reads."""

import numpy as np
import torch


def raw_numpy(t: torch.Tensor) -> np.ndarray:
    """Stored bit patterns of a CPU tensor: float32 as float32, bfloat16 as
    uint16 patterns, float8_e4m3fn as uint8 codes, integer tensors as is."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype == torch.float8_e4m3fn:
        return t.view(torch.uint8).numpy()
    return t.numpy()


def dtype_tag(t: torch.Tensor) -> str:
    return {torch.float32: "f32", torch.bfloat16: "bf16", torch.float8_e4m3fn: "e4m3"}[t.dtype]


def oracle_on_workload(wl, blocks=None, taus=None):
    """Run the float64 oracle on a workloads.Workload (host tensors)."""
    import oracle

    cfg = wl.cfg
    return oracle.commit_step(
        raw_numpy(wl.hidden), dtype_tag(wl.hidden),
        raw_numpy(wl.weight), dtype_tag(wl.weight),
        None if wl.weight_scale is None else raw_numpy(wl.weight_scale),
        raw_numpy(wl.pos_masked), raw_numpy(wl.block_flags),
        cfg.n_seq, cfg.n_slots, cfg.block_len, wl.mask_token_id,
        wl.tau if taus is None else taus, blocks=blocks)
