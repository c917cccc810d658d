"""Stored bit patterns of host tensors as numpy arrays (format glue only)."""

import numpy as np
import torch


def raw_numpy(t: torch.Tensor) -> np.ndarray:
    """float32 as float32, bfloat16 as uint16 patterns, float8_e4m3fn as uint8
    codes, integer tensors as they are."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype == torch.float8_e4m3fn:
        return t.view(torch.uint8).numpy()
    return t.numpy()


def dtype_tag(t: torch.Tensor) -> str:
    return {torch.float32: "f32", torch.bfloat16: "bf16", torch.float8_e4m3fn: "e4m3"}[t.dtype]
