"""Seeded synthetic inputs for the block-diffusion commit step.

This package only draws random tensors in the shapes, dtypes and value
distributions of the five benchmark workloads. It holds none of the commit
step's arithmetic (no logits, no softmax, no threshold rule): the float64
oracle under ``oracle/`` and the CUDA library both consume what it produces.
"""

from .configs import (B8X2X32_BF16, B32X4X32_TIED, B64X4X64_BF16, B256X8X64_E4M3, CONFIGS, TINY_F32,
                      WorkloadConfig, by_name, scaled)
from .generate import ACTIVE, FALLBACK_ELIGIBLE, Workload, generate

__all__ = [
    "ACTIVE",
    "B256X8X64_E4M3",
    "B32X4X32_TIED",
    "B64X4X64_BF16",
    "B8X2X32_BF16",
    "CONFIGS",
    "FALLBACK_ELIGIBLE",
    "TINY_F32",
    "Workload",
    "WorkloadConfig",
    "by_name",
    "generate",
    "scaled",
]
