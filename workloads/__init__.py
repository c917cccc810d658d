"""Seeded synthetic inputs for the block-diffusion commit step.

This package only draws random tensors in the shapes, dtypes and value
distributions of the five benchmark workloads. It holds none of the commit
step's arithmetic (no logits, no softmax, no threshold rule): the float64
oracle under ``oracle/`` and the CUDA library both consume what it produces.
"""

from .configs import CONFIGS, WorkloadConfig, by_name, scaled
from .generate import ACTIVE, FALLBACK_ELIGIBLE, Workload, generate

__all__ = [
    "ACTIVE",
    "CONFIGS",
    "FALLBACK_ELIGIBLE",
    "Workload",
    "WorkloadConfig",
    "by_name",
    "generate",
    "scaled",
]
