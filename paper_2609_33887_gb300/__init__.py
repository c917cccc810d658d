"""GB300-native (sm_103a) commit step of a multi-block diffusion LM engine,
and the Redline selection of the configuration to deploy.

The work happens in libbdcommit.so (include/bdcommit.h, include/redline.h);
this package holds its sources (csrc/), the in-tree build step (build.py) and
the ctypes bindings (bdcommit.py, redline.py).
"""

from . import bdcommit, redline
from .bdcommit import (
    BD_BLOCK_ACTIVE,
    BD_BLOCK_FALLBACK_ELIGIBLE,
    BD_OK,
    BD_SWEEP_ADMIT,
    BD_SWEEP_ELIGIBLE_OLDEST,
    BdError,
    Nvfp4Head,
    bd_commit_step,
    bd_commit_step_ex,
    bd_commit_sweep,
    bd_get_device_status,
    bd_lmhead_partials,
    bd_merge_commit,
    bd_shutdown,
    bd_status_string,
    bd_verify_step,
    bd_verify_workspace_size,
    bd_version,
    bd_workspace_size,
    commit_step,
    commit_sweep,
    lmhead_partials,
    load_library,
    merge_commit,
    verify_step,
)

__all__ = [
    "BD_BLOCK_ACTIVE",
    "BD_BLOCK_FALLBACK_ELIGIBLE",
    "BD_OK",
    "BD_SWEEP_ADMIT",
    "BD_SWEEP_ELIGIBLE_OLDEST",
    "BdError",
    "Nvfp4Head",
    "bd_commit_step",
    "bd_commit_step_ex",
    "bd_commit_sweep",
    "bd_get_device_status",
    "bd_lmhead_partials",
    "bd_merge_commit",
    "bd_shutdown",
    "bd_status_string",
    "bd_verify_step",
    "bd_verify_workspace_size",
    "bd_version",
    "bd_workspace_size",
    "bdcommit",
    "commit_step",
    "commit_sweep",
    "lmhead_partials",
    "load_library",
    "merge_commit",
    "redline",
    "verify_step",
]
