"""ctypes binding of libbdcommit (include/bdcommit.h).

Argument marshalling only: torch tensors (device memory, streams) become the
plain pointers and sizes of the C ABI, and every step of the commit step runs
in the library's CUDA kernels. There is no fallback: if the shared library is
missing or cannot be loaded, every entry point raises.
"""

from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int, c_int32, c_int64, c_size_t, c_void_p
from dataclasses import dataclass
from typing import Optional, Sequence

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
# BD_LIBRARY selects another build of the library (e.g. the bounds-checked
# libbdcommit_checks.so); by default the in-tree libbdcommit.so
LIB_PATH = os.environ.get("BD_LIBRARY") or os.path.join(_PKG, "libbdcommit.so")

# status codes (bd_status)
BD_OK = 0
BD_ERR_NULL = -1
BD_ERR_SHAPE = -2
BD_ERR_DTYPE = -3
BD_ERR_ALIGN = -4
BD_ERR_TAU = -5
BD_ERR_WORKSPACE = -6
BD_ERR_CUDA = -7
BD_ERR_TIMEOUT = -8
BD_ERR_DEVICE = -9
BD_ERR_ARG = -10
BD_ERR_BOUNDS = -11

# dtypes (bd_dtype)
BD_F32 = 0
BD_BF16 = 1
BD_E4M3 = 2
BD_NVFP4 = 3

BD_BLOCK_ACTIVE = 1
BD_BLOCK_FALLBACK_ELIGIBLE = 2

BD_SWEEP_ADMIT = 1
BD_SWEEP_ELIGIBLE_OLDEST = 2

VARIANT_AUTO = 0
VARIANT_SIMT = 1
VARIANT_TC_ONE_CTA = 2
VARIANT_TC_PAIR = 3

# bd_exec.flags
BD_EXEC_FP8_ACTIVATIONS = 1  # W8A8: E4M3 token rows x E4M3 head on the 8-bit tensor path


class bd_hidden(ctypes.Structure):
    _fields_ = [("data", c_void_p), ("dtype", c_int32), ("rows", c_int64), ("cols", c_int64), ("ld", c_int64)]


class bd_weight(ctypes.Structure):
    _fields_ = [("data", c_void_p), ("dtype", c_int32), ("vocab", c_int64), ("dim", c_int64), ("ld", c_int64),
                ("scale", c_void_p), ("block_scale", c_void_p), ("block_ld", c_int64)]


class bd_mask_state(ctypes.Structure):
    _fields_ = [("n_seq", c_int32), ("n_slots", c_int32), ("block_len", c_int32), ("mask_token_id", c_int32),
                ("pos_masked", c_void_p), ("block_flags", c_void_p)]


class bd_tau_grid(ctypes.Structure):
    _fields_ = [("tau", POINTER(c_float)), ("T", c_int32)]


class bd_exec(ctypes.Structure):
    _fields_ = [("stream", c_void_p), ("workspace", c_void_p), ("workspace_bytes", c_size_t),
                ("out_counts", c_void_p), ("lmhead_event_begin", c_void_p), ("lmhead_event_end", c_void_p),
                ("variant", c_int32), ("flags", c_int32)]


class bd_partials(ctypes.Structure):
    _fields_ = [("m", c_void_p), ("s", c_void_p), ("a", c_void_p)]


class bd_draft(ctypes.Structure):
    _fields_ = [("n_req", c_int32), ("n_draft", c_int32), ("draft", c_void_p)]


class bd_eps_grid(ctypes.Structure):
    _fields_ = [("eps", POINTER(c_float)), ("E", c_int32)]


BD_ACCEPT_LOSSLESS_BIT = 31


class bd_window(ctypes.Structure):
    _fields_ = [("n_seq", c_int32), ("n_slots", c_int32), ("block_len", c_int32), ("mask_token_id", c_int32),
                ("tokens", c_void_p), ("pos_masked", c_void_p), ("block_flags", c_void_p)]


class BdError(RuntimeError):
    def __init__(self, status: int, where: str = "bd_commit_step"):
        self.status = status
        super().__init__(f"{where} failed: {status} ({bd_status_string(status)})")


_lib = None


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Load libbdcommit.so (built in-tree by paper_2609_33887_gb300/build.py)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libbdcommit.so not found at {p}: build it first "
                           "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(p)
    sig = {
        "bd_commit_step": (c_int, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_mask_state),
                                   POINTER(bd_tau_grid), c_void_p, c_void_p, c_void_p]),
        "bd_commit_step_ex": (c_int, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_mask_state),
                                      POINTER(bd_tau_grid), c_void_p, c_void_p, c_void_p, POINTER(bd_exec)]),
        "bd_workspace_size": (c_size_t, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_mask_state),
                                         POINTER(bd_tau_grid)]),
        "bd_step_kernels": (c_int, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_mask_state),
                                    POINTER(bd_tau_grid), POINTER(bd_exec)]),
        "bd_plan_header": (c_int, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_mask_state),
                                   POINTER(bd_tau_grid), POINTER(bd_exec), c_int32, POINTER(c_int32), c_int32]),
        "bd_commit_step_static": (c_int, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_mask_state),
                                          POINTER(bd_tau_grid), c_void_p, c_void_p, c_void_p, c_void_p]),
        "bd_verify_step": (c_int, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_draft), POINTER(bd_eps_grid),
                                   c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, POINTER(bd_exec)]),
        "bd_verify_workspace_size": (c_size_t, [POINTER(bd_hidden), POINTER(bd_weight), POINTER(bd_draft),
                                                POINTER(bd_eps_grid)]),
        "bd_commit_sweep": (c_int, [POINTER(bd_window), c_void_p, c_void_p, c_int32, ctypes.c_uint32, c_void_p,
                                    c_void_p, c_void_p, c_void_p]),
        "bd_lmhead_partials": (c_int, [POINTER(bd_hidden), POINTER(bd_weight), ctypes.c_int64,
                                       POINTER(bd_mask_state), POINTER(bd_partials), POINTER(bd_exec)]),
        "bd_merge_commit": (c_int, [POINTER(bd_partials), ctypes.c_int32, POINTER(bd_mask_state),
                                    POINTER(bd_tau_grid), c_void_p, c_void_p, c_void_p, POINTER(bd_exec)]),
        "bd_get_device_status": (c_int, [c_void_p]),
        "bd_selftest_timeout": (c_int, [c_void_p]),
        "bd_static_device_status": (c_int, [c_void_p]),
        "bd_static_selftest_timeout": (c_int, [c_void_p]),
        "bd_status_string": (ctypes.c_char_p, [c_int]),
        "bd_shutdown": (c_int, []),
        "bd_version": (c_int, []),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


# ------------------------------------------------------------ marshalling --
_DT = {torch.float32: BD_F32, torch.bfloat16: BD_BF16, torch.float8_e4m3fn: BD_E4M3}


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def make_hidden(hidden: torch.Tensor) -> bd_hidden:
    if hidden.dim() != 2 or hidden.stride(1) != 1:
        raise ValueError("hidden must be a 2-D tensor with contiguous rows")
    return bd_hidden(_ptr(hidden), _DT[hidden.dtype], hidden.shape[0], hidden.shape[1], hidden.stride(0))


@dataclass
class Nvfp4Head:
    """An NVFP4 LM head as the library reads it: codes uint8 [vocab, ceil(dim/2)]
    (two E2M1 codes per byte, low nibble first), block_scale uint8
    [vocab, ceil(dim/16)] (E4M3 codes, one per 16 elements) and the width dim.
    The optional per-row float32 scale is passed as the weight scale."""
    codes: torch.Tensor
    block_scale: torch.Tensor
    dim: int


def make_weight(weight, scale: Optional[torch.Tensor] = None) -> bd_weight:
    if isinstance(weight, Nvfp4Head):
        c, b = weight.codes, weight.block_scale
        if c.dtype != torch.uint8 or b.dtype != torch.uint8 or c.dim() != 2 or b.dim() != 2 \
                or c.stride(1) != 1 or b.stride(1) != 1:
            raise ValueError("NVFP4 codes and block scales must be 2-D uint8 tensors with contiguous rows")
        return bd_weight(_ptr(c), BD_NVFP4, c.shape[0], weight.dim, c.stride(0), _ptr(scale), _ptr(b), b.stride(0))
    if weight.dim() != 2 or weight.stride(1) != 1:
        raise ValueError("weight must be a 2-D [vocab, dim] tensor with contiguous rows")
    return bd_weight(_ptr(weight), _DT[weight.dtype], weight.shape[0], weight.shape[1], weight.stride(0),
                     _ptr(scale), None, 0)


def make_mask_state(pos_masked: torch.Tensor, block_flags: torch.Tensor, n_seq: int, n_slots: int,
                    block_len: int, mask_token_id: int = -1) -> bd_mask_state:
    if pos_masked.dtype != torch.uint8 or block_flags.dtype != torch.uint8:
        raise ValueError("pos_masked and block_flags must be uint8")
    if not (pos_masked.is_contiguous() and block_flags.is_contiguous()):
        raise ValueError("pos_masked and block_flags must be contiguous")
    return bd_mask_state(n_seq, n_slots, block_len, mask_token_id, _ptr(pos_masked), _ptr(block_flags))


def make_tau_grid(tau: Sequence[float]):
    arr = (c_float * max(1, len(tau)))(*[float(t) for t in tau])
    return bd_tau_grid(ctypes.cast(arr, POINTER(c_float)), len(tau)), arr


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ------------------------------------------------------------ entry points --
def bd_status_string(status: int) -> str:
    return load_library().bd_status_string(int(status)).decode()


def bd_version() -> int:
    return int(load_library().bd_version())


def bd_shutdown() -> int:
    return int(load_library().bd_shutdown())


def bd_get_device_status(stream=None) -> int:
    return int(load_library().bd_get_device_status(_stream_handle(stream)))


def bd_selftest_timeout(stream=None) -> int:
    """Queue the failure-detection self-test: a bounded wait that runs out (about 1 s)."""
    return int(load_library().bd_selftest_timeout(_stream_handle(stream)))


def bd_workspace_size(hidden, weight, weight_scale, pos_masked, block_flags, n_seq, n_slots, block_len,
                      mask_token_id, tau) -> int:
    h = make_hidden(hidden)
    w = make_weight(weight, weight_scale)
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id)
    tg, _keep = make_tau_grid(tau)
    return int(load_library().bd_workspace_size(ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms),
                                                ctypes.byref(tg)))


def bd_step_kernels(hidden, weight, weight_scale, pos_masked, block_flags, n_seq, n_slots, block_len,
                    mask_token_id, tau, *, variant=VARIANT_AUTO, flags=0) -> int:
    """Kernels one bd_commit_step_ex call with these arguments queues (a
    negative bd_status for invalid arguments). Queues nothing."""
    h = make_hidden(hidden)
    w = make_weight(weight, weight_scale)
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id)
    tg, _keep = make_tau_grid(tau)
    ex = bd_exec()
    ex.variant = variant
    ex.flags = flags
    return int(load_library().bd_step_kernels(ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms),
                                              ctypes.byref(tg), ctypes.byref(ex)))


def bd_plan_header(hidden, weight, weight_scale, pos_masked, block_flags, n_seq, n_slots, block_len,
                   mask_token_id, tau, n_rows, *, variant=VARIANT_AUTO, flags=0):
    """The LM head's work plan for n_rows compacted rows (eight int32 words,
    see include/bdcommit.h), or raises on a negative status."""
    h = make_hidden(hidden)
    w = make_weight(weight, weight_scale)
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id)
    tg, _keep = make_tau_grid(tau)
    ex = bd_exec()
    ex.variant = variant
    ex.flags = flags
    out = (c_int32 * 8)()
    rc = int(load_library().bd_plan_header(ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms), ctypes.byref(tg),
                                           ctypes.byref(ex), int(n_rows), out, 8))
    if rc < 0:
        raise RuntimeError(f"bd_plan_header: {bd_status_string(rc)}")
    return list(out)[:rc]


def bd_commit_step_ex(hidden, weight, weight_scale, pos_masked, block_flags, n_seq, n_slots, block_len,
                      mask_token_id, tau, out_tokens, out_conf, out_commit, *, stream=None, workspace=None,
                      out_counts=None, lmhead_events=None, variant=VARIANT_AUTO, flags=0) -> int:
    """Queue one commit step on `stream` (default: torch's current stream).

    All tensors are device tensors; `tau` is a host sequence of floats.
    Returns the bd_status code (0 on success)."""
    h = make_hidden(hidden)
    w = make_weight(weight, weight_scale)
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id)
    tg, _keep = make_tau_grid(tau)
    ex = bd_exec()
    ex.stream = _stream_handle(stream)
    if workspace is not None:
        ex.workspace = workspace.data_ptr()
        ex.workspace_bytes = workspace.numel() * workspace.element_size()
    ex.out_counts = _ptr(out_counts)
    if lmhead_events is not None:
        ex.lmhead_event_begin = lmhead_events[0].cuda_event
        ex.lmhead_event_end = lmhead_events[1].cuda_event
    ex.variant = variant
    ex.flags = flags
    return int(load_library().bd_commit_step_ex(
        ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms), ctypes.byref(tg),
        _ptr(out_tokens), _ptr(out_conf), _ptr(out_commit), ctypes.byref(ex)))


def bd_commit_step(hidden, weight, weight_scale, pos_masked, block_flags, n_seq, n_slots, block_len,
                   mask_token_id, tau, out_tokens, out_conf, out_commit) -> int:
    """bd_commit_step: default stream, library-owned workspace."""
    h = make_hidden(hidden)
    w = make_weight(weight, weight_scale)
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id)
    tg, _keep = make_tau_grid(tau)
    return int(load_library().bd_commit_step(
        ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms), ctypes.byref(tg),
        _ptr(out_tokens), _ptr(out_conf), _ptr(out_commit)))


def bd_commit_step_static(hidden, weight, weight_scale, pos_masked, block_flags, n_seq, n_slots, block_len,
                          mask_token_id, tau, out_tokens, out_conf, out_commit, *, stream=None) -> int:
    """bd_commit_step_static: the commit step without any device allocation, for
    callers that must not allocate (inside an allocator callback, under a
    framework that owns all device memory, or on a serving path that cannot
    take cudaMalloc's implicit synchronisation). It works in the library's
    fixed 32 MiB device array; see include/bdcommit.h for its limits."""
    h = make_hidden(hidden)
    w = make_weight(weight, weight_scale)
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id)
    tg, _keep = make_tau_grid(tau)
    return int(load_library().bd_commit_step_static(
        ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms), ctypes.byref(tg),
        _ptr(out_tokens), _ptr(out_conf), _ptr(out_commit), _stream_handle(stream)))


def bd_lmhead_partials(hidden, shard, shard_scale, vocab_offset, pos_masked, block_flags, n_seq, n_slots,
                       block_len, mask_token_id, out_m, out_s, out_a, *, stream=None, workspace=None,
                       variant=VARIANT_AUTO) -> int:
    """Queue part 1 of the vocabulary-parallel step: the LM head over head rows
    [vocab_offset, vocab_offset + shard rows) and one (max, sum of exp, global
    argmax) partial per window position into out_m / out_s / out_a (device
    float32 / float32 / int32 [P]). mask_token_id is a global id. Returns the status."""
    h = make_hidden(hidden)
    w = make_weight(shard, shard_scale)
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id)
    out = bd_partials(_ptr(out_m), _ptr(out_s), _ptr(out_a))
    ex = bd_exec()
    ex.stream = _stream_handle(stream)
    if workspace is not None:
        ex.workspace = workspace.data_ptr()
        ex.workspace_bytes = workspace.numel() * workspace.element_size()
    ex.variant = variant
    return int(load_library().bd_lmhead_partials(ctypes.byref(h), ctypes.byref(w), int(vocab_offset),
                                                 ctypes.byref(ms), ctypes.byref(out), ctypes.byref(ex)))


def bd_merge_commit(parts_m, parts_s, parts_a, n_parts, pos_masked, block_flags, n_seq, n_slots, block_len, tau,
                    out_tokens, out_conf, out_commit, *, stream=None, out_counts=None) -> int:
    """Queue part 2: merge the gathered partials ([n_parts, P] device arrays)
    of every position and apply the commit rule for the threshold grid.
    Returns the status."""
    g = bd_partials(_ptr(parts_m), _ptr(parts_s), _ptr(parts_a))
    ms = make_mask_state(pos_masked, block_flags, n_seq, n_slots, block_len, -1)
    tg, _keep = make_tau_grid(tau)
    ex = bd_exec()
    ex.stream = _stream_handle(stream)
    ex.out_counts = _ptr(out_counts)
    return int(load_library().bd_merge_commit(ctypes.byref(g), int(n_parts), ctypes.byref(ms), ctypes.byref(tg),
                                              _ptr(out_tokens), _ptr(out_conf), _ptr(out_commit),
                                              ctypes.byref(ex)))


def lmhead_partials(hidden, shard, vocab_offset, pos_masked, block_flags, n_seq, n_slots, block_len, *,
                    shard_scale=None, mask_token_id=-1, stream=None, workspace=None, variant=VARIANT_AUTO):
    """Allocate the per-position partials on the hidden states' device, queue
    part 1, raise on error. Returns (m float32 [P], s float32 [P], a int32 [P])."""
    P = n_seq * n_slots * block_len
    dev = hidden.device
    m = torch.empty(P, dtype=torch.float32, device=dev)
    s_ = torch.empty(P, dtype=torch.float32, device=dev)
    a = torch.empty(P, dtype=torch.int32, device=dev)
    rc = bd_lmhead_partials(hidden, shard, shard_scale, vocab_offset, pos_masked, block_flags, n_seq, n_slots,
                            block_len, mask_token_id, m, s_, a, stream=stream, workspace=workspace, variant=variant)
    if rc != BD_OK:
        raise BdError(rc, "bd_lmhead_partials")
    return m, s_, a


def merge_commit(parts_m, parts_s, parts_a, pos_masked, block_flags, n_seq, n_slots, block_len, tau, *,
                 stream=None, counts=False):
    """Allocate the outputs, queue part 2 on [n_parts, P] gathered partials,
    raise on error. Returns (tokens, conf, commit, counts or None) as commit_step."""
    P = n_seq * n_slots * block_len
    n_parts = parts_m.numel() // max(1, P)
    dev = parts_m.device
    tokens = torch.empty(P, dtype=torch.int32, device=dev)
    conf = torch.empty(P, dtype=torch.float32, device=dev)
    commit = torch.empty(P, dtype=torch.int32, device=dev)
    cnt = torch.empty((n_seq, len(tau)), dtype=torch.int32, device=dev) if counts else None
    rc = bd_merge_commit(parts_m, parts_s, parts_a, n_parts, pos_masked, block_flags, n_seq, n_slots, block_len, tau,
                         tokens, conf, commit, stream=stream, out_counts=cnt)
    if rc != BD_OK:
        raise BdError(rc, "bd_merge_commit")
    return tokens, conf, commit, cnt


def bd_static_device_status(stream=None) -> int:
    """Synchronise `stream`, then read and clear the status word of
    bd_commit_step_static's array (BD_OK, or BD_ERR_TIMEOUT after a bounded
    wait of a static call gave up)."""
    return int(load_library().bd_static_device_status(_stream_handle(stream)))


def bd_static_selftest_timeout(stream=None) -> int:
    """Queue the failure-detection self-test against the static array's status word."""
    return int(load_library().bd_static_selftest_timeout(_stream_handle(stream)))


def commit_step(hidden, weight, pos_masked, block_flags, n_seq, n_slots, block_len, tau, *,
                weight_scale=None, mask_token_id=-1, stream=None, workspace=None, counts=False,
                variant=VARIANT_AUTO, lmhead_events=None, fp8_activations=False):
    """Allocate the outputs on the hidden states' device, queue the step, raise on error.

    fp8_activations=True selects the W8A8 variant (an E4M3 head only): the
    packed hidden rows are quantised to E4M3 with one scale per row.

    Returns (tokens int32 [P], conf float32 [P], commit int32 [P] holding the
    uint32 bit masks, counts int32 [n_seq, T] or None)."""
    P = n_seq * n_slots * block_len
    dev = hidden.device
    tokens = torch.empty(P, dtype=torch.int32, device=dev)
    conf = torch.empty(P, dtype=torch.float32, device=dev)
    commit = torch.empty(P, dtype=torch.int32, device=dev)
    cnt = torch.empty((n_seq, len(tau)), dtype=torch.int32, device=dev) if counts else None
    rc = bd_commit_step_ex(hidden, weight, weight_scale, pos_masked, block_flags, n_seq, n_slots, block_len,
                           mask_token_id, tau, tokens, conf, commit, stream=stream, workspace=workspace,
                           out_counts=cnt, lmhead_events=lmhead_events, variant=variant,
                           flags=BD_EXEC_FP8_ACTIVATIONS if fp8_activations else 0)
    if rc != BD_OK:
        raise BdError(rc)
    return tokens, conf, commit, cnt


def bd_commit_sweep(tokens, pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id, step_tokens,
                    step_commit, tau_index, options, out_cache_tokens, out_n_committed, out_n_resolved=None,
                    stream=None) -> int:
    """The block-buffer update after a commit step (include/bdcommit.h); returns the status.
    tokens int32 [P], pos_masked uint8 [P], block_flags uint8 [n_seq * n_slots] are updated in place."""
    win = bd_window(n_seq, n_slots, block_len, mask_token_id, _ptr(tokens), _ptr(pos_masked), _ptr(block_flags))
    return load_library().bd_commit_sweep(ctypes.byref(win), _ptr(step_tokens), _ptr(step_commit), int(tau_index),
                                          int(options), _ptr(out_cache_tokens), _ptr(out_n_committed),
                                          _ptr(out_n_resolved), _stream_handle(stream))


def commit_sweep(tokens, pos_masked, block_flags, n_seq, n_slots, block_len, step_tokens, step_commit, tau_index,
                 *, mask_token_id=-1, options=0, stream=None):
    """Allocate the outputs on the window's device, queue the sweep, raise on error.

    Returns (cache int32 [P]: committed blocks of sequence s at blocks s * n_slots + j, j < n_committed[s];
    n_committed int32 [n_seq]; n_resolved int32 [n_seq])."""
    for t, dt in ((tokens, torch.int32), (pos_masked, torch.uint8), (block_flags, torch.uint8),
                  (step_tokens, torch.int32), (step_commit, torch.int32)):
        if t.dtype != dt or not t.is_contiguous():
            raise ValueError("window and step tensors must be contiguous int32 / uint8 tensors")
    dev = tokens.device
    cache = torch.full((tokens.numel(),), -1, dtype=torch.int32, device=dev)
    n_committed = torch.empty(n_seq, dtype=torch.int32, device=dev)
    n_resolved = torch.empty(n_seq, dtype=torch.int32, device=dev)
    rc = bd_commit_sweep(tokens, pos_masked, block_flags, n_seq, n_slots, block_len, mask_token_id, step_tokens,
                         step_commit, tau_index, options, cache, n_committed, n_resolved, stream=stream)
    if rc != BD_OK:
        raise BdError(rc, "bd_commit_sweep")
    return cache, n_committed, n_resolved


def make_eps_grid(eps: Sequence[float]):
    arr = (c_float * max(1, len(eps)))(*[float(e) for e in eps])
    return bd_eps_grid(ctypes.cast(arr, POINTER(c_float)), len(eps)), arr


def bd_verify_workspace_size(hidden, weight, weight_scale, draft, n_req, n_draft, eps) -> int:
    h, w = make_hidden(hidden), make_weight(weight, weight_scale)
    dr = bd_draft(n_req, n_draft, _ptr(draft))
    eg, _keep = make_eps_grid(eps)
    return int(load_library().bd_verify_workspace_size(ctypes.byref(h), ctypes.byref(w), ctypes.byref(dr),
                                                       ctypes.byref(eg)))


def bd_verify_step(hidden, weight, weight_scale, draft, n_req, n_draft, eps, out_tokens, out_p_draft, out_entropy,
                   out_accept, out_accepted, stream=None, workspace=None, lmhead_events=None, variant=0) -> int:
    """Speculative-decoding verification (include/bdcommit.h); returns the status."""
    h, w = make_hidden(hidden), make_weight(weight, weight_scale)
    dr = bd_draft(n_req, n_draft, _ptr(draft))
    eg, _keep = make_eps_grid(eps)
    ex = bd_exec()
    ex.stream = _stream_handle(stream)
    if workspace is not None:
        ex.workspace = workspace.data_ptr()
        ex.workspace_bytes = workspace.numel() * workspace.element_size()
    if lmhead_events is not None:
        ex.lmhead_event_begin = lmhead_events[0].cuda_event
        ex.lmhead_event_end = lmhead_events[1].cuda_event
    ex.variant = variant
    return load_library().bd_verify_step(ctypes.byref(h), ctypes.byref(w), ctypes.byref(dr), ctypes.byref(eg),
                                         _ptr(out_tokens), _ptr(out_p_draft), _ptr(out_entropy), _ptr(out_accept),
                                         _ptr(out_accepted), ctypes.byref(ex))


def verify_step(hidden, weight, draft, n_req, n_draft, eps, *, weight_scale=None, stream=None, workspace=None,
                variant=VARIANT_AUTO, lmhead_events=None):
    """Allocate the outputs on the hidden states' device, queue the verification, raise on error.

    Returns a dict of tensors: tokens int32 [R], p_draft float32 [R], entropy float32 [R],
    accept int32 [R] (uint32 bit masks), accepted int32 [n_req, E + 1]."""
    R = n_req * (n_draft + 1)
    dev = hidden.device
    out = {"tokens": torch.empty(R, dtype=torch.int32, device=dev),
           "p_draft": torch.empty(R, dtype=torch.float32, device=dev),
           "entropy": torch.empty(R, dtype=torch.float32, device=dev),
           "accept": torch.empty(R, dtype=torch.int32, device=dev),
           "accepted": torch.empty((n_req, len(eps) + 1), dtype=torch.int32, device=dev)}
    rc = bd_verify_step(hidden, weight, weight_scale, draft, n_req, n_draft, eps, out["tokens"], out["p_draft"],
                        out["entropy"], out["accept"], out["accepted"], stream=stream, workspace=workspace,
                        lmhead_events=lmhead_events, variant=variant)
    if rc != BD_OK:
        raise BdError(rc, "bd_verify_step")
    return out
