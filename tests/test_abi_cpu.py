"""The C-ABI library without a GPU: it builds, loads, exports every symbol
the headers under include/ declare (and nothing else), and its argument
checks reject bad calls before any CUDA call."""

import ctypes
import math
import os
import re
import shutil
import subprocess

import pytest

from paper_2609_33887_gb300 import bdcommit as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INCLUDE = os.path.join(ROOT, "include")
HEADERS = sorted(os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE) if f.endswith(".h"))


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no CUDA toolkit")
    import __graft_entry__

    __graft_entry__.build()
    return B.load_library()


def declared_functions():
    names = set()
    for h in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"^\s*(?:int|size_t|const char\*)\s+(bd_\w+)\s*\(", text, flags=re.M))
    return sorted(names)


def test_header_declares_the_abi():
    assert declared_functions() == sorted([
        "bd_commit_step", "bd_commit_step_ex", "bd_commit_step_static", "bd_commit_sweep", "bd_get_device_status",
        "bd_selftest_timeout", "bd_static_device_status", "bd_static_selftest_timeout", "bd_shutdown",
        "bd_lmhead_partials", "bd_merge_commit",
        "bd_status_string", "bd_version", "bd_workspace_size", "bd_step_kernels", "bd_plan_header", "bd_verify_step", "bd_verify_workspace_size",
        "bd_binom_cdf", "bd_redline_violations", "bd_redline_pvalues", "bd_redline_test", "bd_redline_deploy",
        "bd_redline_select", "bd_redline_sweep", "bd_redline_critical_count", "bd_redline_power",
        "bd_redline_min_calibration", "bd_redline_tpf"])


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_library_exports_nothing_else(lib):
    nm = shutil.which("nm")
    if nm is None:
        pytest.skip("no nm")
    out = subprocess.run([nm, "-D", "--defined-only", B.LIB_PATH], capture_output=True, text=True).stdout
    names = sorted(l.split()[-1] for l in out.splitlines() if " T " in l)
    assert names == declared_functions()


def test_bounds_checked_build_exports_the_same_abi():
    """The bounds-checked variant (-DBD_CHECKS, libbdcommit_checks.so) builds
    and exports exactly the declared C ABI."""
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no CUDA toolkit")
    from paper_2609_33887_gb300 import build as bld

    path = bld.build(checks=True)
    assert os.path.basename(path) == "libbdcommit_checks.so"
    nm = shutil.which("nm")
    if nm is None:
        pytest.skip("no nm")
    out = subprocess.run([nm, "-D", "--defined-only", path], capture_output=True, text=True).stdout
    assert sorted(l.split()[-1] for l in out.splitlines() if " T " in l) == declared_functions()


def test_status_strings_and_version(lib):
    for code in range(-11, 1):
        s = B.bd_status_string(code)
        assert s and s != "unknown status"
    assert B.bd_status_string(-99) == "unknown status"
    assert B.bd_version() == 100


# ----------------------------------------------------- argument checks --
FAKE = 1 << 20  # a non-null, 256-byte aligned address that is never dereferenced


def _args(**kw):
    p = dict(n_seq=2, n_slots=2, L=32, d=128, V=1000, hdt=B.BD_BF16, wdt=B.BD_BF16, mask=-1,
             taus=[0.5, 0.9], hptr=FAKE, wptr=FAKE, scale=None, rows=None, hld=None, wld=None)
    p.update(kw)
    P = p["n_seq"] * p["n_slots"] * p["L"]
    h = B.bd_hidden(p["hptr"], p["hdt"], P if p["rows"] is None else p["rows"], p["d"],
                    p["d"] if p["hld"] is None else p["hld"])
    w = B.bd_weight(p["wptr"], p["wdt"], p["V"], p["d"], p["d"] if p["wld"] is None else p["wld"], p["scale"])
    ms = B.bd_mask_state(p["n_seq"], p["n_slots"], p["L"], p["mask"], FAKE, FAKE)
    arr = (ctypes.c_float * max(1, len(p["taus"])))(*p["taus"])
    tg = B.bd_tau_grid(ctypes.cast(arr, ctypes.POINTER(ctypes.c_float)), len(p["taus"]))
    return h, w, ms, tg, arr


def _call(lib, variant=0, flags=0, outs=(FAKE, FAKE, FAKE), **kw):
    h, w, ms, tg, _keep = _args(**kw)
    ex = B.bd_exec()
    ex.variant = variant
    ex.flags = flags
    return lib.bd_commit_step_ex(ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms), ctypes.byref(tg),
                                 outs[0], outs[1], outs[2], ctypes.byref(ex))


@pytest.mark.parametrize("kw,code", [
    (dict(taus=[]), B.BD_ERR_TAU),
    (dict(taus=[0.1] * 33), B.BD_ERR_TAU),
    (dict(taus=[0.5, math.nan]), B.BD_ERR_TAU),
    (dict(L=65), B.BD_ERR_SHAPE),
    (dict(L=0), B.BD_ERR_SHAPE),
    (dict(rows=100), B.BD_ERR_SHAPE),
    (dict(hld=64), B.BD_ERR_SHAPE),
    (dict(V=0), B.BD_ERR_SHAPE),
    (dict(hdt=B.BD_F32), B.BD_ERR_DTYPE),
    (dict(hdt=B.BD_BF16, wdt=B.BD_F32), B.BD_ERR_DTYPE),
    (dict(hdt=7), B.BD_ERR_DTYPE),
    (dict(wdt=B.BD_E4M3), B.BD_ERR_NULL),
    (dict(mask=1000), B.BD_ERR_ARG),
    (dict(mask=-2), B.BD_ERR_ARG),
    (dict(hptr=FAKE + 2), B.BD_ERR_ALIGN),
    (dict(wptr=FAKE + 8), B.BD_ERR_ALIGN),
    (dict(d=100, hld=100, wld=100), B.BD_ERR_ALIGN),
    (dict(hptr=None), B.BD_ERR_NULL),
])
def test_argument_checks(lib, kw, code):
    assert _call(lib, **kw) == code


def test_variant_flags_and_outputs_checked(lib):
    assert _call(lib, variant=4) == B.BD_ERR_ARG
    assert _call(lib, flags=2) == B.BD_ERR_ARG
    # W8A8 (BD_EXEC_FP8_ACTIVATIONS): E4M3 heads only, on the CTA-pair kernel, rows of 16-byte multiples
    assert _call(lib, flags=B.BD_EXEC_FP8_ACTIVATIONS) == B.BD_ERR_ARG
    e4 = dict(wdt=B.BD_E4M3, scale=FAKE)
    assert _call(lib, flags=B.BD_EXEC_FP8_ACTIVATIONS | 2, **e4) == B.BD_ERR_ARG
    assert _call(lib, variant=2, flags=B.BD_EXEC_FP8_ACTIVATIONS, **e4) == B.BD_ERR_ARG
    assert _call(lib, variant=1, flags=B.BD_EXEC_FP8_ACTIVATIONS, **e4) == B.BD_ERR_ARG
    assert _call(lib, flags=B.BD_EXEC_FP8_ACTIVATIONS, wld=136, **e4) == B.BD_ERR_ALIGN
    assert _call(lib, flags=B.BD_EXEC_FP8_ACTIVATIONS, wptr=FAKE + 8, **e4) == B.BD_ERR_ALIGN
    assert _call(lib, variant=2, hdt=B.BD_F32, wdt=B.BD_F32) == B.BD_ERR_DTYPE
    assert _call(lib, outs=(None, FAKE, FAKE)) == B.BD_ERR_NULL
    assert _call(lib, outs=(FAKE + 1, FAKE, FAKE)) == B.BD_ERR_ALIGN


def test_null_structs_rejected(lib):
    h, w, ms, tg, _keep = _args()
    assert lib.bd_commit_step(None, ctypes.byref(w), ctypes.byref(ms), ctypes.byref(tg), FAKE, FAKE, FAKE) == \
        B.BD_ERR_NULL
    assert lib.bd_workspace_size(ctypes.byref(h), None, ctypes.byref(ms), ctypes.byref(tg)) == 0
    assert lib.bd_step_kernels(ctypes.byref(h), None, ctypes.byref(ms), ctypes.byref(tg), None) == B.BD_ERR_NULL


def test_empty_window_is_a_no_op(lib):
    # zero sequences: nothing to compute, nothing queued, no CUDA call
    assert _call(lib, n_seq=0, hptr=None, wptr=None, outs=(None, None, None)) == B.BD_OK


# ------------------------------------------------ commit sweep argument checks --
def _sweep(lib, n_seq=2, n_slots=4, L=32, tau_index=0, options=0, ptrs=(FAKE,) * 3, step=(FAKE, FAKE),
           cache=FAKE, n_committed=FAKE):
    win = B.bd_window(n_seq, n_slots, L, -1, *ptrs)
    return lib.bd_commit_sweep(ctypes.byref(win), step[0], step[1], tau_index, options, cache, n_committed, None, 0)


@pytest.mark.parametrize("kw,code", [
    (dict(L=0), B.BD_ERR_SHAPE),
    (dict(L=65), B.BD_ERR_SHAPE),
    (dict(n_slots=0), B.BD_ERR_SHAPE),
    (dict(n_slots=65, L=1), B.BD_ERR_SHAPE),
    (dict(n_seq=-1), B.BD_ERR_SHAPE),
    (dict(tau_index=32), B.BD_ERR_ARG),
    (dict(tau_index=-1), B.BD_ERR_ARG),
    (dict(options=4), B.BD_ERR_ARG),
    (dict(ptrs=(None, FAKE, FAKE)), B.BD_ERR_NULL),
    (dict(step=(FAKE, None)), B.BD_ERR_NULL),
    (dict(cache=None), B.BD_ERR_NULL),
    (dict(n_committed=None), B.BD_ERR_NULL),
])
def test_sweep_argument_checks(lib, kw, code):
    assert _sweep(lib, **kw) == code


def test_sweep_empty_window_is_a_no_op(lib):
    assert _sweep(lib, n_seq=0, ptrs=(None, None, None), step=(None, None), cache=None, n_committed=None) == B.BD_OK
    assert lib.bd_commit_sweep(None, FAKE, FAKE, 0, 0, FAKE, FAKE, None, 0) == B.BD_ERR_NULL


# ------------------------------------------------ verification argument checks --
# every case fails a check before any CUDA call (none may reach a launch)
def _verify(lib, n_req=4, n_draft=4, rows=None, eps=(0.1, 0.3), d=128, V=1000, hdt=B.BD_BF16, wdt=B.BD_BF16,
            draft=FAKE, outs=(FAKE,) * 5, counts=None, variant=0, hptr=FAKE):
    R = n_req * (n_draft + 1) if rows is None else rows
    h = B.bd_hidden(hptr, hdt, R, d, d)
    w = B.bd_weight(FAKE, wdt, V, d, d, None)
    dr = B.bd_draft(n_req, n_draft, draft)
    arr = (ctypes.c_float * max(1, len(eps)))(*eps)
    eg = B.bd_eps_grid(ctypes.cast(arr, ctypes.POINTER(ctypes.c_float)), len(eps))
    ex = B.bd_exec()
    ex.variant = variant
    ex.out_counts = counts
    return lib.bd_verify_step(ctypes.byref(h), ctypes.byref(w), ctypes.byref(dr), ctypes.byref(eg), *outs,
                              ctypes.byref(ex))


@pytest.mark.parametrize("kw,code", [
    (dict(eps=()), B.BD_ERR_TAU),
    (dict(eps=(0.1,) * 32), B.BD_ERR_TAU),
    (dict(eps=(0.0,)), B.BD_ERR_TAU),
    (dict(eps=(1.5,)), B.BD_ERR_TAU),
    (dict(eps=(math.nan,)), B.BD_ERR_TAU),
    (dict(n_draft=0), B.BD_ERR_SHAPE),
    (dict(n_draft=33), B.BD_ERR_SHAPE),
    (dict(rows=19), B.BD_ERR_SHAPE),
    (dict(V=0), B.BD_ERR_SHAPE),
    (dict(hdt=B.BD_F32), B.BD_ERR_DTYPE),
    (dict(variant=2, hdt=B.BD_F32, wdt=B.BD_F32), B.BD_ERR_DTYPE),
    (dict(variant=5), B.BD_ERR_ARG),
    (dict(counts=FAKE), B.BD_ERR_ARG),
    (dict(draft=None), B.BD_ERR_NULL),
    (dict(draft=FAKE + 2), B.BD_ERR_ALIGN),
    (dict(hptr=FAKE + 4), B.BD_ERR_ALIGN),
    (dict(outs=(FAKE, FAKE, None, FAKE, FAKE)), B.BD_ERR_NULL),
    (dict(outs=(FAKE, FAKE, FAKE, FAKE + 2, FAKE)), B.BD_ERR_ALIGN),
])
def test_verify_argument_checks(lib, kw, code):
    assert _verify(lib, **kw) == code


def test_verify_empty_batch_is_a_no_op(lib):
    assert _verify(lib, n_req=0, draft=None, hptr=None, outs=(None,) * 5) == B.BD_OK


# ------------------------------------------------------- NVFP4 head checks --
def _nvfp4_call(lib, ld=64, bs=FAKE, bld=4, d=128, hdt=B.BD_BF16, variant=0):
    h, _w, ms, tg, _keep = _args(d=d, hdt=hdt)
    w = B.bd_weight(FAKE, B.BD_NVFP4, 1000, d, ld, None, bs, bld)
    ex = B.bd_exec()
    ex.variant = variant
    return lib.bd_commit_step_ex(ctypes.byref(h), ctypes.byref(w), ctypes.byref(ms), ctypes.byref(tg),
                                 FAKE, FAKE, FAKE, ctypes.byref(ex))


@pytest.mark.parametrize("kw,code", [
    (dict(bs=None), B.BD_ERR_NULL),
    (dict(bld=7, d=128), B.BD_ERR_SHAPE),      # ceil(128 / 16) = 8 scales per row
    (dict(ld=63), B.BD_ERR_SHAPE),             # fewer than ceil(128 / 2) bytes per row
    (dict(ld=72, bld=8), B.BD_ERR_ALIGN),      # row stride not a multiple of 16 bytes
    (dict(hdt=B.BD_F32, bld=8), B.BD_ERR_DTYPE),
])
def test_nvfp4_argument_checks(lib, kw, code):
    assert _nvfp4_call(lib, **kw) == code
