"""ctypes binding of the Redline entry points of libbdcommit (include/redline.h).

Argument marshalling only: every count, p-value, test and deployment is
computed by the library. Inputs are host arrays (numpy or anything
`numpy.ascontiguousarray` accepts); a nonzero status raises BdError.
"""

from __future__ import annotations

import ctypes
from ctypes import POINTER, c_double, c_int, c_int32, c_int64, c_void_p
from typing import Optional, Sequence

import numpy as np

from .bdcommit import BdError, load_library

BD_REDLINE_HOLM = 0
BD_REDLINE_BONFERRONI = 1
BD_REDLINE_FIXED_SEQUENCE = 2
PROCEDURES = {"holm": BD_REDLINE_HOLM, "bonferroni": BD_REDLINE_BONFERRONI,
              "fixed_sequence": BD_REDLINE_FIXED_SEQUENCE}


class bd_redline_grid(ctypes.Structure):
    _fields_ = [("m", c_int32), ("n", c_int64), ("violations", c_void_p), ("cost", c_void_p),
                ("ref_index", c_int32), ("higher_is_better", c_int32)]


class bd_redline_rule(ctypes.Structure):
    _fields_ = [("delta", c_double), ("procedure", c_int32), ("order", c_void_p)]


_SIG = {
    "bd_binom_cdf": [c_int64, c_int64, c_double, POINTER(c_double)],
    "bd_redline_violations": [c_void_p, c_int64, c_int32, c_int64, c_int32, c_void_p],
    "bd_redline_pvalues": [c_void_p, c_int32, c_int64, c_double, c_void_p],
    "bd_redline_test": [c_void_p, c_int32, POINTER(bd_redline_rule), c_void_p],
    "bd_redline_deploy": [c_void_p, c_void_p, c_int32, c_int32, c_int32, POINTER(c_int32)],
    "bd_redline_select": [POINTER(bd_redline_grid), c_double, POINTER(bd_redline_rule), c_void_p, c_void_p,
                          POINTER(c_int32)],
    "bd_redline_sweep": [POINTER(bd_redline_grid), c_void_p, c_int32, POINTER(bd_redline_rule), c_void_p, c_void_p,
                         POINTER(c_int32)],
    "bd_redline_critical_count": [c_int64, c_double, c_double, POINTER(c_int64)],
    "bd_redline_power": [c_int64, c_double, c_double, c_double, POINTER(c_double)],
    "bd_redline_min_calibration": [c_double, c_double, c_double, c_double, c_int64, POINTER(c_int64)],
    "bd_redline_tpf": [c_void_p, c_int32, c_int32, c_int64, c_int32, c_void_p],
}
_lib = None


def _L():
    global _lib
    if _lib is None:
        lib = load_library()
        for name, args in _SIG.items():
            fn = getattr(lib, name)
            fn.restype = c_int
            fn.argtypes = args
        _lib = lib
    return _lib


def _check(st: int, where: str):
    if st != 0:
        raise BdError(st, where)


def _arr(x, dtype):
    return np.ascontiguousarray(np.asarray(x), dtype=dtype)


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def _rule(delta: float, procedure, order) -> tuple:
    proc = PROCEDURES[procedure] if isinstance(procedure, str) else int(procedure)
    o = None if order is None else _arr(order, np.int32)
    return bd_redline_rule(float(delta), proc, _p(o)), o


def _grid(violations, cost, n: int, ref_index: int, higher_is_better: bool) -> tuple:
    V = _arr(violations, np.int64)
    C = _arr(cost, np.float64)
    if V.ndim != 1 or C.shape != V.shape:
        raise ValueError("violations and cost must be 1-D arrays of one length")
    return bd_redline_grid(V.size, int(n), _p(V), _p(C), int(ref_index), int(bool(higher_is_better))), V, C


def bd_binom_cdf(k: int, n: int, p: float) -> float:
    out = c_double()
    _check(_L().bd_binom_cdf(int(k), int(n), float(p), ctypes.byref(out)), "bd_binom_cdf")
    return out.value


def bd_redline_violations(outcomes, ref_index: int) -> np.ndarray:
    """V per configuration from a [n, m] correctness matrix (nonzero = correct)."""
    O = _arr(outcomes, np.uint8)
    if O.ndim != 2:
        raise ValueError("outcomes must be [n, m]")
    V = np.empty(O.shape[1], dtype=np.int64)
    _check(_L().bd_redline_violations(_p(O), O.shape[0], O.shape[1], O.shape[1], int(ref_index), _p(V)),
           "bd_redline_violations")
    return V


def bd_redline_pvalues(violations, n: int, alpha: float) -> np.ndarray:
    V = _arr(violations, np.int64)
    p = np.empty(V.size, dtype=np.float64)
    _check(_L().bd_redline_pvalues(_p(V), V.size, int(n), float(alpha), _p(p)), "bd_redline_pvalues")
    return p


def bd_redline_test(p, delta: float = 0.10, procedure="holm", order: Optional[Sequence[int]] = None) -> np.ndarray:
    P = _arr(p, np.float64)
    rule, _o = _rule(delta, procedure, order)
    valid = np.empty(P.size, dtype=np.uint8)
    _check(_L().bd_redline_test(_p(P), P.size, ctypes.byref(rule), _p(valid)), "bd_redline_test")
    return valid.astype(bool)


def bd_redline_deploy(valid, cost, ref_index: int, higher_is_better: bool = True) -> int:
    Vd = _arr(valid, np.uint8)
    C = _arr(cost, np.float64)
    out = c_int32()
    _check(_L().bd_redline_deploy(_p(Vd), _p(C), Vd.size, int(bool(higher_is_better)), int(ref_index),
                                  ctypes.byref(out)), "bd_redline_deploy")
    return out.value


def bd_redline_select(violations, cost, n: int, alpha: float, ref_index: int, *, delta: float = 0.10,
                      procedure="holm", order=None, higher_is_better: bool = True) -> dict:
    """Steps (ii)-(iv) at one budget: {'p', 'valid', 'deployed'}."""
    grid, _V, _C = _grid(violations, cost, n, ref_index, higher_is_better)
    rule, _o = _rule(delta, procedure, order)
    p = np.empty(grid.m, dtype=np.float64)
    valid = np.empty(grid.m, dtype=np.uint8)
    dep = c_int32()
    _check(_L().bd_redline_select(ctypes.byref(grid), float(alpha), ctypes.byref(rule), _p(p), _p(valid),
                                  ctypes.byref(dep)), "bd_redline_select")
    return {"p": p, "valid": valid.astype(bool), "deployed": dep.value}


def bd_redline_sweep(violations, cost, n: int, alphas, ref_index: int, *, delta: float = 0.10, procedure="holm",
                     order=None, higher_is_better: bool = True) -> dict:
    """Redline at every budget: {'deployed', 'n_valid', 'first_gain'}."""
    grid, _V, _C = _grid(violations, cost, n, ref_index, higher_is_better)
    rule, _o = _rule(delta, procedure, order)
    A = _arr(alphas, np.float64)
    dep = np.empty(A.size, dtype=np.int32)
    nv = np.empty(A.size, dtype=np.int32)
    fg = c_int32()
    _check(_L().bd_redline_sweep(ctypes.byref(grid), _p(A), A.size, ctypes.byref(rule), _p(dep), _p(nv),
                                 ctypes.byref(fg)), "bd_redline_sweep")
    return {"deployed": dep, "n_valid": nv, "first_gain": fg.value}


def bd_redline_critical_count(n: int, alpha: float, level: float) -> int:
    out = c_int64()
    _check(_L().bd_redline_critical_count(int(n), float(alpha), float(level), ctypes.byref(out)),
           "bd_redline_critical_count")
    return out.value


def bd_redline_power(n: int, risk: float, alpha: float, level: float) -> float:
    out = c_double()
    _check(_L().bd_redline_power(int(n), float(risk), float(alpha), float(level), ctypes.byref(out)),
           "bd_redline_power")
    return out.value


def bd_redline_min_calibration(risk: float, alpha: float, level: float, target: float, n_max: int) -> int:
    out = c_int64()
    _check(_L().bd_redline_min_calibration(float(risk), float(alpha), float(level), float(target), int(n_max),
                                           ctypes.byref(out)), "bd_redline_min_calibration")
    return out.value


def bd_redline_tpf(counts, n_seq: int) -> np.ndarray:
    """TPF per accept threshold from per-forward commit counts [steps, T]."""
    Cn = _arr(counts, np.int32)
    if Cn.ndim != 2:
        raise ValueError("counts must be [steps, T]")
    out = np.empty(Cn.shape[1], dtype=np.float64)
    _check(_L().bd_redline_tpf(_p(Cn), Cn.shape[0], Cn.shape[1], Cn.shape[1], int(n_seq), _p(out)),
           "bd_redline_tpf")
    return out
