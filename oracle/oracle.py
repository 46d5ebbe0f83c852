"""CPU oracle for frontier accounting -- TEST INFRASTRUCTURE.

Thin numpy wrapper over ``sforacle.c``, the literal restatement of the
paper's definitions (Sec. 3 Eq. 1-2, Sec. 4 Eq. 4, App. A-C).  Only the test
suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg may
import this module; the product path never does.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libsforacle.so")

OK, NEGATIVE, RANGE, BADARG = 0, 1, 2, 3

L_FRONTIER_ACCOUNTING = 1 << 0
L_DIRECT_EXPOSURE = 1 << 1
L_SYNC_WAIT_DEPENDENT = 1 << 2
L_CO_CRITICAL = 1 << 3
L_ROLE_AWARE_NEEDED = 1 << 4
L_TELEMETRY_LIMITED = 1 << 5
L_RAW_ONLY = 1 << 6


class OracleError(RuntimeError):
    def __init__(self, rc: int):
        super().__init__({NEGATIVE: "negative duration", RANGE: "value out of range",
                          BADARG: "bad arguments"}.get(rc, f"error {rc}"))
        self.rc = rc


class _Ratio(ctypes.Structure):
    _fields_ = [("num", ctypes.c_int64), ("den", ctypes.c_int64)]


class Config(ctypes.Structure):
    _fields_ = [(n, _Ratio) for n in ("gamma_A", "gamma_G", "eta_A", "eta_G", "tau_C", "eta_Q",
                                      "gamma_switch", "gamma_elig", "closure_max", "overlap_max")] + \
               [("denom_floor_ns", ctypes.c_int64), ("max_missing_ranks", ctypes.c_int32),
                ("model_fit_mask", ctypes.c_uint32)]


def build_lib(force: bool = False) -> str:
    src = os.path.join(_HERE, "sforacle.c")
    hdr = os.path.join(_HERE, "sforacle.h")
    newest = max(os.path.getmtime(src), os.path.getmtime(hdr))
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < newest:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-fPIC", "-shared", "-o", tmp, src], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int64


def lib():
    global _lib
    if _lib is None:
        build_lib()
        L = ctypes.CDLL(_LIB_PATH)
        L.sfo_frontier.argtypes = [_P, _I, _I, _I, _P, _P, _P, _P, _P]
        L.sfo_windows.argtypes = [_P, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P]
        L.sfo_topk.argtypes = [_P, _P, _I, _I, _I, ctypes.c_int32, _P, _P, _P, _P]
        L.sfo_window_median.argtypes = [_P, _I, _I, _I, _I, _P]
        L.sfo_direct_gain.argtypes = [_P, _I, _I, _I, _I, _P, _P]
        L.sfo_label_windows.argtypes = [_P, _I, _I, _I, _I, _P, _P, _P, ctypes.c_int32,
                                        ctypes.POINTER(Config), _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                        _P, _P]
        L.sfo_baselines.argtypes = [_P, _I, _I, _I, _I, _I, _P, _P, _P, _P]
        L.sfo_baselines.restype = ctypes.c_int
        L.sfo_rank_lag.argtypes = [_P, _I, _I, _I, _P, _P, _P]
        L.sfo_rank_lag.restype = ctypes.c_int
        L.sfo_raw_spread.argtypes = [_P, _I, _I, _I, _I, _I, _P]
        L.sfo_rank_lag_windows.argtypes = [_P, _I, _I, _I, _I, _I, _P, _P]
        L.sfo_rank_lag_windows.restype = ctypes.c_int
        L.sfo_raw_spread.restype = ctypes.c_int
        L.sfo_group_windows.argtypes = [_P, _I, _I, _I, _P, _I, _I, _I, _P, _P]
        L.sfo_group_windows.restype = ctypes.c_int
        L.sfo_stage_group_sum.argtypes = [_P, _I, _I, _P, _I, _P]
        L.sfo_stage_group_sum.restype = ctypes.c_int
        L.sfo_config_default.argtypes = [ctypes.POINTER(Config)]
        for f in ("sfo_frontier", "sfo_windows", "sfo_topk", "sfo_window_median", "sfo_direct_gain",
                  "sfo_label_windows"):
            getattr(L, f).restype = ctypes.c_int
        L.sfo_config_default.restype = None
        _lib = L
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def _check(rc: int):
    if rc != OK:
        raise OracleError(rc)


def _d(d) -> np.ndarray:
    d = np.ascontiguousarray(d, dtype=np.int64)
    assert d.ndim == 3, "d must be [T][R][S]"
    return d


def default_config() -> Config:
    c = Config()
    lib().sfo_config_default(ctypes.byref(c))
    return c


@dataclass
class Frontier:
    F: np.ndarray      # [T][S] frontier F_{t,s}
    a: np.ndarray      # [T][S] increments a_{t,s}
    lead: np.ndarray   # [T][S] lowest rank attaining F_{t,s}
    ties: np.ndarray   # [T][S] number of ranks attaining F_{t,s}
    makespan: np.ndarray  # [T] F_{t,S}


def frontier(d) -> Frontier:
    """Sec. 3 Eq. 1 on every step of d[T][R][S]."""
    d = _d(d)
    T, R, S = d.shape
    F = np.empty((T, S), np.int64)
    a = np.empty((T, S), np.int64)
    lead = np.empty((T, S), np.int32)
    ties = np.empty((T, S), np.int32)
    mk = np.empty(T, np.int64)
    _check(lib().sfo_frontier(_ptr(d), T, R, S, _ptr(F), _ptr(a), _ptr(lead), _ptr(ties), _ptr(mk)))
    return Frontier(F, a, lead, ties, mk)


def num_windows(t0: int, T: int, W: int) -> int:
    return (t0 + T - 1) // W - t0 // W + 1


@dataclass
class Windows:
    X: np.ndarray   # [nW][S]
    D: np.ndarray   # [nW]
    E: np.ndarray   # [nW][S][R]
    C: np.ndarray   # [nW][S][R]
    step_lead: np.ndarray  # [T] uint8


def windows(d, W: int, t0: int = 0) -> Windows:
    """Sec. 3 Eq. 2 numerators/denominators and lead-rank credit per window."""
    d = _d(d)
    T, R, S = d.shape
    nW = num_windows(t0, T, W)
    X = np.empty((nW, S), np.int64)
    D = np.empty(nW, np.int64)
    E = np.empty((nW, S, R), np.int64)
    C = np.empty((nW, S, R), np.int32)
    sl = np.empty(T, np.uint8)
    _check(lib().sfo_windows(_ptr(d), T, R, S, t0, W, _ptr(X), _ptr(D), _ptr(E), _ptr(C), _ptr(sl)))
    return Windows(X, D, E, C, sl)


@dataclass
class TopK:
    stage: np.ndarray        # [nW][k]
    stage_value: np.ndarray  # [nW][k]
    pair: np.ndarray         # [nW][k][2] (stage, rank)
    pair_value: np.ndarray   # [nW][k]


def topk(X, E, k: int) -> TopK:
    X = np.ascontiguousarray(X, dtype=np.int64)
    E = np.ascontiguousarray(E, dtype=np.int64)
    nW, S = X.shape
    R = E.shape[2]
    st = np.empty((nW, k), np.int32)
    sv = np.empty((nW, k), np.int64)
    pr = np.empty((nW, k, 2), np.int32)
    pv = np.empty((nW, k), np.int64)
    _check(lib().sfo_topk(_ptr(X), _ptr(E), nW, S, R, k, _ptr(st), _ptr(sv), _ptr(pr), _ptr(pv)))
    return TopK(st, sv, pr, pv)


def window_median(d, W: int) -> np.ndarray:
    d = _d(d)
    T, R, S = d.shape
    nW = (T + W - 1) // W
    m = np.empty((nW, R, S), np.int64)
    _check(lib().sfo_window_median(_ptr(d), T, R, S, W, _ptr(m)))
    return m


def direct_gain(d, W: int, m) -> np.ndarray:
    d = _d(d)
    T, R, S = d.shape
    nW = (T + W - 1) // W
    m = np.ascontiguousarray(m, dtype=np.int64)
    Y = np.empty((nW, S), np.int64)
    _check(lib().sfo_direct_gain(_ptr(d), T, R, S, W, _ptr(m), _ptr(Y)))
    return Y


@dataclass
class Labels:
    labels: np.ndarray      # [nW] uint32 bitmask
    route_mask: np.ndarray  # [nW] uint32
    amb_mask: np.ndarray    # [nW] uint32
    share: np.ndarray       # [nW][S] fp64
    gain: np.ndarray        # [nW][S] fp64
    X: np.ndarray
    D: np.ndarray
    Y: np.ndarray
    m: np.ndarray
    n_confident: np.ndarray
    n_switch: np.ndarray


def label_windows(d, W: int, role=None, missing=None, wall=None, other_stage: int = -1,
                  cfg: Optional[Config] = None) -> Labels:
    d = _d(d)
    T, R, S = d.shape
    nW = (T + W - 1) // W
    cfg = cfg if cfg is not None else default_config()
    role = None if role is None else np.ascontiguousarray(role, dtype=np.int32)
    missing = None if missing is None else np.ascontiguousarray(missing, dtype=np.int32)
    wall = None if wall is None else np.ascontiguousarray(wall, dtype=np.int64)
    out = Labels(np.empty(nW, np.uint32), np.empty(nW, np.uint32), np.empty(nW, np.uint32),
                 np.empty((nW, S)), np.empty((nW, S)), np.empty((nW, S), np.int64),
                 np.empty(nW, np.int64), np.empty((nW, S), np.int64), np.empty((nW, R, S), np.int64),
                 np.empty(nW, np.int32), np.empty(nW, np.int32))
    _check(lib().sfo_label_windows(_ptr(d), T, R, S, W, _ptr(role), _ptr(missing), _ptr(wall),
                                   other_stage, ctypes.byref(cfg), _ptr(out.labels),
                                   _ptr(out.route_mask), _ptr(out.amb_mask), _ptr(out.share),
                                   _ptr(out.gain), _ptr(out.X), _ptr(out.D), _ptr(out.Y),
                                   _ptr(out.m), _ptr(out.n_confident), _ptr(out.n_switch)))
    return out


@dataclass
class Baselines:
    M: np.ndarray      # [nW][S] sum_t max_r d
    SUM: np.ndarray    # [nW][S] sum_t sum_r d (Python ints, exact)
    SLOW: np.ndarray   # [nW][S] slowest-rank breakdown
    RANK0: np.ndarray  # [nW][S] rank-0 local total


def baselines(d, W: int, t0: int = 0) -> Baselines:
    """Routing baselines of Sec. 3 (per-stage max / average) and Sec. 6."""
    d = _d(d)
    T, R, S = d.shape
    nW = num_windows(t0, T, W)
    M = np.empty((nW, S), np.int64)
    SUM = np.empty((nW, S, 2), np.uint64)
    SLOW = np.empty((nW, S), np.int64)
    R0 = np.empty((nW, S), np.int64)
    _check(lib().sfo_baselines(_ptr(d), T, R, S, t0, W, _ptr(M), _ptr(SUM), _ptr(SLOW), _ptr(R0)))
    total = np.array([[int(SUM[w, s, 1]) << 64 | int(SUM[w, s, 0]) for s in range(S)] for w in range(nW)],
                     dtype=object)
    return Baselines(M, total, SLOW, R0)


@dataclass
class Lag:
    L: np.ndarray   # [T][S] F - median_r P
    dL: np.ndarray  # [T][S] increment of L over stages
    G: np.ndarray   # [T][S] max-minus-second-max gap


def rank_lag(d) -> Lag:
    """Sec. 4 localization evidence per step and stage."""
    d = _d(d)
    T, R, S = d.shape
    out = Lag(np.empty((T, S), np.int64), np.empty((T, S), np.int64), np.empty((T, S), np.int64))
    _check(lib().sfo_rank_lag(_ptr(d), T, R, S, _ptr(out.L), _ptr(out.dL), _ptr(out.G)))
    return out


def raw_spread(d, W: int, t0: int = 0) -> np.ndarray:
    """Sec. 6 raw rank spread per window and stage."""
    d = _d(d)
    T, R, S = d.shape
    out = np.empty((num_windows(t0, T, W), S), np.int64)
    _check(lib().sfo_raw_spread(_ptr(d), T, R, S, t0, W, _ptr(out)))
    return out


@dataclass
class GroupWindows:
    X: np.ndarray  # [G][nW][S] sum of the group frontier's increments
    D: np.ndarray  # [G][nW] sum of the group makespans


def group_windows(d, group, G: int, W: int, t0: int = 0) -> GroupWindows:
    """Frontier within role groups (App. A role check, Sec. 3 Eq. 1 per group)."""
    d = _d(d)
    T, R, S = d.shape
    group = np.ascontiguousarray(group, dtype=np.int32)
    assert group.shape == (R,)
    nW = num_windows(t0, T, W)
    out = GroupWindows(np.empty((G, nW, S), np.int64), np.empty((G, nW), np.int64))
    _check(lib().sfo_group_windows(_ptr(d), T, R, S, _ptr(group), G, t0, W, _ptr(out.X), _ptr(out.D)))
    return out


def stage_group_sum(X, stage_group, K: int) -> np.ndarray:
    """Reporting groups aggregated after the frontier (Sec. 3)."""
    X = np.ascontiguousarray(X, dtype=np.int64)
    nW, S = X.shape
    stage_group = np.ascontiguousarray(stage_group, dtype=np.int32)
    assert stage_group.shape == (S,)
    Y = np.empty((nW, K), np.int64)
    _check(lib().sfo_stage_group_sum(_ptr(X), nW, S, _ptr(stage_group), K, _ptr(Y)))
    return Y


def rank_lag_windows(d, W: int, t0: int = 0):
    """Sec. 4 lag evidence summed per window: (LW, GW), each [nW][S]."""
    d = _d(d)
    T, R, S = d.shape
    nW = num_windows(t0, T, W)
    LW = np.empty((nW, S), np.int64)
    GW = np.empty((nW, S), np.int64)
    _check(lib().sfo_rank_lag_windows(_ptr(d), T, R, S, t0, W, _ptr(LW), _ptr(GW)))
    return LW, GW
