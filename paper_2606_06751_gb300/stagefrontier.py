"""Python binding of libstagefrontier: argument marshalling only.

Each function carries the name of the C entry point it calls and forwards
torch tensors as raw device pointers plus the current CUDA stream; every step
of the computation runs in the library's CUDA kernels.  Torch is used for
device memory and streams only.  Missing output tensors are allocated here
(torch.empty) for convenience.  There is no CPU fallback: importing this
module fails if the shared library cannot be loaded.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libstagefrontier.so")

SF_OK, SF_EINVAL, SF_EINVAL_ALIGN, SF_EUNSUPPORTED, SF_ECUDA, SF_EWORKSPACE = 0, -1, -2, -3, -4, -5
SF_ST_NEGATIVE, SF_ST_RANGE, SF_ST_TIMEOUT, SF_ST_INDEX = 1, 2, 4, 8
SF_STEP_CONFIDENT = 0x80
LABEL_NAMES = ("frontier_accounting", "direct_exposure", "sync_wait_dependent", "co_critical",
               "role_aware_needed", "telemetry_limited", "raw_only")


class SFError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {_lib.sf_status_str(code).decode()} ({code})")
        self.code = code


class Ratio(ctypes.Structure):
    _fields_ = [("num", ctypes.c_int64), ("den", ctypes.c_int64)]


class LabelConfig(ctypes.Structure):
    _fields_ = [(n, Ratio) for n in ("gamma_A", "gamma_G", "eta_A", "eta_G", "tau_C", "eta_Q",
                                     "gamma_switch", "gamma_elig", "closure_max", "overlap_max")] + \
               [("denom_floor_ns", ctypes.c_int64), ("max_missing_ranks", ctypes.c_int32),
                ("model_fit_mask", ctypes.c_uint32)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libstagefrontier.so not built at {LIB_PATH}; run "
                          "`python -m paper_2606_06751_gb300.build`")
    L = ctypes.CDLL(LIB_PATH)
    P, I, I32, S = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p
    sigs = {
        "sf_frontier": [P, I, I, I, P, P, P, P, S],
        "sf_frontier_ties": [P, I, I, I, P, P, P, S],
        "sf_window_aggregate": [P, I, I, I, I, I, P, P, P, P, P, I32, P, S],
        "sf_topk_suspects": [P, P, I, I, I, I32, P, P, P, P, S],
        "sf_window_baselines": [P, I, I, I, I, I, P, P, P, P, I32, P, S],
        "sf_rank_lag": [P, I, I, I, P, P, P, P, ctypes.c_size_t, P, S],
        "sf_rank_lag_windows": [P, I, I, I, I, I, P, P, I32, P, ctypes.c_size_t, P, S],
        "sf_group_aggregate": [P, I, I, I, P, I, I, I, P, P, I32, P, S],
        "sf_stage_group_sum": [P, I, I, P, I, P, S],
        "sf_raw_spread": [P, I, I, I, I, I, P, I32, P, ctypes.c_size_t, P, S],
        "sf_window_median": [P, I, I, I, I, P, P, S],
        "sf_direct_gain": [P, I, I, I, I, P, P, I32, Ratio, P, P, P, P, P, P, P, P, S],
        "sf_label_gates": [I, I, I, I, P, P, P, P, P, P, P, ctypes.POINTER(LabelConfig), P, P, P, P,
                           P, P, P, S],
        "sf_label_windows": [P, I, I, I, I, P, P, P, I32, ctypes.POINTER(LabelConfig), P,
                             ctypes.c_size_t, P, P, P, P, P, P, P, P, P, S],
        "sf_label_windows_noalloc": [P, I, I, I, I, P, P, P, I32, ctypes.POINTER(LabelConfig), P, P, P,
                                     P, P, P, P, P, P, S],
        "sf_stream_windows": [P, I, I, I, I, I32, I, ctypes.POINTER(LabelConfig), P, ctypes.c_size_t, P,
                              ctypes.c_size_t, P, P, P, P, P, P, P, P, P, P, P, P, P, P, S, S],
        "sf_stream_gathered_windows": [P, I, I, I, I, I32, I, ctypes.POINTER(LabelConfig), P, ctypes.c_size_t, P,
                                       ctypes.c_size_t, P, P, P, P, P, P, P, P, P, P, P, P, P, P, S, S],
        "sf_gathered_to_steps": [P, I, I, I, I, P, S],
    }
    for name, argt in sigs.items():
        f = getattr(L, name)
        f.argtypes = argt
        f.restype = ctypes.c_int
    L.sf_status_str.argtypes = [ctypes.c_int]
    L.sf_status_str.restype = ctypes.c_char_p
    L.sf_num_windows.argtypes = [I, I, I]
    L.sf_num_windows.restype = I
    L.sf_selftest_bounded_wait.argtypes = [ctypes.c_uint64, P, S]
    L.sf_selftest_bounded_wait.restype = ctypes.c_int
    L.sf_launch_count.argtypes = []
    L.sf_launch_count.restype = ctypes.c_uint64
    L.sf_label_config_default.argtypes = [ctypes.POINTER(LabelConfig)]
    L.sf_label_config_default.restype = None
    L.sf_label_windows_workspace_size.argtypes = [I, I, I, I]
    L.sf_label_windows_workspace_size.restype = ctypes.c_size_t
    L.sf_rank_workspace_size.argtypes = [I, I, I]
    L.sf_rank_workspace_size.restype = ctypes.c_size_t
    for name in ("sf_stream_windows_staging_size", "sf_stream_gathered_staging_size"):
        getattr(L, name).argtypes = [I, I, I, I]
        getattr(L, name).restype = ctypes.c_size_t
    return L


_lib = _load()


def lib():
    return _lib


def _p(t: Optional[torch.Tensor]):
    return None if t is None else t.data_ptr()


def _stream(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _hold(tensors, *streams):
    """Temporaries the binding allocated for work enqueued on `streams`: the
    caching allocator may reuse their memory only once that work is done."""
    cur = torch.cuda.current_stream()
    for st in streams:
        if st is not None and st != cur:
            for t in tensors:
                if t is not None:
                    t.record_stream(st)


def _check(rc: int, where: str):
    if rc != SF_OK:
        raise SFError(rc, where)


def _dev(t: torch.Tensor, dtype, name: str) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda or t.dtype != dtype or not t.is_contiguous():
        raise TypeError(f"{name} must be a contiguous CUDA tensor of {dtype}")
    return t


def _d3(d: torch.Tensor):
    _dev(d, torch.int64, "d")
    if d.dim() != 3:
        raise ValueError("d must be [T][R][S]")
    return d.shape


def _empty(shape, dtype, like: torch.Tensor):
    return torch.empty(shape, dtype=dtype, device=like.device)


def num_windows(t0: int, T: int, W: int) -> int:
    return int(_lib.sf_num_windows(t0, T, W))


def launch_count() -> int:
    return int(_lib.sf_launch_count())


def default_config() -> LabelConfig:
    c = LabelConfig()
    _lib.sf_label_config_default(ctypes.byref(c))
    return c


def new_status(device) -> torch.Tensor:
    return torch.zeros(1, dtype=torch.int32, device=device)


@dataclass
class Frontier:
    a: Optional[torch.Tensor]
    lead: Optional[torch.Tensor]
    makespan: Optional[torch.Tensor]


def sf_frontier(d, a=None, lead=None, makespan=None, status=None, stream=None, outputs=("a", "lead", "makespan")):
    T, R, S = _d3(d)
    if a is None and "a" in outputs:
        a = _empty((T, S), torch.int64, d)
    if lead is None and "lead" in outputs:
        lead = _empty((T, S), torch.int32, d)
    if makespan is None and "makespan" in outputs:
        makespan = _empty((T,), torch.int64, d)
    _check(_lib.sf_frontier(_p(d), T, R, S, _p(a), _p(lead), _p(makespan), _p(status), _stream(stream)),
           "sf_frontier")
    return Frontier(a, lead, makespan)


def sf_frontier_ties(d, a=None, ties=None, status=None, stream=None):
    """ties[t, s]: how many ranks reach the frontier F[t, s] (Sec. 4's tie set);
    `a` are sf_frontier's increments on the same d (computed here when absent)."""
    T, R, S = _d3(d)
    if a is None:
        a = sf_frontier(d, status=status, stream=stream, outputs=("a",)).a
    ties = ties if ties is not None else _empty((T, S), torch.int32, d)
    _check(_lib.sf_frontier_ties(_p(d), T, R, S, _p(a), _p(ties), _p(status), _stream(stream)),
           "sf_frontier_ties")
    return ties


@dataclass
class Windows:
    X: torch.Tensor
    D: torch.Tensor
    E: Optional[torch.Tensor]
    C: Optional[torch.Tensor]
    step_lead: Optional[torch.Tensor]


def sf_window_aggregate(d, W: int, t0: int = 0, X=None, D=None, E=None, C=None, step_lead=None,
                        accumulate: bool = False, want=("E", "C", "step_lead"), status=None, stream=None):
    T, R, S = _d3(d)
    nW = num_windows(t0, T, W)
    X = X if X is not None else _empty((nW, S), torch.int64, d)
    D = D if D is not None else _empty((nW,), torch.int64, d)
    if E is None and "E" in want:
        E = _empty((nW, S, R), torch.int64, d)
    if C is None and "C" in want:
        C = _empty((nW, S, R), torch.int32, d)
    if step_lead is None and "step_lead" in want:
        step_lead = _empty((T,), torch.uint8, d)
    _check(_lib.sf_window_aggregate(_p(d), T, R, S, t0, W, _p(X), _p(D), _p(E), _p(C), _p(step_lead),
                                    1 if accumulate else 0, _p(status), _stream(stream)),
           "sf_window_aggregate")
    return Windows(X, D, E, C, step_lead)


@dataclass
class TopK:
    stage: torch.Tensor
    stage_value: torch.Tensor
    pair: Optional[torch.Tensor]
    pair_value: Optional[torch.Tensor]


def sf_topk_suspects(X, E, k: int, stream=None, out: Optional[TopK] = None):
    _dev(X, torch.int64, "X")
    nW, S = X.shape
    R = E.shape[2] if E is not None else 1
    if out is None:
        out = TopK(_empty((nW, k), torch.int32, X), _empty((nW, k), torch.int64, X),
                   None if E is None else _empty((nW, k, 2), torch.int32, X),
                   None if E is None else _empty((nW, k), torch.int64, X))
    _check(_lib.sf_topk_suspects(_p(X), _p(E), nW, S, R, k, _p(out.stage), _p(out.stage_value),
                                 _p(out.pair), _p(out.pair_value), _stream(stream)), "sf_topk_suspects")
    return out


def sf_window_median(d, W: int, m=None, status=None, stream=None):
    T, R, S = _d3(d)
    nW = (T + W - 1) // W
    m = m if m is not None else _empty((nW, R, S), torch.int64, d)
    _check(_lib.sf_window_median(_p(d), T, R, S, W, _p(m), _p(status), _stream(stream)), "sf_window_median")
    return m


@dataclass
class Evidence:
    X: torch.Tensor
    Y: torch.Tensor
    D: torch.Tensor
    step_lead: torch.Tensor
    quality: Optional[torch.Tensor]
    E: Optional[torch.Tensor] = None
    C: Optional[torch.Tensor] = None


def sf_direct_gain(d, W: int, m, wall=None, other_stage: int = -1, eta_Q=(1, 20), out: Optional[Evidence] = None,
                   lead_credit: bool = False, status=None, stream=None):
    T, R, S = _d3(d)
    nW = (T + W - 1) // W
    if out is None:
        q = _empty((nW, 6), torch.uint64, d) if (wall is not None or other_stage >= 0) else None
        out = Evidence(_empty((nW, S), torch.int64, d), _empty((nW, S), torch.int64, d),
                       _empty((nW,), torch.int64, d), _empty((T,), torch.uint8, d), q)
        if lead_credit:
            out.E = _empty((nW, S, R), torch.int64, d)
            out.C = _empty((nW, S, R), torch.int32, d)
    _check(_lib.sf_direct_gain(_p(d), T, R, S, W, _p(m), _p(wall), other_stage, Ratio(*eta_Q), _p(out.X),
                               _p(out.Y), _p(out.D), _p(out.E), _p(out.C), _p(out.step_lead), _p(out.quality),
                               _p(status), _stream(stream)), "sf_direct_gain")
    return out


@dataclass
class Labels:
    labels: torch.Tensor
    route_mask: torch.Tensor
    amb_mask: torch.Tensor
    share: torch.Tensor
    gain: torch.Tensor
    n_confident: Optional[torch.Tensor] = None
    n_switch: Optional[torch.Tensor] = None
    X: Optional[torch.Tensor] = None
    Y: Optional[torch.Tensor] = None
    D: Optional[torch.Tensor] = None


def _label_out(nW, S, like):
    return Labels(_empty((nW,), torch.int32, like), _empty((nW,), torch.int32, like),
                  _empty((nW,), torch.int32, like), _empty((nW, S), torch.float64, like),
                  _empty((nW, S), torch.float64, like))


def sf_label_gates(T: int, R: int, S: int, W: int, ev: Evidence, role=None, missing=None, cfg=None,
                   out: Optional[Labels] = None, stream=None):
    nW = (T + W - 1) // W
    cfg = cfg if cfg is not None else default_config()
    if out is None:
        out = _label_out(nW, S, ev.X)
        out.n_confident = _empty((nW,), torch.int32, ev.X)
        out.n_switch = _empty((nW,), torch.int32, ev.X)
    _check(_lib.sf_label_gates(T, R, S, W, _p(ev.X), _p(ev.Y), _p(ev.D), _p(ev.step_lead), _p(ev.quality),
                               _p(role), _p(missing), ctypes.byref(cfg), _p(out.labels), _p(out.route_mask),
                               _p(out.amb_mask), _p(out.share), _p(out.gain), _p(out.n_confident),
                               _p(out.n_switch), _stream(stream)), "sf_label_gates")
    return out


def workspace_size(T: int, R: int, S: int, W: int) -> int:
    return int(_lib.sf_label_windows_workspace_size(T, R, S, W))


def sf_label_windows(d, W: int, role=None, missing=None, wall=None, other_stage: int = -1, cfg=None,
                     workspace=None, out: Optional[Labels] = None, evidence: bool = True, status=None,
                     stream=None):
    T, R, S = _d3(d)
    nW = (T + W - 1) // W
    cfg = cfg if cfg is not None else default_config()
    need = workspace_size(T, R, S, W)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=d.device)
        _hold([workspace], stream)
    if out is None:
        out = _label_out(nW, S, d)
        if evidence:
            out.X = _empty((nW, S), torch.int64, d)
            out.Y = _empty((nW, S), torch.int64, d)
            out.D = _empty((nW,), torch.int64, d)
    _check(_lib.sf_label_windows(_p(d), T, R, S, W, _p(role), _p(missing), _p(wall), other_stage,
                                 ctypes.byref(cfg), _p(workspace), workspace.numel(), _p(out.labels),
                                 _p(out.route_mask), _p(out.amb_mask), _p(out.share), _p(out.gain),
                                 _p(out.X), _p(out.Y), _p(out.D), _p(status), _stream(stream)),
           "sf_label_windows")
    return out


STATIC_SCRATCH_BYTES = 16 * 1024 * 1024


def sf_label_windows_noalloc(d, W: int, role=None, missing=None, wall=None, other_stage: int = -1,
                             cfg=None, out: Labels = None, status=None, stream=None):
    """The labeler with its intermediates in the library's static device
    scratch (no workspace; the outputs are still the caller's tensors)."""
    T, R, S = _d3(d)
    cfg = cfg if cfg is not None else default_config()
    if out is None:
        raise ValueError("pass preallocated outputs (Labels with X, Y, D) to the no-allocation entry point")
    _check(_lib.sf_label_windows_noalloc(_p(d), T, R, S, W, _p(role), _p(missing), _p(wall), other_stage,
                                         ctypes.byref(cfg), _p(out.labels), _p(out.route_mask),
                                         _p(out.amb_mask), _p(out.share), _p(out.gain), _p(out.X),
                                         _p(out.Y), _p(out.D), _p(status), _stream(stream)),
           "sf_label_windows_noalloc")
    return out


@dataclass
class Streamed:
    X: torch.Tensor
    Y: torch.Tensor
    D: torch.Tensor
    E: Optional[torch.Tensor]
    C: Optional[torch.Tensor]
    top_stage: torch.Tensor
    top_pair: Optional[torch.Tensor]
    top_pair_value: Optional[torch.Tensor]
    labels: torch.Tensor
    route_mask: torch.Tensor
    amb_mask: torch.Tensor
    share: torch.Tensor
    gain: torch.Tensor


class StreamBuffers:
    """Device staging, workspace and outputs for sf_stream_windows, reusable across calls."""

    def __init__(self, T: int, R: int, S: int, W: int, k: int, chunk_steps: int, device, lead_credit=True,
                 gathered=False):
        nW = (T + W - 1) // W
        e = lambda shape, dt: torch.empty(shape, dtype=dt, device=device)  # noqa: E731
        self.shape = (T, R, S, W, k, chunk_steps)
        size = _lib.sf_stream_gathered_staging_size if gathered else _lib.sf_stream_windows_staging_size
        self.staging = e((int(size(T, R, S, chunk_steps)),), torch.uint8)
        self.workspace = e((workspace_size(min(chunk_steps, T), R, S, W),), torch.uint8)
        self.out = Streamed(e((nW, S), torch.int64), e((nW, S), torch.int64), e((nW,), torch.int64),
                            e((nW, S, R), torch.int64) if lead_credit else None,
                            e((nW, S, R), torch.int32) if lead_credit else None,
                            e((nW, k), torch.int32), e((nW, k, 2), torch.int32) if lead_credit else None,
                            e((nW, k), torch.int64) if lead_credit else None,
                            e((nW,), torch.int32), e((nW,), torch.int32), e((nW,), torch.int32),
                            e((nW, S), torch.float64), e((nW, S), torch.float64))


def sf_stream_windows(h_d: torch.Tensor, W: int, k: int, chunk_steps: int, bufs: StreamBuffers = None,
                      cfg=None, status=None, stream=None, copy_stream=None) -> Streamed:
    """h_d: [T][R][S] int64 CPU tensor (pin it for copy/compute overlap)."""
    if h_d.is_cuda or h_d.dtype != torch.int64 or not h_d.is_contiguous() or h_d.dim() != 3:
        raise TypeError("h_d must be a contiguous [T][R][S] int64 host tensor")
    T, R, S = h_d.shape
    cfg = cfg if cfg is not None else default_config()
    dev = torch.device("cuda", torch.cuda.current_device())
    cs = copy_stream if copy_stream is not None else (stream if stream is not None else torch.cuda.current_stream())
    if bufs is None:
        # staging and workspace are used by both streams: keep them until that work is done
        bufs = StreamBuffers(T, R, S, W, k, chunk_steps, dev)
        _hold([bufs.staging, bufs.workspace], cs, stream)
    o = bufs.out
    _check(_lib.sf_stream_windows(h_d.data_ptr(), T, R, S, W, k, chunk_steps, ctypes.byref(cfg),
                                  _p(bufs.staging), bufs.staging.numel(), _p(bufs.workspace), bufs.workspace.numel(),
                                  _p(o.X), _p(o.Y), _p(o.D), _p(o.E), _p(o.C), _p(o.top_stage), _p(o.top_pair),
                                  _p(o.top_pair_value), _p(o.labels), _p(o.route_mask), _p(o.amb_mask), _p(o.share),
                                  _p(o.gain), _p(status), _stream(stream), cs.cuda_stream), "sf_stream_windows")
    return o


def sf_selftest_bounded_wait(limit_ns: int, status: torch.Tensor, stream=None):
    _check(_lib.sf_selftest_bounded_wait(limit_ns, _p(status), _stream(stream)), "sf_selftest_bounded_wait")


@dataclass
class Baselines:
    M: torch.Tensor      # [nW][S] sum_t max_r d
    SUM: torch.Tensor    # [nW][S][2] uint64 (lo, hi) of sum_t sum_r d
    SLOW: torch.Tensor   # [nW][S] slowest-rank breakdown
    RANK0: torch.Tensor  # [nW][S] rank-0 local total


def sf_window_baselines(d, W: int, t0: int = 0, out: Optional[Baselines] = None, accumulate: bool = False,
                        status=None, stream=None) -> Baselines:
    T, R, S = _d3(d)
    nW = num_windows(t0, T, W)
    if out is None:
        out = Baselines(_empty((nW, S), torch.int64, d), _empty((nW, S, 2), torch.uint64, d),
                        _empty((nW, S), torch.int64, d), _empty((nW, S), torch.int64, d))
    _check(_lib.sf_window_baselines(_p(d), T, R, S, t0, W, _p(out.M), _p(out.SUM), _p(out.SLOW), _p(out.RANK0),
                                    1 if accumulate else 0, _p(status), _stream(stream)), "sf_window_baselines")
    return out


@dataclass
class Lag:
    L: Optional[torch.Tensor]   # [T][S] F - median_r P
    dL: Optional[torch.Tensor]  # [T][S] increment of the lag over stages
    G: Optional[torch.Tensor]   # [T][S] max-minus-second-max gap


def rank_workspace(T: int, R: int, S: int, device) -> torch.Tensor:
    """Device scratch for sf_rank_lag / sf_raw_spread (reusable across calls)."""
    return torch.empty(int(_lib.sf_rank_workspace_size(T, R, S)), dtype=torch.uint8, device=device)


def sf_rank_lag(d, out: Optional[Lag] = None, workspace=None, status=None, stream=None) -> Lag:
    T, R, S = _d3(d)
    if out is None:
        out = Lag(_empty((T, S), torch.int64, d), _empty((T, S), torch.int64, d), _empty((T, S), torch.int64, d))
    ws = workspace
    if ws is None:
        ws = rank_workspace(T, R, S, d.device)
        _hold([ws], stream)
    _check(_lib.sf_rank_lag(_p(d), T, R, S, _p(out.L), _p(out.dL), _p(out.G), _p(ws), ws.numel(), _p(status),
                            _stream(stream)), "sf_rank_lag")
    return out


def sf_raw_spread(d, W: int, t0: int = 0, spread=None, accumulate: bool = False, workspace=None, status=None,
                  stream=None):
    T, R, S = _d3(d)
    spread = spread if spread is not None else _empty((num_windows(t0, T, W), S), torch.int64, d)
    ws = workspace
    if ws is None:
        ws = rank_workspace(T, R, S, d.device)
        _hold([ws], stream)
    _check(_lib.sf_raw_spread(_p(d), T, R, S, t0, W, _p(spread), 1 if accumulate else 0, _p(ws), ws.numel(),
                              _p(status), _stream(stream)), "sf_raw_spread")
    return spread


@dataclass
class GroupWindows:
    X: torch.Tensor  # [nW][G][S] sums of the group frontier's increments
    D: torch.Tensor  # [nW][G] sums of the group makespans


def sf_group_aggregate(d, group, G: int, W: int, t0: int = 0, out: Optional[GroupWindows] = None,
                       accumulate: bool = False, status=None, stream=None) -> GroupWindows:
    T, R, S = _d3(d)
    group = _dev(group, torch.int32, "group")
    nW = num_windows(t0, T, W)
    if out is None:
        out = GroupWindows(_empty((nW, G, S), torch.int64, d), _empty((nW, G), torch.int64, d))
    _check(_lib.sf_group_aggregate(_p(d), T, R, S, _p(group), G, t0, W, _p(out.X), _p(out.D),
                                   1 if accumulate else 0, _p(status), _stream(stream)), "sf_group_aggregate")
    return out


def sf_stage_group_sum(X, stage_group, K: int, Y=None, stream=None):
    """stage_group: a host sequence of S group ids in [0, K)."""
    nW, S = X.shape
    sg = (ctypes.c_int32 * S)(*[int(v) for v in stage_group])
    Y = Y if Y is not None else _empty((nW, K), torch.int64, X)
    _check(_lib.sf_stage_group_sum(_p(X), nW, S, sg, K, _p(Y), _stream(stream)), "sf_stage_group_sum")
    return Y


def sf_stream_gathered_windows(h_g: torch.Tensor, T: int, R: int, S: int, W: int, k: int, chunk_steps: int,
                               bufs: StreamBuffers = None, cfg=None, status=None, stream=None,
                               copy_stream=None) -> Streamed:
    """h_g: int64 CPU tensor holding the windows' gathered [R][n][S] blocks one
    after another (T*R*S values; pin it for copy/compute overlap)."""
    if h_g.is_cuda or h_g.dtype != torch.int64 or not h_g.is_contiguous() or h_g.numel() != T * R * S:
        raise TypeError("h_g must be a contiguous int64 host tensor of T*R*S values")
    cfg = cfg if cfg is not None else default_config()
    dev = torch.device("cuda", torch.cuda.current_device())
    cs = copy_stream if copy_stream is not None else (stream if stream is not None else torch.cuda.current_stream())
    if bufs is None:
        bufs = StreamBuffers(T, R, S, W, k, chunk_steps, dev, gathered=True)
        _hold([bufs.staging, bufs.workspace], cs, stream)
    o = bufs.out
    _check(_lib.sf_stream_gathered_windows(h_g.data_ptr(), T, R, S, W, k, chunk_steps, ctypes.byref(cfg),
                                           _p(bufs.staging), bufs.staging.numel(), _p(bufs.workspace),
                                           bufs.workspace.numel(), _p(o.X), _p(o.Y), _p(o.D), _p(o.E), _p(o.C),
                                           _p(o.top_stage), _p(o.top_pair), _p(o.top_pair_value), _p(o.labels),
                                           _p(o.route_mask), _p(o.amb_mask), _p(o.share), _p(o.gain), _p(status),
                                           _stream(stream), cs.cuda_stream), "sf_stream_gathered_windows")
    return o


def sf_gathered_to_steps(src: torch.Tensor, T: int, R: int, S: int, N: int, dst=None, stream=None):
    """src: device int64 holding ceil(T/N) gathered [R][n][S] blocks; returns [T][R][S]."""
    if not src.is_cuda or src.dtype != torch.int64 or not src.is_contiguous() or src.numel() != T * R * S:
        raise TypeError("src must be a contiguous int64 CUDA tensor of T*R*S values")
    dst = dst if dst is not None else torch.empty((T, R, S), dtype=torch.int64, device=src.device)
    _check(_lib.sf_gathered_to_steps(_p(src), T, R, S, N, _p(dst), _stream(stream)), "sf_gathered_to_steps")
    return dst


def sf_rank_lag_windows(d, W: int, t0: int = 0, Lw=None, Gw=None, accumulate: bool = False, workspace=None,
                        status=None, stream=None):
    """Window sums of the lag and the gap: (Lw, Gw), each [nW][S]."""
    T, R, S = _d3(d)
    nW = num_windows(t0, T, W)
    Lw = Lw if Lw is not None else _empty((nW, S), torch.int64, d)
    Gw = Gw if Gw is not None else _empty((nW, S), torch.int64, d)
    ws = workspace
    if ws is None:
        ws = rank_workspace(T, R, S, d.device)
        _hold([ws], stream)
    _check(_lib.sf_rank_lag_windows(_p(d), T, R, S, t0, W, _p(Lw), _p(Gw), 1 if accumulate else 0, _p(ws),
                                    ws.numel(), _p(status), _stream(stream)), "sf_rank_lag_windows")
    return Lw, Gw
