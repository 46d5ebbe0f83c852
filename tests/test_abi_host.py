"""The C ABI library without a GPU: it loads, exports every declared entry
point, and rejects bad arguments on the host before touching CUDA."""
import ctypes
import os
import re

import pytest

from paper_2606_06751_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def sf():
    B.build()
    from paper_2606_06751_gb300 import stagefrontier
    return stagefrontier


def declared_symbols():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            txt = open(os.path.join(inc, f)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names |= set(re.findall(r"\b(sf_[a-z0-9_]+)\s*\(", txt))
    return names


def test_exports_every_declared_symbol(sf):
    syms = declared_symbols()
    assert {"sf_frontier", "sf_window_aggregate", "sf_topk_suspects", "sf_label_windows"} <= syms
    lib = ctypes.CDLL(sf.LIB_PATH)
    missing = [s for s in sorted(syms) if not hasattr(lib, s)]
    assert not missing, missing


def test_status_strings_and_helpers(sf):
    L = sf.lib()
    assert L.sf_status_str(0) == b"ok"
    assert L.sf_status_str(-5).startswith(b"workspace")
    assert sf.num_windows(0, 100, 10) == 10
    assert sf.num_windows(5, 37, 7) == 6
    assert sf.num_windows(0, 0, 7) == 0
    c = sf.default_config()
    assert (c.gamma_A.num, c.gamma_A.den) == (2, 5) and (c.tau_C.num, c.tau_C.den) == (4, 5)
    assert L.sf_label_windows_workspace_size(1000, 8, 6, 100) > 10 * 8 * 6 * 8
    assert L.sf_label_windows_workspace_size(0, 8, 6, 100) == 0


FAKE = 1 << 20  # a well-aligned address that is never dereferenced: every call below fails validation


def test_host_validation(sf):
    L = sf.lib()
    # tie-set sizes: null d / a / ties, bad shape, misaligned d
    assert L.sf_frontier_ties(None, 10, 4, 4, FAKE, FAKE, None, None) == sf.SF_EINVAL
    assert L.sf_frontier_ties(FAKE, 10, 4, 4, None, FAKE, None, None) == sf.SF_EINVAL
    assert L.sf_frontier_ties(FAKE, 10, 4, 4, FAKE, None, None, None) == sf.SF_EINVAL
    assert L.sf_frontier_ties(FAKE, 0, 4, 4, FAKE, FAKE, None, None) == sf.SF_EINVAL
    assert L.sf_frontier_ties(FAKE + 8, 10, 4, 4, FAKE, FAKE, None, None) == sf.SF_EINVAL_ALIGN
    # null input, bad shapes, no outputs
    assert L.sf_frontier(None, 10, 4, 4, FAKE, None, None, None, None) == sf.SF_EINVAL
    assert L.sf_frontier(FAKE, 0, 4, 4, FAKE, None, None, None, None) == sf.SF_EINVAL
    assert L.sf_frontier(FAKE, 10, 65537, 4, FAKE, None, None, None, None) == sf.SF_EINVAL
    assert L.sf_frontier(FAKE, 10, 4, 33, FAKE, None, None, None, None) == sf.SF_EINVAL
    assert L.sf_frontier(FAKE, 10, 4, 4, None, None, None, None, None) == sf.SF_EINVAL
    # alignment
    assert L.sf_frontier(FAKE + 8, 10, 4, 4, FAKE, None, None, None, None) == sf.SF_EINVAL_ALIGN
    assert L.sf_frontier(FAKE, 10, 4, 4, FAKE + 4, None, None, None, None) == sf.SF_EINVAL_ALIGN
    # window aggregate: W out of range, accumulate flag, missing X
    agg = L.sf_window_aggregate
    assert agg(FAKE, 10, 4, 4, 0, 0, FAKE, FAKE, None, None, None, 0, None, None) == sf.SF_EINVAL
    assert agg(FAKE, 10, 4, 4, 0, 65537, FAKE, FAKE, None, None, None, 0, None, None) == sf.SF_EINVAL
    assert agg(FAKE, 10, 4, 4, 0, 5, FAKE, FAKE, None, None, None, 2, None, None) == sf.SF_EINVAL
    assert agg(FAKE, 10, 4, 4, -1, 5, FAKE, FAKE, None, None, None, 0, None, None) == sf.SF_EINVAL
    assert agg(FAKE, 10, 4, 4, 0, 5, None, FAKE, None, None, None, 0, None, None) == sf.SF_EINVAL
    # top-k: k range, pairs without E
    assert L.sf_topk_suspects(FAKE, FAKE, 3, 4, 4, 0, FAKE, None, None, None, None) == sf.SF_EINVAL
    assert L.sf_topk_suspects(FAKE, FAKE, 3, 4, 4, 33, FAKE, None, None, None, None) == sf.SF_EINVAL
    assert L.sf_topk_suspects(FAKE, None, 3, 4, 4, 2, None, None, FAKE, None, None) == sf.SF_EINVAL
    # labeler: bad config, workspace too small or misaligned
    cfg = sf.default_config()
    bad = sf.default_config()
    bad.tau_C.den = 0
    lw = L.sf_label_windows
    assert lw(FAKE, 10, 4, 4, 5, None, None, None, -1, ctypes.byref(bad), FAKE, 1 << 20, FAKE, FAKE,
              FAKE, None, None, None, None, None, None, None) == sf.SF_EINVAL
    assert lw(FAKE, 10, 4, 4, 5, None, None, None, 4, ctypes.byref(cfg), FAKE, 1 << 20, FAKE, FAKE,
              FAKE, None, None, None, None, None, None, None) == sf.SF_EINVAL
    assert lw(FAKE, 10, 4, 4, 5, None, None, None, -1, ctypes.byref(cfg), FAKE, 16, FAKE, FAKE,
              FAKE, None, None, None, None, None, None, None) == sf.SF_EWORKSPACE
    assert lw(FAKE, 10, 4, 4, 5, None, None, None, -1, ctypes.byref(cfg), FAKE + 16, 1 << 20, FAKE,
              FAKE, FAKE, None, None, None, None, None, None, None) == sf.SF_EINVAL_ALIGN
    # evidence pass: bad eta ratio and residual stage index
    dg = L.sf_direct_gain
    assert dg(FAKE, 10, 4, 4, 5, FAKE, None, -1, sf.Ratio(1, 0), FAKE, FAKE, FAKE, None, None, FAKE, None,
              None, None) == sf.SF_EINVAL
    assert dg(FAKE, 10, 4, 4, 5, FAKE, None, -2, sf.Ratio(1, 20), FAKE, FAKE, FAKE, None, None, FAKE, None,
              None, None) == sf.SF_EINVAL
    assert dg(FAKE, 10, 4, 4, 5, FAKE, None, -1, sf.Ratio(1, 20), FAKE, FAKE, FAKE, FAKE + 4, None, FAKE,
              None, None, None) == sf.SF_EINVAL_ALIGN
    assert L.sf_window_median(FAKE, 10, 4, 4, 0, FAKE, None, None) == sf.SF_EINVAL
    # cross-rank order statistics: no outputs, bad window, misaligned output
    assert L.sf_rank_lag(FAKE, 10, 4, 4, None, None, None, FAKE, 1 << 20, None, None) == sf.SF_EINVAL
    assert L.sf_rank_lag(FAKE, 10, 4, 4, FAKE + 4, None, None, FAKE, 1 << 20, None, None) == sf.SF_EINVAL_ALIGN
    assert L.sf_rank_lag(FAKE, 10, 4, 4, FAKE, None, None, FAKE + 16, 1 << 20, None, None) == sf.SF_EINVAL_ALIGN
    assert L.sf_rank_lag(FAKE, 10, 4, 4, FAKE, None, None, FAKE, 64, None, None) == sf.SF_EWORKSPACE
    assert L.sf_rank_lag(FAKE, 10, 4, 4, FAKE, None, None, None, 1 << 20, None, None) == sf.SF_EWORKSPACE
    assert L.sf_raw_spread(FAKE, 10, 4, 4, 0, 0, FAKE, 0, FAKE, 1 << 20, None, None) == sf.SF_EINVAL
    assert L.sf_raw_spread(FAKE, 10, 4, 4, 0, 5, None, 0, FAKE, 1 << 20, None, None) == sf.SF_EINVAL
    assert L.sf_raw_spread(FAKE, 10, 4, 4, 0, 5, FAKE, 3, FAKE, 1 << 20, None, None) == sf.SF_EINVAL
    assert L.sf_raw_spread(FAKE, 10, 4, 4, 0, 5, FAKE + 4, 0, FAKE, 1 << 20, None, None) == sf.SF_EINVAL_ALIGN
    assert L.sf_rank_lag_windows(FAKE, 10, 4, 4, 0, 5, None, None, 0, FAKE, 1 << 20, None, None) == sf.SF_EINVAL
    assert L.sf_rank_lag_windows(FAKE, 10, 4, 4, 0, 0, FAKE, None, 0, FAKE, 1 << 20, None, None) == sf.SF_EINVAL
    assert L.sf_rank_lag_windows(FAKE, 10, 4, 4, 0, 5, FAKE, None, 0, FAKE, 8, None, None) == sf.SF_EWORKSPACE
    assert L.sf_rank_workspace_size(8192, 8192, 8) >= 8 * 8192 * 4
    assert L.sf_rank_workspace_size(0, 8, 8) == 0
    # role groups: group count, G*S limit, stage-group ids (host array)
    ga = L.sf_group_aggregate
    assert ga(FAKE, 10, 4, 4, FAKE, 0, 0, 5, FAKE, FAKE, 0, None, None) == sf.SF_EINVAL
    assert ga(FAKE, 10, 4, 8, FAKE, 1000, 0, 5, FAKE, FAKE, 0, None, None) == sf.SF_EINVAL
    assert ga(FAKE, 10, 4, 4, None, 2, 0, 5, FAKE, FAKE, 0, None, None) == sf.SF_EINVAL
    assert ga(FAKE, 10, 4, 4, FAKE + 2, 2, 0, 5, FAKE, FAKE, 0, None, None) == sf.SF_EINVAL_ALIGN
    sg = (ctypes.c_int32 * 4)(0, 1, 0, 5)
    assert L.sf_stage_group_sum(FAKE, 3, 4, sg, 2, FAKE, None) == sf.SF_EINVAL
    sg = (ctypes.c_int32 * 4)(0, 1, 0, 1)
    assert L.sf_stage_group_sum(FAKE, 3, 4, sg, 33, FAKE, None) == sf.SF_EINVAL
    assert L.sf_stage_group_sum(FAKE + 4, 3, 4, sg, 2, FAKE, None) == sf.SF_EINVAL_ALIGN
    # rank-major ingest: block length, in-place conversion, alignment
    assert L.sf_gathered_to_steps(FAKE, 10, 4, 4, 0, FAKE + (1 << 16), None) == sf.SF_EINVAL
    assert L.sf_gathered_to_steps(FAKE, 10, 4, 4, 5, FAKE + 64, None) == sf.SF_EINVAL
    assert L.sf_gathered_to_steps(FAKE + 8, 10, 4, 4, 5, FAKE + (1 << 16), None) == sf.SF_EINVAL_ALIGN
    # nothing was launched by any of the rejected calls
    assert sf.launch_count() == 0


def test_no_cpu_fallback_in_binding():
    src = open(os.path.join(ROOT, "paper_2606_06751_gb300", "stagefrontier.py")).read()
    assert "oracle" not in src and "numpy" not in src
