"""GPU parity of the cross-rank order statistics: the Sec. 4 lag, its
increment over stages and the max-minus-second-max gap per step, and the
Sec. 6 raw rank spread per window, against the CPU oracle, bit-exact."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from synth import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sf():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_06751_gb300 import build as B
    B.build()
    from paper_2606_06751_gb300 import stagefrontier
    return stagefrontier


def dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def host(t):
    return t.cpu().numpy()


def make(T, R, S, seed, kind):
    rng = np.random.default_rng(seed)
    if kind == "ties":
        return rng.integers(0, 6, size=(T, R, S), dtype=np.int64)
    if kind == "zeros":
        d = rng.integers(0, 1000, size=(T, R, S), dtype=np.int64)
        d[rng.random((T, R, S)) < 0.6] = 0
        return d
    if kind == "wide":      # offsets spanning 5-6 bytes: every radix pass runs
        return rng.integers(0, 1 << 41, size=(T, R, S), dtype=np.int64)
    med = rng.uniform(1e6, 5e7, size=S)
    d = np.rint(med * np.exp(0.1 * rng.standard_normal((T, R, S)))).astype(np.int64)
    if kind == "sampleskew":  # the first 4 ranks of every 32 far faster: a sample of them misleads
        d[:, (np.arange(R) % 32) < 4, :] //= 4
    if kind == "cluster":   # 70 % of the values equal: the median sits in one heavy tie
        d[rng.random((T, R, S)) < 0.7] = int(med[0])
    if kind == "boundary":  # values around 2^27..2^29: the 32-bit encode's limits for 16, 8 and 4 stages
        edges = np.array([(1 << b) + o for b in (27, 28, 29) for o in (-2, -1, 0, 1)], dtype=np.int64)
        return edges[rng.integers(0, len(edges), size=(T, R, S))]
    if kind == "refwide":   # rank 0 alone far from the rest at one stage
        d[:, 0, S // 2] += 1 << 31
    if kind == "mixed":     # a few steps with a multi-second stall on one rank (64-bit path)
        for t in rng.choice(T, size=max(1, T // 7), replace=False):
            d[t, rng.integers(R), rng.integers(S)] += int(rng.integers(1 << 31, 1 << 33))
    return d


# templated stage counts (4, 6, 8, 10, 16) and the generic kernel; R = 1 and 2,
# odd and even R, R above the CTA width, the largest R
SHAPES = [(20, 1, 1), (9, 2, 3), (37, 3, 5), (11, 7, 32), (6, 5, 18), (50, 2, 8),
          (1000, 8, 6), (123, 64, 4), (97, 40, 10), (77, 64, 16), (31, 257, 8),
          (13, 1024, 10), (7, 8192, 8), (5, 4096, 16), (3, 32768, 4), (2, 65536, 2), (2, 65535, 7),
          (2, 32768, 16), (3, 9000, 9), (2, 65536, 32),
          (5, 1023, 4), (4, 2048, 5), (3, 2049, 7), (3, 4097, 3), (2, 6001, 12)]


@pytest.mark.parametrize("T,R,S", SHAPES)
@pytest.mark.parametrize("kind", ["ties", "zeros", "lognormal", "wide", "mixed", "sampleskew", "cluster", "boundary",
                                  "refwide"])
def test_rank_lag_parity(sf, T, R, S, kind):
    d_np = make(T, R, S, T * 17 + R * 5 + S, kind)
    o = O.rank_lag(d_np)
    st = sf.new_status("cuda")
    g = sf.sf_rank_lag(dev(d_np), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(g.L), o.L)
    assert np.array_equal(host(g.dL), o.dL)
    assert np.array_equal(host(g.G), o.G)


def make_stream(T, R, S, seed, kind):
    """Inputs for the streaming pass, where a CTA walks many consecutive steps
    and predicts each step's median from the last: smooth steps, steps whose
    level jumps up and down (the prediction misses on both sides), heavy ties
    (candidate segments overflow), rare wide values (the 64-bit fallback) and
    values at the 32-bit limits of the main pass."""
    rng = np.random.default_rng(seed)
    if kind in ("lognormal", "mixed", "cluster", "boundary", "ties"):
        return make(T, R, S, seed, kind)
    med = rng.uniform(1e6, 5e7, size=S)
    d = np.rint(med * np.exp(0.1 * rng.standard_normal((T, R, S)))).astype(np.int64)
    if kind == "jumps":      # every step's level drawn anew: 0.2x .. 5x
        d = np.rint(d * np.exp(rng.uniform(-1.6, 1.6, size=(T, 1, 1)))).astype(np.int64)
    if kind == "drift":      # a slow trend with occasional 3x steps
        f = np.exp(np.cumsum(rng.normal(0, 0.02, size=T)))
        f[rng.random(T) < 0.05] *= 3
        d = np.rint(d * f[:, None, None]).astype(np.int64)
    if kind == "narrow":     # the spread collapses for some steps: few distinct values
        sel = rng.random(T) < 0.3
        d[sel] = (d[sel] // 100000) * 100000
    return d


@pytest.mark.parametrize("T,R,S", [(3000, 1024, 8), (2000, 2048, 4), (1500, 1024, 16), (700, 4096, 8)])
@pytest.mark.parametrize("kind", ["lognormal", "jumps", "drift", "narrow", "mixed", "cluster", "ties", "boundary"])
def test_rank_lag_streaming_many_steps(sf, T, R, S, kind):
    """Many steps per CTA (the grid holds two CTAs per SM), so most steps are
    resolved from the predicted bracket and the rest by the exact fallback."""
    d_np = make_stream(T, R, S, T + R + S, kind)
    o = O.rank_lag(d_np)
    st = sf.new_status("cuda")
    g = sf.sf_rank_lag(dev(d_np), status=st)
    sp = sf.sf_raw_spread(dev(d_np), 100, t0=7, status=st)
    lw = sf.sf_rank_lag_windows(dev(d_np), 100, t0=7, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(g.L), o.L)
    assert np.array_equal(host(g.dL), o.dL)
    assert np.array_equal(host(g.G), o.G)
    assert np.array_equal(host(sp), O.raw_spread(d_np, 100, 7))
    LW, GW = O.rank_lag_windows(d_np, 100, t0=7)
    assert np.array_equal(host(lw[0]), LW) and np.array_equal(host(lw[1]), GW)


def test_rank_lag_optional_outputs(sf):
    d_np = make(40, 33, 6, 5, "lognormal")
    o = O.rank_lag(d_np)
    d = dev(d_np)
    e = lambda: torch.empty((40, 6), dtype=torch.int64, device="cuda")  # noqa: E731
    only_g = sf.sf_rank_lag(d, out=sf.Lag(None, None, e()))
    only_dl = sf.sf_rank_lag(d, out=sf.Lag(None, e(), None))    # the lag is formed in dL and converted in place
    l_dl = sf.sf_rank_lag(d, out=sf.Lag(e(), e(), None))
    torch.cuda.synchronize()
    assert np.array_equal(host(only_g.G), o.G)
    assert np.array_equal(host(only_dl.dL), o.dL)
    assert np.array_equal(host(l_dl.L), o.L) and np.array_equal(host(l_dl.dL), o.dL)


@pytest.mark.parametrize("T,R,S,steps_per_chunk", [(50, 100, 8, 1), (37, 1025, 6, 3), (12, 4096, 16, 5),
                                                   (9, 7, 32, 2)])
@pytest.mark.parametrize("kind", ["lognormal", "mixed"])
def test_rank_lag_small_workspace_many_chunks(sf, T, R, S, steps_per_chunk, kind):
    """A workspace that holds only a few steps: every chunk reuses the same
    scratch (and its discarded L2 lines) for the next."""
    d_np = make(T, R, S, T + R, kind)
    o = O.rank_lag(d_np)
    one = int(sf.lib().sf_rank_workspace_size(1, R, S))
    ws = torch.empty(one * steps_per_chunk, dtype=torch.uint8, device="cuda")
    g = sf.sf_rank_lag(dev(d_np), workspace=ws)
    sp = sf.sf_raw_spread(dev(d_np), 4, t0=3, workspace=ws)
    torch.cuda.synchronize()
    assert np.array_equal(host(g.L), o.L) and np.array_equal(host(g.dL), o.dL) and np.array_equal(host(g.G), o.G)
    assert np.array_equal(host(sp), O.raw_spread(d_np, 4, 3))


def test_rank_lag_workspace_too_small_is_rejected(sf):
    d = dev(make(4, 64, 8, 1, "lognormal"))
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(RuntimeError):
        sf.sf_rank_lag(d, workspace=ws)


@pytest.mark.parametrize("T,R,S", [(20, 1, 1), (37, 3, 5), (301, 64, 4), (97, 40, 10), (1000, 8, 6),
                                   (23, 1024, 10), (9, 8192, 8), (4, 65536, 2)])
@pytest.mark.parametrize("t0,W", [(0, 1), (0, 7), (5, 10), (3, 1000)])
def test_raw_spread_parity(sf, T, R, S, t0, W):
    d_np = make(T, R, S, T + R + S + W, "ties" if R < 100 else "lognormal")
    o = O.raw_spread(d_np, W, t0)
    st = sf.new_status("cuda")
    got = sf.sf_raw_spread(dev(d_np), W, t0=t0, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(got), o)


@pytest.mark.parametrize("T,R,S", [(9, 8192, 8), (5, 4096, 3), (3, 65536, 2)])
@pytest.mark.parametrize("kind", ["sampleskew", "cluster"])
def test_raw_spread_misleading_sample(sf, T, R, S, kind):
    d_np = make(T, R, S, T * 3 + R + S, kind)
    o = O.raw_spread(d_np, 4, 0)
    st = sf.new_status("cuda")
    got = sf.sf_raw_spread(dev(d_np), 4, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(got), o)


def test_raw_spread_accumulates_across_chunks(sf):
    T, R, S, W = 2500, 128, 8, 1000
    d_np = make(T, R, S, 11, "lognormal")
    o = O.raw_spread(d_np, W)
    out = torch.zeros((3, S), dtype=torch.int64, device="cuda")
    for t0 in (0, 700, 1900):
        t1 = {0: 700, 700: 1900, 1900: 2500}[t0]
        w0 = t0 // W
        part = out[w0:]
        sf.sf_raw_spread(dev(d_np[t0:t1]), W, t0=t0, spread=part, accumulate=True)
    torch.cuda.synchronize()
    assert np.array_equal(host(out), o)


def test_rank_lag_status_bits(sf):
    d_np = make(8, 16, 4, 3, "lognormal")
    d_np[3, 5, 2] = -1
    st = sf.new_status("cuda")
    sf.sf_rank_lag(dev(d_np), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & sf.SF_ST_NEGATIVE
    d_np = make(8, 16, 4, 3, "lognormal")
    d_np[2, 1, 1] = 1 << 50
    st = sf.new_status("cuda")
    sf.sf_raw_spread(dev(d_np), 4, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & sf.SF_ST_RANGE


@pytest.mark.parametrize("name", ["tiny", "ddp128", "fsdp1024", "accum8192"])
def test_rank_lag_on_workloads(sf, name):
    """The workload generators (sync stages absorbing skew, stalls, Pareto
    tails, node slowdowns) on a prefix of steps, lag and spread exact."""
    w = wl.by_name(name)
    n = {"tiny": 1000, "ddp128": 3000, "fsdp1024": 600, "accum8192": 40}[name]
    d_np = w.generate(0, n)
    o = O.rank_lag(d_np)
    g = sf.sf_rank_lag(dev(d_np))
    sp = sf.sf_raw_spread(dev(d_np), w.W)
    torch.cuda.synchronize()
    assert np.array_equal(host(g.L), o.L) and np.array_equal(host(g.dL), o.dL)
    assert np.array_equal(host(g.G), o.G)
    assert np.array_equal(host(sp), O.raw_spread(d_np, w.W))


@pytest.mark.parametrize("T,R,S,t0,W", [(37, 3, 5, 0, 7), (300, 64, 8, 5, 100), (45, 1024, 10, 0, 20),
                                        (9, 8192, 8, 3, 4), (20, 1, 1, 0, 3)])
def test_rank_lag_windows_parity(sf, T, R, S, t0, W):
    d_np = make(T, R, S, T * R + S, "lognormal" if R > 3 else "ties")
    oL, oG = O.rank_lag_windows(d_np, W, t0)
    st = sf.new_status("cuda")
    Lw, Gw = sf.sf_rank_lag_windows(dev(d_np), W, t0=t0, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(Lw), oL) and np.array_equal(host(Gw), oG)


def test_back_to_back_calls_share_the_workspace(sf):
    """Calls queued back to back on one stream reuse one workspace: a call's
    first chunk must not overwrite the scratch the previous call's last
    chunk is still selecting from (several chunks per call, odd and even
    chunk counts)."""
    T, R, S, W = 700, 2048, 8, 100
    d_np = make(T, R, S, 77, "lognormal")
    d = dev(d_np)
    one = int(sf.lib().sf_rank_workspace_size(1, R, S))
    o_sp = O.raw_spread(d_np, W)
    o_lag = O.rank_lag(d_np)
    for steps_per_chunk in (64, 100, 233):
        ws = torch.empty(one * steps_per_chunk, dtype=torch.uint8, device="cuda")
        outs = []
        for _ in range(4):
            outs.append(sf.sf_raw_spread(d, W, workspace=ws))
            outs.append(sf.sf_rank_lag(d, out=sf.Lag(None, None, torch.empty((T, S), dtype=torch.int64,
                                                                             device="cuda")), workspace=ws).G)
        torch.cuda.synchronize()
        for i in range(0, len(outs), 2):
            assert np.array_equal(host(outs[i]), o_sp), (steps_per_chunk, i)
            assert np.array_equal(host(outs[i + 1]), o_lag.G), (steps_per_chunk, i)
