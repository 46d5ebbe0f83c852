"""GPU parity of the role-group frontier (App. A role check, Sec. 3 Eq. 1 per
group) and of the reporting-group sums after the frontier (Sec. 3), against
the CPU oracle, bit-exact."""
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
    med = rng.uniform(1e6, 5e7, size=S)
    return np.rint(med * np.exp(0.1 * rng.standard_normal((T, R, S)))).astype(np.int64)


def groups(R, G, kind, seed):
    rng = np.random.default_rng(seed)
    if kind == "blocks":     # contiguous node groups (warp-uniform fast path)
        return (np.arange(R) * G // R).astype(np.int32)
    return rng.integers(0, G, size=R).astype(np.int32)   # scattered roles (per-lane path)


CASES = [(37, 3, 5, 2), (20, 1, 1, 1), (11, 7, 32, 3), (50, 64, 8, 4), (301, 128, 8, 2), (97, 40, 10, 5),
         (23, 1024, 10, 8), (7, 8192, 8, 64), (5, 4096, 16, 16), (3, 65536, 2, 512), (9, 300, 6, 682),
         (4, 100, 1, 4096)]


@pytest.mark.parametrize("T,R,S,G", CASES)
@pytest.mark.parametrize("gkind", ["blocks", "random"])
@pytest.mark.parametrize("t0,W", [(0, 10), (7, 3)])
def test_group_aggregate_parity(sf, T, R, S, G, gkind, t0, W):
    d_np = make(T, R, S, T + R + S + G, "ties" if R < 100 else "lognormal")
    grp = groups(R, G, gkind, R + G)
    o = O.group_windows(d_np, grp, G, W, t0)
    st = sf.new_status("cuda")
    g = sf.sf_group_aggregate(dev(d_np), dev(grp), G, W, t0=t0, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(g.X), np.transpose(o.X, (1, 0, 2)))
    assert np.array_equal(host(g.D), o.D.T)


def test_group_aggregate_one_group_matches_window_aggregate(sf):
    w = wl.by_name("fsdp1024")
    d = dev(w.generate(0, 1000))
    g = sf.sf_group_aggregate(d, torch.zeros(w.R, dtype=torch.int32, device="cuda"), 1, w.W)
    a = sf.sf_window_aggregate(d, w.W)
    torch.cuda.synchronize()
    assert torch.equal(g.X[:, 0, :], a.X) and torch.equal(g.D[:, 0], a.D)


def test_group_aggregate_node_groups_accum(sf):
    """8192 ranks in 64 nodes of 128 with a node-correlated slowdown."""
    w = wl.by_name("accum8192")
    d_np = w.generate(0, 60)
    grp = (np.arange(w.R) // 128).astype(np.int32)
    o = O.group_windows(d_np, grp, 64, 25)
    g = sf.sf_group_aggregate(dev(d_np), dev(grp), 64, 25)
    torch.cuda.synchronize()
    assert np.array_equal(host(g.X), np.transpose(o.X, (1, 0, 2))) and np.array_equal(host(g.D), o.D.T)


def test_group_aggregate_accumulates_across_chunks(sf):
    T, R, S, W, G = 2500, 256, 8, 1000, 4
    d_np = make(T, R, S, 3, "lognormal")
    grp = groups(R, G, "random", 1)
    o = O.group_windows(d_np, grp, G, W)
    out = sf.GroupWindows(torch.zeros((3, G, S), dtype=torch.int64, device="cuda"),
                          torch.zeros((3, G), dtype=torch.int64, device="cuda"))
    for t0, t1 in ((0, 700), (700, 1900), (1900, 2500)):
        w0 = t0 // W
        part = sf.GroupWindows(out.X[w0:], out.D[w0:])
        sf.sf_group_aggregate(dev(d_np[t0:t1]), dev(grp), G, W, t0=t0, out=part, accumulate=True)
    torch.cuda.synchronize()
    assert np.array_equal(host(out.X), np.transpose(o.X, (1, 0, 2))) and np.array_equal(host(out.D), o.D.T)


def test_group_aggregate_bad_group_ids_are_skipped_and_flagged(sf):
    T, R, S, W, G = 30, 96, 4, 10, 3
    d_np = make(T, R, S, 8, "lognormal")
    grp = groups(R, G, "random", 2)
    bad = grp.copy()
    bad[[5, 40, 77]] = [-1, 3, 1 << 20]
    keep = np.ones(R, bool)
    keep[[5, 40, 77]] = False
    o = O.group_windows(d_np[:, keep, :], grp[keep], G, W)
    st = sf.new_status("cuda")
    g = sf.sf_group_aggregate(dev(d_np), dev(bad), G, W, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & sf.SF_ST_INDEX
    assert np.array_equal(host(g.X), np.transpose(o.X, (1, 0, 2))) and np.array_equal(host(g.D), o.D.T)


@pytest.mark.parametrize("S,K,seed", [(8, 2, 0), (8, 8, 1), (6, 1, 2), (32, 5, 3), (1, 1, 4)])
def test_stage_group_sum_parity(sf, S, K, seed):
    rng = np.random.default_rng(seed)
    d_np = make(240, 16, S, seed, "lognormal")
    X = O.windows(d_np, 25).X
    sg = rng.integers(0, K, size=S).astype(np.int32)
    Y = sf.sf_stage_group_sum(dev(X), list(sg), K)
    torch.cuda.synchronize()
    assert np.array_equal(host(Y), O.stage_group_sum(X, sg, K))
