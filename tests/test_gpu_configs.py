"""GPU parity at the full workload sizes, in the launch configuration the
benchmark uses: every integer output against the CPU oracle where the oracle
finishes in seconds (frontier and window aggregates on every step of every
workload), and the labeler on whole windows sampled from each workload."""
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


def _to_dev(d_np):
    return torch.from_numpy(d_np).cuda()


@pytest.mark.parametrize("name", ["tiny", "ddp128", "fsdp1024", "accum8192"])
def test_workload_full_aggregate(sf, name):
    w = wl.by_name(name)
    d_np = w.generate()
    d = _to_dev(d_np)
    st = sf.new_status("cuda")
    g = sf.sf_window_aggregate(d, w.W, status=st)
    top = sf.sf_topk_suspects(g.X, g.E, w.k)
    f = sf.sf_frontier(d, status=st, outputs=("makespan",))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    o = O.windows(d_np, w.W)
    for k in ("X", "D", "E", "C", "step_lead"):
        assert np.array_equal(getattr(g, k).cpu().numpy(), getattr(o, k)), k
    ot = O.topk(o.X, o.E, w.k)
    assert np.array_equal(top.stage.cpu().numpy(), ot.stage)
    assert np.array_equal(top.pair.cpu().numpy(), ot.pair)
    assert np.array_equal(top.pair_value.cpu().numpy(), ot.pair_value)
    # makespans: sampled steps against the oracle frontier, and Theorem 1 over windows
    idx = np.random.default_rng(0).choice(w.T, size=min(w.T, 64), replace=False)
    of = O.frontier(d_np[np.sort(idx)])
    assert np.array_equal(f.makespan.cpu().numpy()[np.sort(idx)], of.makespan)
    assert np.array_equal(o.X.sum(axis=1), o.D)
    del d


@pytest.mark.parametrize("name,windows", [("tiny", None), ("ddp128", 4), ("fsdp1024", 6),
                                          ("accum8192", 2)])
def test_workload_labels_sampled(sf, name, windows):
    w = wl.by_name(name)
    n = w.T if windows is None else windows * w.W
    t0 = 0 if windows is None else (w.T // 2) // w.W * w.W   # whole windows from the middle
    d_np = w.generate(t0=t0, nsteps=n)
    o = O.label_windows(d_np, w.W)
    st = sf.new_status("cuda")
    lab = sf.sf_label_windows(_to_dev(d_np), w.W, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(lab.labels.cpu().numpy().astype(np.uint32), o.labels)
    assert np.array_equal(lab.route_mask.cpu().numpy().astype(np.uint32), o.route_mask)
    assert np.array_equal(lab.amb_mask.cpu().numpy().astype(np.uint32), o.amb_mask)
    assert np.array_equal(lab.Y.cpu().numpy(), o.Y)
    np.testing.assert_allclose(lab.share.cpu().numpy(), o.share, rtol=1e-12, atol=0)
    np.testing.assert_allclose(lab.gain.cpu().numpy(), o.gain, rtol=1e-12, atol=0)


@pytest.mark.parametrize("R", wl.SWEEP_R)
@pytest.mark.parametrize("S", wl.SWEEP_S)
def test_sweep_frontier_full(sf, R, S):
    w = wl.sweep(R, S)
    d_np = w.generate()
    st = sf.new_status("cuda")
    d = _to_dev(d_np)
    f = sf.sf_frontier(d, status=st)
    ties = sf.sf_frontier_ties(d, a=f.a, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    o = O.frontier(d_np)
    assert np.array_equal(f.a.cpu().numpy(), o.a)
    assert np.array_equal(f.lead.cpu().numpy(), o.lead)
    assert np.array_equal(f.makespan.cpu().numpy(), o.makespan)
    assert np.array_equal(ties.cpu().numpy(), o.ties)


def test_streamed_chunks_match_resident(sf):
    """The 2000-step chunked pass over the largest workload (accumulating
    windows across chunk calls) equals the whole-tensor pass."""
    w = wl.accum8192(steps=6000)
    d_np = w.generate()
    d = _to_dev(d_np)
    whole = sf.sf_window_aggregate(d, w.W)
    nW = sf.num_windows(0, w.T, w.W)
    X = torch.zeros((nW, w.S), dtype=torch.int64, device="cuda")
    D = torch.zeros(nW, dtype=torch.int64, device="cuda")
    E = torch.zeros((nW, w.S, w.R), dtype=torch.int64, device="cuda")
    for t0 in range(0, w.T, 2000):
        sf.sf_window_aggregate(d[t0:t0 + 2000], w.W, t0=t0, X=X[t0 // w.W:], D=D[t0 // w.W:],
                               E=E[t0 // w.W:], want=(), accumulate=True)
    assert torch.equal(X, whole.X) and torch.equal(D, whole.D) and torch.equal(E, whole.E)
