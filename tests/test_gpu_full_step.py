"""The benchmark's launch configuration at full size: the 8192-rank x 8-stage
x 20000-step workload (10.5 GB) resident on the device, every entry point
called once on the whole tensor exactly as bench.py times it, and sampled
outputs checked against the oracle on the samples alone (windows and steps
are independent, so a sample's oracle is the oracle of the whole)."""
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


@pytest.fixture(scope="module")
def full(sf):
    w = wl.by_name("accum8192")
    d_np = w.generate()
    return w, d_np, torch.from_numpy(d_np).cuda()


def test_bench_step_sampled_windows(sf, full):
    w, d_np, d = full
    st = sf.new_status("cuda")
    m = sf.sf_window_median(d, w.W, status=st)
    ev = sf.sf_direct_gain(d, w.W, m, lead_credit=True, status=st)
    top = sf.sf_topk_suspects(ev.X, ev.E, w.k)
    lab = sf.sf_label_gates(w.T, w.R, w.S, w.W, ev)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for wi in (0, 11, w.T // w.W - 1):
        part = d_np[wi * w.W:(wi + 1) * w.W]
        ol = O.label_windows(part, w.W)
        ow = O.windows(part, w.W)
        ot = O.topk(ow.X, ow.E, w.k)
        assert np.array_equal(m[wi].cpu().numpy(), O.window_median(part, w.W)[0]), wi
        assert np.array_equal(ev.X[wi].cpu().numpy(), ow.X[0]) and np.array_equal(ev.Y[wi].cpu().numpy(), ol.Y[0])
        assert np.array_equal(ev.E[wi].cpu().numpy(), ow.E[0]) and np.array_equal(ev.C[wi].cpu().numpy(), ow.C[0])
        assert np.array_equal(top.stage[wi].cpu().numpy(), ot.stage[0])
        assert np.array_equal(top.pair[wi].cpu().numpy(), ot.pair[0])
        assert int(lab.labels[wi]) == int(ol.labels[0]) and int(lab.route_mask[wi]) == int(ol.route_mask[0])
        assert int(lab.amb_mask[wi]) == int(ol.amb_mask[0])
        np.testing.assert_allclose(lab.share[wi].cpu().numpy(), ol.share[0], rtol=1e-12, atol=0)
        np.testing.assert_allclose(lab.gain[wi].cpu().numpy(), ol.gain[0], rtol=1e-12, atol=0)


def test_lag_spread_group_full_sampled(sf, full):
    w, d_np, d = full
    st = sf.new_status("cuda")
    ws = sf.rank_workspace(w.T, w.R, w.S, d.device)
    lag = sf.sf_rank_lag(d, workspace=ws, status=st)
    sp = sf.sf_raw_spread(d, w.W, workspace=ws, status=st)
    G = w.R // 128
    grp = (torch.arange(w.R, device="cuda", dtype=torch.int32) * G // w.R).to(torch.int32)
    ga = sf.sf_group_aggregate(d, grp, G, w.W, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    steps = np.sort(np.random.default_rng(1).choice(w.T, size=24, replace=False))
    ol = O.rank_lag(d_np[steps])
    assert np.array_equal(lag.L.cpu().numpy()[steps], ol.L)
    assert np.array_equal(lag.dL.cpu().numpy()[steps], ol.dL)
    assert np.array_equal(lag.G.cpu().numpy()[steps], ol.G)
    wi = 7
    assert np.array_equal(sp[wi].cpu().numpy(), O.raw_spread(d_np[wi * w.W:(wi + 1) * w.W], w.W)[0])
    og = O.group_windows(d_np, grp.cpu().numpy(), G, w.W)
    assert np.array_equal(ga.X.cpu().numpy(), np.transpose(og.X, (1, 0, 2)))
    assert np.array_equal(ga.D.cpu().numpy(), og.D.T)


def test_ingest_full_round_trip(sf, full):
    w, d_np, d = full
    nW = w.T // w.W
    g = d.view(nW, w.W, w.R, w.S).permute(0, 2, 1, 3).contiguous().view(-1)
    back = sf.sf_gathered_to_steps(g, w.T, w.R, w.S, w.W)
    torch.cuda.synchronize()
    assert torch.equal(back, d)
