"""sf_stream_windows: the whole hot path over a host-resident tensor streamed
to the GPU in chunks of whole windows, against the CPU oracle (small
workload, ragged last chunk) and against the device-resident calls (largest
workload's rank count, 2000-step chunks)."""
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


def test_stream_matches_oracle_ragged(sf):
    w = wl.ddp128(steps=2500)
    d_np = w.generate()
    W, k, chunk = 500, 3, 1000                     # 3 chunks, the last one half full
    h = torch.from_numpy(d_np).pin_memory()
    st = sf.new_status("cuda")
    out = sf.sf_stream_windows(h, W, k, chunk, status=st, copy_stream=torch.cuda.Stream())
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ow = O.windows(d_np, W)
    ol = O.label_windows(d_np, W)
    ot = O.topk(ow.X, ow.E, k)
    for name, ref in (("X", ow.X), ("D", ow.D), ("E", ow.E), ("C", ow.C), ("Y", ol.Y),
                      ("top_stage", ot.stage), ("top_pair", ot.pair), ("top_pair_value", ot.pair_value)):
        assert np.array_equal(getattr(out, name).cpu().numpy(), ref), name
    assert np.array_equal(out.labels.cpu().numpy().astype(np.uint32), ol.labels)
    assert np.array_equal(out.route_mask.cpu().numpy().astype(np.uint32), ol.route_mask)
    assert np.array_equal(out.amb_mask.cpu().numpy().astype(np.uint32), ol.amb_mask)
    np.testing.assert_allclose(out.share.cpu().numpy(), ol.share, rtol=1e-12, atol=0)
    np.testing.assert_allclose(out.gain.cpu().numpy(), ol.gain, rtol=1e-12, atol=0)


def test_stream_matches_resident_large(sf):
    w = wl.accum8192(steps=6000)
    d_np = w.generate()
    h = torch.from_numpy(d_np).pin_memory()
    out = sf.sf_stream_windows(h, w.W, w.k, 2000, copy_stream=torch.cuda.Stream())
    d = h.cuda()
    m = sf.sf_window_median(d, w.W)
    ev = sf.sf_direct_gain(d, w.W, m, lead_credit=True)
    top = sf.sf_topk_suspects(ev.X, ev.E, w.k)
    lab = sf.sf_label_gates(w.T, w.R, w.S, w.W, ev)
    torch.cuda.synchronize()
    for a, b in ((out.X, ev.X), (out.Y, ev.Y), (out.D, ev.D), (out.E, ev.E), (out.C, ev.C),
                 (out.top_stage, top.stage), (out.top_pair, top.pair), (out.labels, lab.labels),
                 (out.route_mask, lab.route_mask), (out.amb_mask, lab.amb_mask), (out.share, lab.share),
                 (out.gain, lab.gain)):
        assert torch.equal(a, b)
    # and the first two windows against the oracle
    ol = O.label_windows(d_np[:2000], w.W)
    assert np.array_equal(out.labels[:2].cpu().numpy().astype(np.uint32), ol.labels)
    assert np.array_equal(out.Y[:2].cpu().numpy(), ol.Y)


def test_stream_rejects_unaligned_chunks(sf):
    h = torch.zeros((10, 4, 4), dtype=torch.int64)
    with pytest.raises(sf.SFError):
        sf.sf_stream_windows(h, 4, 2, 6)           # 6 steps is not a multiple of W = 4
