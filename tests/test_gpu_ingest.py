"""Rank-major ingest (the window-boundary gather of Sec. 5 delivers each
window as an [R][n][S] block): the device conversion to [T][R][S] is an exact
copy, and the host-streamed path over gathered windows gives the same
outputs as the step-major path and the oracle."""
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


def gathered(d, N):
    """The gather's layout: for each block of N steps, every rank's [n][S] rows in rank order."""
    T = d.shape[0]
    return np.concatenate([np.ascontiguousarray(d[b:b + N].transpose(1, 0, 2)).reshape(-1)
                           for b in range(0, T, N)])


@pytest.mark.parametrize("T,R,S,N", [(10, 3, 5, 4), (7, 1, 1, 7), (12, 8, 6, 5), (20, 64, 8, 20), (9, 33, 7, 2),
                                     (5, 4096, 16, 3), (3, 65536, 2, 1), (6, 100, 10, 100), (1000, 8, 6, 100)])
def test_gathered_to_steps_is_an_exact_copy(sf, T, R, S, N):
    rng = np.random.default_rng(T + R + S + N)
    d = rng.integers(0, 1 << 46, size=(T, R, S), dtype=np.int64)
    src = torch.from_numpy(gathered(d, N)).cuda()
    out = sf.sf_gathered_to_steps(src, T, R, S, N)
    torch.cuda.synchronize()
    assert np.array_equal(out.cpu().numpy(), d)


def test_gathered_to_steps_rejects_in_place(sf):
    buf = torch.zeros(4 * 8 * 6, dtype=torch.int64, device="cuda")
    with pytest.raises(RuntimeError):
        sf.sf_gathered_to_steps(buf, 4, 8, 6, 2, dst=buf.view(4, 8, 6))


def test_stream_gathered_matches_oracle_ragged(sf):
    w = wl.ddp128(steps=2500)
    d_np = w.generate()
    W, k, chunk = 500, 3, 1000                     # 3 chunks, the last one half full
    h = torch.from_numpy(gathered(d_np, W)).pin_memory()
    st = sf.new_status("cuda")
    out = sf.sf_stream_gathered_windows(h, w.T, w.R, w.S, W, k, chunk, status=st, copy_stream=torch.cuda.Stream())
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


def test_stream_gathered_matches_step_major_large(sf):
    w = wl.accum8192(steps=4500)                  # 3 chunks of 2000 steps, the last one short
    d_np = w.generate()
    hs = torch.from_numpy(d_np).pin_memory()
    hg = torch.from_numpy(gathered(d_np, w.W)).pin_memory()
    a = sf.sf_stream_windows(hs, w.W, w.k, 2000, copy_stream=torch.cuda.Stream())
    b = sf.sf_stream_gathered_windows(hg, w.T, w.R, w.S, w.W, w.k, 2000, copy_stream=torch.cuda.Stream())
    torch.cuda.synchronize()
    for name in ("X", "Y", "D", "E", "C", "top_stage", "top_pair", "top_pair_value", "labels", "route_mask",
                 "amb_mask", "share", "gain"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
