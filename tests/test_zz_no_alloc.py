"""sf_label_windows_noalloc, the labeler for callers that cannot allocate
device memory (a monitor running inside a training job whose framework owns
the device memory, where a cudaMalloc from the hook could stall the step it
measures).  Its intermediates live in the library's static device scratch.

Both entry points are called through the C ABI on the same inputs; the
no-allocation one must agree with the workspace one and with the CPU oracle
on two calls in a row (the second on different data, so stale scratch from
the first call would show), and must refuse a problem larger than its static
scratch.  This file
is collected last so a failure here does not hide the rest of the suite."""
import ctypes

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


def _outputs(nW, S):
    z = lambda shape, dt: torch.full(shape, 7, dtype=dt, device="cuda")  # noqa: E731  (not zeroed on purpose)
    return [z((nW,), torch.int32), z((nW,), torch.int32), z((nW,), torch.int32),
            z((nW, S), torch.float64), z((nW, S), torch.float64), z((nW, S), torch.int64),
            z((nW, S), torch.int64), z((nW,), torch.int64)]


def _call(sf, d, W, use_static, missing=None):
    L = sf.lib()
    T, R, S = d.shape
    nW = (T + W - 1) // W
    outs = _outputs(nW, S)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    cfg = sf.default_config()
    stream = torch.cuda.current_stream().cuda_stream
    mp = None if missing is None else missing.data_ptr()
    ptrs = [o.data_ptr() for o in outs]
    if use_static:
        rc = L.sf_label_windows_noalloc(d.data_ptr(), T, R, S, W, None, mp, None, -1, ctypes.byref(cfg),
                                        *ptrs, status.data_ptr(), stream)
    else:
        ws = torch.empty(L.sf_label_windows_workspace_size(T, R, S, W), dtype=torch.uint8, device="cuda")
        rc = L.sf_label_windows(d.data_ptr(), T, R, S, W, None, mp, None, -1, ctypes.byref(cfg),
                                ws.data_ptr(), ws.numel(), *ptrs, status.data_ptr(), stream)
    assert rc == sf.SF_OK
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return [o.cpu().numpy() for o in outs]


def _same(a, b):
    for i, (x, y) in enumerate(zip(a, b)):
        if x.dtype == np.float64:
            np.testing.assert_allclose(x, y, rtol=1e-12, atol=0)
        else:
            assert np.array_equal(x, y), i


def _oracle(d_np, W, missing):
    o = O.label_windows(d_np, W, missing=missing)
    return [o.labels, o.route_mask, o.amb_mask, o.share, o.gain, o.X, o.Y, o.D]


def test_noalloc_matches_workspace_entry_point_twice(sf):
    first = wl.fsdp1024(steps=1000).generate()          # 2 windows of 500 steps
    second = wl.accum8192(steps=120, seed=3).generate()  # different shape and data
    for d_np, W in ((first, 500), (second, 40)):
        d = torch.from_numpy(d_np).cuda()
        nW = (d.shape[0] + W - 1) // W
        missing = torch.zeros(nW, dtype=torch.int32, device="cuda")
        ref = _call(sf, d, W, use_static=False, missing=missing)
        got = _call(sf, d, W, use_static=True, missing=missing)
        _same(got, ref)
        # the CPU oracle on the same input: integer outputs bit-exact, the
        # fp64 shares and gains within 1e-12 relative
        orc = _oracle(d_np, W, np.zeros(nW, np.int32))
        _same([g.astype(o.dtype) for g, o in zip(got, orc)], orc)
        # a second call in a row on the same data sees the scratch the first one left
        _same(_call(sf, d, W, use_static=True, missing=missing), ref)


def test_noalloc_refuses_oversized_problem(sf):
    L = sf.lib()
    T, R, S, W = 20000, 8192, 8, 1000          # medians alone need 10.5 MB per 20 windows ...
    T *= 4                                       # ... so 80000 steps need ~42 MB > 16 MiB
    assert L.sf_label_windows_workspace_size(T, R, S, W) > sf.STATIC_SCRATCH_BYTES
    cfg = sf.default_config()
    n0 = sf.launch_count()
    rc = L.sf_label_windows_noalloc(1 << 20, T, R, S, W, None, None, None, -1, ctypes.byref(cfg),
                                    1 << 20, 1 << 20, 1 << 20, None, None, None, None, None, None,
                                    torch.cuda.current_stream().cuda_stream)
    assert rc == sf.SF_EWORKSPACE and sf.launch_count() == n0
