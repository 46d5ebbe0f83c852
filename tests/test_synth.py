"""The seeded input generator: determinism, chunking, and the workload shapes."""
import numpy as np
import pytest

from synth import workloads as wl


def test_thread_count_and_chunk_independence():
    w = wl.ddp128(steps=300)
    a = w.generate(threads=1)
    b = w.generate(threads=7)
    assert (a == b).all()
    c = np.concatenate([w.generate(t0=0, nsteps=120), w.generate(t0=120, nsteps=180)])
    assert (a == c).all()


def test_seed_changes_data():
    a = wl.tiny(seed=0).generate()
    b = wl.tiny(seed=1).generate()
    assert not (a == b).all()


@pytest.mark.parametrize("name,steps", [("tiny", None), ("ddp128", 50), ("fsdp1024", 8),
                                        ("accum8192", 2)])
def test_shapes_and_ranges(name, steps):
    w = wl.by_name(name, steps=steps)
    d = w.generate()
    assert d.shape == (w.T, w.R, w.S) and d.dtype == np.int64
    assert (d > 0).all() and (d.sum(axis=2) < (1 << 47)).all()


def test_sync_stage_releases_ranks_together():
    """Clock simulation: after a sync stage every rank's elapsed time is the
    common release time plus its own intrinsic work, so the spread of the
    prefix right after the sync is far below the spread right before it."""
    w = wl.ddp128(steps=20)
    d = w.generate()
    P = np.cumsum(d, axis=2)
    before = P[:, :, 2].max(axis=1) - P[:, :, 2].min(axis=1)
    after = P[:, :, 3].max(axis=1) - P[:, :, 3].min(axis=1)
    assert (after < before).all()


def test_tiny_stall_injected():
    w = wl.tiny()
    d = w.generate()
    (tb, te, r, s, delta), = w.stalls
    assert d[tb, r, s] > 40 * wl.MS and delta == 30 * wl.MS


def test_sweep_sizes():
    for R in wl.SWEEP_R:
        for S in wl.SWEEP_S:
            w = wl.sweep(R, S)
            assert w.nbytes == 1 << 30
