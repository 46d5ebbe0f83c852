"""GPU parity: every output of the CUDA path against the CPU oracle, element
by element, on seeded inputs that span several tiles, ragged tails, both
streaming regimes and the generic path.  Integer outputs must be bit-exact;
fp64 shares/gains within 1e-12 relative (they are one IEEE division of the
same integers, so equality is expected)."""
import numpy as np
import pytest
import torch

from oracle import oracle as O
from synth import workloads as wl

pytestmark = pytest.mark.gpu

RTOL = 1e-12


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
    if kind == "ties":      # tiny value range: ties at almost every boundary
        return rng.integers(0, 6, size=(T, R, S), dtype=np.int64)
    if kind == "zeros":     # many zero durations and equal prefixes
        d = rng.integers(0, 1000, size=(T, R, S), dtype=np.int64)
        d[rng.random((T, R, S)) < 0.6] = 0
        return d
    # lognormal around ms medians with one sync stage (realistic skew)
    med = rng.uniform(1e6, 5e7, size=S)
    x = np.rint(med * np.exp(0.1 * rng.standard_normal((T, R, S)))).astype(np.int64)
    if kind == "mixed":     # wide rows among narrow ones (the kernels' 32-bit path takes only
        # rows whose values stay below 2^(31 - ceil(log2 S))): one long stage in some rows, and
        # copies of the rank below with a 2^32 ns last stage, equal prefixes across the two paths
        t1, r1 = np.nonzero(rng.random((T, R)) < 0.05)
        x[t1, r1, rng.integers(0, S, size=t1.size)] = rng.integers(1 << 26, 1 << 33, size=t1.size)
        if R > 1:
            t2, r2 = np.nonzero(rng.random((T, R - 1)) < 0.05)
            x[t2, r2 + 1] = x[t2, r2]
            x[t2, r2 + 1, S - 1] += 1 << 32
    return x


# (T, R, S): generic path; fast path with warp-owned tiles of whole steps
# (<= 12 KB steps); fast path one-step-per-CTA with overlapped last tile.
SHAPES = [
    (37, 3, 5), (20, 1, 1), (11, 7, 32), (9, 65, 3), (6, 5, 18),          # generic
    (1000, 8, 6), (301, 128, 8), (123, 64, 4), (77, 64, 16), (50, 2, 8),   # one step per warp
    (301, 16, 2), (97, 40, 10), (45, 24, 14), (33, 120, 12),
    (13, 1024, 10), (7, 8192, 8), (5, 4096, 16), (3, 32768, 4),            # one step per CTA
    (9, 520, 12), (6, 1000, 14), (4, 512, 8), (3, 65536, 2),
]

# one-step-per-CTA shapes whose steps are one or two tiles go to two or four
# warp groups in turn, each group flushing its own window sums
GROUPED = [(9, 520, 12), (6, 1000, 14), (4, 512, 8), (3000, 512, 4), (700, 768, 6), (301, 2048, 2)]


# small steps (R*S <= 768, S in {2, 4, 8, 16}) taken G = 2, 4 or 8 steps per
# warp instruction: every (S, G) pair, rank counts that are not a multiple of
# the lanes per step, step counts that are not a multiple of the tile; then
# 6-12 KB steps just past that path (one step per warp, every S)
LANES = [(257, 376, 2), (300, 104, 2), (999, 40, 2), (211, 184, 4), (405, 52, 4), (333, 44, 4),
         (150, 94, 8), (97, 64, 8), (260, 46, 8), (70, 48, 16), (88, 33, 16),
         (61, 53, 16), (77, 100, 8), (99, 236, 4), (45, 440, 2),
         (45, 90, 16), (33, 180, 8), (50, 300, 4), (40, 696, 2)]


# generic path (odd S with R*S not a multiple of 16, even S with R*S not a
# multiple of 16, more than 16 stages): every stage bound of its kernels
# (S <= 4, <= 8, <= 16, <= 32)
GENERIC = [(23, 9, 11), (10, 5, 14), (17, 33, 7), (12, 101, 4), (8, 30, 24), (300, 1000, 5)]
# generic shapes with many steps (at least 4 x 8 per SM): one warp per step
GENERIC_MANY = [(6000, 9, 11), (6000, 33, 7), (6000, 10, 3), (6000, 5, 14), (6000, 7, 6)]


@pytest.mark.parametrize("T,R,S", SHAPES + GROUPED[4:] + LANES + GENERIC + GENERIC_MANY)
@pytest.mark.parametrize("kind", ["ties", "zeros", "lognormal", "mixed"])
def test_frontier_parity(sf, T, R, S, kind):
    d_np = make(T, R, S, T * 131 + R * 7 + S, kind)
    o = O.frontier(d_np)
    st = sf.new_status("cuda")
    f = sf.sf_frontier(dev(d_np), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(f.a), o.a)
    assert np.array_equal(host(f.lead), o.lead)
    assert np.array_equal(host(f.makespan), o.makespan)


@pytest.mark.parametrize("T,R,S", SHAPES[:10] + SHAPES[14:] + LANES[:6] + GENERIC)
@pytest.mark.parametrize("kind", ["ties", "zeros", "lognormal"])
def test_frontier_ties_parity(sf, T, R, S, kind):
    """Size of the lead rank's tie set per step and stage against the oracle."""
    d_np = make(T, R, S, T * 7 + R + S, kind)
    o = O.frontier(d_np)
    st = sf.new_status("cuda")
    ties = sf.sf_frontier_ties(dev(d_np), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(ties), o.ties)


@pytest.mark.parametrize("T,R,S", [(40, 64, 4), (30, 128, 8), (200, 256, 4), (20, 512, 4), (300, 1000, 10),
                                   (12, 1024, 10), (9, 4096, 2), (25, 48, 16), (7, 300, 6)])
@pytest.mark.parametrize("wide_even", [True, False])
def test_frontier_ties_across_narrow_and_wide_rows(sf, T, R, S, wide_even):
    """Every rank has the same durations except a 2^32 ns last stage on every
    other rank, so at every boundary before the last all ranks reach the
    frontier together, half of them on the 32-bit path and half on the 64-bit
    one: the lead rank must be rank 0 either way, and rank 0 or 1 at the last."""
    rng = np.random.default_rng(T + R + S)
    row = rng.integers(1, 1000, size=(T, 1, S), dtype=np.int64)
    d_np = np.repeat(row, R, axis=1)
    d_np[:, (0 if wide_even else 1)::2, S - 1] += 1 << 32
    o = O.frontier(d_np)
    st = sf.new_status("cuda")
    f = sf.sf_frontier(dev(d_np), status=st)
    g = sf.sf_window_aggregate(dev(d_np), 5, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(f.a), o.a) and np.array_equal(host(f.lead), o.lead)
    assert (o.lead[:, :S - 1] == 0).all()
    ow = O.windows(d_np, 5)
    for name in ("X", "D", "E", "C", "step_lead"):
        assert np.array_equal(host(getattr(g, name)), getattr(ow, name)), name


# Long step ranges: every CTA streams many tiles, so every ring stage is reused
# many times (both regimes, both passes).
LONG = [(200000, 8, 6), (20000, 64, 4), (8000, 128, 8), (3000, 512, 4), (1500, 1024, 10),
        (600, 4096, 8), (30000, 94, 8), (60000, 40, 2), (20000, 53, 16)]


@pytest.mark.parametrize("T,R,S", LONG)
def test_long_ranges_reuse_ring(sf, T, R, S):
    d_np = make(T, R, S, T + R, "ties" if R <= 64 else "lognormal")
    W = 100
    o = O.frontier(d_np)
    ow = O.windows(d_np, W)
    st = sf.new_status("cuda")
    d = dev(d_np)
    f = sf.sf_frontier(d, status=st)
    g = sf.sf_window_aggregate(d, W, status=st)
    m = sf.sf_window_median(d, W)
    ev = sf.sf_direct_gain(d, W, m, lead_credit=True, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(f.a), o.a) and np.array_equal(host(f.lead), o.lead)
    assert np.array_equal(host(f.makespan), o.makespan)
    for name in ("X", "D", "E", "C", "step_lead"):
        assert np.array_equal(host(getattr(g, name)), getattr(ow, name)), name
    assert np.array_equal(host(ev.X), ow.X) and np.array_equal(host(ev.D), ow.D)
    assert np.array_equal(host(ev.E), ow.E) and np.array_equal(host(ev.C), ow.C)
    assert np.array_equal(host(ev.step_lead) & 31, ow.step_lead)
    # gain numerators on the first two windows (the literal oracle is S x slower)
    m2 = O.window_median(d_np[:2 * W], W)
    assert np.array_equal(host(m)[:2], m2)
    assert np.array_equal(host(ev.Y)[:2], O.direct_gain(d_np[:2 * W], W, m2))


@pytest.mark.parametrize("T,R,S", SHAPES[:4] + SHAPES[5:9] + SHAPES[14:18] + GROUPED + LANES + GENERIC
                         + GENERIC_MANY)
@pytest.mark.parametrize("t0,W", [(0, 7), (13, 10), (0, 1000)])
def test_window_aggregate_parity(sf, T, R, S, t0, W):
    d_np = make(T, R, S, T + R + S + t0, "ties" if R < 100 else "lognormal")
    o = O.windows(d_np, W, t0)
    st = sf.new_status("cuda")
    g = sf.sf_window_aggregate(dev(d_np), W, t0=t0, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for name in ("X", "D", "E", "C", "step_lead"):
        assert np.array_equal(host(getattr(g, name)), getattr(o, name)), name


# fewer steps than SMs over many ranks: each step's ranks are split over a
# thread-block cluster (up to 16 CTAs) and combined through distributed
# shared memory; ragged rank splits included (R = 9000)
@pytest.mark.parametrize("T,R,S", [(1, 8192, 8), (8, 8192, 8), (64, 8192, 8), (1, 65536, 8), (8, 65536, 8),
                                   (64, 65536, 8), (3, 9000, 16), (100, 8192, 4), (20, 2048, 2)])
@pytest.mark.parametrize("kind", ["lognormal", "ties"])
def test_few_steps_split_ranks(sf, T, R, S, kind):
    d_np = make(T, R, S, T * 31 + R + S, kind)
    d = dev(d_np)
    st = sf.new_status("cuda")
    f = sf.sf_frontier(d, status=st)
    t0, W = 3, 7
    win = sf.sf_window_aggregate(d, W, t0=t0, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    o = O.frontier(d_np)
    assert np.array_equal(host(f.a), o.a)
    assert np.array_equal(host(f.lead), o.lead)
    assert np.array_equal(host(f.makespan), o.makespan)
    ow = O.windows(d_np, W, t0=t0)
    assert np.array_equal(host(win.X), ow.X) and np.array_equal(host(win.D), ow.D)
    assert np.array_equal(host(win.E), ow.E) and np.array_equal(host(win.C), ow.C)
    assert np.array_equal(host(win.step_lead), ow.step_lead)


def test_window_aggregate_chunked_accumulate(sf):
    T, R, S, W, chunk = 90, 64, 8, 25, 35
    d_np = make(T, R, S, 5, "lognormal")
    o = O.windows(d_np, W, 0)
    d = dev(d_np)
    nW = sf.num_windows(0, T, W)
    X = torch.zeros((nW, S), dtype=torch.int64, device="cuda")
    D = torch.zeros(nW, dtype=torch.int64, device="cuda")
    E = torch.zeros((nW, S, R), dtype=torch.int64, device="cuda")
    C = torch.zeros((nW, S, R), dtype=torch.int32, device="cuda")
    for t0 in range(0, T, chunk):
        w0 = t0 // W
        n = min(chunk, T - t0)
        sf.sf_window_aggregate(d[t0:t0 + n], W, t0=t0, X=X[w0:], D=D[w0:], E=E[w0:], C=C[w0:],
                               want=(), accumulate=True)
    assert np.array_equal(host(X), o.X) and np.array_equal(host(D), o.D)
    assert np.array_equal(host(E), o.E) and np.array_equal(host(C), o.C)


@pytest.mark.parametrize("nW,S,R,k", [(3, 5, 7, 6), (4, 8, 128, 2), (2, 10, 1024, 5), (1, 32, 3, 32),
                                      (5, 1, 1, 3)])
def test_topk_parity(sf, nW, S, R, k):
    rng = np.random.default_rng(nW * S * R)
    X = rng.integers(0, 4, size=(nW, S)).astype(np.int64)
    E = rng.integers(0, 4, size=(nW, S, R)).astype(np.int64)
    o = O.topk(X, E, k)
    t = sf.sf_topk_suspects(dev(X), dev(E), k)
    assert np.array_equal(host(t.stage), o.stage) and np.array_equal(host(t.stage_value), o.stage_value)
    assert np.array_equal(host(t.pair), o.pair) and np.array_equal(host(t.pair_value), o.pair_value)


@pytest.mark.parametrize("T,R,S,W", [(7, 3, 5, 1), (9, 4, 3, 2), (33, 2, 3, 3),
                                     (100, 8, 6, 100), (250, 4, 3, 32), (130, 5, 4, 64), (300, 2, 8, 128),
                                     (700, 3, 2, 256), (1100, 2, 4, 512), (2100, 1, 4, 1000),
                                     (2200, 2, 2, 1024), (2500, 1, 3, 1100), (45, 1024, 10, 20),
                                     (1200, 3, 2, 1000), (600, 2, 3, 200), (1990, 2, 4, 995)])
@pytest.mark.parametrize("kind", ["ties", "lognormal", "wide", "zeros", "ranges", "clusters"])
def test_median_parity(sf, T, R, S, W, kind):
    rng = np.random.default_rng(T + W)
    if kind == "wide":  # signed values spanning more than 2^32: the 64-bit search path
        d_np = rng.integers(-(1 << 40), 1 << 40, size=(T, R, S), dtype=np.int64)
    elif kind == "ranges":  # per-column range from 1 to 32 bits (the last at the 32-bit edge)
        bits = rng.integers(0, 33, size=(1, R, S))
        bits[0, 0, 0] = 32
        d_np = (rng.integers(0, 1 << 62, size=(T, R, S), dtype=np.int64) % (np.int64(1) << bits)) + (1 << 33)
    elif kind == "clusters":  # a few tight clusters: the chosen top-digit bin is large or just fits
        centers = rng.integers(0, 1 << 30, size=(4,))
        d_np = centers[rng.integers(0, 4, size=(T, R, S))] + rng.integers(0, 3, size=(T, R, S))
    else:
        d_np = make(T, R, S, T + W, kind)
    o = O.window_median(d_np, W)
    m = sf.sf_window_median(dev(d_np), W)
    assert np.array_equal(host(m), o)


@pytest.mark.parametrize("T,R,S,W", [(120, 8, 6, 50), (64, 128, 8, 30), (40, 1024, 10, 16),
                                     (33, 3, 5, 10), (20, 8192, 8, 8), (30, 64, 16, 30), (9, 5, 4, 1),
                                     (11, 40, 8, 2), (23, 9, 11, 5), (17, 33, 7, 4), (8, 30, 24, 3),
                                     (12, 101, 4, 6), (10, 5, 14, 3), (6000, 9, 11, 100), (6000, 33, 7, 250),
                                     (6000, 10, 3, 1000), (6000, 5, 14, 64)])
def test_direct_gain_parity(sf, T, R, S, W):
    d_np = make(T, R, S, R + S, "lognormal")
    m_np = O.window_median(d_np, W)
    Y = O.direct_gain(d_np, W, m_np)
    ow = O.windows(d_np, W)
    ev = sf.sf_direct_gain(dev(d_np), W, dev(m_np), lead_credit=True)
    assert np.array_equal(host(ev.Y), Y)
    assert np.array_equal(host(ev.D), [ow.D[w] for w in range(len(ow.D))])
    assert np.array_equal(host(ev.X), ow.X)
    assert np.array_equal(host(ev.E), ow.E) and np.array_equal(host(ev.C), ow.C)
    assert np.array_equal(host(ev.step_lead) & 31, ow.step_lead)


def compare_labels(sf, d_np, W, role=None, missing=None, wall=None, other_stage=-1, cfg=None):
    o = O.label_windows(d_np, W, role=role, missing=missing, wall=wall, other_stage=other_stage, cfg=cfg)
    args = {}
    for name, v in (("role", role), ("missing", missing), ("wall", wall)):
        if v is not None:
            args[name] = dev(v)
    cfg_sf = None
    if cfg is not None:
        cfg_sf = sf.default_config()
        cfg_sf.model_fit_mask = cfg.model_fit_mask
    st = sf.new_status("cuda")
    lab = sf.sf_label_windows(dev(d_np), W, other_stage=other_stage, cfg=cfg_sf, status=st, **args)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(lab.labels).astype(np.uint32), o.labels)
    assert np.array_equal(host(lab.route_mask).astype(np.uint32), o.route_mask)
    assert np.array_equal(host(lab.amb_mask).astype(np.uint32), o.amb_mask)
    assert np.array_equal(host(lab.X), o.X) and np.array_equal(host(lab.Y), o.Y)
    assert np.array_equal(host(lab.D), o.D)
    np.testing.assert_allclose(host(lab.share), o.share, rtol=RTOL, atol=0)
    np.testing.assert_allclose(host(lab.gain), o.gain, rtol=RTOL, atol=0)
    # the gates entry point also reports the leader-switch evidence
    ev = sf.sf_direct_gain(dev(d_np), W, sf.sf_window_median(dev(d_np), W))
    g = sf.sf_label_gates(d_np.shape[0], d_np.shape[1], d_np.shape[2], W, ev)
    assert np.array_equal(host(g.n_confident), o.n_confident)
    assert np.array_equal(host(g.n_switch), o.n_switch)
    return o


U = 1_000_000


def test_label_fixtures(sf):
    base = np.full((10, 4, 3), 10 * U, np.int64)
    base[0:4, 0, 0] += 30 * U                                     # intermittent data stall
    o = compare_labels(sf, base, 10)
    assert o.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_DIRECT_EXPOSURE
    compare_labels(sf, base, 10, missing=np.array([1], np.int32))
    compare_labels(sf, base, 10, role=np.array([0, 0, 1, 1], np.int32))
    tot = base.sum(axis=2)
    compare_labels(sf, base, 10, wall=tot + tot // 10)
    compare_labels(sf, base, 10, wall=tot - tot // 50)
    compare_labels(sf, base, 10, other_stage=2)
    sharp = np.repeat(np.array([[[10, 0], [0, 10]]], np.int64) * 10**9, 20, axis=0)
    o = compare_labels(sf, sharp, 20)
    assert o.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_CO_CRITICAL and o.amb_mask[0] == 3
    cfg = O.default_config()
    cfg.model_fit_mask = 1
    compare_labels(sf, sharp, 20, cfg=cfg)
    tie = np.full((10, 2, 2), 10 * U, np.int64)
    tie[0::2, 0, 0] += 30 * U
    tie[1::2, 0, 1] += 30 * U
    compare_labels(sf, tie, 10)
    compare_labels(sf, np.zeros((5, 3, 4), np.int64), 5)
    compare_labels(sf, np.concatenate([base, np.full((3, 4, 3), 10 * U, np.int64)]), 10)


@pytest.mark.parametrize("name,steps", [("tiny", None), ("ddp128", 3000), ("fsdp1024", 1000),
                                        ("accum8192", 60)])
def test_labels_on_workloads(sf, name, steps):
    w = wl.by_name(name, steps=steps)
    d_np = w.generate()
    W = min(w.W, max(1, steps // 3)) if steps else w.W
    rng = np.random.default_rng(1)
    missing = (rng.random((d_np.shape[0] + W - 1) // W) < 0.3).astype(np.int32)
    compare_labels(sf, d_np, W)
    compare_labels(sf, d_np, W, missing=missing, wall=w.wall(d_np), other_stage=w.S - 1)


def test_device_status_bits(sf):
    d_np = np.ones((16, 64, 8), np.int64)
    d_np[3, 5, 2] = -4
    st = sf.new_status("cuda")
    sf.sf_frontier(dev(d_np), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & sf.SF_ST_NEGATIVE
    d_np[3, 5, 2] = 1 << 47
    st.zero_()
    sf.sf_window_aggregate(dev(d_np), 4, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & sf.SF_ST_RANGE
    d_np[3, 5, 2] = 1 << 46
    d_np[3, 5, 3] = 1 << 46                          # rank total reaches 2^47
    st.zero_()
    sf.sf_frontier(dev(d_np), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == sf.SF_ST_RANGE
    d_np = np.ones((16, 3, 5), np.int64)             # generic path
    d_np[0, 0, 0] = -1
    st.zero_()
    sf.sf_frontier(dev(d_np), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & sf.SF_ST_NEGATIVE


def test_deterministic_repeat(sf):
    d = dev(make(200, 256, 8, 3, "ties"))
    a = sf.sf_window_aggregate(d, 50)
    b = sf.sf_window_aggregate(d, 50)
    for name in ("X", "D", "E", "C", "step_lead"):
        assert torch.equal(getattr(a, name), getattr(b, name))


def test_bounded_wait_times_out_cleanly(sf):
    """A device wait that can never complete gives up after its limit, reports
    SF_ST_TIMEOUT through the status word, and leaves the context usable."""
    st = sf.new_status("cuda")
    sf.sf_selftest_bounded_wait(50_000_000, st)      # 50 ms
    torch.cuda.synchronize()
    assert int(st.item()) == sf.SF_ST_TIMEOUT
    d = dev(make(40, 64, 8, 1, "lognormal"))          # the context still runs work
    f = sf.sf_frontier(d)
    assert np.array_equal(host(f.a), O.frontier(host(d)).a)


@pytest.mark.parametrize("T,R,S", SHAPES[:4] + SHAPES[5:9] + SHAPES[14:18] + GROUPED + GENERIC + GENERIC_MANY
                         + [(200000, 8, 6)])
@pytest.mark.parametrize("t0,W", [(0, 7), (13, 100)])
def test_baselines_parity(sf, T, R, S, t0, W):
    """Per-stage max, sum (128-bit), slowest-rank breakdown and rank-0 total
    per window against the oracle, on every streaming path."""
    d_np = make(T, R, S, T + 3 * R + S, "ties" if R < 100 else "lognormal")
    o = O.baselines(d_np, W, t0)
    st = sf.new_status("cuda")
    b = sf.sf_window_baselines(dev(d_np), W, t0=t0, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert np.array_equal(host(b.M), o.M)
    assert np.array_equal(host(b.SLOW), o.SLOW) and np.array_equal(host(b.RANK0), o.RANK0)
    s2 = host(b.SUM)
    got = [[int(s2[w, s, 1]) << 64 | int(s2[w, s, 0]) for s in range(S)] for w in range(s2.shape[0])]
    assert got == [list(r) for r in o.SUM]
