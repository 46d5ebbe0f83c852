"""Pins of the CPU oracle to facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: the paper's
worked examples (golden fixtures), Theorem 1, the slack identity, the bounds
of Propositions 1-3 with their tightness constructions, special cases that
reduce to a library routine (numpy sort / median / argmax, Python sorted),
brute-force single-rank-stall constructions, and hand-derived label fixtures.
"""
import itertools

import numpy as np
import pytest

from oracle import oracle as O
from tests.golden import fixtures

LIMIT47 = 1 << 47


def rand_d(rng, T, R, S, hi=10**6, zero_frac=0.0):
    d = rng.integers(0, hi, size=(T, R, S), dtype=np.int64)
    if zero_frac:
        d[rng.random((T, R, S)) < zero_frac] = 0
    return d


# ---------------------------------------------------------------- worked examples

def test_fig1_motivating_example():
    g = fixtures.load("fig1_motivating.txt")
    f = O.frontier(g["d"])
    u = g["unit_ns"]
    assert (f.a[0] == g["a"] * u).all()
    assert f.makespan[0] == g["makespan"][0] * u
    assert (f.lead[0] == g["lead"]).all()       # tie at bwd goes to the lowest rank, r0
    assert (f.ties[0] == g["ties"]).all()
    # the per-stage maximum the paper contrasts with the frontier
    assert g["d"][0].max(axis=0).sum() == g["per_stage_max_total"][0] * u


def test_fig2_frontier_example():
    g = fixtures.load("fig2_frontier.txt")
    f = O.frontier(g["d"])
    u = g["unit_ns"]
    assert (f.F[0] == g["F"] * u).all()
    assert (f.a[0] == g["a"] * u).all()
    assert f.makespan[0] == g["makespan"][0] * u
    assert (f.lead[0] == g["lead"]).all()


def test_sharp_cocritical_example():
    g = fixtures.load("sharp_cocritical.txt")
    W = int(g["W"][0])
    d = np.repeat(g["d"], W, axis=0)
    f = O.frontier(d)
    u = g["unit_ns"]
    assert (f.F == g["F"] * u).all() and (f.a == g["a"] * u).all() and (f.lead == g["lead"]).all()
    L = O.label_windows(d, W)
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_CO_CRITICAL
    assert L.amb_mask[0] == sum(1 << s for s in g["amb"])
    assert L.route_mask[0] == 0b01
    assert (L.Y == 0).all()


# ---------------------------------------------------------------- Theorem 1 / identities

@pytest.mark.parametrize("T,R,S", [(50, 1, 1), (40, 3, 5), (30, 17, 8), (10, 64, 13)])
def test_telescoping_exact(T, R, S):
    rng = np.random.default_rng(T * 1000 + R * 10 + S)
    d = rand_d(rng, T, R, S, zero_frac=0.2)
    f = O.frontier(d)
    assert (f.a >= 0).all()
    assert (f.a.sum(axis=1) == f.makespan).all()          # Theorem 1, exact in int64
    assert (f.makespan == d.sum(axis=2).max(axis=1)).all()  # F_{t,S} is the largest rank total


@pytest.mark.parametrize("seed", range(4))
def test_slack_identity(seed):
    rng = np.random.default_rng(seed)
    T, R, S = 25, 7, 6
    d = rand_d(rng, T, R, S, zero_frac=0.3)
    f = O.frontier(d)
    P = np.cumsum(d, axis=2)
    Fprev = np.concatenate([np.zeros((T, 1), np.int64), f.F[:, :-1]], axis=1)
    Pprev = np.concatenate([np.zeros((T, R, 1), np.int64), P[:, :, :-1]], axis=2)
    lam = Fprev[:, None, :] - Pprev            # slack lambda_{t,r,s} >= 0
    assert (lam >= 0).all()
    assert (f.a == (d - lam).max(axis=1)).all()


@pytest.mark.parametrize("seed", range(3))
def test_prop1_prop2_bounds(seed):
    rng = np.random.default_rng(100 + seed)
    T, R, S = 40, 9, 5
    d = rand_d(rng, T, R, S, zero_frac=0.3)
    f = O.frontier(d)
    M = d.max(axis=1).sum(axis=1)
    Mbar_R = d.sum(axis=1).sum(axis=1)          # R * average summary, kept integral
    F = f.makespan
    assert (F <= M).all() and (M <= min(R, S) * F).all()
    assert (F <= Mbar_R).all() and (Mbar_R <= R * F).all()


@pytest.mark.parametrize("R,S", [(3, 5), (5, 3), (4, 4)])
def test_prop1_tightness(R, S):
    # min(R,S) distinct rank-stage pairs of duration D, no rank holding two
    Dv = 7_000_000
    d = np.zeros((1, R, S), np.int64)
    for i in range(min(R, S)):
        d[0, i, i] = Dv
    f = O.frontier(d)
    M = d.max(axis=1).sum()
    assert M == min(R, S) * f.makespan[0]


def test_prop2_tightness():
    R, S = 6, 4
    d = np.zeros((1, R, S), np.int64)
    d[0, 2] = [1, 2, 3, 4]                      # one rank with total D, all others zero
    f = O.frontier(d)
    assert d.sum() == f.makespan[0]             # R * Mbar == F, i.e. Mbar = F / R


@pytest.mark.parametrize("seed", range(4))
def test_prop3_stability(seed):
    rng = np.random.default_rng(200 + seed)
    T, R, S, eps = 30, 6, 7, 1000
    d = rand_d(rng, T, R, S, hi=10**6) + eps
    delta = rng.integers(-eps, eps + 1, size=d.shape)
    f0, f1 = O.frontier(d), O.frontier(d + delta)
    s1 = np.arange(1, S + 1)                    # 1-based stage index
    assert (np.abs(f1.F - f0.F) <= s1 * eps).all()
    assert (np.abs(f1.a - f0.a) <= (2 * s1 - 1) * eps).all()


# ---------------------------------------------------------------- special cases

def test_single_rank_reduces_to_its_vector():
    rng = np.random.default_rng(7)
    d = rand_d(rng, 20, 1, 9)
    f = O.frontier(d)
    assert (f.a == d[:, 0, :]).all() and (f.lead == 0).all() and (f.ties == 1).all()


def test_identical_ranks():
    rng = np.random.default_rng(8)
    base = rand_d(rng, 15, 1, 6)
    d = np.repeat(base, 11, axis=1)
    f = O.frontier(d)
    assert (f.a == base[:, 0, :]).all() and (f.lead == 0).all() and (f.ties == 11).all()


@pytest.mark.parametrize("R,S", [(2, 2), (3, 4), (5, 6)])
def test_single_rank_stall_brute_force(R, S):
    """Identical ranks, no sync stage, a stall Delta on (r*, s*): only a[s*]
    grows, by exactly Delta, and r* leads every boundary from s* on."""
    rng = np.random.default_rng(R * 10 + S)
    base = rng.integers(1, 10**6, size=S, dtype=np.int64)
    for r_star, s_star in itertools.product(range(R), range(S)):
        Delta = int(rng.integers(1, 10**6))
        d = np.tile(base, (1, R, 1))
        d[0, r_star, s_star] += Delta
        f = O.frontier(d)
        exp_a = base.copy()
        exp_a[s_star] += Delta
        assert (f.a[0] == exp_a).all()
        exp_lead = np.where(np.arange(S) >= s_star, r_star, 0)
        assert (f.lead[0] == exp_lead).all()


def test_rank_permutation_invariance():
    rng = np.random.default_rng(9)
    d = rand_d(rng, 12, 6, 5, hi=50)           # small values: many ties
    perm = rng.permutation(6)
    f0, f1 = O.frontier(d), O.frontier(d[:, perm, :])
    assert (f0.F == f1.F).all() and (f0.a == f1.a).all() and (f0.ties == f1.ties).all()


def test_input_errors():
    d = np.ones((2, 3, 4), np.int64)
    d[1, 2, 3] = -1
    with pytest.raises(O.OracleError) as e:
        O.frontier(d)
    assert e.value.rc == O.NEGATIVE
    d[1, 2, 3] = LIMIT47
    with pytest.raises(O.OracleError) as e:
        O.frontier(d)
    assert e.value.rc == O.RANGE
    d[1, 2, 3] = LIMIT47 // 2
    d[1, 2, 2] = LIMIT47 // 2                   # prefix reaches 2^47
    with pytest.raises(O.OracleError) as e:
        O.frontier(d)
    assert e.value.rc == O.RANGE


# ---------------------------------------------------------------- windows (Eq. 2)

@pytest.mark.parametrize("t0,W", [(0, 7), (5, 7), (13, 4), (0, 100)])
def test_window_invariants(t0, W):
    rng = np.random.default_rng(t0 + W)
    T, R, S = 37, 5, 4
    d = rand_d(rng, T, R, S, hi=30, zero_frac=0.2)   # many ties
    w = O.windows(d, W, t0)
    f = O.frontier(d)
    nW = O.num_windows(t0, T, W)
    assert w.X.shape == (nW, S)
    assert (w.X.sum(axis=1) == w.D).all()
    assert (w.E.sum(axis=2) == w.X).all()
    g = np.arange(T) + t0
    widx = g // W - t0 // W
    n_w = np.bincount(widx, minlength=nW)
    assert (w.C.sum(axis=2) == n_w[:, None]).all()
    assert (w.step_lead == np.argmax(f.a, axis=1)).all()   # numpy argmax: first maximum
    for i in range(nW):
        sel = widx == i
        assert (w.X[i] == f.a[sel].sum(axis=0)).all() and w.D[i] == f.makespan[sel].sum()


def test_window_chunk_additivity():
    rng = np.random.default_rng(11)
    T, R, S, W = 60, 4, 3, 25
    d = rand_d(rng, T, R, S)
    whole = O.windows(d, W, 0)
    a = O.windows(d[:35], W, 0)      # windows 0..1
    b = O.windows(d[35:], W, 35)     # windows 1..2
    X = np.zeros_like(whole.X)
    X[:2] += a.X
    X[1:] += b.X
    assert (X == whole.X).all()


# ---------------------------------------------------------------- top-k

@pytest.mark.parametrize("seed", range(3))
def test_topk_against_sorted(seed):
    rng = np.random.default_rng(300 + seed)
    nW, S, R, k = 3, 5, 7, 6
    X = rng.integers(0, 4, size=(nW, S)).astype(np.int64)
    E = rng.integers(0, 4, size=(nW, S, R)).astype(np.int64)
    t = O.topk(X, E, k)
    for w in range(nW):
        st = sorted([(-X[w, s], s) for s in range(S) if X[w, s] > 0])[:k]
        exp = [s for _, s in st] + [-1] * (k - len(st))
        assert list(t.stage[w]) == exp
        pr = sorted([(-E[w, s, r], s, r) for s in range(S) for r in range(R) if E[w, s, r] > 0])[:k]
        exp_p = [[s, r] for _, s, r in pr] + [[-1, -1]] * (k - len(pr))
        assert t.pair[w].tolist() == exp_p
        assert list(t.pair_value[w]) == [-v for v, _, _ in pr] + [0] * (k - len(pr))


# ---------------------------------------------------------------- median and gain (Eq. 4)

@pytest.mark.parametrize("T,W", [(30, 10), (31, 10), (9, 4), (5, 16)])
def test_median_is_lower_median(T, W):
    rng = np.random.default_rng(T + W)
    R, S = 3, 4
    d = rand_d(rng, T, R, S, hi=20)
    m = O.window_median(d, W)
    for w in range((T + W - 1) // W):
        blk = d[w * W:(w + 1) * W]
        n = blk.shape[0]
        assert (m[w] == np.sort(blk, axis=0)[(n - 1) // 2]).all()
        if n % 2 == 1:
            assert (m[w] == np.median(blk, axis=0)).all()


@pytest.mark.parametrize("seed", range(4))
def test_gain_closed_form_and_sign(seed):
    """Replacing one stage shifts only the prefixes at and after it, so
    F'_S = max_r (P_{t,r,S} - max(0, d_{t,r,s} - m_{r,s})); G_s >= 0."""
    rng = np.random.default_rng(400 + seed)
    T, R, S, W = 23, 6, 5, 8
    d = rand_d(rng, T, R, S, hi=1000, zero_frac=0.1)
    m = O.window_median(d, W)
    Y = O.direct_gain(d, W, m)
    assert (Y >= 0).all()
    PS = d.sum(axis=2)
    FS = PS.max(axis=1)
    exp = np.zeros_like(Y)
    for t in range(T):
        w = t // W
        cut = np.maximum(0, d[t] - m[w])            # [R][S]
        Fp = (PS[t][:, None] - cut).max(axis=0)     # [S]
        exp[w] += FS[t] - Fp
    assert (Y == exp).all()


def test_gain_single_rank_and_constant_window():
    rng = np.random.default_rng(5)
    d = rand_d(rng, 20, 1, 4)
    W = 10
    m = O.window_median(d, W)
    Y = O.direct_gain(d, W, m)
    for w in range(2):
        assert (Y[w] == np.maximum(0, d[w * W:(w + 1) * W, 0, :] - m[w, 0]).sum(axis=0)).all()
    const = np.repeat(rand_d(rng, 1, 5, 4), 12, axis=0)
    assert (O.direct_gain(const, 6, O.window_median(const, 6)) == 0).all()


# ---------------------------------------------------------------- labels: hand-derived fixtures

U = 1_000_000  # 1 ms


def _intermittent_data_stall():
    """R=4, S=3, W=10, every duration 10 ms; r0's data +30 ms on steps 0-3.
    Stalled steps: a=(40,10,10), F_S=60; others a=(10,10,10), F_S=30.
    X=(220,100,100), D=420 -> A_data=0.524>0.4.  r0's data median over
    {40 x4, 10 x6} is 10, so the clipped replacement removes the stall:
    Y_data=4*(60-30)=120, G=0.286>=0.1 -> direct_exposure.  C_A=C_G={data}.
    Only the 4 stalled steps are confident (margin 30 >= 0.05*60), all data."""
    d = np.full((10, 4, 3), 10 * U, np.int64)
    d[0:4, 0, 0] += 30 * U
    return d


def test_label_direct_exposure():
    L = O.label_windows(_intermittent_data_stall(), 10)
    assert (L.X[0] == np.array([220, 100, 100]) * U).all() and L.D[0] == 420 * U
    assert (L.Y[0] == np.array([120, 0, 0]) * U).all()
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_DIRECT_EXPOSURE
    assert L.amb_mask[0] == 0b001
    # cumulative X: 220 < 336, 320 < 336, 420 >= 336 = 0.8*420
    assert L.route_mask[0] == 0b111
    assert L.n_confident[0] == 4 and L.n_switch[0] == 0
    assert L.share[0, 0] == 220 / 420 and L.gain[0, 0] == 120 / 420


def test_label_sync_wait_dependent_with_model_fit():
    g = fixtures.load("sharp_cocritical.txt")
    d = np.repeat(g["d"], 20, axis=0)
    cfg = O.default_config()
    cfg.model_fit_mask = 0b01                       # W_data = 1
    L = O.label_windows(d, 20, cfg=cfg)
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_SYNC_WAIT_DEPENDENT
    assert L.amb_mask[0] == 0b11


def test_label_telemetry_limited_missing_rank():
    L = O.label_windows(_intermittent_data_stall(), 10, missing=np.array([1]))
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_TELEMETRY_LIMITED


def test_label_telemetry_limited_closure_and_overlap():
    d = _intermittent_data_stall()
    tot = d.sum(axis=2)
    ok = O.label_windows(d, 10, wall=tot + tot // 25)          # 4 % residual: under 5 %
    assert ok.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_DIRECT_EXPOSURE
    bad = O.label_windows(d, 10, wall=tot + tot // 10)         # 10 % residual
    assert bad.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_TELEMETRY_LIMITED
    ovl = O.label_windows(d, 10, wall=tot - tot // 50)         # 2 % overlap > 1 %
    assert ovl.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_TELEMETRY_LIMITED
    # a recorded residual stage (stage 2 as "other") carrying 100/420 of the time
    oth = O.label_windows(d, 10, other_stage=2)
    assert oth.labels[0] & O.L_TELEMETRY_LIMITED


def test_label_role_aware_needed():
    L = O.label_windows(_intermittent_data_stall(), 10, role=np.array([0, 0, 1, 1]))
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_ROLE_AWARE_NEEDED
    same = O.label_windows(_intermittent_data_stall(), 10, role=np.array([3, 3, 3, 3]))
    assert same.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_DIRECT_EXPOSURE


def test_label_two_stage_tie():
    """R=2, S=2, W=10, base 10 ms; even steps r0 data +30, odd steps r0 bwd
    +30: a alternates (40,10)/(10,40), X=(250,250), D=500 -> C_A={0,1};
    every step is confident with alternating leaders (9 switches of 10);
    medians of r0 are 10 so Y=(150,150), G=0.3 each (a gain tie)."""
    d = np.full((10, 2, 2), 10 * U, np.int64)
    d[0::2, 0, 0] += 30 * U
    d[1::2, 0, 1] += 30 * U
    L = O.label_windows(d, 10)
    assert (L.X[0] == [250 * U, 250 * U]).all() and (L.Y[0] == [150 * U, 150 * U]).all()
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_CO_CRITICAL
    assert L.amb_mask[0] == 0b11 and L.n_confident[0] == 10 and L.n_switch[0] == 9


def test_label_leader_switch_only():
    """Even steps r0 data +50, odd steps r0 bwd +30 (base 10, R=2, W=10):
    a = (60,10) / (10,40); X=(350,250), D=600: C_A={data} (gap 100 >= 30),
    A_data=0.583 high; r0 medians: data {60x5,10x5}->10, bwd {40x5,10x5}->10,
    so Y=(250,150), G_data=0.417 (direct evidence), C_G={data} (gap 100).
    All 10 steps are confident and alternate -> high switch -> co_critical,
    and direct_exposure is downgraded."""
    d = np.full((10, 2, 2), 10 * U, np.int64)
    d[0::2, 0, 0] += 50 * U
    d[1::2, 0, 1] += 30 * U
    L = O.label_windows(d, 10)
    assert (L.X[0] == [350 * U, 250 * U]).all() and L.D[0] == 600 * U
    assert (L.Y[0] == [250 * U, 150 * U]).all()
    assert L.n_switch[0] == 9
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_CO_CRITICAL
    assert L.amb_mask[0] == 0b01


def test_label_raw_only_zero_window():
    L = O.label_windows(np.zeros((5, 3, 4), np.int64), 5)
    assert L.labels[0] == O.L_FRONTIER_ACCOUNTING | O.L_TELEMETRY_LIMITED | O.L_RAW_ONLY
    assert L.route_mask[0] == 0 and L.amb_mask[0] == 0 and (L.share == 0).all()


def test_label_partial_last_window():
    d = np.concatenate([_intermittent_data_stall(), np.full((3, 4, 3), 10 * U, np.int64)])
    L = O.label_windows(d, 10)
    assert L.labels.shape == (2,)
    # last window: 3 identical steps, three-way share tie, no confident leader
    assert L.labels[1] == O.L_FRONTIER_ACCOUNTING | O.L_CO_CRITICAL
    assert L.amb_mask[1] == 0b111 and L.n_confident[1] == 0


# ---------------------------------------------------------------- routing baselines (Sec. 3, Sec. 6)

@pytest.mark.parametrize("seed", range(3))
def test_baselines_bounds_and_identities(seed):
    """Props 1-2 summed over a window: D <= sum_s M <= min(R,S) D and
    D <= sum_s SUM <= R D; the slowest rank's breakdown sums to D exactly (its
    total is the makespan); rank 0's total never exceeds D."""
    rng = np.random.default_rng(500 + seed)
    T, R, S, W = 45, 7, 5, 10
    d = rand_d(rng, T, R, S, hi=1000, zero_frac=0.2)
    b = O.baselines(d, W)
    w = O.windows(d, W)
    for i in range(len(w.D)):
        Dw = int(w.D[i])
        assert Dw <= int(b.M[i].sum()) <= min(R, S) * Dw
        assert Dw <= sum(b.SUM[i]) <= R * Dw
        assert int(b.SLOW[i].sum()) == Dw
        assert int(b.RANK0[i].sum()) <= Dw
    # against numpy reductions of the same definitions
    lead = O.frontier(d).lead[:, -1]
    for i in range(len(w.D)):
        blk = slice(i * W, (i + 1) * W)
        assert (b.M[i] == d[blk].max(axis=1).sum(axis=0)).all()
        assert list(b.SUM[i]) == [int(x) for x in d[blk].sum(axis=(0, 1))]
        assert (b.SLOW[i] == d[blk][np.arange(d[blk].shape[0]), lead[blk]].sum(axis=0)).all()
        assert (b.RANK0[i] == d[blk, 0, :].sum(axis=0)).all()


def test_baselines_special_cases():
    rng = np.random.default_rng(9)
    one = rand_d(rng, 12, 1, 4)
    b, w = O.baselines(one, 5), O.windows(one, 5)
    for arr in (b.M, b.SLOW, b.RANK0):                 # R = 1: every summary is the accounting
        assert (arr == w.X).all()
    base = rand_d(rng, 12, 1, 4)
    same = np.repeat(base, 6, axis=1)                  # identical ranks
    b, w = O.baselines(same, 5), O.windows(same, 5)
    assert (b.M == w.X).all() and (b.SLOW == w.X).all()
    assert [list(r) for r in b.SUM] == [[6 * int(x) for x in row] for row in w.X]
    # Prop 1 tightness: min(R,S) pairs of duration Dv, no rank holding two
    dt = np.zeros((1, 3, 5), np.int64)
    for i in range(3):
        dt[0, i, i] = 7
    b, w = O.baselines(dt, 1), O.windows(dt, 1)
    assert b.M[0].sum() == 3 * w.D[0]


def test_baselines_big_sums_are_exact():
    d = np.full((4, 3, 1), (1 << 46) + 12345, np.int64)  # each rank total just under 2^47
    b = O.baselines(d, 4)
    assert b.SUM[0][0] == 12 * ((1 << 46) + 12345)    # above 2^49, exact


# ---------------------------------------------------------------- localization evidence (Sec. 4) and spread (Sec. 6)

@pytest.mark.parametrize("seed", range(3))
def test_lag_against_library_routines(seed):
    rng = np.random.default_rng(600 + seed)
    T, R, S = 20, 9, 5                                   # odd R: lower median == np.median
    d = rand_d(rng, T, R, S, hi=50, zero_frac=0.2)
    g = O.rank_lag(d)
    P = np.cumsum(d, axis=2)
    F = P.max(axis=1)
    assert (g.L == F - np.median(P, axis=1).astype(np.int64)).all()
    assert (g.G == F - np.sort(P, axis=1)[:, -2, :]).all()
    assert (g.dL == np.diff(np.concatenate([np.zeros((T, 1), np.int64), g.L], axis=1), axis=1)).all()
    assert (g.L >= 0).all() and (g.G >= 0).all()
    assert (F == O.frontier(d).F).all()                  # the lag's maximum is the frontier


def test_lag_special_cases():
    rng = np.random.default_rng(3)
    one = rand_d(rng, 6, 1, 4)
    g = O.rank_lag(one)
    assert (g.L == 0).all() and (g.G == 0).all()          # R = 1: no cross-rank evidence
    same = np.repeat(rand_d(rng, 6, 1, 4), 5, axis=1)
    g = O.rank_lag(same)
    assert (g.L == 0).all() and (g.G == 0).all()          # identical ranks: no lag, tied top
    # a stall Delta on one rank of otherwise identical ranks (R >= 3, no sync):
    # from the stalled stage on, the lag and the gap are both exactly Delta
    base = rng.integers(1, 1000, size=4).astype(np.int64)
    d = np.tile(base, (1, 5, 1))
    d[0, 2, 1] += 777
    g = O.rank_lag(d)
    assert list(g.L[0]) == [0, 777, 777, 777] and list(g.G[0]) == [0, 777, 777, 777]
    assert list(g.dL[0]) == [0, 777, 0, 0]


def test_raw_spread():
    rng = np.random.default_rng(11)
    T, R, S, W = 30, 7, 4, 8
    d = rand_d(rng, T, R, S, hi=100)
    sp = O.raw_spread(d, W)
    per_step = d.max(axis=1) - np.median(d, axis=1).astype(np.int64)
    for w in range(sp.shape[0]):
        assert (sp[w] == per_step[w * W:(w + 1) * W].sum(axis=0)).all()
    assert (O.raw_spread(np.repeat(d[:, :1], 5, axis=1), W) == 0).all()


# ---------------------------------------------------------------- role groups (App. A) and reporting groups (Sec. 3)

@pytest.mark.parametrize("seed", range(3))
def test_group_windows_one_group_is_the_global_frontier(seed):
    rng = np.random.default_rng(700 + seed)
    T, R, S, W = 25, 6, 4, 7
    d = rand_d(rng, T, R, S, hi=80, zero_frac=0.2)
    gw = O.group_windows(d, np.zeros(R, np.int32), 1, W, t0=3)
    w = O.windows(d, W, t0=3)
    assert (gw.X[0] == w.X).all() and (gw.D[0] == w.D).all()


def test_group_windows_singletons_are_rank_sums():
    # one rank per group: the group frontier is the rank's own prefix, so the
    # increments are its durations and the makespan its total
    rng = np.random.default_rng(5)
    T, R, S, W = 12, 5, 3, 4
    d = rand_d(rng, T, R, S, hi=60)
    gw = O.group_windows(d, np.arange(R, dtype=np.int32), R, W)
    for g in range(R):
        for w in range(gw.X.shape[1]):
            assert (gw.X[g, w] == d[w * W:(w + 1) * W, g, :].sum(axis=0)).all()
            assert gw.D[g, w] == d[w * W:(w + 1) * W, g, :].sum()


def test_group_windows_invariants_and_empty_groups():
    rng = np.random.default_rng(9)
    T, R, S, W = 40, 9, 5, 10
    d = rand_d(rng, T, R, S, hi=50, zero_frac=0.3)
    group = rng.integers(0, 3, size=R).astype(np.int32)
    group[group == 2] = 1                                # group 2 left empty, group 3 too
    gw = O.group_windows(d, group, 4, W)
    w = O.windows(d, W)
    assert (gw.X >= 0).all()                             # group frontiers are monotone in s
    assert (gw.X.sum(axis=2) == gw.D).all()              # Theorem 1 inside each group
    assert (gw.X[2] == 0).all() and (gw.D[2] == 0).all() and (gw.D[3] == 0).all()
    assert (gw.D <= w.D).all() and (w.D <= gw.D.sum(axis=0)).all()
    # permuting ranks together with their group ids changes nothing
    perm = rng.permutation(R)
    gp = O.group_windows(d[:, perm, :], group[perm], 4, W)
    assert (gp.X == gw.X).all() and (gp.D == gw.D).all()


def test_stage_group_sum():
    rng = np.random.default_rng(4)
    d = rand_d(rng, 30, 4, 8, hi=90)
    w = O.windows(d, 10)
    assert (O.stage_group_sum(w.X, np.arange(8), 8) == w.X).all()          # singletons: identity
    assert (O.stage_group_sum(w.X, np.zeros(8), 1)[:, 0] == w.D).all()     # one group: Theorem 1
    fb = np.array([0, 1] * 4)                                              # f1 b1 f2 b2 ... -> fwd, bwd
    y = O.stage_group_sum(w.X, fb, 2)
    assert (y[:, 0] == w.X[:, 0::2].sum(axis=1)).all() and (y.sum(axis=1) == w.D).all()


def _lower_median_by_counting(col):
    """The smallest value v of the column with #{x <= v} >= ceil(n/2): for an
    even n this is the lower of the two middle values, for an odd n the median."""
    n = len(col)
    return min(v for v in col if sum(1 for x in col if x <= v) >= (n + 1) // 2)


@pytest.mark.parametrize("R", [2, 4, 8, 64])
def test_lag_even_ranks_take_the_lower_median(R):
    """Sec. 4 lag L = max_r P - median_r P with an even number of ranks: the
    median is the lower of the two middle prefixes (the reading that keeps the
    lag an exact integer).  Checked against numpy's 'lower' percentile and a
    brute-force count, on data with many ties."""
    rng = np.random.default_rng(800 + R)
    T, S = 9, 4
    d = rand_d(rng, T, R, S, hi=6, zero_frac=0.3)           # few distinct values: ties
    g = O.rank_lag(d)
    P = np.cumsum(d, axis=2)
    F = P.max(axis=1)
    lower = np.percentile(P, 50, axis=1, method="lower").astype(np.int64)
    assert (g.L == F - lower).all()
    for t in range(T):
        for s in range(S):
            assert g.L[t, s] == F[t, s] - _lower_median_by_counting(list(P[t, :, s]))
    second = np.sort(P, axis=1)[:, -2, :]
    assert (g.G == F - second).all()
    # the upper middle value would give a different lag somewhere on this data
    upper = np.sort(P, axis=1)[:, R // 2, :]
    assert (lower != upper).any()


def test_lag_and_spread_four_rank_fixture():
    """Hand fixture for the even-R reading: one step, one stage, four ranks
    with durations (= prefixes) 5, 9, 1, 2.  Sorted 1 2 5 9: the lower middle
    value is 2, so L = 9 - 2 = 7 (the upper middle would give 4, the mean of
    the two 5.5); the gap to the second largest is 9 - 5 = 4; the raw spread
    of the window is the same 7."""
    d = np.array([[[5], [9], [1], [2]]], np.int64)
    g = O.rank_lag(d)
    assert g.L.tolist() == [[7]] and g.G.tolist() == [[4]] and g.dL.tolist() == [[7]]
    assert O.raw_spread(d, 1).tolist() == [[7]]
    # two stages: prefixes (5,8) (9,9) (1,11) (2,2) -> stage 1 column 8 9 11 2,
    # sorted 2 8 9 11, lower middle 8: L = 11 - 8 = 3, delta-lag 3 - 7 = -4
    d2 = np.array([[[5, 3], [9, 0], [1, 10], [2, 0]]], np.int64)
    g2 = O.rank_lag(d2)
    assert g2.L.tolist() == [[7, 3]] and g2.dL.tolist() == [[7, -4]] and g2.G.tolist() == [[4, 2]]
    # spread of the durations: stage 0 as above (7); stage 1 column 3 0 10 0,
    # sorted 0 0 3 10, lower middle 0: 10 - 0 = 10
    assert O.raw_spread(d2, 1).tolist() == [[7, 10]]


@pytest.mark.parametrize("R", [2, 8, 64])
def test_raw_spread_even_ranks_take_the_lower_median(R):
    rng = np.random.default_rng(900 + R)
    T, S, W = 14, 3, 5
    d = rand_d(rng, T, R, S, hi=5, zero_frac=0.2)
    sp = O.raw_spread(d, W)
    per_step = d.max(axis=1) - np.percentile(d, 50, axis=1, method="lower").astype(np.int64)
    for w in range(sp.shape[0]):
        assert (sp[w] == per_step[w * W:(w + 1) * W].sum(axis=0)).all()
    t, s = 3, 1
    assert per_step[t, s] == d[t, :, s].max() - _lower_median_by_counting(list(d[t, :, s]))


def test_lag_windows():
    # window sums of the per-step evidence; a stall Delta on one of otherwise
    # identical ranks at step t contributes Delta to every stage from the
    # stalled one on, in the window of t only
    rng = np.random.default_rng(21)
    base = rng.integers(1, 1000, size=(7, 1, 4)).astype(np.int64)
    d = np.repeat(base, 5, axis=1)
    d[4, 3, 2] += 555
    LW, GW = O.rank_lag_windows(d, 3, t0=1)          # windows: steps {0,1}, {2,3,4}, {5,6}
    assert LW.shape == (3, 4)
    assert (LW[0] == 0).all() and (LW[2] == 0).all() and list(LW[1]) == [0, 0, 555, 555]
    assert (GW == LW).all()
    d2 = rand_d(rng, 20, 6, 3, hi=40, zero_frac=0.2)
    g = O.rank_lag(d2)
    LW2, GW2 = O.rank_lag_windows(d2, 7)
    for w in range(LW2.shape[0]):
        assert (LW2[w] == g.L[w * 7:(w + 1) * 7].sum(axis=0)).all()
        assert (GW2[w] == g.G[w * 7:(w + 1) * 7].sum(axis=0)).all()
