"""Pins of the oracle's worker-configuration model (Sec. 4.1: Eq. TP compute,
the all-reduce overhead, M = N_g m_gpu - m_model, Eq. max throughput) and of
the worker-count model of Sec. 5.2 (Eq. total_worker_pre), against numbers
worked by hand, closed forms of the arithmetic series, limiting cases and a
library least-squares fit."""
import math

import numpy as np
import pytest

BASE = dict(k1=0.001, c1=10.0, k2=2e-4, c2=0.05, c3=8.0, h=1, j=0, T_pre=1000.0, T_dec=50.0,
            gamma=0.5, theta=1.0, K=8192)


def test_tp_config_hand(orc):
    # k4 = 30, c4 = 10, kc = 4, 4 GPUs: (30/4 + 10 + 4 * 3/4) / (30 + 10) = 20.5 / 40
    M, s = orc.tp_config(30.0, 10.0, 4.0, 80_000.0, 30_000.0, 4)
    assert M == 4 * 80_000.0 - 30_000.0
    assert s == pytest.approx(0.5125, rel=1e-15)
    M1, s1 = orc.tp_config(30.0, 10.0, 4.0, 80_000.0, 30_000.0, 1)
    assert M1 == 50_000.0 and s1 == 1.0
    # many GPUs: the compute term vanishes, the all-reduce term tends to kc
    _, s_big = orc.tp_config(30.0, 10.0, 4.0, 80_000.0, 30_000.0, 1 << 20)
    assert s_big == pytest.approx(14.0 / 40.0, rel=1e-5)


def test_trace_demand_closed_form(orc):
    """A request (a, r) holds a + s tokens in its s-th iteration: summed over
    s = 1..r that is r a + r (r + 1) / 2, so the iteration-averaged context
    is sum(r a + r (r + 1) / 2) / sum(r), and KV = h context + j."""
    rng = np.random.default_rng(1)
    a = rng.integers(0, 2000, 300)
    r = rng.integers(1, 1000, 300)
    p = dict(BASE, h=3, j=5)
    m_r, l_ave = orc.trace_demand(p, a, r)
    ctx = float(np.sum(r * a + r * (r + 1) // 2)) / float(np.sum(r))
    assert l_ave == pytest.approx(ctx, rel=1e-14)
    assert m_r == pytest.approx(3 * ctx + 5, rel=1e-14)
    # one request (100, 100): 100 + 101/2 = 150.5
    assert orc.trace_demand(BASE, [100], [100]) == (150.5, 150.5)


@pytest.mark.parametrize("g,M,scale,want,bound", [
    # b_kv = 65536 / 150.5 = 435.455; t(b_kv) = 8 + 0.05 b_kv + 2e-4 * 65536 = 42.880 ms;
    # 435.455 / 42.880 = 10.1552 tokens/ms, below the SLO bound 524.345 / 50 = 10.4869
    (1, 65536.0, 1.0, 10.155214117, "kv"),
    # s = 1/sqrt(2): B = (50 sqrt(2) - 8) / 0.0801 = 782.905, 782.905 / (2 * 50) = 7.82905,
    # below the KV bound 870.910 / (2 * 54.985) = 7.91959
    (2, 131072.0, 1.0 / math.sqrt(2.0), 7.829048454, "slo"),
])
def test_max_throughput_hand(orc, g, M, scale, want, bound):
    t = orc.max_throughput(BASE, g, M, scale, 150.5, 150.5)
    assert t == pytest.approx(want, rel=1e-9)


def test_max_throughput_limits(orc):
    """T_dec without bound: only the KV term, b_kv / (g t(b_kv)); KV without
    bound: only the SLO term B / (g T_dec) with B from Eq. input limit."""
    m_r, l = 640.0, 640.0
    t = orc.max_throughput(dict(BASE, T_dec=1e12), 2, 131072.0, 0.8, m_r, l)
    b = 131072.0 / m_r
    assert t == pytest.approx(b / (2 * 0.8 * (8 + 0.05 * b + 2e-4 * b * l)), rel=1e-12)
    t = orc.max_throughput(BASE, 4, 1e15, 0.5, m_r, l)
    B = (50.0 / 0.5 - 8.0) / (0.05 + 2e-4 * l)
    assert t == pytest.approx(B / (4 * 50.0), rel=1e-12)


def test_pick_config(orc):
    gpus = [1, 2, 4, 8]
    M = [65536.0 * g for g in gpus]
    sc = [1.0 / math.sqrt(g) for g in gpus]
    best, t = orc.pick_config(BASE, gpus, M, sc, 150.5, 150.5)
    assert best == 0 and t[0] == pytest.approx(10.155214117, rel=1e-9)
    assert np.all(t[1:] < t[0])
    # perfectly parallel workers (latency / GPUs, KV x GPUs): every option
    # has the same per-GPU throughput once the KV bound binds, first wins
    best, t = orc.pick_config(dict(BASE, T_dec=1e12, c2=0.0, c3=0.0), gpus, M,
                              [1.0 / g for g in gpus], 150.5, 150.5)
    assert best == 0 and np.allclose(t, t[0], rtol=1e-12)


def test_fit_workers_exact_line(orc):
    rates = np.array([250.0, 500.0, 750.0, 1000.0, 1500.0, 2000.0])
    nw = (0.06 * rates + 4).astype(np.int32)   # exact integers: 19, 34, 49, 64, 94, 124
    k5, c5, used = orc.fit_workers(rates, nw)
    assert used == 6
    assert k5 == pytest.approx(0.06, rel=1e-12) and c5 == pytest.approx(4.0, rel=1e-12)
    assert orc.predict_workers(k5, c5, 1234.0) == math.ceil(0.06 * 1234.0 + 4.0)


def test_fit_workers_least_squares(orc):
    rng = np.random.default_rng(3)
    rates = rng.uniform(100, 3000, 12)
    nw = (0.05 * rates + 7 + rng.integers(-3, 4, 12)).astype(np.int32)
    R = 400.0
    k5, c5, used = orc.fit_workers(rates, nw, R)
    sel = rates > R
    assert used == int(sel.sum())
    want = np.polyfit(rates[sel], nw[sel].astype(np.float64), 1)
    assert k5 == pytest.approx(want[0], rel=1e-9) and c5 == pytest.approx(want[1], rel=1e-9)
    # fewer than two points above R: no fit
    assert orc.fit_workers([100.0, 5000.0], [3, 9], 1000.0) == (0.0, 0.0, 1)
