"""Pins of the oracle's prediction-error handling and Algorithm 2 (Sec. 4.3,
re-balancing with prediction error): execution that follows real output
lengths with re-prediction, the per-worker error indicators, and the
re-balancing moves, against hand-worked numbers, closed forms and the
reduction to exact predictions."""
import math

import numpy as np
import pytest

BASE = dict(k1=0.001, c1=10.0, k2=2e-4, c2=0.05, c3=8.0, h=1, j=0, T_pre=1000.0, T_dec=50.0,
            gamma=0.5, theta=1.0, K=8192)
NORM = math.sqrt(2e-4 ** 2 + 0.05 ** 2)


def test_repredicted_execution_closed_form(orc):
    """A request (prompt 100, predicted 10, real 15) runs alone: after 10
    iterations it is re-predicted to 20 (l^e += 10, b^e += 1), then finishes
    at 15, before its new prediction (l^e += 15 - 20, b^e -= 1). Its ATGT is
    the 15-iteration decode sum over 15 tokens:
    sum_{s=1}^{15} (c3 + c2 + k2 (100 + s)) = 15 (8.05 + 0.02) + 2e-4 * 120."""
    cl = orc.Cluster(BASE, [10**6], [1.0], 8)
    cl.place_round([100], [10], [0.0], crid=[3])
    real = np.zeros(8, np.int32)
    real[0] = 15
    rep = np.arange(1, 8194, dtype=np.int32)
    rep[10] = 20
    cl.set_real(real, rep)
    ev = np.zeros(2, np.int64)
    rid, val, kind = cl.advance(0.0, 10_000.0, events=ev)
    assert list(ev) == [1, 1]
    assert cl.le[0] == 10 + (15 - 20) and cl.be[0] == 0
    D = 15 * (8.0 + 0.05 + 2e-4 * 100) + 2e-4 * 120
    assert list(kind) == [0, 1] and val[1] == pytest.approx(D / 15, rel=1e-12)
    assert cl.n[0] == 0


def test_exact_predictions_change_nothing(orc, synth):
    """Without prediction errors there are no events, Algorithm 2 moves
    nothing, and the simulation is the one without re-balancing."""
    tr = synth.diurnal_trace(5, 400, 40.0, 10.0)
    p = dict(synth.BASE_PARAMS)
    a = orc.simulate(p, 4, 256, 65536, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    b = orc.simulate(dict(p, rebalance=1), 4, 256, 65536, 1.0, tr, 100.0, stop_at_fail=False,
                     drain=True)
    assert a == b
    assert b["moved"] == 0 and b["repredictions"] == 0 and b["early_finishes"] == 0


def three_on_worker0(orc, M1=10**6, W=2, loads=None):
    """W workers; the three requests of the round (prompts 200, predictions
    100, 300, 50) all go to worker 0 (Algorithm 1: empty workers tie, then
    worker 0 has the largest capacity_norm)."""
    cl = orc.Cluster(BASE, [10**6] + [M1] * (W - 1), [1.0] * W, 16,
                     np.array([0] + [0] + list(np.cumsum(loads or [0] * (W - 1))), np.int32)
                     if loads else None,
                     *([np.full(sum(loads), 300, np.int32), np.zeros(sum(loads), np.int32),
                        np.full(sum(loads), 400, np.int32)] if loads else [None] * 3))
    cin, cpred, cw = [200, 200, 200], [100, 300, 50], [0.0, 0.0, 0.0]
    pl = cl.place_round(cin, cpred, cw)
    assert list(pl) == [0, 0, 0]
    return cl, cin, cpred, cw, pl


def test_rebalance_hand_example(orc):
    """e = k2 l^e + c2 b^e: worker 0 (l^e 500, b^e 2) e0 = 0.2, worker 1
    (l^e -400, b^e -1) e1 = -0.13. Request 0 (d = k2 100 + c2 = 0.07): gain
    (0.2 + 0.13) - 0.13 - 0.06 = 0.14 > 0, moves: e = (0.13, -0.06). Request 1
    (d = 0.11): gain 0.19 - 0.02 - 0.05 = 0.12, moves: e = (0.02, 0.05).
    Request 2: worker 1 is no longer under-utilized, it stays."""
    cl, cin, cpred, cw, pl = three_on_worker0(orc)
    mv, before, after = cl.rebalance(cin, cpred, cw, pl, [500, -400], [2, -1])
    assert list(pl) == [1, 1, 0] and mv == 2
    assert before == pytest.approx((0.2 + 0.13) / NORM, rel=1e-12)
    assert after == pytest.approx((0.02 + 0.05) / NORM, rel=1e-9)
    assert list(cl.n) == [1, 2]
    assert sorted(cl.pred[16:18].tolist()) == [100, 300] and cl.pred[0] == 50
    assert np.all(cl.pend[16:18] == 1)


def test_rebalance_needs_a_feasible_target(orc):
    """Worker 1 cannot hold any of the requests (KV capacity 240 < 200 + 50):
    nothing moves although it is under-utilized."""
    cl, cin, cpred, cw, pl = three_on_worker0(orc, M1=240)
    mv, before, after = cl.rebalance(cin, cpred, cw, pl, [500, -400], [2, -1])
    assert mv == 0 and list(pl) == [0, 0, 0] and before == after


@pytest.mark.parametrize("loads,target", [([3, 1, 2], 2), ([3, 2, 1], 1)])
def test_rebalance_tie_goes_to_larger_capacity_norm(orc, loads, target):
    """Two under-utilized workers with the same error give the same gain
    (2 d, d below both errors); the request goes to the one of larger
    capacity_norm, whatever its index."""
    roff = np.concatenate([[0], np.cumsum(loads)]).astype(np.int32)
    n = int(roff[-1])
    cl = orc.Cluster(BASE, [10**6] * 3, [1.0] * 3, 16, roff, np.full(n, 300, np.int32),
                     np.zeros(n, np.int32), np.full(n, 400, np.int32))
    pl = cl.place_round([200], [100], [0.0])
    assert list(pl) == [0]          # worker 0 has the largest capacity_norm
    mv, before, after = cl.rebalance([200], [100], [0.0], pl, [10**4, -10**4, -10**4],
                                     [0, 0, 0])
    assert mv == 1 and list(pl) == [target]
    assert after == pytest.approx(before - 2 * (2e-4 * 100 + 0.05) / NORM, rel=1e-12)


def test_rebalance_lowers_the_objective(orc, synth):
    rng = np.random.default_rng(8)
    total = 0
    for trial in range(12):
        wl = synth.config("tiny", per_worker_random=True, seed=500 + trial, per_worker=10,
                          n_cand=40, b_cap=128, params=dict(T_pre=400.0, T_dec=40.0))
        oc = orc.Cluster.from_workload(wl)
        pl = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        le = rng.integers(-3000, 3000, wl.n_workers)
        be = rng.integers(-4, 5, wl.n_workers).astype(np.int32)
        n0 = oc.n.copy()
        mv, before, after = oc.rebalance(wl.cand_in, wl.cand_pred, wl.cand_wait, pl, le, be)
        total += mv
        assert after <= before + 1e-12
        assert (mv == 0) == (after == before)
        assert oc.n.sum() == n0.sum()
        # a move only leaves a worker with positive error for one with negative
        e = 2e-4 * le + 0.05 * be
        assert np.all(oc.n[e <= 0] >= n0[e <= 0]) and np.all(oc.n[e >= 0] <= n0[e >= 0])
    assert total > 0


def test_simulation_with_prediction_errors(orc, synth):
    """Noisy predictions: requests are re-predicted and finish early, and
    Algorithm 2 moves requests; every admitted request is still counted."""
    tr = synth.with_prediction_error(synth.diurnal_trace(9, 1500, 60.0, 15.0), 0.5, 9)
    p = dict(synth.BASE_PARAMS, T_dec=30.0)
    off = orc.simulate(p, 5, 256, 40000, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    on = orc.simulate(dict(p, rebalance=1), 5, 256, 40000, 1.0, tr, 100.0, stop_at_fail=False,
                      drain=True)
    for r in (off, on):
        assert r["repredictions"] > 0 and r["early_finishes"] > 0
        assert r["placed"] + (r["failed"] - r["violations"]) == 1500
    assert off["moved"] == 0 and on["moved"] > 0
