"""Parity of prediction-error handling and Algorithm 2 (Sec. 4.3,
re-balancing with prediction error) with the oracle, through the C ABI:
aladdin_rebalance on placed rounds, and simulations and worker searches of
traces whose requests run to real lengths different from their
predictions."""
import math

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

BASE = dict(k1=0.001, c1=10.0, k2=2e-4, c2=0.05, c3=8.0, h=1, j=0, T_pre=1000.0, T_dec=50.0,
            gamma=0.5, theta=1.0, K=8192)


@pytest.fixture(scope="module")
def A():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.init()
    from paper_2405_06856_gb300 import build
    build.build()
    from paper_2405_06856_gb300 import aladdin
    return aladdin


def state_multiset(n, inp, gen, pred, pend, cap):
    out = []
    for w in range(len(n)):
        s = w * cap
        k = int(n[w])
        out.append(sorted(zip(inp[s:s + k].tolist(), gen[s:s + k].tolist(), pred[s:s + k].tolist(),
                              pend[s:s + k].tolist())))
    return out


def assert_same_state(cl, oc, label):
    n, i, g, p, pe = cl.state()
    assert np.array_equal(n, oc.n), label
    assert state_multiset(n, i, g, p, pe, cl.b_cap) == \
        state_multiset(oc.n, oc.inp, oc.gen, oc.pred, oc.pend, oc.cap), label


def both(A, orc, params, M, loads, cap=32):
    W = len(M)
    roff = np.concatenate([[0], np.cumsum(loads)]).astype(np.int32)
    n = int(roff[-1])
    ins, gen, pred = np.full(n, 300, np.int32), np.zeros(n, np.int32), np.full(n, 400, np.int32)
    g = A.Cluster(params, [1] * W, M, [1.0] * W, cap, roff, ins, gen, pred)
    o = orc.Cluster(params, M, [1.0] * W, cap, roff, ins, gen, pred)
    o.tdec[:] = params["theta"] * params["T_dec"] * o.gen   # the library's default history
    o.has_tdec = True
    return g, o


def test_rebalance_hand_example(A, orc):
    """The oracle's hand-worked case: two of the three requests move."""
    g, o = both(A, orc, BASE, [10**6, 10**6], [0, 0])
    with g:
        cin, cpr, cw = [200, 200, 200], [100, 300, 50], [0.0, 0.0, 0.0]
        pl = g.place_round(cin, cpr, cw)
        rl = o.place_round(cin, cpr, cw)
        assert list(pl) == list(rl) == [0, 0, 0]
        mv, b0, b1 = g.rebalance(cin, cpr, cw, pl, [500, -400], [2, -1])
        omv, ob0, ob1 = o.rebalance(cin, cpr, cw, rl, [500, -400], [2, -1])
        assert list(pl) == list(rl) == [1, 1, 0] and mv == omv == 2
        assert b0 == pytest.approx(ob0, rel=1e-12) and b1 == pytest.approx(ob1, rel=1e-12)
        assert_same_state(g, o, "hand")


def random_case(A, orc, synth, seed):
    """A placed round on a mixed-load tiny cluster with random errors,
    re-balanced on both sides; returns the moves."""
    rng = np.random.default_rng(seed)
    wl = synth.config("tiny", per_worker_random=True, seed=seed, per_worker=10, n_cand=60,
                      b_cap=128, params=dict(T_pre=400.0, T_dec=40.0))
    h = (wl.req_gen * rng.uniform(10.0, 40.0, len(wl.req_gen))).astype(np.float32)
    oc = orc.Cluster.from_workload(wl, tdec=h.astype(np.float64))
    le = rng.integers(-4000, 4000, wl.n_workers)
    be = rng.integers(-5, 6, wl.n_workers).astype(np.int32)
    with A.Cluster.from_workload(wl, tdec_ms=h) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        rl = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, rl)
        mv, b0, b1 = cl.rebalance(wl.cand_in, wl.cand_pred, wl.cand_wait, pl, le, be)
        omv, ob0, ob1 = oc.rebalance(wl.cand_in, wl.cand_pred,
                                     wl.cand_wait.astype(np.float32).astype(np.float64), rl, le, be)
        assert np.array_equal(pl, rl) and mv == omv
        assert b0 == pytest.approx(ob0, rel=1e-12) and b1 == pytest.approx(ob1, rel=1e-12)
        assert_same_state(cl, oc, "random-%d" % seed)
        # the scoring state after the moves (tables and ranks rebuilt)
        g = cl.score(wl.cand_in[:20], wl.cand_pred[:20], wl.cand_wait[:20])
        r = oc.score(wl.cand_in[:20], wl.cand_pred[:20], wl.cand_wait[:20])
        ok = r["near"] > 1e-5
        assert np.array_equal(g["flags"][ok], r["flags"][ok])
        order = oc.order()
        for c in range(20):
            feas = r["flags"][c][order] == 15
            if ok[c].all():
                assert g["argbest"][c] == (int(order[np.argmax(feas)]) if feas.any() else -1)
    return mv


def test_rebalance_random_matches_oracle(A, orc, synth):
    assert sum(random_case(A, orc, synth, s) for s in (601, 602, 603, 604, 605, 606)) > 0


def test_rebalance_1024_slots(A, orc, synth):
    """Workers of 1,024 request slots (the cooperative table rebuild)."""
    rng = np.random.default_rng(620)
    wl = synth.make_cluster("big", 620, 24, 300, 1_000_000, 400, per_worker_random=True,
                            b_cap=1024, params=dict(T_pre=400.0, T_dec=60.0))
    oc = orc.Cluster.from_workload(wl)
    oc.tdec[:] = wl.params["theta"] * wl.params["T_dec"] * oc.gen
    oc.has_tdec = True
    le = rng.integers(-20000, 20000, wl.n_workers)
    be = rng.integers(-20, 21, wl.n_workers).astype(np.int32)
    with A.Cluster.from_workload(wl) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        rl = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, rl)
        mv, _, _ = cl.rebalance(wl.cand_in, wl.cand_pred, wl.cand_wait, pl, le, be)
        omv, _, _ = oc.rebalance(wl.cand_in, wl.cand_pred,
                                 wl.cand_wait.astype(np.float32).astype(np.float64), rl, le, be)
        assert np.array_equal(pl, rl) and mv == omv and mv > 0
        assert_same_state(cl, oc, "1024")


def sim_gpu(A, p, N, M, tr, stop, drain, cap=256):
    out = np.zeros(A.SIMULATE_OUT)
    A.aladdin_simulate(A.make_params(p, cap), A.make_cfgs([1], [M], [1.0])[0], N,
                       A.trace_of(tr), 100.0, int(stop), int(drain), out)
    return out


@pytest.mark.parametrize("rebalance", [0, 1])
@pytest.mark.parametrize("sigma", [0.3, 0.6])
def test_simulation_with_prediction_errors(A, orc, synth, rebalance, sigma):
    tr = synth.with_prediction_error(synth.diurnal_trace(9, 1500, 60.0, 15.0), sigma, 9)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, rebalance=rebalance)
    for N in (4, 6):
        ref = orc.simulate(p, N, 256, 40000, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
        out = sim_gpu(A, p, N, 40000, tr, False, True)
        lab = (sigma, rebalance, N, out, ref)
        assert int(out[0]) == ref["failed"] and int(out[1]) == ref["placed"], lab
        assert int(out[2]) == ref["heartbeats"], lab
        assert out[3] == pytest.approx(ref["max_ttft"], rel=1e-12), lab
        assert out[4] == pytest.approx(ref["max_atgt"], rel=1e-12), lab
        assert int(out[5]) == ref["violations"], lab
        assert int(out[6]) == ref["repredictions"] and int(out[7]) == ref["early_finishes"], lab
        assert int(out[8]) == ref["moved"], lab
        assert out[6] > 0 and out[7] > 0
        assert (out[8] > 0) == bool(rebalance)


@pytest.mark.parametrize("theta", [0.5, 0.6])
def test_min_workers_with_prediction_errors(A, orc, synth, theta):
    """With prediction errors only a tighter SLO knob (theta, Sec. 4.2) finds
    worker counts without violations; searches match the oracle."""
    tr = synth.with_prediction_error(synth.diurnal_trace(6, 300, 30.0, 7.5), 0.4, 6)
    for rebalance in (0, 1):
        p = dict(synth.BASE_PARAMS, T_dec=30.0, rebalance=rebalance, theta=theta)
        ref = orc.min_workers(p, [1, 2], [32768, 65536], [1.0, 1.0 / math.sqrt(2.0)], 256, tr,
                              100.0, 32)
        got = np.zeros(2, np.int32)
        A.aladdin_min_workers(A.make_params(p, 256),
                              A.make_cfgs([1, 2], [32768, 65536], [1.0, 1.0 / math.sqrt(2.0)]),
                              A.trace_of(tr), 100.0, 32, got)
        assert np.array_equal(got, ref), (rebalance, got, ref)
        assert (got > 0).any()
