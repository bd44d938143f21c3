"""Parity of decode instances (split-phase inference, Sec. 5.1) and of the JSQ
and power-of-two-choices placement baselines (Sec. 6.1, Sec. 6.4) with the
oracle, through the C ABI: scoring, placement rounds, the execution step with
its realized-violation counts, the fleet simulation and the minimum-worker
search."""
import json
import os

import numpy as np
import pytest

from parity import check_argbest, compare_pairs

pytestmark = pytest.mark.gpu

GOLD = os.path.join(os.path.dirname(__file__), "golden")


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


def history(wl, seed, lo, hi):
    rng = np.random.default_rng(seed)
    return (wl.req_gen * rng.uniform(lo, hi, len(wl.req_gen))).astype(np.float32)


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


def trace_of(t, i, p):
    class T:
        pass
    tr = T()
    tr.t_arr = np.asarray(t, np.float64)
    tr.req_in = np.asarray(i, np.int32)
    tr.req_pred = np.asarray(p, np.int32)
    return tr


def simulate_gpu(A, p, b_cap, M, scale, N, tr, stop_at_fail, drain):
    out = np.zeros(A.SIMULATE_OUT)
    A.aladdin_simulate(A.make_params(p, b_cap), A.make_cfgs([1], [M], [scale])[0], N,
                       A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0,
                       int(stop_at_fail), int(drain), out)
    return out


def same_simulation(out, ref, label):
    assert int(out[0]) == ref["failed"] and int(out[1]) == ref["placed"], (label, out, ref)
    assert int(out[2]) == ref["heartbeats"], (label, out, ref)
    assert out[3] == pytest.approx(ref["max_ttft"], rel=1e-12), label
    assert out[4] == pytest.approx(ref["max_atgt"], rel=1e-12), label
    assert int(out[5]) == ref["violations"], (label, out, ref)


# --------------------------------------------------------------------------
# Decode instances: scoring without stall or TTFT.

@pytest.mark.parametrize("seed,tdec,mode", [(401, 10.5, 0), (402, 11.0, 1), (403, 9.5, 0),
                                            (404, 12.0, 1)])
def test_decode_scoring_tiny(A, orc, synth, seed, tdec, mode):
    wl = synth.config("tiny", per_worker_random=True, seed=seed, per_worker=16, kv_per_gpu=8192,
                      n_cand=300, params=dict(T_pre=1.0, T_dec=tdec, theta=0.9, mode=mode,
                                              phase=1))
    h = history(wl, seed, 0.5 * tdec, 0.95 * tdec)
    with A.Cluster.from_workload(wl, tdec_ms=h) as cl:
        g = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait, detail=True)
    oc = orc.Cluster.from_workload(wl, tdec=h.astype(np.float64))
    ref = oc.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    compare_pairs(ref, g["flags"], g["margin"], wl.cand_in, g["kvpeak"], g["tcand"],
                  "decode-%d" % seed)
    check_argbest(oc.order(), g["flags"], g["argbest"], "decode-%d" % seed)
    assert np.all(g["flags"] & 2)                  # TTFT is not tested (T_pre = 1 ms)
    if mode == 1:
        assert np.all(g["flags"] & 4)              # no stall: (d) is vacuous
    assert 0.0 < (g["flags"] == 15).mean() < 1.0


@pytest.mark.parametrize("mode,T_dec", [(0, 20.0), (1, 19.5)])
def test_decode_round_then_score_w256(A, orc, synth, mode, T_dec):
    """A decode-instance round (placements pending), then scoring that sees
    them, then an execution step: placements, pairs and state match."""
    wl = synth.config("w256", n_cand=1024, b_cap=128,
                      params=dict(T_dec=T_dec, theta=0.95, mode=mode, phase=1))
    h = history(wl, 410 + mode, 0.5 * T_dec, T_dec)
    oc = orc.Cluster.from_workload(wl, tdec=h.astype(np.float64))
    with A.Cluster.from_workload(wl, tdec_ms=h) as cl:
        pl = cl.place_round(wl.cand_in[:512], wl.cand_pred[:512], wl.cand_wait[:512])
        ref = oc.place_round(wl.cand_in[:512], wl.cand_pred[:512], wl.cand_wait[:512])
        assert np.array_equal(pl, ref), np.argwhere(pl != ref)[:5]
        assert 0 < (pl >= 0).mean() < 1
        assert_same_state(cl, oc, "decode-round")
        g = cl.score(wl.cand_in[512:], wl.cand_pred[512:], wl.cand_wait[512:], detail=True)
        r2 = oc.score(wl.cand_in[512:], wl.cand_pred[512:], wl.cand_wait[512:])
        compare_pairs(r2, g["flags"], g["margin"], wl.cand_in[512:], g["kvpeak"], g["tcand"],
                      "decode-after-round")
        st = cl.advance(100.0)
        v = np.zeros(3, np.int64)
        oc.advance(0.0, 100.0, violations=v)
        assert_same_state(cl, oc, "decode-advance")
        assert st[2] == 0.0                       # no TTFT on a decode instance
        assert np.array_equal(st[4:7].astype(np.int64), v)


# --------------------------------------------------------------------------
# JSQ and power of two: rounds, execution, violations.

@pytest.mark.parametrize("policy", [1, 2])
@pytest.mark.parametrize("phase", [0, 1])
def test_queue_rounds_and_advance(A, orc, synth, policy, phase):
    """Two rounds (the power-of-two request ids continue across calls), then
    scoring of the new state, then execution with its violation counts."""
    wl = synth.config("w256", n_cand=2048, b_cap=256, kv_per_gpu=52000,
                      params=dict(T_dec=24.0, policy=policy, phase=phase, seed=77))
    h = history(wl, 420 + 2 * policy + phase, 8.0, 24.0)
    oc = orc.Cluster.from_workload(wl, tdec=h.astype(np.float64))
    with A.Cluster.from_workload(wl, tdec_ms=h) as cl:
        pa = cl.place_round(wl.cand_in[:1000], wl.cand_pred[:1000], wl.cand_wait[:1000])
        pb = cl.place_round(wl.cand_in[1000:], wl.cand_pred[1000:], wl.cand_wait[1000:])
        ra = oc.place_round(wl.cand_in[:1000], wl.cand_pred[:1000], wl.cand_wait[:1000],
                            crid=np.arange(1000))
        rb = oc.place_round(wl.cand_in[1000:], wl.cand_pred[1000:], wl.cand_wait[1000:],
                            crid=np.arange(1000, 2048))
        assert np.array_equal(pa, ra) and np.array_equal(pb, rb)
        assert (pa >= 0).all() and (pb >= 0).all()
        assert_same_state(cl, oc, "queue-round")
        g = cl.score(wl.cand_in[:200], wl.cand_pred[:200], wl.cand_wait[:200], detail=True)
        r2 = oc.score(wl.cand_in[:200], wl.cand_pred[:200], wl.cand_wait[:200])
        compare_pairs(r2, g["flags"], g["margin"], wl.cand_in[:200], g["kvpeak"], g["tcand"],
                      "queue-score")
        v = np.zeros(3, np.int64)
        for k in range(4):
            st = cl.advance(100.0)
            oc.advance(100.0 * k, 100.0, violations=v)
            assert_same_state(cl, oc, "queue-advance-%d" % k)
            assert np.array_equal(st[4:7].astype(np.int64), v), (k, st, v)
        assert v.sum() > 0       # the tight capacity and SLO are broken somewhere


def test_queue_capacity_error(A, orc, synth):
    """A JSQ choice without a free slot: ALADDIN_ERR_CAPACITY, the placements
    before it kept, the later ones ALADDIN_NONE."""
    p = dict(synth.BASE_PARAMS, policy=1)
    wl = synth.make_cluster("cap", 5, 2, 31, 10**6, 3, params=p)
    with A.Cluster.from_workload(wl, b_cap=32) as cl:
        pl = np.zeros(3, np.int32)
        with pytest.raises(A.AladdinError) as e:
            A.aladdin_place_round(cl.handle, 3, wl.cand_in, wl.cand_pred, None, pl)
        assert e.value.code == A.ERR_CAPACITY
        assert list(pl) == [0, 1, -1]


@pytest.mark.parametrize("policy,fails", [(0, 0), (1, 2)])
def test_jsq_paper_example(A, policy, fails):
    """Sec. 4.2 example on two workers of KV capacity 9: executing JSQ's
    placement overflows both workers (two violations), best-fit's none."""
    with open(os.path.join(GOLD, "jsq_example.json")) as f:
        g = json.load(f)
    p = dict(g["params"], policy=policy)
    seq = [g[k] for k in g["arrival_order"]]
    tr = trace_of([0.0] * 4, [s["in"] for s in seq], [s["pred"] for s in seq])
    out = np.zeros(A.SIMULATE_OUT)
    A.aladdin_simulate(A.make_params(p, 32), A.make_cfgs([1], [g["capacity"]], [1.0])[0], 2,
                       A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 0, 1, out)
    assert int(out[1]) == 4 and int(out[5]) == fails and int(out[0]) == fails


@pytest.mark.parametrize("policy,phase", [(0, 1), (1, 0), (1, 1), (2, 0), (2, 1)])
def test_simulate_policies(A, orc, synth, policy, phase):
    tr = synth.diurnal_trace(21, 1200, 60.0, 15.0)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, policy=policy, phase=phase, seed=3)
    for N in (2, 4, 7):
        ref = orc.simulate(p, N, 256, 40000, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
        out = simulate_gpu(A, p, 256, 40000, 1.0, N, tr, False, True)
        same_simulation(out, ref, "sim-%d-%d-N%d" % (policy, phase, N))
    ref = orc.simulate(p, 2, 256, 40000, 1.0, tr, 100.0, stop_at_fail=True, drain=policy != 0)
    out = simulate_gpu(A, p, 256, 40000, 1.0, 2, tr, True, policy != 0)
    assert ref["failed"] > 0 and int(out[0]) > 0
    assert int(out[2]) == ref["heartbeats"]


@pytest.mark.parametrize("policy,phase", [(1, 1), (2, 1), (0, 1), (1, 0), (2, 0)])
def test_min_workers_policies(A, orc, synth, policy, phase):
    tr = synth.diurnal_trace(6, 300, 30.0, 7.5)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, policy=policy, phase=phase, seed=5)
    gpus = [1, 2]
    M = [32768, 65536]
    sc = [1.0, 1.0 / np.sqrt(2.0)]
    ref = orc.min_workers(p, gpus, M, sc, 256, tr, 100.0, 16)
    got = np.zeros(2, np.int32)
    A.aladdin_min_workers(A.make_params(p, 256), A.make_cfgs(gpus, M, sc),
                          A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 16, got)
    assert np.array_equal(got, ref), (got, ref)
    assert (got > 0).all()
