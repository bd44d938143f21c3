"""Parity of the greedy round (aladdin_place_round), the execution step
(aladdin_cluster_advance) and the fleet simulation / minimum-worker search
with the oracle, through the C ABI."""
import numpy as np
import pytest

from parity import compare_pairs

pytestmark = pytest.mark.gpu


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


def assert_same_state(A_cl, oc, label):
    n, i, g, p, pe = A_cl.state()
    assert np.array_equal(n, oc.n), label
    a = state_multiset(n, i, g, p, pe, A_cl.b_cap)
    b = state_multiset(oc.n, oc.inp, oc.gen, oc.pred, oc.pend, oc.cap)
    assert a == b, label


@pytest.mark.parametrize("seed,tdec", [(201, 12.0), (202, 20.0), (203, 16.0)])
def test_round_tiny(A, orc, synth, seed, tdec):
    wl = synth.config("tiny", per_worker_random=True, seed=seed, b_cap=128,
                      params=dict(T_pre=300.0, T_dec=tdec))
    with A.Cluster.from_workload(wl) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        oc = orc.Cluster.from_workload(wl)
        ref = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, ref), (pl, ref)
        assert_same_state(cl, oc, "round-tiny")
        # scoring after the round sees the pending requests
        g = cl.score(wl.cand_in[:32], wl.cand_pred[:32], wl.cand_wait[:32], detail=True)
        r2 = oc.score(wl.cand_in[:32], wl.cand_pred[:32], wl.cand_wait[:32])
        compare_pairs(r2, g["flags"], g["margin"], wl.cand_in[:32], g["kvpeak"], g["tcand"],
                      "after-round")


def test_round_w256(A, orc, synth):
    wl = synth.config("w256", n_cand=512, b_cap=128)
    with A.Cluster.from_workload(wl) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        oc = orc.Cluster.from_workload(wl)
        ref = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, ref)
        assert_same_state(cl, oc, "round-w256")
        assert (pl >= 0).any()


def test_round_capacity_error(A, synth):
    wl = synth.make_cluster("cap", 210, 2, 30, 10**6, 40, params=dict(T_pre=1e6, T_dec=1e6),
                            b_cap=32)
    with A.Cluster.from_workload(wl) as cl:
        with pytest.raises(A.AladdinError) as e:
            cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert e.value.code == A.ERR_CAPACITY


def test_rounds_and_advance(A, orc, synth):
    """Several heartbeats: round, then execute 100 ms; state, realized
    latencies and later scoring match the oracle."""
    wl = synth.config("tiny", per_worker_random=True, seed=220, b_cap=128,
                      params=dict(T_pre=400.0, T_dec=30.0))
    rng = np.random.default_rng(3)
    oc = orc.Cluster.from_workload(wl, tdec=None)
    oc.tdec[:] = 0.0
    # the oracle's "no history" reading is bank 0: give it the same explicit history
    for w in range(oc.W):
        s = w * oc.cap
        k = int(oc.n[w])
        oc.tdec[s:s + k] = wl.params["theta"] * wl.params["T_dec"] * oc.gen[s:s + k]
    oc.has_tdec = True
    with A.Cluster.from_workload(wl) as cl:
        t = 0.0
        for hb in range(6):
            C = 40
            cin = rng.integers(16, 1500, C).astype(np.int32)
            cpr = rng.integers(8, 600, C).astype(np.int32)
            cw = rng.uniform(0, 100, C).astype(np.float32)
            pl = cl.place_round(cin, cpr, cw)
            ref = oc.place_round(cin, cpr, cw.astype(np.float64))
            assert np.array_equal(pl, ref), hb
            st = cl.advance(100.0)
            oc.advance(t, 100.0)
            t += 100.0
            assert_same_state(cl, oc, "hb%d" % hb)
            g = cl.score(cin, cpr, cw, detail=True)
            r2 = oc.score(cin, cpr, cw.astype(np.float64))
            compare_pairs(r2, g["flags"], g["margin"], cin, g["kvpeak"], g["tcand"], "hb%d" % hb)
        assert st[0] > 0 and st[1] > 0
        assert st[2] <= wl.params["T_pre"] + 1e-6
        assert st[3] <= wl.params["T_dec"] * wl.params["theta"] + 1e-6


def test_simulate_matches_oracle(A, orc, synth):
    tr = synth.diurnal_trace(5, 400, 40.0, 10.0)
    p = dict(synth.BASE_PARAMS)
    for N in (2, 4, 6):
        ref = orc.simulate(p, N, 256, 65536, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
        out = np.zeros(5)
        A.aladdin_simulate(A.make_params(p, 256), A.make_cfgs([1], [65536], [1.0])[0], N,
                           A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 0, 1, out)
        assert int(out[0]) == ref["failed"] and int(out[1]) == ref["placed"], (N, out, ref)
        assert int(out[2]) == ref["heartbeats"]
        assert out[3] == pytest.approx(ref["max_ttft"], rel=1e-12)
        assert out[4] == pytest.approx(ref["max_atgt"], rel=1e-12)


def test_simulate_stop_at_fail(A, orc, synth):
    tr = synth.diurnal_trace(8, 500, 60.0, 15.0)
    p = dict(synth.BASE_PARAMS, T_dec=30.0)
    ref = orc.simulate(p, 1, 256, 32768, 1.0, tr, 100.0, stop_at_fail=True)
    out = np.zeros(5)
    A.aladdin_simulate(A.make_params(p, 256), A.make_cfgs([1], [32768], [1.0])[0], 1,
                       A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 1, 0, out)
    assert ref["failed"] > 0
    assert int(out[0]) == ref["failed"] and int(out[2]) == ref["heartbeats"]


def test_min_workers_matches_oracle(A, orc, synth):
    tr = synth.diurnal_trace(6, 300, 30.0, 7.5)
    p = dict(synth.BASE_PARAMS, T_dec=30.0)
    gpus = [1, 2]
    M = [32768, 65536]
    sc = [1.0, 1.0 / np.sqrt(2.0)]
    ref = orc.min_workers(p, gpus, M, sc, 256, tr, 100.0, 16)
    got = np.zeros(2, np.int32)
    best, total = A.aladdin_min_workers(A.make_params(p, 256), A.make_cfgs(gpus, M, sc),
                                        A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 16,
                                        got)
    assert np.array_equal(got, ref), (got, ref)
    tot = [g * n if n > 0 else 10**9 for g, n in zip(gpus, ref)]
    assert total == min(tot) and best == int(np.argmin(tot))


@pytest.mark.parametrize("W,b_cap,seed,per_worker,tpre,tdec", [
    (1500, 512, 230, 12, 60.0, 12.0), (4096, 128, 231, 12, 60.0, 12.0),
    (1500, 512, 232, 40, 40.0, 11.0)])
def test_round_many_slices(A, orc, synth, W, b_cap, seed, per_worker, tpre, tdec):
    """Clusters whose worker state does not fit one CTA's shared memory: the
    round runs as a cooperative grid of worker slices exchanging per-slice
    bests each candidate."""
    wl = synth.make_cluster("slices", seed, W, per_worker, 60000, 1000, per_worker_random=True,
                            b_cap=b_cap, params=dict(T_pre=tpre, T_dec=tdec))
    with A.Cluster.from_workload(wl) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        oc = orc.Cluster.from_workload(wl)
        ref = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, ref), np.argwhere(pl != ref)[:5]
        assert 0 < (pl >= 0).mean() < 1
        assert_same_state(cl, oc, "slices-%d" % W)
        assert cl.status() == A.OK


def test_simulate_many_slices(A, orc, synth):
    """Fleet simulation on 450 workers of 512 slots (several worker slices):
    waiting list, failures and realized latencies match the oracle."""
    tr = synth.diurnal_trace(11, 6000, 3000.0, 500.0)
    p = dict(synth.BASE_PARAMS, T_pre=100.0, T_dec=14.0)
    ref = orc.simulate(p, 450, 512, 12000, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    out = np.zeros(5)
    A.aladdin_simulate(A.make_params(p, 512), A.make_cfgs([1], [12000], [1.0])[0], 450,
                       A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 0, 1, out)
    assert ref["failed"] > 0
    assert int(out[0]) == ref["failed"] and int(out[1]) == ref["placed"], (out, ref)
    assert int(out[2]) == ref["heartbeats"]
    assert out[3] == pytest.approx(ref["max_ttft"], rel=1e-12)
    assert out[4] == pytest.approx(ref["max_atgt"], rel=1e-12)
