"""Parity of the approximate mode (the placement MIP's own decode constraints
(b), with Eq. input limit, and (d), Sec. 4.2) with the oracle, through the C
ABI: scoring, greedy rounds and the fleet simulation."""
import numpy as np
import pytest

from parity import check_argbest, compare_pairs

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


def history(wl, seed, lo=8.0, hi=45.0):
    """Decode time so far: each generated token took lo..hi ms."""
    rng = np.random.default_rng(seed)
    return (wl.req_gen * rng.uniform(lo, hi, len(wl.req_gen))).astype(np.float32)


def score_both(A, orc, wl, tdec, label):
    with A.Cluster.from_workload(wl, tdec_ms=tdec) as cl:
        g = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait, detail=True)
    oc = orc.Cluster.from_workload(wl, tdec=None if tdec is None else tdec.astype(np.float64))
    ref = oc.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    near = compare_pairs(ref, g["flags"], g["margin"], wl.cand_in, g["kvpeak"], g["tcand"], label)
    check_argbest(oc.order(), g["flags"], g["argbest"], label)
    return g, ref, near


@pytest.mark.parametrize("seed,tpre,tdec_slo,theta", [
    (301, 60.0, 30.0, 0.9), (302, 1000.0, 50.0, 0.8), (303, 30.0, 20.0, 0.95),
    (304, 80.0, 14.0, 1.0)])
def test_approx_scoring_tiny(A, orc, synth, seed, tpre, tdec_slo, theta):
    wl = synth.config("tiny", per_worker_random=True, seed=seed, n_cand=300,
                      params=dict(T_pre=tpre, T_dec=tdec_slo, theta=theta, mode=1))
    g, ref, near = score_both(A, orc, wl, history(wl, seed, 0.3 * tdec_slo, 0.95 * tdec_slo),
                              "approx-%d" % seed)
    assert 0.0 < (g["flags"] == 15).mean() < 1.0


def test_approx_every_group_binds(A, orc, synth):
    seen = 0
    for seed, tpre, tdec_slo in ((311, 22.0, 16.0), (312, 40.0, 11.0), (313, 14.0, 40.0),
                                 (314, 40.0, 9.0)):
        wl = synth.config("tiny", per_worker_random=True, seed=seed, n_cand=200,
                          params=dict(T_pre=tpre, T_dec=tdec_slo, theta=0.9, mode=1))
        g, ref, near = score_both(A, orc, wl, history(wl, seed, 0.5 * tdec_slo, tdec_slo),
                                  "approx-groups-%d" % seed)
        for b in range(4):
            if ((g["flags"] >> b) & 1 == 0).any():
                seen |= 1 << b
    assert seen == 15


def test_approx_no_history(A, orc, synth):
    """Without a decode history every request has used its theta-scaled
    budget exactly: with theta < 1 the saved time is (1 - theta) T_dec l_out."""
    wl = synth.config("tiny", per_worker_random=True, seed=320, n_cand=200,
                      params=dict(T_pre=200.0, T_dec=40.0, theta=0.7, mode=1))
    score_both(A, orc, wl, None, "approx-nohist")


def test_approx_w256_and_ragged(A, orc, synth):
    wl = synth.config("w256", n_cand=1024, params=dict(theta=0.9, mode=1))
    g, ref, near = score_both(A, orc, wl, history(wl, 330, 10.0, 50.0), "approx-w256")
    for W, C, seed in ((7, 257, 331), (33, 513, 332)):  # scalar store path, chunk tails
        wl = synth.make_cluster("edge", seed, W, 20, 30000, C, per_worker_random=True,
                                params=dict(T_pre=50.0, T_dec=25.0, K=4096, theta=0.9, mode=1))
        score_both(A, orc, wl, history(wl, seed, 5.0, 25.0), "approx-edge-W%d" % W)


def test_approx_differs_from_exact(A, synth):
    """The two modes share the KV and TTFT bits and differ in the others."""
    wl = synth.config("tiny", per_worker_random=True, seed=340, n_cand=300,
                      params=dict(T_pre=60.0, T_dec=30.0, theta=0.9))
    tdec = history(wl, 340, 10.0, 33.0)
    with A.Cluster.from_workload(wl, tdec_ms=tdec) as cl:
        ex = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    wa = synth.config("tiny", per_worker_random=True, seed=340, n_cand=300,
                      params=dict(T_pre=60.0, T_dec=30.0, theta=0.9, mode=1))
    with A.Cluster.from_workload(wa, tdec_ms=tdec) as cl:
        ap = cl.score(wa.cand_in, wa.cand_pred, wa.cand_wait)
    assert np.array_equal(ex["flags"] & 3, ap["flags"] & 3)
    assert (ex["flags"] != ap["flags"]).any()


def test_approx_round_and_simulation(A, orc, synth):
    wl = synth.config("w256", n_cand=512, b_cap=128, params=dict(theta=0.9, T_dec=30.0, mode=1))
    tdec = history(wl, 350, 10.0, 30.0)
    with A.Cluster.from_workload(wl, tdec_ms=tdec) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
    oc = orc.Cluster.from_workload(wl, tdec=tdec.astype(np.float64))
    ref = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
    assert np.array_equal(pl, ref), np.argwhere(pl != ref)[:5]
    assert 0 < (pl >= 0).mean() < 1

    tr = synth.diurnal_trace(12, 1500, 60.0, 15.0)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, theta=0.9, mode=1)
    for N in (3, 6):
        ref = orc.simulate(p, N, 256, 65536, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
        out = np.zeros(A.SIMULATE_OUT)
        A.aladdin_simulate(A.make_params(p, 256), A.make_cfgs([1], [65536], [1.0])[0], N,
                           A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 0, 1, out)
        assert int(out[0]) == ref["failed"] and int(out[1]) == ref["placed"], (N, out, ref)
        assert int(out[2]) == ref["heartbeats"]
        assert out[3] == pytest.approx(ref["max_ttft"], rel=1e-12)
        assert out[4] == pytest.approx(ref["max_atgt"], rel=1e-12)
