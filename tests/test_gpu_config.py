"""Parity of the worker-configuration model (Sec. 4.1: trace demand, Eq. max
throughput, the optimal configuration) and of the worker-count model of
Sec. 5.2 (Eq. total_worker_pre fitted to minimum-worker searches) with the
oracle, through the C ABI."""
import math

import numpy as np
import pytest

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


@pytest.mark.parametrize("h,j", [(1, 0), (3, 5)])
def test_trace_demand_matches_oracle(A, orc, synth, h, j):
    tr = synth.diurnal_trace(4, 100_000, 2000.0, 500.0, out_law=(256.0, 1.2, 8, 4096))
    p = dict(synth.BASE_PARAMS, h=h, j=j)
    got = A.aladdin_trace_demand(A.make_params(p, 256), A.make_trace(tr.t_arr, tr.req_in,
                                                                       tr.req_pred))
    want = orc.trace_demand(p, tr.req_in, tr.req_pred)
    assert got == want      # exact integer sums, one division each


@pytest.mark.parametrize("T_dec", [50.0, 20.0, 200.0])
def test_pick_config_matches_oracle(A, orc, synth, T_dec):
    tr = synth.diurnal_trace(7, 20_000, 500.0, 500.0)
    p = dict(synth.BASE_PARAMS, T_dec=T_dec)
    trace = A.make_trace(tr.t_arr, tr.req_in, tr.req_pred)
    m_r, l_ave = orc.trace_demand(p, tr.req_in, tr.req_pred)
    for gpus, M, sc in (
            ([1, 2, 4, 8], [65536 * g for g in [1, 2, 4, 8]],
             [1.0 / math.sqrt(g) for g in [1, 2, 4, 8]]),
            ([1, 2, 4, 8], None, None)):            # from the tensor-parallel model
        if M is None:
            cfgs = A.aladdin_tp_configs(A.aladdin_tp_model(30.0, 6.0, 5.0, 40_000.0, 26_000.0),
                                        gpus)
        else:
            cfgs = A.make_cfgs(gpus, M, sc)
        t = np.zeros(len(gpus))
        best = A.aladdin_pick_config(A.make_params(p, 256), cfgs, trace, t)
        wb, wt = orc.pick_config(p, gpus, [c.kv_capacity for c in cfgs],
                                 [c.lat_scale for c in cfgs], m_r, l_ave)
        assert np.allclose(t, wt, rtol=1e-12, atol=0), (t, wt)
        assert best == wb


def constant_rate_traces(synth, rates, n, seed0):
    return [synth.diurnal_trace(seed0 + k, n, r, r) for k, r in enumerate(rates)]


@pytest.mark.parametrize("policy,phase", [(0, 0), (1, 1)])
def test_fit_workers_matches_oracle(A, orc, synth, policy, phase):
    rates = [20.0, 40.0, 60.0, 80.0, 100.0]
    trs = constant_rate_traces(synth, rates, 1500, 30)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, policy=policy, phase=phase, seed=9)
    cfg = A.make_cfgs([1], [32768], [1.0])[0]
    nw = np.zeros(len(rates), np.int32)
    R = 30.0
    k5, c5 = A.aladdin_fit_workers(A.make_params(p, 256), cfg,
                                   [A.make_trace(t.t_arr, t.req_in, t.req_pred) for t in trs],
                                   rates, R, 100.0, 64, nw)
    want = [int(orc.min_workers(p, [1], [32768], [1.0], 256, t, 100.0, 64)[0]) for t in trs]
    assert nw.tolist() == want
    wk, wc, used = orc.fit_workers(rates, want, R)
    assert used == 4
    assert k5 == pytest.approx(wk, rel=1e-12) and c5 == pytest.approx(wc, rel=1e-12, abs=1e-12)
    assert A.aladdin_predict_workers(k5, c5, 70.0) == orc.predict_workers(wk, wc, 70.0)


def test_fit_workers_needs_two_rates(A, synth):
    trs = constant_rate_traces(synth, [40.0], 500, 50)
    p = dict(synth.BASE_PARAMS, T_dec=30.0)
    nw = np.zeros(1, np.int32)
    with pytest.raises(A.AladdinError) as e:
        A.aladdin_fit_workers(A.make_params(p, 256), A.make_cfgs([1], [32768], [1.0])[0],
                              [A.make_trace(t.t_arr, t.req_in, t.req_pred) for t in trs],
                              [40.0], 0.0, 100.0, 64, nw)
    assert e.value.code == A.ERR_ARG and nw[0] > 0
