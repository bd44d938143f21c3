"""Pins of the oracle's serving settings and placement policies.

Decode instances of split-phase inference (Sec. 5.1: no prefill on the
worker, so no stall and no TTFT test), the JSQ and power-of-two-choices
baselines (Sec. 6.1, Sec. 6.4) and the realized-violation accounting of the
execution step are checked against hand-worked numbers, the paper's JSQ
example (Sec. 4.2), closed forms, reductions to the mixed setting, and the
published SplitMix64 test vectors.
"""
import json
import os

import numpy as np
import pytest

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def one_worker(orc, params, M, reqs, cap=16, scale=1.0):
    ins = np.array([r[0] for r in reqs], np.int32)
    gen = np.array([r[1] for r in reqs], np.int32)
    pred = np.array([r[2] for r in reqs], np.int32)
    return orc.Cluster(params, [M], [scale], cap, np.array([0, len(reqs)], np.int32), ins, gen,
                       pred)


class Trace:
    def __init__(self, t, i, p):
        self.t_arr = np.asarray(t, np.float64)
        self.req_in = np.asarray(i, np.int32)
        self.req_pred = np.asarray(p, np.int32)


# --------------------------------------------------------------------------
# SplitMix64 and the power-of-two draws.

def test_splitmix64_published_vectors(orc):
    for st in load("splitmix64.json")["streams"]:
        for n, v in enumerate(st["outputs"], start=1):
            assert orc.splitmix64(st["seed"], n) == int(v, 0)


def test_po2_draw_mapping(orc):
    """Draw k of request rid is output 2 rid + k + 1, its upper 32 bits
    scaled to [0, W)."""
    outs = [int(v) for v in load("splitmix64.json")["streams"][1]["outputs"]]
    for W in (1, 2, 7, 1000, 16384):
        for rid in (0, 1):
            for k in (0, 1):
                x = outs[2 * rid + k]
                assert orc.po2_draw(1234567, rid, k, W) == ((x >> 32) * W) >> 32


def test_po2_draws_uniform(orc):
    W, n = 10, 20000
    counts = np.bincount([orc.po2_draw(99, rid, k, W) for rid in range(n // 2) for k in (0, 1)],
                         minlength=W)
    assert counts.sum() == n and counts.min() > 0
    sd = np.sqrt(n * (1 / W) * (1 - 1 / W))
    assert np.all(np.abs(counts - n / W) < 5 * sd), counts


# --------------------------------------------------------------------------
# JSQ and power of two choices.

def test_jsq_paper_example_placement(orc):
    """Sec. 4.2: with JSQ the two long-prompt requests share one worker and the
    two long-output requests the other."""
    g = load("jsq_example.json")
    p = dict(g["params"], policy=1)
    cl = orc.Cluster(p, [g["capacity"]] * 2, [1.0, 1.0], 8)
    seq = [g[k] for k in g["arrival_order"]]
    pl = cl.place_round([s["in"] for s in seq], [s["pred"] for s in seq])
    assert list(pl) == [0, 1, 0, 1]
    assert [g["arrival_order"][i] for i in (0, 2)] == ["long_prompt"] * 2


@pytest.mark.parametrize("policy,fails", [(0, 0), (1, 2)])
def test_jsq_paper_example_executes_over_capacity(orc, policy, fails):
    """Executing the JSQ placement, each worker's KV demand reaches 10 > 9 in
    one decode iteration (the two long prompts in their only iteration, the
    two long outputs in their last), which counts two violations; best-fit's
    placement peaks at 7 and counts none."""
    g = load("jsq_example.json")
    p = dict(g["params"], policy=policy)
    seq = [g[k] for k in g["arrival_order"]]
    tr = Trace([0.0] * 4, [s["in"] for s in seq], [s["pred"] for s in seq])
    res = orc.simulate(p, 2, 8, g["capacity"], 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    assert res["placed"] == 4
    assert res["violations"] == fails and res["failed"] == fails


def test_jsq_round_robin_from_empty(orc, synth):
    """On empty workers JSQ (fewest requests, lowest index on ties) deals the
    requests out in turn: request c goes to worker c mod N."""
    p = dict(synth.BASE_PARAMS, policy=1)
    rng = np.random.default_rng(3)
    for N in (1, 3, 8):
        cl = orc.Cluster(p, [10**6] * N, [1.0] * N, 64)
        C = 5 * N + 2
        pl = cl.place_round(rng.integers(1, 500, C), rng.integers(1, 500, C))
        assert list(pl) == [c % N for c in range(C)]


def test_jsq_balances_counts(orc, synth):
    wl = synth.config("tiny", per_worker_random=True, seed=5, per_worker=20)
    p = dict(wl.params, policy=1)
    cl = orc.Cluster(p, wl.kv_capacity, wl.lat_scale, 128, wl.roff, wl.req_in, wl.req_gen,
                     wl.req_pred)
    n0 = cl.n.copy()
    pl = cl.place_round(wl.cand_in, wl.cand_pred)
    n = n0.copy()
    for c, w in enumerate(pl):
        assert n[w] == n.min() and w == int(np.flatnonzero(n == n.min())[0]), c
        n[w] += 1
    assert np.array_equal(n, cl.n)


def test_po2_placements_from_published_outputs(orc, synth):
    """Two requests (ids 0 and 1) under seed 1234567 on 5 workers holding
    3, 0, 2, 1, 4 requests: each picks, of its two drawn workers, the one
    holding fewer requests (the first drawn on ties)."""
    outs = [int(v) for v in load("splitmix64.json")["streams"][1]["outputs"]]
    W = 5
    counts = [3, 0, 2, 1, 4]
    draws = [((x >> 32) * W) >> 32 for x in outs[:4]]
    reqs = []
    for w, k in enumerate(counts):
        reqs += [(w, 10, 0, 50)] * k
    roff = np.cumsum([0] + counts).astype(np.int32)
    ins = np.array([r[1] for r in reqs], np.int32)
    p = dict(synth.BASE_PARAMS, policy=2, seed=1234567)
    cl = orc.Cluster(p, [10**6] * W, [1.0] * W, 16, roff, ins, np.zeros(len(reqs), np.int32),
                     np.full(len(reqs), 50, np.int32))
    pl = cl.place_round([10, 10], [50, 50], crid=[0, 1])
    n = list(counts)
    for c in range(2):
        w1, w2 = draws[2 * c], draws[2 * c + 1]
        want = w2 if n[w2] < n[w1] else w1
        assert pl[c] == want
        n[want] += 1


def test_policy_full_worker(orc, synth):
    """A JSQ choice without a free slot is a capacity error in a fixed-cluster
    round and a failed request in the simulation."""
    p = dict(synth.BASE_PARAMS, policy=1)
    cl = orc.Cluster(p, [10**6], [1.0], 2)
    with pytest.raises(OverflowError):
        cl.place_round([10, 10, 10], [5, 5, 5])
    tr = Trace([0.0] * 3, [10] * 3, [5] * 3)
    res = orc.simulate(p, 1, 2, 10**6, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    assert res["placed"] == 2 and res["failed"] == 1 and res["violations"] == 0


# --------------------------------------------------------------------------
# Decode instances (split-phase inference).

@pytest.mark.parametrize("T_dec,flags,margin", [
    # request 2 (r = 1): t(1) = 8.1568 + 0.0002 l <= 20, l <= 59,216; request 1
    # (r = 3): 24.3122 + 0.0004 l <= 60, l <= 89,219.5; candidate (r = 2):
    # 16.2596 + 0.0004 l <= 40, l <= 59,351; KV: 10^6 - 34. No stall, so
    # request 2 binds at 59,216 (the mixed setting's stall made it 1,536).
    (20.0, 15, 59216.0 - 5.0),
    # T_dec 8.1: request 2 (8.1 - 8.1568)/0.0002 = -284, request 1
    # (24.3 - 24.3122)/0.0004 = -30.5, candidate (16.2 - 16.2596)/0.0004 = -149:
    # bits 4 and 8 clear; bit 2 stays set although T_pre = 1 ms (not tested).
    (8.1, 3, -284.0 - 5.0),
])
def test_decode_hand_example(orc, T_dec, flags, margin):
    g = load("hand_example.json")
    p = dict(g["params"], T_pre=1.0, T_dec=T_dec, phase=1)
    reqs = list(zip(g["worker"]["in"], g["worker"]["gen"], g["worker"]["pred"]))
    cl = one_worker(orc, p, 10**6, reqs)
    r = cl.score([g["candidate"]["in"]], [g["candidate"]["pred"]], [500.0])
    assert int(r["flags"][0, 0]) == flags
    assert r["margin"][0, 0] == pytest.approx(margin, rel=1e-9, abs=1e-9)
    assert int(r["kvpeak"][0, 0]) == 39
    assert r["tcand"][0, 0] == pytest.approx(16.2616, rel=1e-12)


@pytest.mark.parametrize("mode", [0, 1])
def test_decode_is_mixed_without_prefill(orc, synth, mode):
    """A decode instance scores like a mixed worker whose prefill costs
    nothing (k1 = c1 = 0) and whose TTFT SLO never binds, including with
    placements pending in an open round."""
    wl = synth.config("tiny", per_worker_random=True, seed=17, per_worker=16, kv_per_gpu=8192,
                      params=dict(T_pre=60.0, T_dec=10.5, theta=0.9, mode=mode))
    tdec = wl.params["theta"] * wl.params["T_dec"] * wl.req_gen * 0.97
    dec = orc.Cluster(wl.params | dict(phase=1), wl.kv_capacity, wl.lat_scale, wl.b_cap, wl.roff,
                      wl.req_in, wl.req_gen, wl.req_pred, tdec)
    ref = orc.Cluster(wl.params | dict(k1=0.0, c1=0.0, T_pre=1e300), wl.kv_capacity,
                      wl.lat_scale, wl.b_cap, wl.roff, wl.req_in, wl.req_gen, wl.req_pred, tdec)
    for cl in (dec, ref):
        cl.place_round(wl.cand_in[:6], wl.cand_pred[:6], wl.cand_wait[:6])
    a = dec.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    b = ref.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    assert np.array_equal(a["flags"], b["flags"])
    assert np.array_equal(a["margin"], b["margin"])
    assert np.array_equal(a["argbest"], b["argbest"])
    assert 0 < (a["flags"] == 15).mean() < 1
    assert np.all(a["flags"] & 2)
    assert 0 < ((a["flags"] & 1) > 0).mean() < 1 and 0 < ((a["flags"] & 8) > 0).mean() < 1


def test_decode_advance_closed_form(orc, synth):
    """On a decode instance a placed request joins the batch at the worker's
    next boundary with no prefill: no TTFT record, and its ATGT is the
    empty-worker decode sum over its r iterations divided by r."""
    p = dict(synth.BASE_PARAMS, phase=1)
    cl = orc.Cluster(p, [10**6], [0.8], 8)
    cl.place_round([300], [40], [12.5], crid=[7])
    rid, val, kind = cl.advance(0.0, 10_000.0)
    assert list(rid) == [7] and list(kind) == [1]
    D = 0.8 * (40 * (p["c3"] + p["c2"] + p["k2"] * 300) + p["k2"] * 40 * 41 / 2)
    assert val[0] == pytest.approx(D / 40, rel=1e-12)


def test_decode_unplaced_fails_at_once(orc, synth):
    """Two requests arrive together; one worker can hold only one. On a decode
    instance the second fails at its first heartbeat; in the mixed setting it
    waits (its TTFT allows) and is placed once the first has finished."""
    base = dict(synth.BASE_PARAMS, T_pre=10_000.0)
    tr = Trace([0.0, 0.0], [500, 500], [100, 100])
    M = 700
    dec = orc.simulate(dict(base, phase=1), 1, 8, M, 1.0, tr, 100.0, stop_at_fail=False,
                       drain=True)
    assert dec["placed"] == 1 and dec["failed"] == 1 and dec["violations"] == 0
    mix = orc.simulate(base, 1, 8, M, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    assert mix["placed"] == 2 and mix["failed"] == 0


@pytest.mark.parametrize("phase", [0, 1])
def test_atgt_violation_count(orc, synth, phase):
    """Two requests (prompt 100, output 10) decoding together take
    t(s) = 8 + 0.05*2 + 2e-4 * 2 (100 + s) = 8.14 + 4e-4 s, so
    ATGT = (81.4 + 4e-4 * 55) / 10 = 8.1422 ms > T_dec = 8.1: JSQ puts both
    on the one worker and both violate; alone a request takes
    (80.7 + 2e-4 * 55) / 10 = 8.0711 ms, so best-fit admits one; the other
    fails on a decode instance and, in the mixed setting, waits one
    heartbeat and then runs alone."""
    base = dict(synth.BASE_PARAMS, T_dec=8.1, phase=phase)
    tr = Trace([0.0, 0.0], [100, 100], [10, 10])
    jsq = orc.simulate(dict(base, policy=1), 1, 8, 10**6, 1.0, tr, 100.0, stop_at_fail=False,
                       drain=True)
    assert jsq["placed"] == 2 and jsq["violations"] == 2 and jsq["failed"] == 2
    assert jsq["max_atgt"] == pytest.approx(8.1422, rel=1e-12)
    bf = orc.simulate(base, 1, 8, 10**6, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    assert bf["placed"] == 2 - phase and bf["violations"] == 0 and bf["failed"] == phase
    assert bf["max_atgt"] == pytest.approx(8.0711, rel=1e-12)


def test_ttft_violation_count(orc, synth):
    """Mixed setting, T_pre = 10.1 ms: a 200-token prompt's prefill takes
    0.001 * 200 + 10 = 10.2 ms. JSQ places it anyway (one TTFT violation);
    best-fit finds no worker and the request fails unplaced."""
    base = dict(synth.BASE_PARAMS, T_pre=10.1)
    tr = Trace([0.0], [200], [5])
    jsq = orc.simulate(dict(base, policy=1), 1, 8, 10**6, 1.0, tr, 100.0, stop_at_fail=False,
                       drain=True)
    assert jsq["violations"] == 1 and jsq["max_ttft"] == pytest.approx(10.2, rel=1e-12)
    bf = orc.simulate(base, 1, 8, 10**6, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    assert bf["placed"] == 0 and bf["failed"] == 1 and bf["violations"] == 0


@pytest.mark.parametrize("policy,phase", [(1, 1), (2, 1), (0, 1), (1, 0)])
def test_min_workers_linear_scan_policies(orc, synth, policy, phase):
    tr = synth.diurnal_trace(6, 300, 30.0, 7.5)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, policy=policy, phase=phase, seed=5)
    drain = policy != 0
    oks = [orc.simulate(p, n, 256, 32768, 1.0, tr, 100.0, drain=drain)["failed"] == 0
           for n in range(1, 13)]
    assert True in oks
    first = oks.index(True) + 1
    assert all(oks[first - 1:]), oks
    got = orc.min_workers(p, [1], [32768], [1.0], 256, tr, 100.0, 16)
    assert got[0] == first
