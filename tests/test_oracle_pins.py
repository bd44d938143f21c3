"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test checks the oracle against something other than itself: numbers
worked by hand from the paper's equations, the numbers of the paper's JSQ
example, closed forms of arithmetic series, the structure the paper states
(KV peaks just before a request finishes), brute force over small inputs and
exhaustive search of the placement MIP.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def one_worker(orc, params, M, reqs, cap=16, scale=1.0, tdec=None, off=0.0):
    ins = np.array([r[0] for r in reqs], np.int32)
    gen = np.array([r[1] for r in reqs], np.int32)
    pred = np.array([r[2] for r in reqs], np.int32)
    roff = np.array([0, len(reqs)], np.int32)
    return orc.Cluster(params, [M], [scale], cap, roff, ins, gen, pred,
                       None if tdec is None else np.asarray(tdec, np.float64), off=[off])


# --------------------------------------------------------------------------
# Hand-worked example of Eq. kv cache, Eq. prefill iter time, Eq. iter time.

@pytest.mark.parametrize("case", range(3))
def test_hand_example(orc, case):
    g = load("hand_example.json")
    c = g["cases"][case]
    p = dict(g["params"], T_pre=c["T_pre"], T_dec=c["T_dec"])
    reqs = list(zip(g["worker"]["in"], g["worker"]["gen"], g["worker"]["pred"]))
    cl = one_worker(orc, p, c["M"], reqs)
    r = cl.score([g["candidate"]["in"]], [g["candidate"]["pred"]], [g["candidate"]["wait"]])
    assert int(r["kvpeak"][0, 0]) == c["kv_peak"]
    assert r["tcand"][0, 0] == pytest.approx(c["t_cand"], rel=1e-12)
    assert int(r["flags"][0, 0]) == c["flags"]
    assert r["margin"][0, 0] == pytest.approx(c["margin"], rel=1e-9, abs=1e-9)


def test_hand_kv_curve(orc):
    g = load("hand_example.json")
    reqs = list(zip(g["worker"]["in"], g["worker"]["gen"], g["worker"]["pred"]))
    cl = one_worker(orc, g["params"], 40, reqs)
    assert list(cl.kv_curve(0, 5, 2)) == [39, 19, 13]
    assert list(cl.kv_curve(0, 0, 0)) == [33, 12, 13]


def test_prefill_example(orc, synth):
    """Tiny-workload prefill model: 10 ms + 0.1 ms per 100 tokens, so a 512-token
    prompt takes 10.512 ms. With T_pre = 11.012 ms the TTFT bound on an empty
    worker is (11.012 - 10)/0.001 = 1012 tokens."""
    p = dict(synth.BASE_PARAMS, T_pre=11.012)
    cl = one_worker(orc, p, 10**6, [])
    r = cl.score([512], [1], [0.0])
    assert r["flags"][0, 0] == 15
    assert r["margin"][0, 0] == pytest.approx(1012 - 512, abs=1e-6)
    # 0.6 ms more wait leaves 0.4 ms - 0.512 ms < 0: TTFT fails.
    r = cl.score([512], [1], [0.6])
    assert r["flags"][0, 0] == 15 - 2


# --------------------------------------------------------------------------
# The paper's JSQ example (Sec. 4.2, Fig. example).

def test_jsq_example_peaks(orc):
    g = load("jsq_example.json")
    lp, lo = g["long_prompt"], g["long_output"]
    p = g["params"]
    for reqs, want in (([lp, lp], g["peak_two_long_prompt"]), ([lo, lo], g["peak_two_long_output"]),
                       ([lp, lo], g["peak_mixed"])):
        cl = one_worker(orc, p, g["capacity"], [(reqs[0]["in"], 0, reqs[0]["pred"])])
        r = cl.score([reqs[1]["in"]], [reqs[1]["pred"]])
        assert int(r["kvpeak"][0, 0]) == want
        assert bool(r["flags"][0, 0] & 1) == (want <= g["capacity"])


def test_jsq_example_best_fit(orc):
    g = load("jsq_example.json")
    p = g["params"]
    cl = orc.Cluster(p, [g["capacity"]] * 2, [1.0, 1.0], 8)
    seq = [g[k] for k in g["arrival_order"]]
    pl = cl.place_round([s["in"] for s in seq], [s["pred"] for s in seq])
    assert list(pl) == g["best_fit_placement"]


# --------------------------------------------------------------------------
# Closed forms of the arithmetic series behind Eq. iter time.

def test_empty_worker_closed_form(orc, synth):
    rng = np.random.default_rng(11)
    p = dict(synth.BASE_PARAMS, h=3, j=7)
    cl = one_worker(orc, p, 10**7, [], scale=0.7)
    a = rng.integers(1, 3000, 50)
    r = rng.integers(1, 3000, 50)
    out = cl.score(a, r)
    for i in range(50):
        ai, ri = float(a[i]), float(r[i])
        s = 0.7
        # sum_{s=1}^{r} (c3 + c2 + k2 (a + s)) = r (c3 + c2 + k2 a) + k2 r (r + 1) / 2
        D = s * (ri * (p["c3"] + p["c2"] + p["k2"] * ai) + p["k2"] * ri * (ri + 1) / 2)
        assert out["tcand"][i, 0] == pytest.approx(D, rel=1e-12)
        assert out["kvpeak"][i, 0] == p["h"] * (a[i] + r[i]) + p["j"]


def test_single_segment_closed_form(orc, synth):
    """All requests (and the candidate) finish together: one segment, b = n + 1
    throughout, so D = r (c3 + c2 b + k2 sum a) + k2 b r (r + 1) / 2."""
    rng = np.random.default_rng(12)
    p = dict(synth.BASE_PARAMS)
    for trial in range(20):
        n = int(rng.integers(1, 10))
        r = int(rng.integers(1, 500))
        ins = rng.integers(1, 1000, n)
        gens = rng.integers(0, 300, n)
        reqs = [(int(ins[q]), int(gens[q]), int(gens[q]) + r) for q in range(n)]
        cl = one_worker(orc, p, 10**8, reqs)
        a_c = int(rng.integers(1, 1000))
        out = cl.score([a_c], [r])
        b = n + 1
        suma = float(np.sum(ins + gens) + a_c)
        D = r * (p["c3"] + p["c2"] * b + p["k2"] * suma) + p["k2"] * b * r * (r + 1) / 2
        assert out["tcand"][0, 0] == pytest.approx(D, rel=1e-12)
        assert out["kvpeak"][0, 0] == int(suma) + b * r


# --------------------------------------------------------------------------
# Structure: KV peaks just before a request finishes (Sec. 1; vector w of (e)).

def test_kv_peak_at_breakpoints(orc, synth):
    rng = np.random.default_rng(13)
    p = dict(synth.BASE_PARAMS, h=2, j=5)
    for trial in range(30):
        n = int(rng.integers(0, 12))
        pred = rng.integers(1, 200, n)
        gen = np.array([int(rng.integers(0, x)) for x in pred], np.int64)
        ins = rng.integers(1, 300, n)
        reqs = [(int(ins[q]), int(gen[q]), int(pred[q])) for q in range(n)]
        cl = one_worker(orc, p, 10**7, reqs)
        a_c, r_c = int(rng.integers(1, 300)), int(rng.integers(1, 250))
        curve = cl.kv_curve(0, a_c, r_c)
        out = cl.score([a_c], [r_c])
        assert curve.max() == out["kvpeak"][0, 0]
        ends = set(int(x) for x in (pred - gen)) | {r_c}
        s_star = int(np.argmax(curve)) + 1
        assert s_star in ends
        # strictly increasing inside every segment between finishing times
        for s in range(1, len(curve)):
            if s not in ends:
                assert curve[s] > curve[s - 1]


# --------------------------------------------------------------------------
# The margin is the largest admissible prompt length minus a_c: moving the
# prompt across it flips feasibility (the flags are computed from the slack at
# a_c directly, the bound from slack(0)/slope).

def test_margin_is_tight(orc, synth):
    wl = synth.config("tiny", per_worker_random=True, seed=21,
                      params=dict(T_pre=40.0, T_dec=30.0))
    cl = orc.Cluster.from_workload(wl)
    out = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    checked = 0
    for c in range(wl.n_cand):
        for w in range(wl.n_workers):
            m = out["margin"][c, w]
            if not np.isfinite(m):
                continue
            bound = m + wl.cand_in[c]
            lo = math.floor(bound)
            if lo < 0 or abs(bound - round(bound)) < 1e-6 or lo > 10**6:
                continue
            sub = orc.Cluster.from_workload(wl)
            r = sub.score_pairs([0, 1], [w, w], [lo, lo + 1], [wl.cand_pred[c]] * 2,
                                [wl.cand_wait[c]] * 2)
            assert r["flags"][0] == 15, (c, w, bound)
            assert r["flags"][1] != 15, (c, w, bound)
            checked += 1
            if checked > 150:
                return
    assert checked > 20


def test_infinite_slo_reduces_to_kv_packing(orc, synth):
    wl = synth.config("tiny", per_worker_random=True, seed=22,
                      params=dict(T_pre=1e12, T_dec=1e12))
    cl = orc.Cluster.from_workload(wl)
    out = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    M = wl.kv_capacity[None, :]
    assert np.array_equal(out["flags"] == 15, out["kvpeak"] <= M)
    assert np.all(out["flags"] & 14 == 14)


def test_infinite_kv_reduces_to_slo_packing(orc, synth):
    wl = synth.config("tiny", per_worker_random=True, seed=23, kv_per_gpu=10**9,
                      params=dict(T_pre=200.0, T_dec=12.0))
    cl = orc.Cluster.from_workload(wl)
    out = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    assert np.all(out["flags"] & 1)
    assert 0 < np.mean(out["flags"] == 15) < 1


def test_latency_scale(orc, synth):
    """Scaling every latency coefficient by s scales every projected latency by s."""
    wl = synth.config("tiny", per_worker_random=True, seed=24)
    a = orc.Cluster.from_workload(wl)
    b = orc.Cluster(wl.params, wl.kv_capacity, np.full(wl.n_workers, 0.5), wl.b_cap, wl.roff,
                    wl.req_in, wl.req_gen, wl.req_pred)
    ra = a.score(wl.cand_in[:8], wl.cand_pred[:8])
    rb = b.score(wl.cand_in[:8], wl.cand_pred[:8])
    assert np.allclose(rb["tcand"], 0.5 * ra["tcand"], rtol=1e-12)
    assert np.array_equal(ra["kvpeak"], rb["kvpeak"])


# --------------------------------------------------------------------------
# Algorithm 1: the chosen worker is the feasible one with the largest
# capacity_norm, lowest index on ties (brute force over all workers).

def capacity_norms(wl, gamma):
    out = []
    for w in range(wl.n_workers):
        a, b = wl.roff[w], wl.roff[w + 1]
        B = float(b - a)
        L = float(np.sum(wl.req_in[a:b])) + gamma * float(np.sum(wl.req_pred[a:b]))
        out.append(math.hypot(B, L))
    return np.array(out)


def test_argbest_brute_force(orc, synth):
    for seed in (31, 32, 33):
        wl = synth.config("tiny", per_worker_random=True, seed=seed,
                          params=dict(T_pre=60.0, T_dec=35.0))
        cl = orc.Cluster.from_workload(wl)
        out = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        norms = capacity_norms(wl, wl.params["gamma"])
        for c in range(wl.n_cand):
            best, bw = -1.0, -1
            for w in range(wl.n_workers):
                if out["flags"][c, w] == 15 and norms[w] > best:
                    best, bw = norms[w], w
            assert out["argbest"][c] == bw


def test_argbest_ties_lowest_index(orc, synth):
    p = dict(synth.BASE_PARAMS)
    cl = orc.Cluster(p, [10**6] * 4, [1.0] * 4, 8, np.array([0, 1, 2, 3, 4]),
                     np.array([100, 100, 100, 100]), np.array([0, 0, 0, 0]),
                     np.array([50, 50, 50, 50]))
    out = cl.score([10, 10], [5, 5])
    assert list(out["argbest"]) == [0, 0]


# --------------------------------------------------------------------------
# Greedy round = repeated single placements; MIP optimum as a lower bound.

def test_round_is_sequential_argbest(orc, synth):
    wl = synth.config("tiny", per_worker_random=True, seed=41,
                      params=dict(T_pre=300.0, T_dec=12.0))
    a = orc.Cluster.from_workload(wl, cap=96)
    b = orc.Cluster.from_workload(wl, cap=96)
    pl = a.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
    for c in range(wl.n_cand):
        one = b.score(wl.cand_in[c:c + 1], wl.cand_pred[c:c + 1], wl.cand_wait[c:c + 1])
        w = int(one["argbest"][0])
        assert pl[c] == w
        if w >= 0:
            s = w * b.cap + int(b.n[w])
            b.inp[s], b.gen[s], b.pred[s] = wl.cand_in[c], 0, wl.cand_pred[c]
            b.pend[s], b.wait[s] = 1, wl.cand_wait[c]
            b.n[w] += 1
    assert np.array_equal(a.n, b.n)
    assert (pl >= 0).sum() > 0 and (pl < 0).sum() > 0


def test_round_pending_stall_accumulates(orc, synth):
    """Each placement adds its prompt to the worker's pending prefill: with a TTFT
    budget for exactly two 100-token prompts, the third goes elsewhere."""
    p = dict(synth.BASE_PARAMS, T_pre=10.0 + 0.2 + 1e-6, k1=0.001, c1=10.0)
    cl = orc.Cluster(p, [10**6, 10**6], [1.0, 1.0], 8)
    pl = cl.place_round([100, 100, 100], [4, 4, 4])
    assert list(pl) == [0, 0, 1]


def set_feasible(orc, p, M, items):
    cl = orc.Cluster(p, [M], [1.0], 16)
    pl = cl.place_round([i[0] for i in items], [i[1] for i in items])
    return bool(np.all(pl >= 0))


def test_greedy_vs_mip_optimum(orc, synth):
    """Exhaustive search over assignments of <= 6 requests to <= 3 empty workers
    (the MIP of Sec. 4.2); greedy best-fit never uses fewer workers."""
    rng = np.random.default_rng(51)
    p = dict(synth.BASE_PARAMS, T_pre=1e9, T_dec=1e9)
    M = 60
    for trial in range(12):
        n = int(rng.integers(2, 7))
        items = [(int(rng.integers(1, 25)), int(rng.integers(1, 25))) for _ in range(n)]
        if any(a + r > M for a, r in items):
            continue
        best = None
        for assign in itertools.product(range(3), repeat=n):
            groups = [[items[i] for i in range(n) if assign[i] == g] for g in range(3)]
            if all(set_feasible(orc, p, M, g) for g in groups if g):
                used = sum(1 for g in groups if g)
                best = used if best is None else min(best, used)
        cl = orc.Cluster(p, [M] * n, [1.0] * n, 16)
        pl = cl.place_round([a for a, _ in items], [r for _, r in items])
        assert np.all(pl >= 0)
        assert best is not None and len(set(pl.tolist())) >= best


# --------------------------------------------------------------------------
# Execution: realized latencies follow the same models; admitted requests meet
# their SLOs when predictions are exact.

def test_advance_single_request_closed_form(orc, synth):
    p = dict(synth.BASE_PARAMS)
    cl = orc.Cluster(p, [10**6], [0.8], 8)
    pl = cl.place_round([300], [40], [12.5], crid=[7])
    assert pl[0] == 0
    rid, val, kind = cl.advance(0.0, 10_000.0)
    s = 0.8
    tau = s * (p["k1"] * 300 + p["c1"])
    assert list(rid) == [7, 7] and list(kind) == [0, 1]
    assert val[0] == pytest.approx(12.5 + tau, rel=1e-12)
    D = s * (40 * (p["c3"] + p["c2"] + p["k2"] * 300) + p["k2"] * 40 * 41 / 2)
    assert val[1] == pytest.approx(D / 40, rel=1e-12)


def test_advance_matches_projection(orc, synth):
    """A candidate's projected decode time (score) equals its realized decode
    time (advance) when nothing else is placed later."""
    wl = synth.config("tiny", per_worker_random=True, seed=61, per_worker=6,
                      params=dict(T_pre=1e6, T_dec=1e6))
    for w in range(4):
        cl = orc.Cluster.from_workload(wl)
        cl.has_tdec = True
        proj = cl.score(wl.cand_in[w:w + 1], wl.cand_pred[w:w + 1])
        cl2 = orc.Cluster.from_workload(wl)
        # place the candidate on worker w only
        s = w * cl2.cap + int(cl2.n[w])
        cl2.inp[s], cl2.gen[s], cl2.pred[s], cl2.pend[s] = wl.cand_in[w], 0, wl.cand_pred[w], 1
        cl2.rid[s] = 999
        cl2.n[w] += 1
        rid, val, kind = cl2.advance(0.0, 1e9)
        atgt = val[(rid == 999) & (kind == 1)]
        assert len(atgt) == 1
        assert atgt[0] * wl.cand_pred[w] == pytest.approx(proj["tcand"][0, w], rel=1e-9)


def test_simulation_meets_slos(orc, synth):
    """With exact predictions every request best-fit admits meets its SLOs
    (P100, Sec. 6.4): on this trace 8 workers serve every request, and with 4
    the unplaced requests fail while the admitted ones still meet TTFT, ATGT
    and KV capacity."""
    tr = synth.diurnal_trace(5, 600, 120.0, 30.0)
    p = dict(synth.BASE_PARAMS, T_dec=25.0, T_pre=400.0)
    ok = orc.simulate(p, 8, 256, 32768, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    short = orc.simulate(p, 4, 256, 32768, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    assert ok["failed"] == 0 and ok["placed"] == 600
    assert short["failed"] > 0 and short["placed"] + short["failed"] == 600
    for res in (ok, short):
        assert res["violations"] == 0
        assert res["max_ttft"] <= p["T_pre"] * (1 + 1e-9)
        assert res["max_atgt"] <= p["theta"] * p["T_dec"] * (1 + 1e-9)


def test_min_workers_linear_scan(orc, synth):
    tr = synth.diurnal_trace(6, 300, 30.0, 7.5)
    p = dict(synth.BASE_PARAMS, T_dec=30.0)
    oks = [orc.simulate(p, n, 256, 32768, 1.0, tr, 100.0)["failed"] == 0 for n in range(1, 9)]
    first = oks.index(True) + 1 if True in oks else -1
    assert all(oks[first - 1:]), oks   # monotone on this trace
    got = orc.min_workers(p, [1], [32768], [1.0], 256, tr, 100.0, 16)
    assert got[0] == first


# --------------------------------------------------------------------------
# Approximate mode: the MIP's constraints (b) (with Eq. input limit) and (d)
# as stated in Sec. 4.2, worked by hand.

APPROX = dict(k1=0.01, c1=5.0, k2=0.001, c2=1.0, c3=10.0, h=1, j=0, T_pre=1000.0, T_dec=50.0,
              gamma=0.5, theta=0.8, K=8192, mode=1)


@pytest.mark.parametrize("T_dec,tdec,flags,margin", [
    # (b): L = (100 + 0.5*60) + (300 + 0.5*40) = 450; l_d(3) = (50 - 10 - 3)/0.001
    # = 37,000; bound 0.8*37,000 - 450 - 0.5*30 = 29,135. (d): saved time
    # 0.8*(50*20 - 700) = 240 and 0.8*(50*5 - 200) = 40; stall 0.01*a + 5 <= 40
    # gives a <= 3,500 (binding). TTFT: a <= (1000 - 5)/0.01 = 99,500.
    (50.0, [700.0, 200.0], 15, 3500.0 - 150.0),
    # request 2 saved only 0.8*(250 - 249) = 0.8 ms < the 6.5 ms stall: (d) fails,
    # bound (0.8 - 5)/0.01 = -420
    (50.0, [700.0, 249.0], 11, -420.0 - 150.0),
    # T_dec 10.5: l_d(3) = (10.5 - 10 - 3)/0.001 = -2,500, bound 0.8*(-2,500) - 465
    # = -2,465: (b) fails; saved 0.8*(210 - 150) = 48 and 0.8*(52.5 - 40) = 10
    # keep (d) (a <= 500)
    (10.5, [150.0, 40.0], 7, -2465.0 - 150.0),
])
def test_approx_hand_example(orc, T_dec, tdec, flags, margin):
    p = dict(APPROX, T_dec=T_dec)
    cl = one_worker(orc, p, 10**6, [(100, 20, 60), (300, 5, 40)], tdec=tdec)
    r = cl.score([150], [30], [0.0])
    assert int(r["flags"][0, 0]) == flags
    assert r["margin"][0, 0] == pytest.approx(margin, rel=1e-12)


def test_approx_input_limit_per_request(orc, synth):
    """Each request added to a worker lowers the (b) bound by theta * c2 / k2
    (Eq. input limit's slope in the batch size) plus its own l_in + gamma
    l_pred, whatever the rest of the worker holds."""
    rng = np.random.default_rng(31)
    p = dict(APPROX, T_dec=100.0, T_pre=1e9)
    # every request has generated 10 tokens in no time: (d) allows a stall of
    # 0.8 * 100 * 10 = 800 ms (a <= 79,500), looser than (b) (a <= ~60,000)
    for _ in range(20):
        n = int(rng.integers(1, 12))
        reqs = [(int(rng.integers(16, 500)), 10, int(rng.integers(11, 300))) for _ in range(n)]
        cand_in, cand_pred = int(rng.integers(16, 200)), int(rng.integers(8, 200))
        margins = []
        for k in (n - 1, n):
            cl = one_worker(orc, p, 10**9, reqs[:k], tdec=[0.0] * k)
            margins.append(cl.score([cand_in], [cand_pred], [0.0])["margin"][0, 0])
        added = reqs[n - 1][0] + p["gamma"] * reqs[n - 1][2]
        assert margins[0] - margins[1] == pytest.approx(p["theta"] * p["c2"] / p["k2"] + added,
                                                        rel=1e-12)


def test_approx_and_exact_share_kv_and_ttft(orc, synth):
    """Switching the mode changes only the two decode-SLO groups: the KV and
    TTFT flags and the KV peaks of every pair are the same."""
    wl = synth.config("tiny", per_worker_random=True, seed=32, n_cand=80,
                      params=dict(T_pre=60.0, T_dec=30.0, theta=0.9))
    ex = orc.Cluster.from_workload(wl).score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    ap = orc.Cluster(dict(wl.params, mode=1), wl.kv_capacity, wl.lat_scale, wl.b_cap, wl.roff,
                     wl.req_in, wl.req_gen, wl.req_pred).score(wl.cand_in, wl.cand_pred,
                                                               wl.cand_wait)
    assert np.array_equal(ex["flags"] & 3, ap["flags"] & 3)
    assert np.array_equal(ex["kvpeak"], ap["kvpeak"])
    assert (ex["flags"] != ap["flags"]).any()


# --------------------------------------------------------------------------
# Decode history (Table 1's t^dec) in constraint (d), the iteration-boundary
# offset a straddling execution step leaves, and the prefill stall charged to
# the requests already decoding: worked by hand
# (tests/golden/history_example.json).

@pytest.mark.parametrize("case", range(2))
def test_history_bank(orc, case):
    g = load("history_example.json")["bank"]
    c = g["cases"][case]
    reqs = list(zip(g["worker"]["in"], g["worker"]["gen"], g["worker"]["pred"]))
    cl = one_worker(orc, g["params"], g["M"], reqs, tdec=c["tdec"])
    r = cl.score([g["candidate"]["in"]], [g["candidate"]["pred"]], [g["candidate"]["wait"]])
    assert int(r["flags"][0, 0]) == c["flags"]
    assert r["margin"][0, 0] == pytest.approx(c["margin"], rel=1e-9)
    # the decode time the candidate sees is unchanged by the history
    assert r["tcand"][0, 0] == pytest.approx(8.1578 + 8.1036 + 2 * 2e-4 * 5, rel=1e-12)


def test_history_offset(orc):
    g = load("history_example.json")["offset"]
    reqs = list(zip(g["worker"]["in"], g["worker"]["gen"], g["worker"]["pred"]))
    cl = one_worker(orc, g["params"], g["M"], reqs, tdec=[0.0])
    rid, val, kind = cl.advance(0.0, g["heartbeat_ms"])
    assert len(rid) == 0  # nothing finished
    a = g["after"]
    assert int(cl.gen[0]) == a["gen"]
    assert cl.tdec[0] == pytest.approx(a["tdec"], rel=1e-12)
    assert cl.clock[0] == pytest.approx(a["clock"], rel=1e-12)
    assert cl.off[0] == pytest.approx(a["off"], rel=1e-9)
    for c in g["cases"]:
        r = cl.score([g["candidate"]["in"]], [g["candidate"]["pred"]], [c["wait"]])
        assert int(r["flags"][0, 0]) == c["flags"], c
        assert r["margin"][0, 0] == pytest.approx(c["margin"], rel=1e-9), c


def test_history_stall(orc):
    g = load("history_example.json")["stall"]
    w = g["worker"]
    cl = one_worker(orc, g["params"], g["M"], list(zip(w["in"], w["gen"], w["pred"])),
                    tdec=w["tdec"])
    q = g["placed"]
    pl = cl.place_round([q["in"]], [q["pred"]], [q["wait"]], crid=[q["rid"]])
    assert list(pl) == [0]
    rid, val, kind = cl.advance(0.0, g["heartbeat_ms"])
    got = sorted(zip(rid.tolist(), kind.tolist(), val.tolist()))
    want = sorted((r[0], r[2], r[1]) for r in g["records"])
    assert [(a, b) for a, b, _ in got] == [(a, b) for a, b, _ in want]
    for (_, _, v), (_, _, x) in zip(got, want):
        assert v == pytest.approx(x, rel=1e-12)
    assert int(cl.n[0]) == 0
    assert cl.clock[0] == pytest.approx(g["clock"], rel=1e-12)
