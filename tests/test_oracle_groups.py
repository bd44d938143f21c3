"""Pins of the oracle's grouped (distributed) scheduling, Appendix A: requests
dealt round-robin to G groups, each group scheduling on its own workers. The
grouped simulation must be the union of G independent simulations (one per
group, on its own arrivals and workers), and every placement must stay in
its group."""
import numpy as np
import pytest


class Trace:
    def __init__(self, t, i, p):
        self.t_arr = np.asarray(t, np.float64)
        self.req_in = np.asarray(i, np.int32)
        self.req_pred = np.asarray(p, np.int32)


@pytest.mark.parametrize("policy", [0, 1, 2])
def test_placements_stay_in_their_group(orc, synth, policy):
    wl = synth.config("tiny", per_worker_random=True, seed=31, per_worker=12, n_cand=48,
                      b_cap=128, params=dict(T_pre=500.0, T_dec=40.0, policy=policy, groups=3,
                                             seed=3))
    oc = orc.Cluster.from_workload(wl)
    pl = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
    ok = pl >= 0
    assert ok.sum() > 10
    assert np.all(pl[ok] % 3 == np.arange(len(pl))[ok] % 3)


def test_one_group_is_centralized(orc, synth):
    tr = synth.diurnal_trace(5, 400, 40.0, 10.0)
    p = dict(synth.BASE_PARAMS)
    a = orc.simulate(p, 4, 256, 65536, 1.0, tr, 100.0, stop_at_fail=False, drain=True)
    b = orc.simulate(dict(p, groups=1), 4, 256, 65536, 1.0, tr, 100.0, stop_at_fail=False,
                     drain=True)
    assert a == b


@pytest.mark.parametrize("policy,G,N", [(0, 2, 5), (0, 3, 7), (1, 3, 6)])
def test_grouped_simulation_is_union_of_groups(orc, synth, policy, G, N):
    """Group g serves arrivals q = g, g + G, ... on workers g, g + G, ...; its
    run alone (a trace and a cluster of its own) gives the same outcomes, so
    the grouped totals are the sums (counts) and maxima (latencies) over the
    groups, and the run lasts as long as the longest group's."""
    tr = synth.diurnal_trace(11, 900, 50.0, 12.0)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, policy=policy)
    grouped = orc.simulate(dict(p, groups=G), N, 256, 40000, 1.0, tr, 100.0,
                           stop_at_fail=False, drain=True)
    parts = []
    for g in range(G):
        sel = np.arange(len(tr.t_arr)) % G == g
        sub = Trace(tr.t_arr[sel], tr.req_in[sel], tr.req_pred[sel])
        Ng = len(range(g, N, G))
        parts.append(orc.simulate(p, Ng, 256, 40000, 1.0, sub, 100.0, stop_at_fail=False,
                                  drain=True))
    for k in ("failed", "placed", "violations"):
        assert grouped[k] == sum(r[k] for r in parts), k
    for k in ("max_ttft", "max_atgt"):
        assert grouped[k] == max(r[k] for r in parts), k
    assert grouped["heartbeats"] == max(r["heartbeats"] for r in parts)
    assert grouped["placed"] > 0


def test_grouping_costs_workers(orc, synth):
    """Appendix A expects groups to cost extra workers (each group packs only
    its share of the load); on this trace the grouped search needs at least
    as many workers as the centralized one."""
    tr = synth.diurnal_trace(6, 600, 60.0, 15.0)
    p = dict(synth.BASE_PARAMS, T_dec=30.0)
    n1 = orc.min_workers(p, [1], [32768], [1.0], 256, tr, 100.0, 64)[0]
    n3 = orc.min_workers(dict(p, groups=3), [1], [32768], [1.0], 256, tr, 100.0, 64)[0]
    assert n1 > 0 and n3 >= n1


def test_rebalance_stays_in_group(orc):
    """Algorithm 2 with groups: a request on an over-utilized worker of group 0
    moves only to an under-utilized worker of group 0."""
    p = dict(k1=0.001, c1=10.0, k2=2e-4, c2=0.05, c3=8.0, h=1, j=0, T_pre=1000.0, T_dec=50.0,
             gamma=0.5, theta=1.0, K=8192, groups=2)
    cl = orc.Cluster(p, [10**6] * 4, [1.0] * 4, 16)
    pl = cl.place_round([200], [100], [0.0], crid=[0])   # group 0: workers 0, 2
    assert list(pl) == [0]
    # worker 1 (group 1) is the most under-utilized, worker 2 (group 0) less so
    mv, _, _ = cl.rebalance([200], [100], [0.0], pl, [10**4, -10**5, -10**4, 0], [0, 0, 0, 0],
                            crid=[0])
    assert mv == 1 and list(pl) == [2]


def test_full_worker_stops_only_its_group(orc, synth):
    """With groups, a best-fit group whose chosen worker has no free slot stops
    (that candidate and its later ones stay unplaced); the other group goes on.
    Two groups of one worker each, 4 slots: group 0's worker holds 3 requests,
    so its second candidate finds it full; group 1 places all of its own."""
    p = dict(synth.BASE_PARAMS, groups=2)
    roff = np.array([0, 3, 3], np.int32)
    cl = orc.Cluster(p, [10**6, 10**6], [1.0, 1.0], 4, roff, np.full(3, 100, np.int32),
                     np.zeros(3, np.int32), np.full(3, 50, np.int32))
    pl, full = cl.place_round([100] * 8, [50] * 8, crid=np.arange(8), allow_capacity=True)
    assert full
    assert list(pl) == [0, 1, -1, 1, -1, 1, -1, 1]
    assert list(cl.n) == [4, 4]


# --- the number of groups (Appendix A, Eq. group_arrival_limit) -------------

def _gold_groups():
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", "group_count_example.json")) as f:
        return json.load(f)


def test_group_count_paper_example(orc):
    """e = 10%: every group must keep at least five workers, so 50 workers
    allow at most 10 groups and 49 at most 9."""
    g = _gold_groups()
    e, per = g["e"], g["min_workers_per_group"]
    assert orc.pick_groups(0.0, 1.0, e, 1) == 0              # one worker cannot hold 5
    assert orc.pick_groups(0.0, 1.0, e, per) == 1
    # rate 10x one scheduler's limit needs 10 groups: 10 * 5 workers suffice,
    # 10 * 5 - 1 do not
    assert orc.pick_groups(10.0 * 250.0, 250.0, e, 10 * per) == 10
    assert orc.pick_groups(10.0 * 250.0, 250.0, e, 10 * per - 1) == 0
    # a rate just above 9 schedulers' limit also needs 10
    assert orc.pick_groups(9.5 * 250.0, 250.0, e, 10 * per) == 10
    assert orc.pick_groups(9.0 * 250.0, 250.0, e, 10 * per - 1) == 9


def test_group_count_is_the_fewest_feasible(orc):
    """Brute force in exact rational arithmetic: the fewest G with
    rate_a / G <= rate_max and n / G >= 1 / (2e)."""
    from fractions import Fraction as F
    rng = np.random.default_rng(57)
    checked = 0
    for _ in range(400):
        n = int(rng.integers(1, 400))
        e = float(rng.uniform(0.01, 0.6))
        rmax = float(rng.uniform(50.0, 5000.0))
        ra = float(rng.uniform(0.0, 40.0) * rmax)
        want = 0
        for G in range(1, n + 1):
            if F(ra) <= G * F(rmax) and F(n) * 2 * F(e) >= G:
                want = G
                break
        # skip draws within rounding of a boundary of either condition
        near = any(abs(F(ra) - G * F(rmax)) <= F(ra) * F(1, 10**9) or
                   abs(F(n) * 2 * F(e) - G) <= F(1, 10**9) for G in range(1, n + 1))
        if near:
            continue
        assert orc.pick_groups(ra, rmax, e, n) == want, (ra, rmax, e, n)
        checked += 1
    assert checked > 350


def test_group_count_special_cases(orc):
    # one scheduler keeps up: one group (the central scheduler)
    assert orc.pick_groups(100.0, 1000.0, 0.05, 10) == 1
    # the rate needs more groups than the workers allow
    assert orc.pick_groups(2000.0, 100.0, 0.5, 15) == 0
    # e = 1/2 lets every worker be its own group (one worker a group)
    assert orc.pick_groups(2000.0, 100.0, 0.5, 20) == 20
    # more tolerance allows more, smaller groups; never more groups than needed
    for e in (0.05, 0.1, 0.2, 0.5):
        assert orc.pick_groups(1000.0, 300.0, e, 400) == 4
