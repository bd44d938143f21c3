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


@pytest.mark.parametrize("b_cap,seed", [(32, 205), (64, 206)])
def test_round_small_tables(A, orc, synth, b_cap, seed):
    """Rounds on tables of 32 and 64 slots (one and two rebuild warps, each
    with its look-ahead group): placements and the final state equal the
    oracle's, with runs of candidates on the same worker."""
    wl = synth.make_cluster("small", seed, 300, 6, 30000, 700, per_worker_random=True,
                            b_cap=b_cap, params=dict(T_pre=400.0, T_dec=10.2))
    with A.Cluster.from_workload(wl) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert cl.status() == A.OK
        oc = orc.Cluster.from_workload(wl)
        ref = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, ref), np.argwhere(pl != ref)[:5]
        assert_same_state(cl, oc, "small-%d" % b_cap)
    placed = pl[pl >= 0]
    assert len(placed) > 0
    assert (placed[1:] == placed[:-1]).mean() > 0.3  # runs on one worker


def test_round_w256(A, orc, synth):
    wl = synth.config("w256", n_cand=512, b_cap=128)
    with A.Cluster.from_workload(wl) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        oc = orc.Cluster.from_workload(wl)
        ref = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, ref)
        assert_same_state(cl, oc, "round-w256")
        assert (pl >= 0).any()


@pytest.mark.parametrize("max_slots,chunk", [(3, 0), (0, 97), (5, 131)])
def test_round_incremental_hand_offs(A, orc, synth, max_slots, chunk):
    """The incremental round's two hand-offs on a small cluster: with few
    modified-worker slots the sliced round continues from the candidate that
    needs one more, and with small chunks every chunk of candidates is a
    fresh incremental round from the current state. Both place like the
    oracle, over two calls (the second within the open round)."""
    wl = synth.config("w256", n_cand=900, b_cap=128)
    oc = orc.Cluster.from_workload(wl)
    with A.Cluster.from_workload(wl) as cl:
        A.aladdin_cluster_test_round(cl.handle, max_slots, chunk)
        for lo, hi in ((0, 520), (520, 900)):
            pl = cl.place_round(wl.cand_in[lo:hi], wl.cand_pred[lo:hi], wl.cand_wait[lo:hi])
            ref = oc.place_round(wl.cand_in[lo:hi], wl.cand_pred[lo:hi], wl.cand_wait[lo:hi])
            assert np.array_equal(pl, ref), np.argwhere(pl != ref)[:5]
        assert_same_state(cl, oc, "hand-offs-%d-%d" % (max_slots, chunk))
        assert cl.status() == A.OK
    with A.Cluster.from_workload(wl) as cl:
        with pytest.raises(A.AladdinError) as e:
            A.aladdin_cluster_test_round(cl.handle, -1, 0)
        assert e.value.code == A.ERR_ARG


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
        out = np.zeros(A.SIMULATE_OUT)
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
    out = np.zeros(A.SIMULATE_OUT)
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
    out = np.zeros(A.SIMULATE_OUT)
    A.aladdin_simulate(A.make_params(p, 512), A.make_cfgs([1], [12000], [1.0])[0], 450,
                       A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 0, 1, out)
    assert ref["failed"] > 0
    assert int(out[0]) == ref["failed"] and int(out[1]) == ref["placed"], (out, ref)
    assert int(out[2]) == ref["heartbeats"]
    assert out[3] == pytest.approx(ref["max_ttft"], rel=1e-12)
    assert out[4] == pytest.approx(ref["max_atgt"], rel=1e-12)


def sorted_state(n, inp, gen, pred, pend, cap):
    """Per-worker request multisets as one array sorted by (worker, in, gen,
    pred, pend)."""
    W = len(n)
    slot = np.arange(W * cap) % cap
    w = np.arange(W * cap) // cap
    live = slot < np.repeat(n, cap)
    cols = (w[live], inp[live], gen[live], pred[live], pend[live].astype(np.int32))
    o = np.lexsort(cols[::-1])
    return np.stack([c[o] for c in cols])


def test_w16384_rounds_sampled(A, orc, synth):
    """The 16,384-worker workload (1/2/4/8-GPU workers) at full size: three of
    its consecutive greedy rounds with 100 ms of execution between them.
    Sampled candidates are placed by the oracle on the same state (the others
    take the GPU's placement); after each execution step the whole cluster
    state must equal the oracle's."""
    wl = synth.config("w16384")
    C = wl.n_cand
    bounds = np.linspace(0, C, 11).astype(int)
    oc = orc.Cluster.from_workload(wl)
    for w in range(oc.W):  # explicit "no history" decode time, as the library assumes
        s = w * oc.cap
        k = int(oc.n[w])
        oc.tdec[s:s + k] = wl.params["theta"] * wl.params["T_dec"] * oc.gen[s:s + k]
    oc.has_tdec = True
    rng = np.random.default_rng(17)
    t = 0.0
    with A.Cluster.from_workload(wl) as cl:
        for k in range(3):
            a, b = int(bounds[k]), int(bounds[k + 1])
            pl = cl.place_round(wl.cand_in[a:b], wl.cand_pred[a:b], wl.cand_wait[a:b])
            assert cl.status() == A.OK
            sample = set(rng.choice(b - a, 6, replace=False).tolist()) | {0, b - a - 1}
            for i in range(b - a):
                c = a + i
                if i in sample:
                    ref = oc.place_round(wl.cand_in[c:c + 1], wl.cand_pred[c:c + 1],
                                         wl.cand_wait[c:c + 1].astype(np.float64))
                    assert ref[0] == pl[i], (k, i, ref[0], pl[i])
                elif pl[i] >= 0:
                    oc.commit(pl[i], wl.cand_in[c], wl.cand_pred[c], float(wl.cand_wait[c]), c)
            cl.advance(100.0)
            oc.advance(t, 100.0)
            t += 100.0
            n, i_, g_, p_, pe = cl.state()
            assert np.array_equal(n, oc.n), k
            got = sorted_state(n, i_, g_, p_, pe, cl.b_cap)
            ref = sorted_state(oc.n, oc.inp, oc.gen, oc.pred, oc.pend, oc.cap)
            assert np.array_equal(got, ref), k


def test_capacity_1024(A, orc, synth):
    """Workers of 1,024 request slots (tables built by cooperating warps):
    scoring, a greedy round and an execution step against the oracle."""
    wl = synth.make_cluster("c1024", 250, 40, 700, 400000, 300, per_worker_random=True,
                            b_cap=1024, gpus_cycle=(1, 2, 4, 8),
                            params=dict(T_pre=3000.0, T_dec=120.0))
    assert np.diff(wl.roff).max() > 512
    with A.Cluster.from_workload(wl) as cl:
        g = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait, detail=True)
        oc = orc.Cluster.from_workload(wl)
        ref = oc.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        compare_pairs(ref, g["flags"], g["margin"], wl.cand_in, g["kvpeak"], g["tcand"], "c1024")
        assert 0 < (g["flags"] == 15).mean() < 1
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        rp = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, rp), np.argwhere(pl != rp)[:5]
        assert (pl >= 0).any()
        assert_same_state(cl, oc, "c1024-round")
        for w in range(oc.W):
            s = w * oc.cap
            k = int(oc.n[w])
            oc.tdec[s:s + k] = np.where(oc.pend[s:s + k] == 1, 0.0,
                                        wl.params["theta"] * wl.params["T_dec"] * oc.gen[s:s + k])
        oc.has_tdec = True
        cl.advance(100.0)
        oc.advance(0.0, 100.0)
        assert_same_state(cl, oc, "c1024-advance")


def test_round_rows_beyond_shared_memory(A, orc, synth):
    """20,000 workers of 1,024 slots: each CTA of the round holds about 740
    breakpoint rows per worker (one CTA per SM), fewer than the three heavy
    workers have (about 900 distinct remaining lengths each); their row search
    continues in the table in global memory."""
    import dataclasses
    W = 20000
    wl = synth.make_cluster("rows", 240, W, 3, 65536, 300, per_worker_random=True, b_cap=1024,
                            params=dict(T_pre=2000.0, T_dec=85.0))
    heavy = {7: 900, 9000: 880, 19999: 910}
    counts = np.diff(wl.roff).astype(np.int64)
    ins, gens, preds = [], [], []
    for w in range(W):
        a, b = int(wl.roff[w]), int(wl.roff[w + 1])
        if w in heavy:
            r = np.arange(1, heavy[w] + 1, dtype=np.int32)  # distinct remaining lengths
            ins.append(np.full(len(r), 16, np.int32))
            gens.append(np.ones(len(r), np.int32))
            preds.append(r + 1)
            counts[w] = len(r)
        else:
            ins.append(wl.req_in[a:b])
            gens.append(wl.req_gen[a:b])
            preds.append(wl.req_pred[a:b])
    roff = np.zeros(W + 1, np.int32)
    np.cumsum(counts, out=roff[1:])
    kv = wl.kv_capacity.copy()
    for w in heavy:
        kv[w] = 240000  # the KV constraint binds after some placements
    rng = np.random.default_rng(241)
    wl = dataclasses.replace(wl, roff=roff, req_in=np.concatenate(ins),
                             req_gen=np.concatenate(gens), req_pred=np.concatenate(preds),
                             kv_capacity=kv,
                             cand_pred=rng.integers(1, 2500, wl.n_cand).astype(np.int32))
    with A.Cluster.from_workload(wl) as cl:
        pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        oc = orc.Cluster.from_workload(wl)
        rp = oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(pl, rp), np.argwhere(pl != rp)[:5]
        on_heavy = np.isin(pl, list(heavy))
        assert on_heavy.any() and (~on_heavy).any()
        assert (wl.cand_pred[on_heavy] > 750).any()
        assert_same_state(cl, oc, "rows")


def test_min_workers_four_options(A, orc, synth):
    """The minimum-worker search of the 1/2/4/8-GPU options (KV 65,536 tokens
    per GPU, latency x 1/sqrt(GPUs), 1,024 request slots) on the diurnal
    trace scaled down to 10,000 requests at a peak of 200 req/s."""
    tr = synth.diurnal_trace(14, 10000, 200.0, 50.0)
    p = dict(synth.BASE_PARAMS)
    gpus = [1, 2, 4, 8]
    M = [65536 * g for g in gpus]
    sc = [1.0 / np.sqrt(g) for g in gpus]
    ref = orc.min_workers(p, gpus, M, sc, 1024, tr, 100.0, 256)
    got = np.zeros(4, np.int32)
    best, total = A.aladdin_min_workers(A.make_params(p, 1024), A.make_cfgs(gpus, M, sc),
                                        A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 256,
                                        got)
    assert np.array_equal(got, ref), (got, ref)
    tot = [g * n for g, n in zip(gpus, ref)]
    assert total == min(tot) and best == int(np.argmin(tot))


def test_round_and_simulation_deterministic(A, synth):
    """The same round on two fresh clusters (a cooperative grid of several
    CTAs) gives the same placements and state bytes; the same simulation twice
    gives the same outputs."""
    wl = synth.config("w4096", n_cand=3000, b_cap=256)
    res = []
    for _ in range(2):
        with A.Cluster.from_workload(wl) as cl:
            pl = cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
            cl.advance(100.0)
            res.append((pl.tobytes(),) + tuple(x.tobytes() for x in cl.state()))
    assert res[0] == res[1]
    tr = synth.with_prediction_error(synth.diurnal_trace(8, 3000, 80.0, 20.0), 0.4, 8)
    p = dict(synth.BASE_PARAMS, T_dec=30.0, rebalance=1)
    outs = []
    for _ in range(2):
        out = np.zeros(A.SIMULATE_OUT)
        A.aladdin_simulate(A.make_params(p, 256), A.make_cfgs([1], [40000], [1.0])[0], 9,
                           A.trace_of(tr), 100.0, 0, 1, out)
        outs.append(out.tobytes())
    assert outs[0] == outs[1]


def test_checkpoint_resume(A, synth):
    """A cluster saved with an open round (pending placements, decode history,
    clock) and restored into a fresh cluster of the same shape continues
    exactly like the original: the same scores, placements and state."""
    wl = synth.config("w256", n_cand=1500, b_cap=128, params=dict(T_dec=30.0))
    h = (wl.req_gen * np.random.default_rng(3).uniform(8.0, 30.0, len(wl.req_gen))).astype(
        np.float32)
    with A.Cluster.from_workload(wl, tdec_ms=h) as a:
        a.place_round(wl.cand_in[:400], wl.cand_pred[:400], wl.cand_wait[:400])
        a.advance(100.0)
        a.place_round(wl.cand_in[400:700], wl.cand_pred[400:700], wl.cand_wait[400:700])
        blob = A.aladdin_cluster_save(a.handle)
        with A.Cluster.from_workload(synth.config("w256", n_cand=4, b_cap=128,
                                                  params=dict(T_dec=30.0))) as b:
            A.aladdin_cluster_restore(b.handle, blob)
            outs = []
            for cl in (a, b):
                s = cl.score(wl.cand_in[700:900], wl.cand_pred[700:900], wl.cand_wait[700:900])
                pl = cl.place_round(wl.cand_in[700:], wl.cand_pred[700:], wl.cand_wait[700:])
                st = cl.advance(100.0)
                outs.append([s["flags"].tobytes(), s["margin"].tobytes(), s["argbest"].tobytes(),
                             pl.tobytes()] + [x.tobytes() for x in cl.state()])
            assert outs[0] == outs[1]
    with A.Cluster.from_workload(synth.config("tiny")) as c:
        with pytest.raises(A.AladdinError):
            A.aladdin_cluster_restore(c.handle, blob)       # another shape
        with pytest.raises(A.AladdinError):
            A.aladdin_cluster_restore(c.handle, blob[:100])  # truncated
