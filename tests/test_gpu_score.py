"""Parity of the CUDA scoring path (aladdin_score / aladdin_score_detail)
with the oracle, element by element, through the C ABI."""
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


def run_full(A, orc, wl, detail=True, label=""):
    with A.Cluster.from_workload(wl) as cl:
        g = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait, detail=detail)
    oc = orc.Cluster.from_workload(wl)
    ref = oc.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    near = compare_pairs(ref, g["flags"], g["margin"], wl.cand_in, g.get("kvpeak"), g.get("tcand"),
                         label)
    check_argbest(oc.order(), g["flags"], g["argbest"], label)
    if near == 0:
        assert np.array_equal(g["argbest"], ref["argbest"])
    return g, ref, near


def test_tiny_literal(A, orc, synth):
    wl = synth.config("tiny")
    g, ref, near = run_full(A, orc, wl, label="tiny")


@pytest.mark.parametrize("seed,tpre,tdec", [(101, 40.0, 30.0), (102, 1000.0, 50.0),
                                            (103, 25.0, 20.0), (104, 80.0, 14.0)])
def test_tiny_mixed_load(A, orc, synth, seed, tpre, tdec):
    wl = synth.config("tiny", per_worker_random=True, seed=seed, n_cand=300,
                      params=dict(T_pre=tpre, T_dec=tdec))
    g, ref, near = run_full(A, orc, wl, label="tiny-mixed-%d" % seed)
    frac = (g["flags"] == 15).mean()
    assert 0.0 < frac < 1.0


def test_every_constraint_group_binds(A, orc, synth):
    """Across seeds every flag bit is seen cleared on some pair."""
    seen = 0
    for seed, tpre, tdec in ((110, 22.0, 16.0), (111, 22.0, 11.0), (112, 12.0, 30.0),
                             (113, 40.0, 12.5)):
        wl = synth.config("tiny", per_worker_random=True, seed=seed, n_cand=200,
                          params=dict(T_pre=tpre, T_dec=tdec))
        g, ref, near = run_full(A, orc, wl, label="groups-%d" % seed)
        for b in range(4):
            if ((g["flags"] >> b) & 1 == 0).any():
                seen |= 1 << b
    assert seen == 15


def test_scale_h_j_and_history(A, orc, synth):
    """Non-unit KV coefficients, mixed latency scales and a decode history."""
    wl = synth.config("tiny", per_worker_random=True, seed=120, n_cand=256, gpus_cycle=(1, 2, 4, 8),
                      kv_per_gpu=40000, params=dict(h=2, j=3, T_pre=70.0, T_dec=24.0, theta=0.9))
    rng = np.random.default_rng(5)
    tdec = (wl.req_gen * rng.uniform(8.0, 30.0, len(wl.req_gen))).astype(np.float32)
    with A.Cluster.from_workload(wl, tdec_ms=tdec) as cl:
        g = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait, detail=True)
    oc = orc.Cluster.from_workload(wl, tdec=tdec.astype(np.float64))
    ref = oc.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    compare_pairs(ref, g["flags"], g["margin"], wl.cand_in, g["kvpeak"], g["tcand"], "hist")
    check_argbest(oc.order(), g["flags"], g["argbest"], "hist")


def test_w256(A, orc, synth):
    wl = synth.config("w256")
    g, ref, near = run_full(A, orc, wl, label="w256")
    print("w256: near pairs %d of %d, feasible %.3f" % (near, g["flags"].size,
                                                         (g["flags"] == 15).mean()))


def test_ragged_and_edge_shapes(A, orc, synth):
    """W not a multiple of 4 (scalar store path), one worker, one candidate,
    empty workers, candidates at the sequence limit, and chunk tails."""
    for W, C, seed in ((7, 257, 130), (1, 1, 131), (33, 513, 132), (130, 1000, 133)):
        wl = synth.make_cluster("edge", seed, W, 20, 30000, C, per_worker_random=True,
                                params=dict(T_pre=50.0, T_dec=25.0, K=4096))
        wl.cand_pred[: min(3, C)] = 4096 - wl.cand_in[: min(3, C)]
        run_full(A, orc, wl, label="edge-W%d-C%d" % (W, C))


def test_invalid_candidates(A, orc, synth):
    wl = synth.config("tiny", per_worker_random=True, seed=140, n_cand=40)
    cin, cpr, cw = wl.cand_in.copy(), wl.cand_pred.copy(), wl.cand_wait.copy()
    cin[3] = -1
    cpr[5] = 0
    cpr[7] = wl.params["K"]          # in + pred > K
    cw[9] = np.nan
    cw[11] = -1.0
    bad = [3, 5, 7, 9, 11]
    with A.Cluster.from_workload(wl) as cl:
        g = cl.score(cin, cpr, cw, detail=True)
    assert np.all(g["flags"][bad] == A.FLAG_INVALID)
    assert np.all(np.isnan(g["margin"][bad]))
    assert np.all(g["argbest"][bad] == A.INVALID)
    good = np.setdiff1d(np.arange(40), bad)
    oc = orc.Cluster.from_workload(wl)
    ref = oc.score(cin[good], cpr[good], cw[good])
    compare_pairs(ref, g["flags"][good], g["margin"][good], cin[good], g["kvpeak"][good],
                  g["tcand"][good], "valid-rows")


def test_device_and_host_pointers_agree(A, synth):
    import torch
    wl = synth.config("w256", n_cand=700)
    dev = torch.device("cuda")
    with A.Cluster.from_workload(wl) as cl:
        h = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        C, W = wl.n_cand, wl.n_workers
        f = torch.zeros((C, W), dtype=torch.uint8, device=dev)
        m = torch.zeros((C, W), dtype=torch.float32, device=dev)
        a = torch.zeros(C, dtype=torch.int32, device=dev)
        A.aladdin_score(cl.handle, C, torch.from_numpy(wl.cand_in).to(dev),
                        torch.from_numpy(wl.cand_pred).to(dev), torch.from_numpy(wl.cand_wait).to(dev),
                        f, m, a)
        torch.cuda.synchronize()
        assert np.array_equal(f.cpu().numpy(), h["flags"])
        assert np.array_equal(m.cpu().numpy().view(np.uint32), h["margin"].view(np.uint32))
        assert np.array_equal(a.cpu().numpy(), h["argbest"])
        # argbest only (no pair outputs) gives the same choice
        a2 = torch.zeros(C, dtype=torch.int32, device=dev)
        A.aladdin_score(cl.handle, C, torch.from_numpy(wl.cand_in).to(dev),
                        torch.from_numpy(wl.cand_pred).to(dev), torch.from_numpy(wl.cand_wait).to(dev),
                        None, None, a2)
        torch.cuda.synchronize()
        assert np.array_equal(a2.cpu().numpy(), h["argbest"])


def test_deterministic(A, synth):
    wl = synth.config("w256", n_cand=1500)
    with A.Cluster.from_workload(wl) as cl:
        a = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        b = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    for k in a:
        assert a[k].tobytes() == b[k].tobytes(), k


def test_load_device_state(A, orc, synth):
    """aladdin_cluster_load from device memory equals creation from host memory;
    an invalid request loaded from device memory poisons only its worker."""
    import torch
    wl = synth.config("tiny", per_worker_random=True, seed=150, n_cand=64)
    wl2 = synth.config("tiny", per_worker_random=True, seed=151, n_cand=64)
    dev = torch.device("cuda")
    with A.Cluster.from_workload(wl) as cl:
        t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
        cl.load(t(wl2.roff), t(wl2.req_in), t(wl2.req_gen), t(wl2.req_pred))
        torch.cuda.synchronize()
        g = cl.score(wl2.cand_in, wl2.cand_pred, wl2.cand_wait)
        assert cl.status() == A.OK
        ref = orc.Cluster.from_workload(wl2).score(wl2.cand_in, wl2.cand_pred, wl2.cand_wait)
        compare_pairs(ref, g["flags"], g["margin"], wl2.cand_in, label="load")
        gen = wl2.req_gen.copy()
        w_bad = int(np.argmax(np.diff(wl2.roff) > 0))
        gen[wl2.roff[w_bad]] = wl2.req_pred[wl2.roff[w_bad]]  # gen == pred: invalid
        cl.load(t(wl2.roff), t(wl2.req_in), t(gen), t(wl2.req_pred))
        torch.cuda.synchronize()
        assert cl.status() == A.ERR_STATE
        g2 = cl.score(wl2.cand_in, wl2.cand_pred, wl2.cand_wait)
        assert np.all(g2["flags"][:, w_bad] & 1 == 0)
        keep = np.arange(wl2.n_workers) != w_bad
        assert np.array_equal(g2["flags"][:, keep], g["flags"][:, keep])
    # host path rejects the same state up front
    with pytest.raises(A.AladdinError):
        A.Cluster(wl2.params, wl2.gpus, wl2.kv_capacity, wl2.lat_scale, wl2.b_cap, wl2.roff,
                  wl2.req_in, gen, wl2.req_pred)


@pytest.mark.parametrize("theta,T_dec", [(1.0, 32.0 * (1.0 + 2.0 ** -52)),
                                         (0.8, 50.0), (0.6180339887498949, 47.123456789)])
def test_device_pack_decode_budget(A, synth, theta, T_dec):
    """Requests packed from device arrays without a decode history get the
    decode time of a request that used exactly its budget, theta T_dec l_out,
    as the fp64 product (theta T_dec) * l_out: equal to numpy's for output
    lengths up to 2^16 - 1, ties included (with theta T_dec = 32 (1 + 2^-52)
    the exact product for l_out = 3 * 2^k lies halfway between two doubles),
    and the whole packed state equals the state created from the same host
    arrays."""
    import torch
    wl = synth.make_cluster("pack", 77, 96, 40, 1 << 22, 4, per_worker_random=True,
                            out_law=(3000.0, 1.5, 2, 65000), in_law=(64.0, 0.5, 1, 500),
                            params=dict(theta=theta, T_dec=T_dec, K=65536))
    special = np.array([0, 1, 3, 5, 6, 12, 24576, 32769, 49152, 65534], np.int32)
    k = len(special)
    wl.req_gen[:k] = special
    wl.req_pred[:k] = np.maximum(wl.req_pred[:k], special + 1)
    wl.req_in[:k] = np.minimum(wl.req_in[:k], 65536 - wl.req_pred[:k])
    dev = torch.device("cuda")
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    with A.Cluster.from_workload(wl) as host, A.Cluster.from_workload(wl) as packed:
        packed.load(t(wl.roff), t(wl.req_in), t(wl.req_gen), t(wl.req_pred))
        torch.cuda.synchronize()
        assert packed.status() == A.OK
        ch, cp = A.aladdin_cluster_save(host.handle), A.aladdin_cluster_save(packed.handle)
    assert ch == cp
    # the decode-time section of the checkpoint, against numpy's products
    W, S = wl.n_workers, wl.n_workers * wl.b_cap
    tail = 8 * S + S + 8 * S + 4 * W + 8 * W + 8 * W + 4 * W  # tdec .. be
    td = np.frombuffer(cp[len(cp) - tail:len(cp) - tail + 8 * S], np.float64).reshape(W, wl.b_cap)
    thT = np.float64(theta) * np.float64(T_dec)
    for w in range(W):
        lo, hi = wl.roff[w], wl.roff[w + 1]
        want = thT * wl.req_gen[lo:hi].astype(np.float64)
        assert td[w, :hi - lo].tobytes() == want.tobytes(), w


@pytest.mark.parametrize("W", [700, 5000, 9000, 20000, 30000])
def test_rank_order_with_ties(A, orc, synth, W):
    """The capacity_norm order behind argbest (larger key first, lower index
    first among equal keys) on clusters ranked by the all-pairs count (700,
    5,000 and 30,000 workers) and by the chunk sort and merge (9,000 and
    20,000 workers, 9 and 20 chunks of 1,024): workers share one of
    five request sets, so keys tie across chunks, and their KV capacities
    differ, so the feasible workers of a candidate are scattered through each
    tie group. Every argbest must be the first feasible worker in the oracle's
    order."""
    rng = np.random.default_rng(W)
    sets = [rng.integers(16, 400, size=(k, 2)).astype(np.int32) for k in (1, 2, 3, 5, 8)]
    pick = rng.integers(0, len(sets), W)
    counts = np.array([len(sets[s]) for s in pick], np.int32)
    roff = np.zeros(W + 1, np.int32)
    np.cumsum(counts, out=roff[1:])
    req = np.concatenate([sets[s] for s in pick])
    req_in = req[:, 0].copy()
    req_pred = (req[:, 1] + 8).astype(np.int32)
    req_gen = np.minimum(req[:, 1] // 2, req_pred - 1).astype(np.int32)
    kv = rng.choice(np.array([4000, 6000, 9000, 60000], np.int64), W)
    C = 24
    cand_in = rng.integers(16, 3000, C).astype(np.int32)
    cand_pred = rng.integers(8, 300, C).astype(np.int32)
    wl = synth.Workload("ties", dict(synth.BASE_PARAMS), np.ones(W, np.int32), kv,
                        np.ones(W, np.float32), roff, req_in, req_gen, req_pred, cand_in,
                        cand_pred, np.zeros(C, np.float32), 32)
    with A.Cluster.from_workload(wl) as cl:
        g = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    order = orc.Cluster.from_workload(wl).order()
    f = g["flags"] == 15
    assert 0 < f.mean() < 1
    check_argbest(order, g["flags"], g["argbest"], "ties-W%d" % W)


def test_build_overflow_workers(A, orc, synth):
    """Tables of 256 slots where many workers hold more than the 128 requests
    the first-level warp build takes (the rest are listed and built by the
    second level): created from host arrays and loaded from device arrays,
    the pairs score like the oracle."""
    import torch
    wl = synth.make_cluster("ovf", 160, 300, 220, 400000, 256, per_worker_random=True,
                            b_cap=256, params=dict(T_pre=900.0, T_dec=60.0))
    counts = np.diff(wl.roff)
    assert (counts > 128).sum() > 50 and (counts <= 128).sum() > 50
    ref = orc.Cluster.from_workload(wl).score(wl.cand_in, wl.cand_pred, wl.cand_wait)
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(torch.device("cuda"))
    with A.Cluster.from_workload(wl) as cl:
        g = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        compare_pairs(ref, g["flags"], g["margin"], wl.cand_in, label="ovf-host")
        cl.load(t(wl.roff), t(wl.req_in), t(wl.req_gen), t(wl.req_pred))
        torch.cuda.synchronize()
        g2 = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert cl.status() == A.OK
        for k in ("flags", "margin", "argbest"):
            assert g2[k].tobytes() == g[k].tobytes(), k
    assert 0 < (g["flags"] == 15).mean() < 1


def test_w4096_sampled(A, orc, synth):
    """The 4,096-worker workload at full size, scored by the call bench.py
    times (aladdin_cluster_load_score from device arrays): sampled pairs and
    sampled argbest rows against the oracle, and every byte equal to
    aladdin_score on the loaded state."""
    import torch
    wl = synth.config("w4096")
    C, W = wl.n_cand, wl.n_workers
    dev = torch.device("cuda")
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    with A.Cluster.from_workload(wl) as cl:
        f = torch.zeros((C, W), dtype=torch.uint8, device=dev)
        m = torch.zeros((C, W), dtype=torch.float32, device=dev)
        a = torch.zeros(C, dtype=torch.int32, device=dev)
        cin, cpr, cw = d(wl.cand_in), d(wl.cand_pred), d(wl.cand_wait)
        A.aladdin_cluster_load_score(cl.handle, d(wl.roff), d(wl.req_in), d(wl.req_gen),
                                     d(wl.req_pred), None, C, cin, cpr, cw, f, m, a)
        f2 = torch.zeros_like(f)
        m2 = torch.zeros_like(m)
        a2 = torch.zeros_like(a)
        A.aladdin_score(cl.handle, C, cin, cpr, cw, f2, m2, a2)
        torch.cuda.synchronize()
        assert cl.status() == A.OK
        assert torch.equal(f, f2) and torch.equal(m.view(torch.int32), m2.view(torch.int32))
        assert torch.equal(a, a2)
        del f2, m2, a2
        rng = np.random.default_rng(9)
        pc = rng.integers(0, C, 3000).astype(np.int32)
        pw = rng.integers(0, W, 3000).astype(np.int32)
        oc = orc.Cluster.from_workload(wl)
        ref = oc.score_pairs(pc, pw, wl.cand_in, wl.cand_pred, wl.cand_wait)
        fi = f[torch.from_numpy(pc).long().to(dev), torch.from_numpy(pw).long().to(dev)].cpu().numpy()
        mi = m[torch.from_numpy(pc).long().to(dev), torch.from_numpy(pw).long().to(dev)].cpu().numpy()
        compare_pairs(ref, fi, mi, wl.cand_in[pc], label="w4096-sampled")
        fr = (f == 15).float().mean().item()
        assert fr > 0.05  # the workload as specified is almost entirely feasible
        rows = rng.integers(0, C, 6)
        order = oc.order()
        sub = oc.score(wl.cand_in[rows], wl.cand_pred[rows], wl.cand_wait[rows],
                       want=("flags", "margin", "mscale", "near", "argbest"))
        fr_rows = f[torch.from_numpy(rows).long().to(dev)].cpu().numpy()
        mr_rows = m[torch.from_numpy(rows).long().to(dev)].cpu().numpy()
        compare_pairs(sub, fr_rows, mr_rows, wl.cand_in[rows], label="w4096-rows")
        check_argbest(order, fr_rows, a.cpu().numpy()[rows], "w4096-rows")


def test_w4096_mixed_sampled(A, orc, synth):
    """The 4,096-worker workload with tighter limits and a decode history
    (about half of the pairs feasible, every constraint group binding), at
    full size through the benchmarked call: sampled pairs and argbest rows
    against the oracle, near pairs bounded and reported."""
    import torch
    wl = synth.config("w4096_mixed")
    tdec = synth.decode_history(wl, 18.0, 26.0, synth.MIXED_HISTORY_SEED)
    C, W = wl.n_cand, wl.n_workers
    dev = torch.device("cuda")
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    with A.Cluster.from_workload(wl, tdec_ms=tdec) as cl:
        f = torch.zeros((C, W), dtype=torch.uint8, device=dev)
        m = torch.zeros((C, W), dtype=torch.float32, device=dev)
        a = torch.zeros(C, dtype=torch.int32, device=dev)
        cin, cpr, cw = d(wl.cand_in), d(wl.cand_pred), d(wl.cand_wait)
        A.aladdin_cluster_load_score(cl.handle, d(wl.roff), d(wl.req_in), d(wl.req_gen),
                                     d(wl.req_pred), d(tdec), C, cin, cpr, cw, f, m, a)
        torch.cuda.synchronize()
        assert cl.status() == A.OK
        fr = (f == 15).float().mean().item()
        assert 0.3 < fr < 0.7, fr
        for b in range(4):  # every group is cleared on some pair
            assert ((f >> b) & 1 == 0).any().item(), b
        rng = np.random.default_rng(19)
        pc = rng.integers(0, C, 6000).astype(np.int32)
        pw = rng.integers(0, W, 6000).astype(np.int32)
        oc = orc.Cluster.from_workload(wl, tdec=tdec.astype(np.float64))
        ref = oc.score_pairs(pc, pw, wl.cand_in, wl.cand_pred, wl.cand_wait)
        ip, iw = torch.from_numpy(pc).long().to(dev), torch.from_numpy(pw).long().to(dev)
        rep = {}
        compare_pairs(ref, f[ip, iw].cpu().numpy(), m[ip, iw].cpu().numpy(), wl.cand_in[pc],
                      label="w4096-mixed-sampled", report=rep)
        print("w4096_mixed sampled pairs:", rep)
        rows = rng.integers(0, C, 6)
        sub = oc.score(wl.cand_in[rows], wl.cand_pred[rows], wl.cand_wait[rows],
                       want=("flags", "margin", "mscale", "near", "argbest"))
        fr_rows = f[torch.from_numpy(rows).long().to(dev)].cpu().numpy()
        mr_rows = m[torch.from_numpy(rows).long().to(dev)].cpu().numpy()
        compare_pairs(sub, fr_rows, mr_rows, wl.cand_in[rows], label="w4096-mixed-rows")
        check_argbest(oc.order(), fr_rows, a.cpu().numpy()[rows], "w4096-mixed-rows")


def test_load_score_repeated_calls(A, synth):
    """Repeated aladdin_cluster_load_score calls with the same arrays (the
    library replays its state-load half as a CUDA graph from the second
    call) read the arrays' current contents: each of five calls, with a new
    state and new candidates written into the same device arrays, gives the
    bytes of a separate load and score."""
    import torch
    dev = torch.device("cuda")
    base = synth.config("w256", n_cand=700)
    C, W = base.n_cand, base.n_workers
    N = len(base.req_in)
    roff = torch.from_numpy(base.roff).to(dev)
    rin, rgen, rpred = (torch.empty(N, dtype=torch.int32, device=dev) for _ in range(3))
    cin, cpr = (torch.empty(C, dtype=torch.int32, device=dev) for _ in range(2))
    cw = torch.empty(C, dtype=torch.float32, device=dev)
    f = torch.empty((C, W), dtype=torch.uint8, device=dev)
    m = torch.empty((C, W), dtype=torch.float32, device=dev)
    a = torch.empty(C, dtype=torch.int32, device=dev)
    with A.Cluster.from_workload(base) as cl, A.Cluster.from_workload(base) as ref:
        for seed in range(5):
            wl = synth.config("w256", n_cand=700, seed=40 + seed)
            assert np.array_equal(wl.roff, base.roff)
            for t, x in ((rin, wl.req_in), (rgen, wl.req_gen), (rpred, wl.req_pred),
                         (cin, wl.cand_in), (cpr, wl.cand_pred), (cw, wl.cand_wait)):
                t.copy_(torch.from_numpy(x))
            A.aladdin_cluster_load_score(cl.handle, roff, rin, rgen, rpred, None, C, cin, cpr, cw,
                                         f, m, a)
            ref.load(wl.roff, wl.req_in, wl.req_gen, wl.req_pred)
            g = ref.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
            torch.cuda.synchronize()
            assert cl.status() == A.OK
            assert np.array_equal(f.cpu().numpy(), g["flags"]), seed
            assert np.array_equal(m.cpu().numpy().view(np.int32), g["margin"].view(np.int32)), seed
            assert np.array_equal(a.cpu().numpy(), g["argbest"]), seed


def test_page_locked_host_buffers(A, orc, synth):
    """Page-locked host arrays are read and written in place by the kernels
    (state packed on the device, outputs written over the CPU-GPU link): the
    results equal the device-buffer results byte for byte, and the state
    packed from them scores like the oracle."""
    import torch
    wl = synth.config("w256", n_cand=600)
    dev = torch.device("cuda")
    pin = lambda x: torch.from_numpy(np.ascontiguousarray(x)).pin_memory()
    C, W = wl.n_cand, wl.n_workers
    with A.Cluster.from_workload(wl) as cl:
        cl.load(pin(wl.roff), pin(wl.req_in), pin(wl.req_gen), pin(wl.req_pred))
        assert cl.status() == A.OK
        hf = torch.zeros((C, W), dtype=torch.uint8).pin_memory()
        hm = torch.zeros((C, W), dtype=torch.float32).pin_memory()
        ha = torch.zeros(C, dtype=torch.int32).pin_memory()
        A.aladdin_score(cl.handle, C, pin(wl.cand_in), pin(wl.cand_pred), pin(wl.cand_wait), hf, hm,
                        ha)
        df = torch.zeros((C, W), dtype=torch.uint8, device=dev)
        dm = torch.zeros((C, W), dtype=torch.float32, device=dev)
        da = torch.zeros(C, dtype=torch.int32, device=dev)
        A.aladdin_score(cl.handle, C, torch.from_numpy(wl.cand_in).to(dev),
                        torch.from_numpy(wl.cand_pred).to(dev), torch.from_numpy(wl.cand_wait).to(dev),
                        df, dm, da)
        torch.cuda.synchronize()
        assert np.array_equal(hf.numpy(), df.cpu().numpy())
        assert np.array_equal(hm.numpy().view(np.uint32), dm.cpu().numpy().view(np.uint32))
        assert np.array_equal(ha.numpy(), da.cpu().numpy())
        ref = orc.Cluster.from_workload(wl).score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        compare_pairs(ref, hf.numpy(), hm.numpy(), wl.cand_in, label="pinned")
        hp = torch.zeros(C, dtype=torch.int32).pin_memory()
        A.aladdin_place_round(cl.handle, C, pin(wl.cand_in), pin(wl.cand_pred), pin(wl.cand_wait), hp)
        rp = orc.Cluster.from_workload(wl).place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert np.array_equal(hp.numpy(), rp)


def test_load_score_equals_two_calls(A, synth):
    """aladdin_cluster_load_score (candidates sorted on a second stream while
    the tables are built) gives the bytes of aladdin_cluster_load followed by
    aladdin_score, from device and from host arrays, and leaves the cluster in
    the same state."""
    import torch
    wl = synth.config("w256", n_cand=1500)
    wl2 = synth.config("w256", n_cand=1500, seed=77)   # the state loaded by the step
    dev = torch.device("cuda")
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    C, W = wl.n_cand, wl.n_workers
    outs = []
    for mode in ("two", "one_dev", "one_host"):
        with A.Cluster.from_workload(wl) as cl:
            if mode == "one_host":
                f = np.zeros((C, W), np.uint8)
                m = np.zeros((C, W), np.float32)
                a = np.zeros(C, np.int32)
                A.aladdin_cluster_load_score(cl.handle, wl2.roff, wl2.req_in, wl2.req_gen,
                                             wl2.req_pred, None, C, wl.cand_in, wl.cand_pred,
                                             wl.cand_wait, f, m, a)
            else:
                f = torch.zeros((C, W), dtype=torch.uint8, device=dev)
                m = torch.zeros((C, W), dtype=torch.float32, device=dev)
                a = torch.zeros(C, dtype=torch.int32, device=dev)
                args = (t(wl2.roff), t(wl2.req_in), t(wl2.req_gen), t(wl2.req_pred))
                cand = (t(wl.cand_in), t(wl.cand_pred), t(wl.cand_wait))
                if mode == "two":
                    A.aladdin_cluster_load(cl.handle, *args)
                    A.aladdin_score(cl.handle, C, *cand, f, m, a)
                else:
                    A.aladdin_cluster_load_score(cl.handle, *args, None, C, *cand, f, m, a)
                torch.cuda.synchronize()
                f, m, a = f.cpu().numpy(), m.cpu().numpy(), a.cpu().numpy()
            outs.append((f.tobytes(), m.tobytes(), a.tobytes(),
                         tuple(x.tobytes() for x in cl.state())))
    assert outs[0] == outs[1] == outs[2]


def test_history_hand_cases(A):
    """The kernels reproduce the hand-worked decode-history, offset cases
    (tests/golden/history_example.json): constraint (d) with banked slack
    theta T_dec l_out - t^dec, and the TTFT bound after an execution step
    whose last iteration straddles the heartbeat."""
    import json
    import os
    from parity import REL
    with open(os.path.join(os.path.dirname(__file__), "golden", "history_example.json")) as f:
        g = json.load(f)
    b = g["bank"]
    w = b["worker"]
    arr = lambda x, t=np.int32: np.ascontiguousarray(x, t)
    cand = b["candidate"]
    for c in b["cases"]:
        with A.Cluster(b["params"], [1], [b["M"]], [1.0], 32, arr([0, 2]), arr(w["in"]),
                       arr(w["gen"]), arr(w["pred"]), tdec_ms=arr(c["tdec"], np.float32)) as cl:
            out = cl.score([cand["in"]], [cand["pred"]], [cand["wait"]])
        assert int(out["flags"][0, 0]) == c["flags"], c
        tol = REL * max(abs(c["margin"] + cand["in"]), 1.0)
        assert abs(float(out["margin"][0, 0]) - c["margin"]) <= tol, (out["margin"], c)
    o = g["offset"]
    w = o["worker"]
    with A.Cluster(o["params"], [1], [o["M"]], [1.0], 32, arr([0, 1]), arr(w["in"]), arr(w["gen"]),
                   arr(w["pred"]), tdec_ms=arr([0.0], np.float32)) as cl:
        cl.advance(o["heartbeat_ms"])
        n, i, gen, p, pe = cl.state()
        assert int(n[0]) == 1 and int(gen[0]) == o["after"]["gen"]
        for c in o["cases"]:
            out = cl.score([o["candidate"]["in"]], [o["candidate"]["pred"]], [c["wait"]])
            assert int(out["flags"][0, 0]) == c["flags"], c
            tol = REL * max(abs(c["margin"] + o["candidate"]["in"]), 1.0)
            assert abs(float(out["margin"][0, 0]) - c["margin"]) <= tol, (out["margin"], c)
