"""aladdin_score_noalloc, the scoring call for callers that cannot allocate
device memory while they schedule (a process whose device memory a serving
engine reserved up front for its KV cache, a real-time loop that must not
reach the allocator). It must give the same results as aladdin_score, call
after call, although all calls share one fixed scratch array, and after its
first call on a device it must take no device memory at all. Collected last
so that a failure here stops a -x run only after every other test has run."""
import numpy as np
import pytest

from parity import REL

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


def score_both(A, cl, W, cin, cpr, cw):
    import torch
    dev = torch.device("cuda")
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    C = len(cin)
    din, dpr, dw = t(cin), t(cpr), t(cw)
    out = []
    for fn in (A.aladdin_score, A.aladdin_score_noalloc):
        f = torch.full((C, W), 0xEE, dtype=torch.uint8, device=dev)
        m = torch.full((C, W), 12345.0, dtype=torch.float32, device=dev)
        a = torch.full((C,), 77, dtype=torch.int32, device=dev)
        fn(cl.handle, C, din, dpr, dw, f, m, a)
        torch.cuda.synchronize()
        out.append((f.cpu().numpy(), m.cpu().numpy(), a.cpu().numpy()))
    return out


def assert_same(ref, got):
    (f0, m0, a0), (f1, m1, a1) = ref, got
    assert np.array_equal(f0, f1)
    assert np.array_equal(a0, a1)
    assert np.array_equal(np.isnan(m0), np.isnan(m1))
    assert np.array_equal(np.isneginf(m0), np.isneginf(m1))
    fin = np.isfinite(m0)
    assert np.all(np.abs(m1[fin] - m0[fin]) <= REL * np.maximum(np.abs(m0[fin]), 1.0))


def test_noalloc_matches_score_on_two_calls(A, synth):
    wl = synth.config("w256", n_cand=3000)
    other = synth.config("w256", n_cand=1300, seed=77)
    cin2, cpr2, cw2 = other.cand_in.copy(), other.cand_pred.copy(), other.cand_wait.copy()
    cin2[5] = -3                       # an invalid candidate in the second call
    cpr2[9] = wl.params["K"]
    with A.Cluster.from_workload(wl) as cl:
        first = score_both(A, cl, wl.n_workers, wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert_same(*first)
        second = score_both(A, cl, wl.n_workers, cin2, cpr2, cw2)
        assert_same(*second)
        assert second[1][0][5].max() == A.FLAG_INVALID and second[1][2][9] == A.INVALID
        assert 0 < (first[1][0] == A.FEASIBLE).mean()


def test_noalloc_rejects_what_it_cannot_hold(A, synth):
    import torch
    wl = synth.config("tiny", n_cand=8)
    dev = torch.device("cuda")
    with A.Cluster.from_workload(wl) as cl:
        n = A.NOALLOC_MAX_CAND + 1
        big = torch.ones(n, dtype=torch.int32, device=dev)
        with pytest.raises(A.AladdinError) as e:
            A.aladdin_score_noalloc(cl.handle, n, big, big, None, None, None,
                                    torch.empty(n, dtype=torch.int32, device=dev))
        assert e.value.code == A.ERR_SCRATCH
        with pytest.raises(A.AladdinError) as e:  # host memory would need staging
            A.aladdin_score_noalloc(cl.handle, 8, wl.cand_in, wl.cand_pred, None, None, None,
                                    np.zeros(8, np.int32))
        assert e.value.code == A.ERR_ARG


def test_noalloc_takes_no_device_memory(A, synth):
    """After the first call on the device (which sets the device up), calls
    with every combination of outputs leave the device's free memory
    unchanged: nothing is allocated, not even kernel code."""
    import torch
    wl = synth.config("w256", n_cand=2000)
    dev = torch.device("cuda")
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    C, W = wl.n_cand, wl.n_workers
    din, dpr, dw = t(wl.cand_in), t(wl.cand_pred), t(wl.cand_wait)
    f = torch.empty((C, W), dtype=torch.uint8, device=dev)
    m = torch.empty((C, W), dtype=torch.float32, device=dev)
    a = torch.empty(C, dtype=torch.int32, device=dev)
    ref = torch.empty(C, dtype=torch.int32, device=dev)
    with A.Cluster.from_workload(wl) as cl:
        A.aladdin_score(cl.handle, C, din, dpr, dw, None, None, ref)
        A.aladdin_score_noalloc(cl.handle, 16, din, dpr, dw, None, None, a)  # set-up
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        for outs in ((f, m, a), (f, None, None), (None, m, None), (None, None, a), (f, None, a),
                     (None, m, a), (f, m, None)):
            for n in (C, 7):
                A.aladdin_score_noalloc(cl.handle, n, din, dpr, dw, *outs)
        torch.cuda.synchronize()
        free1 = torch.cuda.mem_get_info()[0]
        assert free1 == free0, "device free memory moved by %d bytes" % (free1 - free0)
        A.aladdin_score_noalloc(cl.handle, C, din, dpr, dw, None, None, a)
        torch.cuda.synchronize()
        assert torch.equal(a, ref)
