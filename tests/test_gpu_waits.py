"""Bounded device waits run out without a fault: a wait that nothing can
complete gives up after its poll limit, the call returns (or the cluster
reports) ALADDIN_ERR_TIMEOUT, and the device stays usable.

The waits are made to run out by design through the library's test hook
(aladdin_cluster_test_waits): the placement round's grid exchange waits for
one arrival more than its CTAs make, and the scoring kernel withholds its
first candidate copy, so nothing ever completes that mbarrier phase. No
kernel faults, traps or hangs: each gives up after a few thousand polls."""
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


def still_usable(A, synth):
    """A fresh cluster scores and places like before: the context survived."""
    wl = synth.config("tiny", per_worker_random=True, seed=7, per_worker=24,
                      params=dict(T_pre=60.0, T_dec=30.0))
    with A.Cluster.from_workload(wl) as cl:
        out = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert cl.status() == A.OK
        assert 0 < (out["flags"] == A.FEASIBLE).mean() < 1


def test_round_grid_wait_runs_out(A, synth):
    """A round of several CTAs (4,096 workers do not fit one CTA's shared
    memory) whose exchange can never complete."""
    wl = synth.make_cluster("slices", 231, 4096, 12, 60000, 200, per_worker_random=True,
                            b_cap=128, params=dict(T_pre=60.0, T_dec=12.0))
    with A.Cluster.from_workload(wl) as cl:
        A.aladdin_cluster_test_waits(cl.handle, 1 << 10, 0, 1)
        with pytest.raises(A.AladdinError) as e:
            cl.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert e.value.code == A.ERR_TIMEOUT
        assert cl.status() == A.ERR_TIMEOUT  # sticky
    still_usable(A, synth)


def test_score_barrier_wait_runs_out(A, synth):
    """The scoring kernel's first candidate chunk never arrives: every CTA
    gives up after the set number of mbarrier polls (waiting for the copy it
    did issue before it leaves), and the cluster reports the timeout."""
    import torch
    wl = synth.config("w256", n_cand=700)
    dev = torch.device("cuda")
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    C, W = wl.n_cand, wl.n_workers
    f = torch.zeros((C, W), dtype=torch.uint8, device=dev)
    m = torch.zeros((C, W), dtype=torch.float32, device=dev)
    a = torch.zeros(C, dtype=torch.int32, device=dev)
    with A.Cluster.from_workload(wl) as cl:
        A.aladdin_cluster_test_waits(cl.handle, 0, 1 << 12, 1)
        A.aladdin_score(cl.handle, C, t(wl.cand_in), t(wl.cand_pred), t(wl.cand_wait), f, m, a)
        torch.cuda.synchronize()
        assert cl.status() == A.ERR_TIMEOUT
    still_usable(A, synth)


def test_wait_hook_rejects_bad_arguments(A, synth):
    wl = synth.config("tiny", n_cand=4)
    with A.Cluster.from_workload(wl) as cl:
        for args in ((-1, 0, 0), (0, -5, 0), (0, 0, 2)):
            with pytest.raises(A.AladdinError) as e:
                A.aladdin_cluster_test_waits(cl.handle, *args)
            assert e.value.code == A.ERR_ARG
        A.aladdin_cluster_test_waits(cl.handle, 0, 0, 0)  # the defaults
        out = cl.score(wl.cand_in, wl.cand_pred, wl.cand_wait)
        assert cl.status() == A.OK and out["argbest"].shape == (4,)
