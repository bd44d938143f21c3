"""The minimum-worker search runs its simulations side by side (options at
once, several doubling steps and bisection levels at once) with placement
rounds on one CTA each; a lone simulation (aladdin_simulate) may place with a
cooperative grid over several CTAs. Both must decide every request alike, so
the worker count the search returns has to pass when simulated alone, and
one worker fewer has to fail (the bisection's last two probes)."""
import math

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

B_CAP = 1024          # 1,024 request slots: one CTA's shared memory holds the
                      # breakpoints of about 108 such workers, so larger
                      # probes take the one-CTA round with fewer rows cached
KV_PER_GPU = 65536


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


def simulate(A, p, cfg, n, trace):
    out = np.zeros(A.SIMULATE_OUT)
    A.aladdin_simulate(A.make_params(p, B_CAP), cfg, int(n), trace, 100.0, 1, 0, out)
    return out


def test_search_boundaries_hold_in_lone_simulations(A, synth):
    tr = synth.diurnal_trace(11, 75_000, 2000.0, 500.0)   # one diurnal period in 60 s
    p = dict(synth.BASE_PARAMS)
    gpus = [1, 2]
    cfgs = A.make_cfgs(gpus, [KV_PER_GPU * g for g in gpus], [1.0 / math.sqrt(g) for g in gpus])
    trace = A.make_trace(tr.t_arr, tr.req_in, tr.req_pred)
    got = np.zeros(len(gpus), np.int32)
    A.aladdin_min_workers(A.make_params(p, B_CAP), cfgs, trace, 100.0, 4096, got)
    assert got[0] > 110, got    # probes beyond one CTA's full row cache took part
    for o in range(len(gpus)):
        n = int(got[o])
        assert simulate(A, p, cfgs[o], n, trace)[0] == 0, (o, n)
        assert simulate(A, p, cfgs[o], n - 1, trace)[0] > 0, (o, n)
    again = np.zeros(len(gpus), np.int32)
    A.aladdin_min_workers(A.make_params(p, B_CAP), cfgs, trace, 100.0, 4096, again)
    assert np.array_equal(got, again)
