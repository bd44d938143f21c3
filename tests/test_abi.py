"""The C ABI library loads, exports every function declared in
include/aladdin.h, and rejects invalid arguments on the host (no GPU needed)."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2405_06856_gb300 import build
    build.build()
    from paper_2405_06856_gb300 import aladdin as A
    return A


def declared_functions():
    src = open(os.path.join(ROOT, "include", "aladdin.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\bint\s+(aladdin_\w+)\s*\(", src)))


def test_header_declares_abi():
    names = declared_functions()
    for n in ("aladdin_cluster_create", "aladdin_cluster_destroy", "aladdin_score",
              "aladdin_place_round", "aladdin_min_workers"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    so = ctypes.CDLL(lib.LIB_PATH)
    for n in declared_functions():
        assert hasattr(so, n), n
    assert sorted(lib.exported_symbols()) == declared_functions()


def test_struct_layout(lib):
    # 5 doubles, h and j, 4 doubles, K b_cap mode phase policy, pad, seed,
    # rebalance, groups
    assert ctypes.sizeof(lib.aladdin_params) == 5 * 8 + 2 * 4 + 4 * 8 + 5 * 4 + 4 + 8 + 4 + 4
    assert lib.aladdin_params.seed.offset == 104
    assert lib.aladdin_params.rebalance.offset == 112
    assert lib.aladdin_params.groups.offset == 116
    assert ctypes.sizeof(lib.aladdin_worker_cfg) == 24
    assert ctypes.sizeof(lib.aladdin_trace) == 48


@pytest.mark.parametrize("bad", [dict(k1=0.0), dict(k2=-1.0), dict(T_dec=5.0), dict(theta=0.0),
                                 dict(theta=1.5), dict(K=1), dict(K=70000), dict(h=0),
                                 dict(j=-1), dict(c1=float("nan")), dict(T_pre=0.0),
                                 dict(phase=2), dict(policy=3), dict(policy=-1),
                                 dict(rebalance=2), dict(groups=-1), dict(groups=70000)])
def test_create_rejects_bad_params(lib, bad):
    from paper_2405_06856_gb300 import synth
    d = dict(synth.BASE_PARAMS)
    d.update(bad)
    p = lib.make_params(d, 32)
    cfg = lib.make_cfgs([1], [1000], [1.0])
    off = np.array([0, 0], np.int32)
    h = ctypes.c_void_p()
    rc = lib._lib.aladdin_cluster_create(ctypes.byref(p), 1, ctypes.cast(cfg, ctypes.c_void_p),
                                         off.ctypes.data, None, None, None, None, None,
                                         ctypes.byref(h))
    assert rc == lib.ERR_ARG and not h.value


@pytest.mark.parametrize("b_cap", [16, 48, 2048])
def test_create_rejects_bad_capacity(lib, b_cap):
    from paper_2405_06856_gb300 import synth
    p = lib.make_params(synth.BASE_PARAMS, b_cap)
    cfg = lib.make_cfgs([1], [1000], [1.0])
    off = np.array([0, 0], np.int32)
    h = ctypes.c_void_p()
    rc = lib._lib.aladdin_cluster_create(ctypes.byref(p), 1, ctypes.cast(cfg, ctypes.c_void_p),
                                         off.ctypes.data, None, None, None, None, None,
                                         ctypes.byref(h))
    assert rc == lib.ERR_ARG


def test_null_arguments(lib):
    assert lib._lib.aladdin_cluster_destroy(None) == lib.ERR_ARG
    assert lib._lib.aladdin_score(None, 1, None, None, None, None, None, None) == lib.ERR_ARG
    assert lib._lib.aladdin_cluster_status(None) == lib.ERR_ARG
    from paper_2405_06856_gb300 import synth
    p = lib.make_params(synth.BASE_PARAMS, 32)
    cfg = lib.make_cfgs([1], [1 << 24], [1.0])  # capacity must be < 2^24
    assert lib._lib.aladdin_simulate(ctypes.byref(p), ctypes.cast(cfg, ctypes.c_void_p), 1, None,
                                     100.0, 1, 0, None, None) == lib.ERR_ARG


# --------------------------------------------------------------------------
# Host-only entry points of the worker-configuration model, against the oracle.

def test_tp_configs_match_oracle(lib, orc):
    tp = lib.aladdin_tp_model(30.0, 10.0, 4.0, 80_000.0, 30_000.0)
    gpus = [1, 2, 4, 8]
    cfgs = lib.aladdin_tp_configs(tp, gpus)
    for o, g in enumerate(gpus):
        M, s = orc.tp_config(30.0, 10.0, 4.0, 80_000.0, 30_000.0, g)
        assert cfgs[o].gpus == g and cfgs[o].kv_capacity == int(np.floor(M))
        assert cfgs[o].lat_scale == pytest.approx(s, rel=1e-15)


@pytest.mark.parametrize("tp,gpus", [((30.0, 10.0, 4.0, 10.0, 30.0), [1]),     # capacity < 1
                                     ((0.0, 0.0, 1.0, 1e5, 0.0), [1]),        # k4 + c4 = 0
                                     ((30.0, -1.0, 4.0, 1e5, 0.0), [1]),
                                     ((30.0, 10.0, 4.0, 1e5, 0.0), [0]),
                                     ((30.0, 10.0, 4.0, 1e7, 0.0), [2])])    # >= 2^24
def test_tp_configs_reject(lib, tp, gpus):
    with pytest.raises(lib.AladdinError):
        lib.aladdin_tp_configs(lib.aladdin_tp_model(*tp), gpus)


def test_predict_workers_matches_oracle(lib, orc):
    for k5, c5, r in ((0.06, 4.0, 1234.0), (0.013, -2.5, 977.0), (1e-3, 0.0, 250.0)):
        assert lib.aladdin_predict_workers(k5, c5, r) == orc.predict_workers(k5, c5, r)
    with pytest.raises(lib.AladdinError):
        lib.aladdin_predict_workers(float("inf"), 0.0, 1.0)


def test_pick_groups_matches_oracle(lib, orc):
    """Appendix A's group count: the library's closed form against the
    oracle's enumeration (0 there = no group count meets both conditions)."""
    rng = np.random.default_rng(91)
    cases = [(0.0, 1.0, 0.1, 5), (2500.0, 250.0, 0.1, 50), (2500.0, 250.0, 0.1, 49),
             (2375.0, 250.0, 0.1, 50), (100.0, 1000.0, 0.05, 10), (2000.0, 100.0, 0.5, 20),
             (2000.0, 100.0, 0.5, 15), (1e300, 1.0, 0.5, 10)]
    for _ in range(300):
        cases.append((float(rng.uniform(0.0, 30.0) * 400.0), float(rng.uniform(100.0, 900.0)),
                      float(rng.uniform(0.02, 0.6)), int(rng.integers(1, 300))))
    for ra, rmax, e, n in cases:
        want = orc.pick_groups(ra, rmax, e, n)
        if want == 0:
            with pytest.raises(lib.AladdinError):
                lib.aladdin_pick_groups(ra, rmax, e, n)
        else:
            assert lib.aladdin_pick_groups(ra, rmax, e, n) == want, (ra, rmax, e, n)
    for bad in ((-1.0, 1.0, 0.1, 5), (1.0, 0.0, 0.1, 5), (1.0, 1.0, 0.0, 5),
                (1.0, 1.0, 0.1, 0), (float("nan"), 1.0, 0.1, 5), (1.0, float("inf"), 0.1, 5)):
        with pytest.raises(lib.AladdinError):
            lib.aladdin_pick_groups(*bad)
