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
    # 5 doubles, h and j, 4 doubles, K b_cap mode phase policy, pad, seed
    assert ctypes.sizeof(lib.aladdin_params) == 5 * 8 + 2 * 4 + 4 * 8 + 5 * 4 + 4 + 8
    assert lib.aladdin_params.seed.offset == 104
    assert ctypes.sizeof(lib.aladdin_worker_cfg) == 24
    assert ctypes.sizeof(lib.aladdin_trace) == 32


@pytest.mark.parametrize("bad", [dict(k1=0.0), dict(k2=-1.0), dict(T_dec=5.0), dict(theta=0.0),
                                 dict(theta=1.5), dict(K=1), dict(K=70000), dict(h=0),
                                 dict(j=-1), dict(c1=float("nan")), dict(T_pre=0.0),
                                 dict(phase=2), dict(policy=3), dict(policy=-1)])
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
