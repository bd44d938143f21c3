"""Python binding of the C ABI in ``include/aladdin.h`` (ctypes).

Argument marshalling only: every function forwards to the function of the
same name in ``libaladdin.so`` and every computation runs in its CUDA kernels.
Arrays may be numpy arrays (host memory) or torch tensors (host or device);
the library decides per pointer whether to copy. Importing this module raises
if the compiled library is missing; there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libaladdin.so")

OK = 0
ERR_ARG, ERR_CAPACITY, ERR_CUDA, ERR_TIMEOUT, ERR_NOMEM, ERR_STATE = -1, -2, -3, -4, -5, -6
ERR_SCRATCH = -7
MODE_EXACT, MODE_APPROX = 0, 1
PHASE_MIXED, PHASE_DECODE = 0, 1
POLICY_BESTFIT, POLICY_JSQ, POLICY_PO2 = 0, 1, 2
ADVANCE_STATS = 9     # doubles written by aladdin_cluster_advance
SIMULATE_OUT = 9      # doubles written by aladdin_simulate
NOALLOC_MAX_CAND = 32768
FLAG_KV, FLAG_TTFT, FLAG_ONGOING, FLAG_NEW, FEASIBLE, FLAG_INVALID = 1, 2, 4, 8, 15, 128
NONE, INVALID = -1, -2

_NAMES = {ERR_ARG: "ALADDIN_ERR_ARG", ERR_CAPACITY: "ALADDIN_ERR_CAPACITY",
          ERR_CUDA: "ALADDIN_ERR_CUDA", ERR_TIMEOUT: "ALADDIN_ERR_TIMEOUT",
          ERR_NOMEM: "ALADDIN_ERR_NOMEM", ERR_STATE: "ALADDIN_ERR_STATE",
          ERR_SCRATCH: "ALADDIN_ERR_SCRATCH"}


class AladdinError(RuntimeError):
    def __init__(self, code, where):
        super().__init__("%s failed: %s (%d)" % (where, _NAMES.get(code, "?"), code))
        self.code = code


if not os.path.exists(LIB_PATH):
    raise ImportError("libaladdin.so is not built (%s); run __graft_entry__.build()" % LIB_PATH)

_lib = C.CDLL(LIB_PATH)


class aladdin_params(C.Structure):
    _fields_ = [("k1", C.c_double), ("c1", C.c_double), ("k2", C.c_double), ("c2", C.c_double),
                ("c3", C.c_double), ("h", C.c_int32), ("j", C.c_int32), ("T_pre", C.c_double),
                ("T_dec", C.c_double), ("gamma", C.c_double), ("theta", C.c_double),
                ("K", C.c_int32), ("b_cap", C.c_int32), ("mode", C.c_int32),
                ("phase", C.c_int32), ("policy", C.c_int32), ("seed", C.c_uint64),
                ("rebalance", C.c_int32), ("groups", C.c_int32)]


class aladdin_worker_cfg(C.Structure):
    _fields_ = [("gpus", C.c_int32), ("kv_capacity", C.c_int64), ("lat_scale", C.c_double)]


class aladdin_tp_model(C.Structure):
    _fields_ = [("k4", C.c_double), ("c4", C.c_double), ("kc", C.c_double),
                ("m_gpu", C.c_double), ("m_model", C.c_double)]


class aladdin_trace(C.Structure):
    _fields_ = [("n", C.c_int64), ("t_arr_ms", C.c_void_p), ("in_", C.c_void_p),
                ("pred", C.c_void_p), ("real", C.c_void_p), ("repred", C.c_void_p)]


_P = C.c_void_p
_sig = {
    "aladdin_cluster_create": [_P, C.c_int32, _P, _P, _P, _P, _P, _P, _P, _P],
    "aladdin_cluster_destroy": [_P],
    "aladdin_cluster_load": [_P, _P, _P, _P, _P, _P],
    "aladdin_score": [_P, C.c_int32, _P, _P, _P, _P, _P, _P],
    "aladdin_score_detail": [_P, C.c_int32, _P, _P, _P, _P, _P, _P, _P, _P],
    "aladdin_score_noalloc": [_P, C.c_int32, _P, _P, _P, _P, _P, _P],
    "aladdin_place_round": [_P, C.c_int32, _P, _P, _P, _P],
    "aladdin_cluster_advance": [_P, C.c_double, _P],
    "aladdin_cluster_state": [_P, _P, _P, _P, _P, _P],
    "aladdin_cluster_status": [_P],
    "aladdin_cluster_test_waits": [_P, C.c_int64, C.c_int64, C.c_int32],
    "aladdin_cluster_test_round": [_P, C.c_int32, C.c_int32],
    "aladdin_cluster_timing": [_P, C.c_int32, _P, _P],
    "aladdin_min_workers": [_P, C.c_int32, _P, _P, C.c_double, C.c_int32, _P, _P, _P, _P],
    "aladdin_simulate": [_P, _P, C.c_int32, _P, C.c_double, C.c_int32, C.c_int32, _P, _P],
    "aladdin_tp_configs": [_P, C.c_int32, _P, _P],
    "aladdin_trace_demand": [_P, _P, _P, _P, _P],
    "aladdin_pick_config": [_P, C.c_int32, _P, _P, _P, _P, _P],
    "aladdin_fit_workers": [_P, _P, C.c_int32, _P, _P, C.c_double, C.c_double, C.c_int32, _P, _P,
                            _P, _P],
    "aladdin_predict_workers": [C.c_double, C.c_double, C.c_double, _P],
    "aladdin_pick_groups": [C.c_double, C.c_double, C.c_double, C.c_int64, _P],
    "aladdin_rebalance": [_P, C.c_int32, _P, _P, _P, _P, _P, _P, _P, _P],
    "aladdin_cluster_save": [_P, _P, _P],
    "aladdin_cluster_load_score": [_P, _P, _P, _P, _P, _P, C.c_int32, _P, _P, _P, _P, _P, _P],
    "aladdin_cluster_restore": [_P, _P, C.c_int64],
}
for _n, _a in _sig.items():
    f = getattr(_lib, _n)
    f.argtypes = _a
    f.restype = C.c_int


def exported_symbols():
    return list(_sig)


def _ptr(x):
    """Address of a numpy array or torch tensor (None stays None)."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("array must be C-contiguous")
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return x.data_ptr()
    raise TypeError("expected a numpy array or a torch tensor, got %r" % type(x))


def _check(rc, where):
    if rc != OK:
        raise AladdinError(rc, where)


def current_stream():
    """The current torch CUDA stream handle, or None (legacy default stream)."""
    try:
        import torch
        if torch.cuda.is_available() and torch.cuda.is_initialized():
            return torch.cuda.current_stream().cuda_stream
    except Exception:
        pass
    return None


def make_params(d, b_cap):
    return aladdin_params(float(d["k1"]), float(d["c1"]), float(d["k2"]), float(d["c2"]),
                          float(d["c3"]), int(d["h"]), int(d["j"]), float(d["T_pre"]),
                          float(d["T_dec"]), float(d["gamma"]), float(d["theta"]), int(d["K"]),
                          int(b_cap), int(d.get("mode", MODE_EXACT)),
                          int(d.get("phase", PHASE_MIXED)), int(d.get("policy", POLICY_BESTFIT)),
                          int(d.get("seed", 0)) & 0xFFFFFFFFFFFFFFFF, int(d.get("rebalance", 0)),
                          int(d.get("groups", 1)))


def make_cfgs(gpus, kv_capacity, lat_scale):
    n = len(gpus)
    arr = (aladdin_worker_cfg * n)()
    for i in range(n):
        arr[i].gpus = int(gpus[i])
        arr[i].kv_capacity = int(kv_capacity[i])
        arr[i].lat_scale = float(lat_scale[i])
    return arr


def make_trace(t_arr, req_in, req_pred, req_real=None, repred=None):
    """An aladdin_trace over host arrays (kept alive by the returned object);
    req_real / repred: prediction errors (see aladdin_trace)."""
    t = np.ascontiguousarray(t_arr, np.float64)
    i = np.ascontiguousarray(req_in, np.int32)
    p = np.ascontiguousarray(req_pred, np.int32)
    r = None if req_real is None else np.ascontiguousarray(req_real, np.int32)
    q = None if repred is None else np.ascontiguousarray(repred, np.int32)
    tr = aladdin_trace(len(t), t.ctypes.data, i.ctypes.data, p.ctypes.data,
                       None if r is None else r.ctypes.data, None if q is None else q.ctypes.data)
    tr._keep = (t, i, p, r, q)
    return tr


def trace_of(tr):
    """make_trace of a synth.Trace (with its prediction errors, if any)."""
    return make_trace(tr.t_arr, tr.req_in, tr.req_pred, getattr(tr, "req_real", None),
                      getattr(tr, "repred", None))


# ---------------------------------------------------------------------------
# The C ABI, one function each.

def aladdin_cluster_create(params, cfgs, req_off, req_in, req_gen, req_pred, tdec_ms=None,
                           stream=None):
    h = C.c_void_p()
    rc = _lib.aladdin_cluster_create(C.byref(params), len(cfgs), C.cast(cfgs, C.c_void_p),
                                     _ptr(req_off), _ptr(req_in), _ptr(req_gen), _ptr(req_pred),
                                     _ptr(tdec_ms), stream, C.byref(h))
    _check(rc, "aladdin_cluster_create")
    return h


def aladdin_cluster_destroy(cl):
    _check(_lib.aladdin_cluster_destroy(cl), "aladdin_cluster_destroy")


def aladdin_cluster_load(cl, req_off, req_in, req_gen, req_pred, tdec_ms=None):
    _check(_lib.aladdin_cluster_load(cl, _ptr(req_off), _ptr(req_in), _ptr(req_gen),
                                     _ptr(req_pred), _ptr(tdec_ms)), "aladdin_cluster_load")


def aladdin_score(cl, n_cand, cand_in, cand_pred, wait_ms, flags, margin, argbest):
    _check(_lib.aladdin_score(cl, int(n_cand), _ptr(cand_in), _ptr(cand_pred), _ptr(wait_ms),
                              _ptr(flags), _ptr(margin), _ptr(argbest)), "aladdin_score")


def aladdin_cluster_load_score(cl, req_off, req_in, req_gen, req_pred, tdec_ms, n_cand, cand_in,
                               cand_pred, wait_ms, flags, margin, argbest):
    """aladdin_cluster_load then aladdin_score in one call (overlapped on the
    device when every array is device memory)."""
    _check(_lib.aladdin_cluster_load_score(cl, _ptr(req_off), _ptr(req_in), _ptr(req_gen),
                                           _ptr(req_pred), _ptr(tdec_ms), int(n_cand),
                                           _ptr(cand_in), _ptr(cand_pred), _ptr(wait_ms),
                                           _ptr(flags), _ptr(margin), _ptr(argbest)),
           "aladdin_cluster_load_score")


def aladdin_score_noalloc(cl, n_cand, cand_in, cand_pred, wait_ms, flags, margin, argbest):
    """aladdin_score without any allocation (device tensors only)."""
    _check(_lib.aladdin_score_noalloc(cl, int(n_cand), _ptr(cand_in), _ptr(cand_pred),
                                      _ptr(wait_ms), _ptr(flags), _ptr(margin), _ptr(argbest)),
           "aladdin_score_noalloc")


def aladdin_score_detail(cl, n_cand, cand_in, cand_pred, wait_ms, flags, margin, argbest,
                         kv_peak, t_cand_ms):
    _check(_lib.aladdin_score_detail(cl, int(n_cand), _ptr(cand_in), _ptr(cand_pred),
                                     _ptr(wait_ms), _ptr(flags), _ptr(margin), _ptr(argbest),
                                     _ptr(kv_peak), _ptr(t_cand_ms)), "aladdin_score_detail")


def aladdin_place_round(cl, n_cand, cand_in, cand_pred, wait_ms, placement):
    _check(_lib.aladdin_place_round(cl, int(n_cand), _ptr(cand_in), _ptr(cand_pred),
                                    _ptr(wait_ms), _ptr(placement)), "aladdin_place_round")


def aladdin_rebalance(cl, n_cand, cand_in, cand_pred, wait_ms, placement, le, be):
    """Algorithm 2 over a placed round; placement is updated in place.
    Returns (moves, summed distance before, after)."""
    mv = C.c_int32(0)
    obj = np.zeros(2)
    _check(_lib.aladdin_rebalance(cl, int(n_cand), _ptr(cand_in), _ptr(cand_pred), _ptr(wait_ms),
                                  _ptr(placement), _ptr(le), _ptr(be), C.byref(mv), _ptr(obj)),
           "aladdin_rebalance")
    return mv.value, obj[0], obj[1]


def aladdin_cluster_save(cl):
    """The cluster's checkpoint as bytes."""
    n = C.c_int64(0)
    _check(_lib.aladdin_cluster_save(cl, None, C.byref(n)), "aladdin_cluster_save")
    buf = np.zeros(n.value, np.uint8)
    _check(_lib.aladdin_cluster_save(cl, buf.ctypes.data, C.byref(n)), "aladdin_cluster_save")
    return buf.tobytes()


def aladdin_cluster_restore(cl, blob):
    buf = np.frombuffer(blob, np.uint8)
    _check(_lib.aladdin_cluster_restore(cl, buf.ctypes.data, len(buf)), "aladdin_cluster_restore")


def aladdin_cluster_advance(cl, dt_ms, stats=None):
    _check(_lib.aladdin_cluster_advance(cl, float(dt_ms), _ptr(stats)), "aladdin_cluster_advance")


def aladdin_cluster_state(cl, n, req_in, req_gen, req_pred, pending):
    _check(_lib.aladdin_cluster_state(cl, _ptr(n), _ptr(req_in), _ptr(req_gen), _ptr(req_pred),
                                      _ptr(pending)), "aladdin_cluster_state")


def aladdin_cluster_status(cl):
    return _lib.aladdin_cluster_status(cl)


def aladdin_cluster_test_waits(cl, grid_polls, mbar_polls, run_out):
    _check(_lib.aladdin_cluster_test_waits(cl, int(grid_polls), int(mbar_polls), int(run_out)),
           "aladdin_cluster_test_waits")


def aladdin_cluster_test_round(cl, max_slots, chunk):
    _check(_lib.aladdin_cluster_test_round(cl, int(max_slots), int(chunk)),
           "aladdin_cluster_test_round")


def aladdin_cluster_timing(cl, enable):
    """Returns (summed scoring-kernel ms, launches) since the previous call."""
    ms = C.c_double(0.0)
    n = C.c_int64(0)
    _check(_lib.aladdin_cluster_timing(cl, int(enable), C.byref(ms), C.byref(n)),
           "aladdin_cluster_timing")
    return ms.value, n.value


def aladdin_min_workers(params, options, trace, heartbeat_ms, n_max, n_workers, stream=None):
    best = C.c_int32(-1)
    total = C.c_int64(-1)
    rc = _lib.aladdin_min_workers(C.byref(params), len(options), C.cast(options, C.c_void_p),
                                  C.byref(trace), float(heartbeat_ms), int(n_max), stream,
                                  _ptr(n_workers), C.byref(best), C.byref(total))
    _check(rc, "aladdin_min_workers")
    return best.value, total.value


def aladdin_simulate(params, cfg, n, trace, heartbeat_ms, stop_at_fail, drain, out, stream=None):
    _check(_lib.aladdin_simulate(C.byref(params), C.byref(cfg), int(n), C.byref(trace),
                                 float(heartbeat_ms), int(stop_at_fail), int(drain), stream,
                                 _ptr(out)), "aladdin_simulate")


def aladdin_tp_configs(tp, gpus):
    """Worker configurations (an aladdin_worker_cfg array) for the GPU counts."""
    g = np.ascontiguousarray(gpus, np.int32)
    out = (aladdin_worker_cfg * len(g))()
    _check(_lib.aladdin_tp_configs(C.byref(tp), len(g), _ptr(g), C.cast(out, C.c_void_p)),
           "aladdin_tp_configs")
    return out


def aladdin_trace_demand(params, trace, stream=None):
    """(m_r, l_ave) of the trace."""
    m = C.c_double()
    l = C.c_double()
    _check(_lib.aladdin_trace_demand(C.byref(params), C.byref(trace), stream, C.byref(m),
                                     C.byref(l)), "aladdin_trace_demand")
    return m.value, l.value


def aladdin_pick_config(params, options, trace, t_max=None, stream=None):
    """Best option (index into options); t_max (float64[n], optional) receives
    each option's Eq. max throughput."""
    best = C.c_int32(-1)
    _check(_lib.aladdin_pick_config(C.byref(params), len(options), C.cast(options, C.c_void_p),
                                    C.byref(trace), stream, _ptr(t_max), C.byref(best)),
           "aladdin_pick_config")
    return best.value


def aladdin_fit_workers(params, cfg, traces, rates, R, heartbeat_ms, n_max, n_workers,
                        stream=None):
    """(k5, c5); n_workers (int32[len(traces)]) receives each search's count."""
    arr = (aladdin_trace * len(traces))(*traces)
    r = np.ascontiguousarray(rates, np.float64)
    k5 = C.c_double()
    c5 = C.c_double()
    _check(_lib.aladdin_fit_workers(C.byref(params), C.byref(cfg), len(traces),
                                    C.cast(arr, C.c_void_p), _ptr(r), float(R),
                                    float(heartbeat_ms), int(n_max), stream, _ptr(n_workers),
                                    C.byref(k5), C.byref(c5)), "aladdin_fit_workers")
    return k5.value, c5.value


def aladdin_predict_workers(k5, c5, rate):
    n = C.c_int64()
    _check(_lib.aladdin_predict_workers(float(k5), float(c5), float(rate), C.byref(n)),
           "aladdin_predict_workers")
    return n.value


def aladdin_pick_groups(rate_a, rate_max, e, n_workers):
    g = C.c_int64()
    _check(_lib.aladdin_pick_groups(float(rate_a), float(rate_max), float(e), int(n_workers),
                                    C.byref(g)), "aladdin_pick_groups")
    return g.value


# ---------------------------------------------------------------------------
# Convenience wrapper owning a cluster handle.

class Cluster:
    def __init__(self, params_dict, gpus, kv_capacity, lat_scale, b_cap, req_off, req_in,
                 req_gen, req_pred, tdec_ms=None, stream=None):
        self.params = make_params(params_dict, b_cap)
        self.cfgs = make_cfgs(gpus, kv_capacity, lat_scale)
        self.W = len(gpus)
        self.b_cap = int(b_cap)
        self.stream = current_stream() if stream is None else stream
        self.handle = aladdin_cluster_create(self.params, self.cfgs, req_off, req_in, req_gen,
                                             req_pred, tdec_ms, self.stream)

    @classmethod
    def from_workload(cls, wl, b_cap=None, tdec_ms=None, stream=None):
        return cls(wl.params, wl.gpus, wl.kv_capacity, wl.lat_scale, b_cap or wl.b_cap, wl.roff,
                   wl.req_in, wl.req_gen, wl.req_pred, tdec_ms, stream)

    def close(self):
        if getattr(self, "handle", None):
            aladdin_cluster_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    def load(self, req_off, req_in, req_gen, req_pred, tdec_ms=None):
        aladdin_cluster_load(self.handle, req_off, req_in, req_gen, req_pred, tdec_ms)

    def score(self, cand_in, cand_pred, wait_ms=None, detail=False):
        """Host convenience: returns numpy outputs."""
        cin = np.ascontiguousarray(cand_in, np.int32)
        cpr = np.ascontiguousarray(cand_pred, np.int32)
        cw = None if wait_ms is None else np.ascontiguousarray(wait_ms, np.float32)
        n = len(cin)
        flags = np.zeros((n, self.W), np.uint8)
        margin = np.zeros((n, self.W), np.float32)
        arg = np.zeros(n, np.int32)
        out = dict(flags=flags, margin=margin, argbest=arg)
        if detail:
            out["kvpeak"] = np.zeros((n, self.W), np.int64)
            out["tcand"] = np.zeros((n, self.W), np.float32)
            aladdin_score_detail(self.handle, n, cin, cpr, cw, flags, margin, arg, out["kvpeak"],
                                 out["tcand"])
        else:
            aladdin_score(self.handle, n, cin, cpr, cw, flags, margin, arg)
        return out

    def place_round(self, cand_in, cand_pred, wait_ms=None):
        cin = np.ascontiguousarray(cand_in, np.int32)
        cpr = np.ascontiguousarray(cand_pred, np.int32)
        cw = None if wait_ms is None else np.ascontiguousarray(wait_ms, np.float32)
        pl = np.zeros(len(cin), np.int32)
        aladdin_place_round(self.handle, len(cin), cin, cpr, cw, pl)
        return pl

    def rebalance(self, cand_in, cand_pred, wait_ms, placement, le, be):
        """Host convenience for aladdin_rebalance (placement: int32 numpy array,
        updated in place)."""
        cin = np.ascontiguousarray(cand_in, np.int32)
        cpr = np.ascontiguousarray(cand_pred, np.int32)
        cw = None if wait_ms is None else np.ascontiguousarray(wait_ms, np.float32)
        return aladdin_rebalance(self.handle, len(cin), cin, cpr, cw, placement,
                                 np.ascontiguousarray(le, np.int64),
                                 np.ascontiguousarray(be, np.int32))

    def advance(self, dt_ms):
        st = np.zeros(ADVANCE_STATS)
        aladdin_cluster_advance(self.handle, dt_ms, st)
        return st

    def state(self):
        n = np.zeros(self.W, np.int32)
        S = self.W * self.b_cap
        i, g, p = np.zeros(S, np.int32), np.zeros(S, np.int32), np.zeros(S, np.int32)
        pe = np.zeros(S, np.uint8)
        aladdin_cluster_state(self.handle, n, i, g, p, pe)
        return n, i, g, p, pe

    def status(self):
        return aladdin_cluster_status(self.handle)
