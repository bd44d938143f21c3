"""ctypes wrapper of the C oracle (``aladdin_oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by the tests, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``; never by the product package.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "aladdin_oracle.c")
LIB = os.path.join(HERE, "_build", "liboracle.so")
# The oracle's own tests build deliberately broken copies of the source (one
# planted mistake each) and check that a pin fails: ALADDIN_ORACLE_SRC names
# such a copy, built beside it.
if os.environ.get("ALADDIN_ORACLE_SRC"):
    SRC = os.path.abspath(os.environ["ALADDIN_ORACLE_SRC"])
    LIB = os.path.splitext(SRC)[0] + ".so"

FLAG_KV, FLAG_TTFT, FLAG_ONGOING, FLAG_NEW = 1, 2, 4, 8
FEASIBLE = 15
PHASE_MIXED, PHASE_DECODE = 0, 1
POLICY_BESTFIT, POLICY_JSQ, POLICY_PO2 = 0, 1, 2


def build(force=False):
    """Compile the oracle with gcc (fp contraction off, so every product and
    sum rounds on its own as written)."""
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    tmp = LIB + ".tmp%d" % os.getpid()
    subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-ffp-contract=off",
                           "-std=c11", "-o", tmp, SRC, "-lm"])
    os.replace(tmp, LIB)
    return LIB


class Params(C.Structure):
    _fields_ = [("k1", C.c_double), ("c1", C.c_double), ("k2", C.c_double),
                ("c2", C.c_double), ("c3", C.c_double), ("h", C.c_int64),
                ("j", C.c_int64), ("T_pre", C.c_double), ("T_dec", C.c_double),
                ("gamma", C.c_double), ("theta", C.c_double), ("K", C.c_int64),
                ("mode", C.c_int64), ("phase", C.c_int64), ("policy", C.c_int64),
                ("seed", C.c_uint64), ("rebalance", C.c_int64), ("groups", C.c_int64)]


class ClusterStruct(C.Structure):
    _fields_ = [("W", C.c_int32), ("cap", C.c_int32),
                ("M", C.c_void_p), ("scale", C.c_void_p), ("off", C.c_void_p),
                ("clock", C.c_void_p), ("n", C.c_void_p), ("inp", C.c_void_p),
                ("gen", C.c_void_p), ("pred", C.c_void_p), ("tdec", C.c_void_p),
                ("pend", C.c_void_p), ("wait", C.c_void_p), ("rid", C.c_void_p),
                ("real", C.c_void_p), ("le", C.c_void_p), ("be", C.c_void_p),
                ("repred", C.c_void_p)]


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        P = C.c_void_p
        _lib.orc_score.argtypes = [P, P, C.c_int32, P, P, P, P, P, P, P, P, P, P]
        _lib.orc_score_pairs.argtypes = [P, P, C.c_int64, P, P, P, P, P, P, P, P, P, P, P]
        _lib.orc_kv_curve.argtypes = [P, P, C.c_int, C.c_int32, C.c_int32, P]
        _lib.orc_kv_curve.restype = C.c_int32
        _lib.orc_place_round.argtypes = [P, P, C.c_int32, P, P, P, P, P]
        _lib.orc_advance.argtypes = [P, P, C.c_double, C.c_double, P, P, P, P, C.c_int64, P, P]
        _lib.orc_rebalance.argtypes = [P, P, C.c_int32, P, P, P, P, P, P, P, P, P]
        _lib.orc_splitmix64.argtypes = [C.c_uint64, C.c_uint64]
        _lib.orc_splitmix64.restype = C.c_uint64
        _lib.orc_po2_draw.argtypes = [C.c_uint64, C.c_int64, C.c_int, C.c_int32]
        _lib.orc_po2_draw.restype = C.c_int32
        _lib.orc_simulate.argtypes = [P, C.c_int32, C.c_int32, C.c_int64, C.c_double, C.c_int64,
                                      P, P, P, P, P, C.c_double, C.c_int32, C.c_int32, P]
        _lib.orc_min_workers.argtypes = [P, C.c_int32, P, P, P, C.c_int32, C.c_int64, P, P, P, P,
                                         P, C.c_double, C.c_int32, P]
        D = C.c_double
        _lib.orc_tp_config.argtypes = [D, D, D, D, D, C.c_int32, P, P]
        _lib.orc_trace_demand.argtypes = [P, C.c_int64, P, P, P, P]
        _lib.orc_max_throughput.argtypes = [P, C.c_int32, D, D, D, D]
        _lib.orc_max_throughput.restype = D
        _lib.orc_pick_config.argtypes = [P, C.c_int32, P, P, P, D, D, P]
        _lib.orc_pick_config.restype = C.c_int32
        _lib.orc_fit_workers.argtypes = [C.c_int32, P, P, D, P, P]
        _lib.orc_fit_workers.restype = C.c_int32
        _lib.orc_predict_workers.argtypes = [D, D, D]
        _lib.orc_predict_workers.restype = C.c_int64
        _lib.orc_pick_groups.argtypes = [D, D, D, C.c_int64]
        _lib.orc_pick_groups.restype = C.c_int64
        _lib.orc_capacity_norm.argtypes = [P, P, C.c_int]
        _lib.orc_capacity_norm.restype = C.c_double
        _lib.orc_order.argtypes = [P, P, P]
    return _lib


def make_params(d):
    return Params(float(d["k1"]), float(d["c1"]), float(d["k2"]), float(d["c2"]),
                  float(d["c3"]), int(d["h"]), int(d["j"]), float(d["T_pre"]),
                  float(d["T_dec"]), float(d["gamma"]), float(d["theta"]), int(d["K"]),
                  int(d.get("mode", 0)), int(d.get("phase", 0)), int(d.get("policy", 0)),
                  int(d.get("seed", 0)) & 0xFFFFFFFFFFFFFFFF, int(d.get("rebalance", 0)),
                  int(d.get("groups", 1)))


def _ptr(a):
    return None if a is None else a.ctypes.data


class Cluster:
    """Oracle cluster state in fixed-stride slots (worker w: slots
    [w*cap, w*cap + n[w]))."""

    def __init__(self, params, kv_capacity, lat_scale, cap, roff=None, req_in=None,
                 req_gen=None, req_pred=None, req_tdec=None, off=None):
        self.params = dict(params)
        W = int(len(kv_capacity))
        self.W, self.cap = W, int(cap)
        self.M = np.ascontiguousarray(kv_capacity, np.int64)
        self.scale = np.ascontiguousarray(lat_scale, np.float64)
        self.off = np.zeros(W) if off is None else np.ascontiguousarray(off, np.float64).copy()
        self.clock = np.zeros(W)
        self.n = np.zeros(W, np.int32)
        S = W * self.cap
        self.inp = np.zeros(S, np.int32)
        self.gen = np.zeros(S, np.int32)
        self.pred = np.ones(S, np.int32)
        self.tdec = np.zeros(S, np.float64)
        self.has_tdec = req_tdec is not None
        self.pend = np.zeros(S, np.uint8)
        self.wait = np.zeros(S, np.float64)
        self.rid = np.zeros(S, np.int64)
        self.real = None          # real output lengths [W*cap], or None (exact)
        self.le = np.zeros(W, np.int64)
        self.be = np.zeros(W, np.int32)
        self.repred = None        # re-prediction table [K+1], or None
        if roff is not None:
            for w in range(W):
                a, b = int(roff[w]), int(roff[w + 1])
                k = b - a
                if k > self.cap:
                    raise ValueError("worker %d has %d requests > cap %d" % (w, k, self.cap))
                s = w * self.cap
                self.n[w] = k
                self.inp[s:s + k] = req_in[a:b]
                self.gen[s:s + k] = req_gen[a:b]
                self.pred[s:s + k] = req_pred[a:b]
                if req_tdec is not None:
                    self.tdec[s:s + k] = req_tdec[a:b]
        self._p = make_params(self.params)

    @classmethod
    def from_workload(cls, wl, cap=None, tdec=None):
        return cls(wl.params, wl.kv_capacity, wl.lat_scale, cap or wl.b_cap, wl.roff,
                   wl.req_in, wl.req_gen, wl.req_pred, tdec)

    def struct(self, with_tdec=None):
        use_tdec = self.has_tdec if with_tdec is None else with_tdec
        return ClusterStruct(self.W, self.cap, _ptr(self.M), _ptr(self.scale), _ptr(self.off),
                             _ptr(self.clock), _ptr(self.n), _ptr(self.inp), _ptr(self.gen),
                             _ptr(self.pred), _ptr(self.tdec) if use_tdec else None,
                             _ptr(self.pend), _ptr(self.wait), _ptr(self.rid), _ptr(self.real),
                             _ptr(self.le), _ptr(self.be), _ptr(self.repred))

    def score(self, cin, cpred, cwait=None, want=("flags", "margin", "mscale", "kvpeak",
                                                    "tcand", "near", "argbest")):
        cin = np.ascontiguousarray(cin, np.int32)
        cpred = np.ascontiguousarray(cpred, np.int32)
        cw = None if cwait is None else np.ascontiguousarray(cwait, np.float64)
        Cn, W = len(cin), self.W
        out = {}
        shapes = dict(flags=(np.uint8, (Cn, W)), margin=(np.float64, (Cn, W)),
                      mscale=(np.float64, (Cn, W)), kvpeak=(np.int64, (Cn, W)),
                      tcand=(np.float64, (Cn, W)), near=(np.float64, (Cn, W)),
                      argbest=(np.int32, (Cn,)))
        for k in shapes:
            if k in want:
                dt, sh = shapes[k]
                out[k] = np.zeros(sh, dt)
        st = self.struct()
        rc = lib().orc_score(C.byref(self._p), C.byref(st), Cn, _ptr(cin), _ptr(cpred), _ptr(cw),
                             *[_ptr(out.get(k)) for k in ("flags", "margin", "mscale", "kvpeak",
                                                          "tcand", "near", "argbest")])
        if rc != 0:
            raise RuntimeError("orc_score failed: %d" % rc)
        return out

    def score_pairs(self, pc, pw, cin, cpred, cwait=None):
        pc = np.ascontiguousarray(pc, np.int32)
        pw = np.ascontiguousarray(pw, np.int32)
        cin = np.ascontiguousarray(cin, np.int32)
        cpred = np.ascontiguousarray(cpred, np.int32)
        cw = None if cwait is None else np.ascontiguousarray(cwait, np.float64)
        n = len(pc)
        out = dict(flags=np.zeros(n, np.uint8), margin=np.zeros(n), mscale=np.zeros(n),
                   kvpeak=np.zeros(n, np.int64), tcand=np.zeros(n), near=np.zeros(n))
        st = self.struct()
        rc = lib().orc_score_pairs(C.byref(self._p), C.byref(st), n, _ptr(pc), _ptr(pw),
                                   _ptr(cin), _ptr(cpred), _ptr(cw),
                                   *[_ptr(out[k]) for k in ("flags", "margin", "mscale", "kvpeak",
                                                            "tcand", "near")])
        if rc != 0:
            raise RuntimeError("orc_score_pairs failed: %d" % rc)
        return out

    def kv_curve(self, w, a_c, r_c):
        buf = np.zeros(int(self.params["K"]) * 2 + 8, np.int64)
        st = self.struct()
        S = lib().orc_kv_curve(C.byref(self._p), C.byref(st), int(w), int(a_c), int(r_c),
                               _ptr(buf))
        if S < 0:
            raise RuntimeError("orc_kv_curve failed")
        return buf[:S].copy()

    def capacity_norm(self, w):
        st = self.struct()
        return lib().orc_capacity_norm(C.byref(self._p), C.byref(st), int(w))

    def order(self):
        o = np.zeros(self.W, np.int32)
        st = self.struct()
        lib().orc_order(C.byref(self._p), C.byref(st), _ptr(o))
        return o

    def place_round(self, cin, cpred, cwait=None, crid=None, allow_capacity=False):
        """One placement round; with allow_capacity a full worker does not
        raise: returns (placements, True) instead."""
        cin = np.ascontiguousarray(cin, np.int32)
        cpred = np.ascontiguousarray(cpred, np.int32)
        cw = None if cwait is None else np.ascontiguousarray(cwait, np.float64)
        cr = None if crid is None else np.ascontiguousarray(crid, np.int64)
        pl = np.zeros(len(cin), np.int32)
        st = self.struct()
        rc = lib().orc_place_round(C.byref(self._p), C.byref(st), len(cin), _ptr(cin),
                                   _ptr(cpred), _ptr(cw), _ptr(cr), _ptr(pl))
        if rc == -2:
            if allow_capacity:
                return pl, True
            raise OverflowError("worker request capacity exceeded")
        if rc != 0:
            raise RuntimeError("orc_place_round failed: %d" % rc)
        return (pl, False) if allow_capacity else pl

    def commit(self, w, a, r, wait=0.0, rid=0):
        """Append request (prompt a, predicted output r) to worker w as a
        placement of the open round (Algorithm 1's commit step, in a pending
        state: gen 0, no decode history)."""
        w = int(w)
        if self.n[w] >= self.cap:
            raise OverflowError("worker request capacity exceeded")
        slot = w * self.cap + int(self.n[w])
        self.inp[slot] = a
        self.gen[slot] = 0
        self.pred[slot] = r
        self.tdec[slot] = 0.0
        self.pend[slot] = 1
        self.wait[slot] = wait
        self.rid[slot] = rid
        self.n[w] += 1

    def set_real(self, real, repred=None):
        """Real output lengths per slot (same layout as pred) and the
        re-prediction table: execution then follows the real lengths."""
        self.real = np.ascontiguousarray(real, np.int32).copy()
        self.repred = None if repred is None else np.ascontiguousarray(repred, np.int32)

    def rebalance(self, cin, cpred, cwait, placement, le, be, crid=None):
        """Algorithm 2 over a round's placements (updated in place); returns
        (moves, objective before, objective after)."""
        cin = np.ascontiguousarray(cin, np.int32)
        cpred = np.ascontiguousarray(cpred, np.int32)
        cw = None if cwait is None else np.ascontiguousarray(cwait, np.float64)
        le = np.ascontiguousarray(le, np.int64)
        be = np.ascontiguousarray(be, np.int32)
        mv = C.c_int32(0)
        obj = np.zeros(2)
        st = self.struct()
        cr = None if crid is None else np.ascontiguousarray(crid, np.int64)
        rc = lib().orc_rebalance(C.byref(self._p), C.byref(st), len(cin), _ptr(cin), _ptr(cpred),
                                 _ptr(cw), _ptr(cr), _ptr(placement), _ptr(le), _ptr(be),
                                 C.byref(mv), _ptr(obj))
        if rc != 0:
            raise RuntimeError("orc_rebalance failed: %d" % rc)
        return mv.value, obj[0], obj[1]

    def advance(self, t_now, dt, rec_cap=1 << 16, violations=None, events=None):
        """Execute every worker for dt ms; returns the realized records (request
        id, value, kind 0 TTFT / 1 ATGT). ``violations`` (int64[3], optional)
        accumulates realized TTFT, ATGT and KV-overflow violations."""
        rr = np.zeros(rec_cap, np.int64)
        rv = np.zeros(rec_cap)
        rk = np.zeros(rec_cap, np.uint8)
        nrec = C.c_int64(0)
        st = self.struct(with_tdec=True)
        self.has_tdec = True
        rc = lib().orc_advance(C.byref(self._p), C.byref(st), float(t_now), float(dt),
                               _ptr(rr), _ptr(rv), _ptr(rk), C.byref(nrec), rec_cap,
                               _ptr(violations), _ptr(events))
        if rc != 0:
            raise RuntimeError("orc_advance failed")
        k = min(nrec.value, rec_cap)
        return rr[:k], rv[:k], rk[:k]

    def worker_requests(self, w):
        s = w * self.cap
        k = int(self.n[w])
        return (self.inp[s:s + k].copy(), self.gen[s:s + k].copy(), self.pred[s:s + k].copy(),
                self.pend[s:s + k].copy())


def splitmix64(seed, n):
    """Output n (n >= 1) of the SplitMix64 stream seeded with ``seed``."""
    return int(lib().orc_splitmix64(int(seed) & 0xFFFFFFFFFFFFFFFF, int(n)))


def po2_draw(seed, rid, k, W):
    """Worker of draw k (0 or 1) of the power-of-two choice for request rid."""
    return int(lib().orc_po2_draw(int(seed) & 0xFFFFFFFFFFFFFFFF, int(rid), int(k), int(W)))


def _trace_real(trace):
    real = getattr(trace, "req_real", None)
    rep = getattr(trace, "repred", None)
    return (None if real is None else np.ascontiguousarray(real, np.int32),
            None if rep is None else np.ascontiguousarray(rep, np.int32))


def simulate(params, N, cap, M, scale, trace, H, stop_at_fail=True, drain=False):
    out = np.zeros(10)
    p = make_params(params)
    t = np.ascontiguousarray(trace.t_arr, np.float64)
    ri = np.ascontiguousarray(trace.req_in, np.int32)
    rp = np.ascontiguousarray(trace.req_pred, np.int32)
    rr, rep = _trace_real(trace)
    rc = lib().orc_simulate(C.byref(p), int(N), int(cap), int(M), float(scale), len(t), _ptr(t),
                            _ptr(ri), _ptr(rp), _ptr(rr), _ptr(rep), float(H), int(stop_at_fail),
                            int(drain), _ptr(out))
    if rc == -2:
        raise OverflowError("worker request capacity exceeded")
    if rc != 0:
        raise RuntimeError("orc_simulate failed: %d" % rc)
    return dict(failed=int(out[0]), placed=int(out[1]), heartbeats=int(out[2]),
                max_ttft=out[3], max_atgt=out[4], violations=int(out[6]),
                repredictions=int(out[7]), early_finishes=int(out[8]), moved=int(out[9]))


def min_workers(params, gpus, M, scale, cap, trace, H, n_max):
    p = make_params(params)
    g = np.ascontiguousarray(gpus, np.int32)
    Mv = np.ascontiguousarray(M, np.int64)
    sv = np.ascontiguousarray(scale, np.float64)
    t = np.ascontiguousarray(trace.t_arr, np.float64)
    ri = np.ascontiguousarray(trace.req_in, np.int32)
    rp = np.ascontiguousarray(trace.req_pred, np.int32)
    n_out = np.zeros(len(g), np.int32)
    rr, rep = _trace_real(trace)
    rc = lib().orc_min_workers(C.byref(p), len(g), _ptr(g), _ptr(Mv), _ptr(sv), int(cap), len(t),
                               _ptr(t), _ptr(ri), _ptr(rp), _ptr(rr), _ptr(rep), float(H),
                               int(n_max), _ptr(n_out))
    if rc != 0:
        raise RuntimeError("orc_min_workers failed: %d" % rc)
    return n_out


# ---------------------------------------------------------------------------
# Worker configuration (Sec. 4.1) and the worker-count model (Sec. 5.2).

def tp_config(k4, c4, kc, m_gpu, m_model, g):
    """(KV capacity, latency multiplier) of a worker of g GPUs."""
    M = C.c_double()
    sc = C.c_double()
    lib().orc_tp_config(float(k4), float(c4), float(kc), float(m_gpu), float(m_model), int(g),
                        C.byref(M), C.byref(sc))
    return M.value, sc.value


def trace_demand(params, req_in, req_pred):
    """(m_r, l_ave): iteration-averaged KV demand and context of a request."""
    p = make_params(params)
    ri = np.ascontiguousarray(req_in, np.int32)
    rp = np.ascontiguousarray(req_pred, np.int32)
    m = C.c_double()
    l = C.c_double()
    lib().orc_trace_demand(C.byref(p), len(ri), _ptr(ri), _ptr(rp), C.byref(m), C.byref(l))
    return m.value, l.value


def max_throughput(params, g, M, scale, m_r, l_ave):
    p = make_params(params)
    return lib().orc_max_throughput(C.byref(p), int(g), float(M), float(scale), float(m_r),
                                    float(l_ave))


def pick_config(params, gpus, M, scale, m_r, l_ave):
    """(best option, T_max per option)."""
    p = make_params(params)
    g = np.ascontiguousarray(gpus, np.int32)
    Mv = np.ascontiguousarray(M, np.float64)
    sv = np.ascontiguousarray(scale, np.float64)
    t = np.zeros(len(g))
    best = lib().orc_pick_config(C.byref(p), len(g), _ptr(g), _ptr(Mv), _ptr(sv), float(m_r),
                                 float(l_ave), _ptr(t))
    return int(best), t


def fit_workers(rates, nw, R=0.0):
    """(k5, c5, points used) of Eq. total_worker_pre."""
    r = np.ascontiguousarray(rates, np.float64)
    n = np.ascontiguousarray(nw, np.int32)
    k5 = C.c_double()
    c5 = C.c_double()
    used = lib().orc_fit_workers(len(r), _ptr(r), _ptr(n), float(R), C.byref(k5), C.byref(c5))
    return k5.value, c5.value, int(used)


def predict_workers(k5, c5, rate):
    return int(lib().orc_predict_workers(float(k5), float(c5), float(rate)))


def pick_groups(rate_a, rate_max, e, n_workers):
    """Appendix A, Eq. group_arrival_limit: the fewest scheduling groups whose
    per-group arrival rate stays within rate_max and that keep at least
    1 / (2e) workers each; 0 if none."""
    return int(lib().orc_pick_groups(float(rate_a), float(rate_max), float(e), int(n_workers)))
