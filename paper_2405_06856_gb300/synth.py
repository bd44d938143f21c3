"""Seeded synthetic workloads shaped like the paper's serving scenarios.

This module only draws random numbers: it holds none of the scheduler's
arithmetic (no KV, latency or feasibility computation). Both the CUDA path and
the CPU oracle read what it produces.

The paper's own lengths come from ShareGPT prompts and Llama2 outputs (Sec. 6.1,
Workload), which are not available here; lognormal lengths with the means,
spreads and clips below stand in for them.

Recipe (all integer lengths are ``int32``):
  * ``lognormal(mean m, sigma s)``: draw from a lognormal whose underlying normal
    has mu = ln m - s^2/2 (so the unclipped mean is m), round to nearest, clip.
  * ongoing requests: input_len ~ lognormal, predicted_out_len ~ lognormal,
    generated ~ uniform integer in [0, predicted_out_len).
  * candidates: input_len and predicted_out_len from the same laws; the wait
    since arrival is uniform in [0, wait_max) ms.
  * worker configs: GPUs per worker from a cyclic list, KV capacity
    proportional to the GPU count, latency coefficients scaled by 1/sqrt(GPUs).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

# Latency model of the workload configs: decode iteration 8 ms + 0.05 ms per
# request + 2e-4 ms per KV token; prefill 10 ms + 0.1 ms per 100 input tokens;
# TTFT SLO 1 s, per-token SLO 50 ms; KV counted in tokens (h = 1, j = 0).
BASE_PARAMS = dict(
    k1=0.001, c1=10.0,            # prefill: ms per input token, ms
    k2=2e-4, c2=0.05, c3=8.0,     # decode: ms per KV token, ms per request, ms
    h=1, j=0,                     # KV slots per context token, per request
    T_pre=1000.0, T_dec=50.0,     # TTFT SLO (ms), per-token decode SLO (ms)
    gamma=0.5, theta=1.0,         # capacity_norm weight, SLO scaling knob
    K=8192,                       # sequence limit: input + output tokens
)


def lognormal_lengths(rng, mean, sigma, lo, hi, size):
    mu = math.log(mean) - 0.5 * sigma * sigma
    x = rng.lognormal(mu, sigma, size)
    return np.clip(np.rint(x), lo, hi).astype(np.int32)


@dataclasses.dataclass
class Workload:
    """A cluster state plus a batch of candidate queries.

    Requests of worker ``w`` are ``[roff[w], roff[w+1])`` of the flat arrays.
    """
    name: str
    params: dict
    gpus: np.ndarray        # int32 [W]
    kv_capacity: np.ndarray  # int64 [W], tokens
    lat_scale: np.ndarray   # float32 [W], multiplies every latency coefficient
    roff: np.ndarray        # int32 [W+1]
    req_in: np.ndarray      # int32 [N]
    req_gen: np.ndarray     # int32 [N]
    req_pred: np.ndarray    # int32 [N]
    cand_in: np.ndarray     # int32 [C]
    cand_pred: np.ndarray   # int32 [C]
    cand_wait: np.ndarray   # float32 [C], ms since arrival
    b_cap: int              # per-worker request capacity of the tables

    @property
    def n_workers(self):
        return int(self.gpus.shape[0])

    @property
    def n_cand(self):
        return int(self.cand_in.shape[0])


def make_cluster(name, seed, n_workers, per_worker, kv_per_gpu, n_cand,
                 in_law=(512.0, 0.8, 16, 2048), out_law=(256.0, 0.9, 8, 1024),
                 gpus_cycle=(1,), wait_max=100.0, params=None, b_cap=None,
                 per_worker_random=False):
    """Draw a cluster and a candidate batch.

    ``per_worker_random``: the number of ongoing requests of each worker is
    uniform in [0, per_worker] instead of exactly ``per_worker`` (a mixed-load
    variant, so that parity cases contain light, heavy and empty workers).
    """
    rng = np.random.default_rng(seed)
    prm = dict(BASE_PARAMS)
    if params:
        prm.update(params)
    W = int(n_workers)
    gpus = np.array([gpus_cycle[i % len(gpus_cycle)] for i in range(W)], np.int32)
    kv = (gpus.astype(np.int64) * int(kv_per_gpu)).astype(np.int64)
    scale = (1.0 / np.sqrt(gpus.astype(np.float64))).astype(np.float32)
    if per_worker_random:
        counts = rng.integers(0, per_worker + 1, W).astype(np.int32)
    else:
        counts = np.full(W, per_worker, np.int32)
    roff = np.zeros(W + 1, np.int32)
    np.cumsum(counts, out=roff[1:])
    N = int(roff[-1])
    im, isg, ilo, ihi = in_law
    om, osg, olo, ohi = out_law
    req_in = lognormal_lengths(rng, im, isg, ilo, ihi, N)
    req_pred = lognormal_lengths(rng, om, osg, olo, ohi, N)
    req_gen = rng.integers(0, req_pred).astype(np.int32)
    cand_in = lognormal_lengths(rng, im, isg, ilo, ihi, n_cand)
    cand_pred = lognormal_lengths(rng, om, osg, olo, ohi, n_cand)
    cand_wait = (rng.random(n_cand) * wait_max).astype(np.float32)
    if b_cap is None:
        b_cap = max(32, 1 << int(math.ceil(math.log2(max(1, 2 * per_worker)))))
    return Workload(name, prm, gpus, kv, scale, roff, req_in, req_gen, req_pred,
                    cand_in, cand_pred, cand_wait, int(b_cap))


HEAVY_OUT = (256.0, 1.2, 8, 4096)


def config(name, **over):
    """The workload configurations, by name.

    tiny     16 workers, KV 16,384, 32 requests each, 64 candidates, seed 0.
    w256     256 workers, KV 65,536, 64 requests each, 2,048 candidates, seed 1.
    w4096    4,096 workers, KV 131,072, 128 requests each, 32,768 candidates,
             output sigma 1.2 clipped at 4,096, seed 2.
    w16384   16,384 workers of 1/2/4/8 GPUs (KV 131,072 per GPU, latency
             coefficients x 1/sqrt(GPUs)), 256 requests each (1,024 request
             slots: an 8-GPU worker meets its SLOs with several hundred),
             131,072 candidates, output law as w4096, seed 3.
    w4096_mixed  w4096's sizes and draws (seed 2) with tighter limits, so that
             about half of the pairs are feasible and every constraint group
             binds somewhere: KV 90,000 tokens, TTFT 95 ms, ATGT 30 ms; pair
             it with decode_history(wl, 18.0, 26.0, MIXED_HISTORY_SEED).
    """
    if name == "tiny":
        kw = dict(seed=0, n_workers=16, per_worker=32, kv_per_gpu=16384, n_cand=64)
    elif name == "w256":
        kw = dict(seed=1, n_workers=256, per_worker=64, kv_per_gpu=65536, n_cand=2048)
    elif name == "w4096":
        kw = dict(seed=2, n_workers=4096, per_worker=128, kv_per_gpu=131072,
                  n_cand=32768, out_law=HEAVY_OUT)
    elif name == "w4096_mixed":
        kw = dict(seed=2, n_workers=4096, per_worker=128, kv_per_gpu=90000,
                  n_cand=32768, out_law=HEAVY_OUT, params=dict(T_pre=95.0, T_dec=30.0))
    elif name == "w16384":
        kw = dict(seed=3, n_workers=16384, per_worker=256, kv_per_gpu=131072,
                  n_cand=131072, out_law=HEAVY_OUT, gpus_cycle=(1, 2, 4, 8),
                  b_cap=1024)
    else:
        raise KeyError(name)
    kw.update(over)
    return make_cluster(name, **kw)


MIXED_HISTORY_SEED = 9


def decode_history(wl, lo_ms, hi_ms, seed):
    """Decode time so far (Table 1's t^dec, ms) of every ongoing request: its
    generated tokens times a per-request rate drawn uniform in [lo_ms, hi_ms)
    ms a token; float32, as the C ABI takes it."""
    rng = np.random.default_rng(seed)
    rate = rng.uniform(lo_ms, hi_ms, len(wl.req_gen))
    return (wl.req_gen.astype(np.float64) * rate).astype(np.float32)


@dataclasses.dataclass
class Trace:
    """Request arrivals: times (ms, non-decreasing), input and predicted lengths;
    optionally the real output lengths (unknown to the scheduler) and the
    re-prediction table a serving system would use when a request outgrows
    its prediction."""
    t_arr: np.ndarray   # float64 [R]
    req_in: np.ndarray  # int32 [R]
    req_pred: np.ndarray  # int32 [R]
    req_real: np.ndarray = None  # int32 [R] or None: predictions are exact
    repred: np.ndarray = None    # int32 [K+1] or None


def repredict_table(out_law, K, n=1_000_000, seed=99):
    """Conditional mean output length given that it exceeds x, for x = 0..K
    (rounded up; x + 1 where no draw exceeds x): what a predictor learned
    from the output-length distribution predicts for a request that has
    generated x tokens without finishing. Drawn from the same law."""
    rng = np.random.default_rng(seed)
    om, osg, olo, ohi = out_law
    L = np.sort(lognormal_lengths(rng, om, osg, olo, ohi, n).astype(np.int64))
    suffix = np.concatenate([np.cumsum(L[::-1])[::-1], [0]])
    x = np.arange(K + 1)
    first = np.searchsorted(L, x, side="right")    # draws > x start here
    cnt = n - first
    mean = np.where(cnt > 0, suffix[first] / np.maximum(cnt, 1), x + 1)
    return np.maximum(np.ceil(mean), x + 1).astype(np.int32)


def with_prediction_error(trace, sigma, seed, out_law=(256.0, 0.9, 8, 1024), K=8192):
    """The same arrivals with the drawn output lengths as the real ones and
    predictions off by a lognormal factor exp(N(0, sigma)), rounded and
    clipped to the output law's range (and to K - input)."""
    rng = np.random.default_rng(seed)
    real = np.asarray(trace.req_pred, np.int32)
    om, osg, olo, ohi = out_law
    noisy = np.rint(real * np.exp(rng.normal(0.0, sigma, len(real))))
    hi = np.minimum(ohi, K - np.asarray(trace.req_in, np.int64))
    pred = np.clip(noisy, olo, hi).astype(np.int32)
    return Trace(trace.t_arr, trace.req_in, pred, real, repredict_table(out_law, K))


def diurnal_trace(seed, n_requests, peak_rate, trough_rate, in_law=(512.0, 0.8, 16, 2048),
                  out_law=(256.0, 0.9, 8, 1024)):
    """Poisson arrivals whose rate follows one sinusoidal day compressed into the
    trace's span (peak:trough as given), drawn by thinning a homogeneous process
    at the peak rate. Rates in requests per second; times in ms."""
    rng = np.random.default_rng(seed)
    mean = 0.5 * (peak_rate + trough_rate)
    amp = 0.5 * (peak_rate - trough_rate)
    span_s = n_requests / mean
    times = []
    t = 0.0
    while len(times) < n_requests:
        gaps = rng.exponential(1.0 / peak_rate, 4096)
        us = rng.random(4096)
        for g, u in zip(gaps, us):
            t += g
            rate = mean - amp * math.cos(2.0 * math.pi * t / span_s)
            if u * peak_rate <= rate:
                times.append(t)
                if len(times) == n_requests:
                    break
    im, isg, ilo, ihi = in_law
    om, osg, olo, ohi = out_law
    return Trace(np.asarray(times) * 1000.0,
                 lognormal_lengths(rng, im, isg, ilo, ihi, n_requests),
                 lognormal_lengths(rng, om, osg, olo, ohi, n_requests))
