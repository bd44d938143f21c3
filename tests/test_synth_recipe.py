"""The seeded synthetic inputs follow the recipe the design states: lognormal
lengths whose pre-clip mean is the stated mean (mu = ln m - sigma^2 / 2),
rounded and clipped; generated tokens uniform below the prediction; waits
uniform in [0, 100) ms; the workloads' sizes; diurnal traces whose rate
follows one sinusoid with the stated peak and trough over the trace's span;
and the prediction-error variant's re-prediction table. Nothing here runs
the method's arithmetic."""
import math

import numpy as np
import pytest

from paper_2405_06856_gb300 import synth


def test_lognormal_lengths_mean_rounding_and_clip():
    rng = np.random.default_rng(3)
    m, s = 512.0, 0.8
    x = synth.lognormal_lengths(rng, m, s, 1, 10**9, 400_000)
    assert x.dtype == np.int32
    # the pre-clip mean is m (rounding moves it by well under a token)
    se = m * math.sqrt(math.exp(s * s) - 1.0) / math.sqrt(len(x))
    assert abs(x.mean() - m) < 5.0 * se + 0.5
    # median of a lognormal is exp(mu) = m exp(-s^2 / 2)
    assert abs(np.median(x) - m * math.exp(-0.5 * s * s)) < 0.01 * m
    y = synth.lognormal_lengths(np.random.default_rng(3), m, s, 16, 2048, 400_000)
    assert y.min() == 16 and y.max() == 2048
    assert np.array_equal(y, np.clip(x, 16, 2048))      # the same draws, clipped


def test_w4096_workload_shape():
    wl = synth.config("w4096")
    assert wl.n_workers == 4096 and wl.n_cand == 32768
    assert np.all(np.diff(wl.roff) == 128)
    assert np.all(wl.kv_capacity == 131072) and np.all(wl.gpus == 1)
    assert wl.req_in.min() >= 16 and wl.req_in.max() <= 2048
    assert wl.req_pred.min() >= 8 and wl.req_pred.max() <= 4096
    assert np.all(wl.req_gen >= 0) and np.all(wl.req_gen < wl.req_pred)
    assert np.all(wl.cand_wait >= 0.0) and np.all(wl.cand_wait < 100.0)
    # heavier output tail (sigma 1.2) than the default law reaches the clip
    assert (wl.req_pred > 1024).mean() > 0.02


def test_w16384_worker_cycle():
    wl = synth.config("w16384")
    assert wl.n_workers == 16384 and wl.n_cand == 131072 and wl.b_cap == 1024
    g = np.array([1, 2, 4, 8] * 4096)
    assert np.array_equal(wl.gpus, g)
    assert np.array_equal(wl.kv_capacity, 131072 * g)
    assert np.allclose(wl.lat_scale, 1.0 / np.sqrt(g))
    assert np.all(np.diff(wl.roff) == 256)


def test_workloads_are_seeded():
    a, b = synth.config("w256"), synth.config("w256")
    for f in ("req_in", "req_gen", "req_pred", "cand_in", "cand_pred", "cand_wait"):
        assert np.array_equal(getattr(a, f), getattr(b, f))
    c = synth.config("w256", seed=2)
    assert not np.array_equal(a.cand_in, c.cand_in)


def test_diurnal_trace_span_and_peak_to_trough():
    n, peak, trough = 200_000, 2000.0, 500.0
    tr = synth.diurnal_trace(4, n, peak, trough)
    t = tr.t_arr / 1000.0
    assert len(t) == n and np.all(np.diff(t) >= 0.0)
    mean = 0.5 * (peak + trough)
    span = n / mean
    assert abs(t[-1] - span) < 0.02 * span
    # one sinusoidal day: the trough at both ends, the peak in the middle
    counts, _ = np.histogram(t, bins=20, range=(0.0, span))
    width = span / 20
    ends = 0.5 * (counts[0] + counts[-1]) / width
    middle = 0.5 * (counts[9] + counts[10]) / width
    assert ends == pytest.approx(trough, rel=0.12)
    assert middle == pytest.approx(peak, rel=0.05)


def test_prediction_error_variant():
    tr = synth.diurnal_trace(9, 20_000, 60.0, 15.0)
    e = synth.with_prediction_error(tr, 0.4, 9)
    assert np.array_equal(e.req_real, tr.req_pred)           # the drawn lengths are the real ones
    assert np.array_equal(e.t_arr, tr.t_arr) and np.array_equal(e.req_in, tr.req_in)
    assert e.req_pred.min() >= 8 and e.req_pred.max() <= 1024
    ratio = np.log(e.req_pred / e.req_real)
    inner = (e.req_pred > 8) & (e.req_pred < 1024)
    assert abs(ratio[inner].std() - 0.4) < 0.05                # lognormal factor exp(N(0, 0.4))
    K = 8192
    rp = e.repred
    assert len(rp) == K + 1
    x = np.arange(K + 1)
    assert np.all(rp >= x + 1)                                 # a re-prediction exceeds x
    assert np.all(np.diff(rp) >= 0)                            # conditional means grow with x
