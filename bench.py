"""Benchmark of the Aladdin scheduler hot path on GB300.

A step is one pass of the hot path over the 4,096-worker workload (128 ongoing
requests per worker, 32,768 candidate queries, KV capacity 131,072, output
lengths lognormal(256, 1.2) clipped at 4,096), one aladdin_cluster_load_score
call: the worker state, resident in HBM, is packed into the cluster and every
worker's projection table is rebuilt (while the candidates are validated and
sorted on a second stream), then every candidate is scored against every
worker with flags, margins and argbest written to HBM.

Prints one JSON line (rank 0). `value` is candidate x worker evaluations per
second over all ranks with inputs resident in HBM; `e2e` is the same metric
through the same C ABI with pinned host buffers (host-to-device copies of the
state and candidates, device-to-host copies of all outputs inside the timed
region). `--impl reference` times the CPU oracle instead (there is no upstream
implementation to install: the paper ships no code).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "candidate x worker placement evaluations/sec"
UNIT = "evals/s"
WORKLOAD = "w4096"
WORKLOAD_DESC = ("4,096 workers x 128 ongoing requests (KV capacity 131,072 tokens), 32,768 candidate "
                 "queries; input lognormal(512, 0.8) clip [16, 2048], output lognormal(256, 1.2) "
                 "clip [8, 4096], generated ~ U[0, output); decode 8 ms + 0.05 ms/request + 2e-4 "
                 "ms/KV token, prefill 10 ms + 0.1 ms/100 tokens, TTFT 1 s, ATGT 50 ms; seed 2")
L2_FLUSH_BYTES = 256 << 20
CLOCK_WINDOW_S = 1.0
# minimum-worker search: KV tokens per GPU and per-worker request slots
MW_KV_PER_GPU = 65536
MW_B_CAP = 1024


def algorithmic_bytes(W, B, C):
    # state in (3 int32 per request) + candidates in (2 int32 + 1 fp32)
    # + flags (u8) and margin (fp32) per pair + argbest (int32) per candidate
    return W * B * 12 + C * 12 + C * W * 5 + C * 4


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        self.path = "/tmp/aladdin_clocks_%d.csv" % os.getpid()
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + q,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def wait_first(self, limit_s=5.0):
        """Block until nvidia-smi has written its first sample (or limit_s)."""
        t0 = time.time()
        while self.proc is not None and time.time() - t0 < limit_s:
            self.f.flush()
            if os.path.getsize(self.path) > 0:
                return
            time.sleep(0.02)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        return clock_summary(lines)


CLOCK_REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")


def clock_summary(lines):
    """Median SM clock, largest max clock and the throttle reasons seen in
    nvidia-smi CSV lines (index, clocks.sm, clocks.max.sm, power.draw,
    reasons.active, then the four reasons of CLOCK_REASONS as Active /
    Not Active); None without a sample."""
    sm, mx, reasons = [], 0.0, set()
    for line in lines:
        parts = [x.strip() for x in line.split(",")]
        if len(parts) < 9:
            continue
        try:
            sm.append(float(parts[1]))
            mx = max(mx, float(parts[2]))
        except ValueError:
            continue
        for k, v in zip(CLOCK_REASONS, parts[5:9]):
            if v.lower() == "active":
                reasons.add(k)
    if not sm:
        return None
    return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
            "samples": len(sm)}


def dist_setup(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        return dist, rank, world, local
    torch.cuda.set_device(0)
    return None, 0, 1, 0


def barrier_max(dist, value, device="cuda"):
    """The largest value over all ranks (every rank gets it)."""
    import torch
    if dist is None:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_value(world, evals_per_replica, step_ms_max):
    """Evaluations per second of the whole job: every replica scores its own
    copy of the workload (weak scaling, no data-path collective), timed by the
    slowest rank."""
    return world * evals_per_replica / (step_ms_max / 1000.0)


def barrier(dist):
    import torch
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()


# ---------------------------------------------------------------------------
# CPU oracle baseline (bounded sample; spawn pool across host cores).

_SLICE_CACHE = {}


def _oracle_slice(args):
    """Every pair of workers `wid` with the first `ncand` candidates, scored by
    the oracle in this (spawned) process; the workload and the sub-cluster are
    built once per process, outside the timed scoring."""
    wid, ncand = args[0], args[1]
    keep = len(args) > 2 and args[2]
    from oracle import oracle as O
    from paper_2405_06856_gb300 import synth
    key = (tuple(wid), ncand)
    if key not in _SLICE_CACHE:
        wl = synth.config(WORKLOAD)
        sub = O.Cluster(wl.params, wl.kv_capacity[wid], wl.lat_scale[wid], wl.b_cap,
                        np.concatenate([[0], np.cumsum(np.diff(wl.roff)[wid])]).astype(np.int32),
                        np.concatenate([wl.req_in[wl.roff[w]:wl.roff[w + 1]] for w in wid]),
                        np.concatenate([wl.req_gen[wl.roff[w]:wl.roff[w + 1]] for w in wid]),
                        np.concatenate([wl.req_pred[wl.roff[w]:wl.roff[w + 1]] for w in wid]))
        _SLICE_CACHE[key] = (sub, wl.cand_in[:ncand].copy(), wl.cand_pred[:ncand].copy(),
                             wl.cand_wait[:ncand].copy())
    sub, cin, cpr, cw = _SLICE_CACHE[key]
    t0 = time.perf_counter()
    out = sub.score(cin, cpr, cw, want=("flags", "margin", "near"))
    dt = time.perf_counter() - t0
    if keep:
        return len(wid) * ncand, dt, wid, out["flags"], out["near"]
    return len(wid) * ncand, dt


def oracle_jobs(workers_per_core, ncand, cores, keep=False):
    return [(list(range(i * workers_per_core, (i + 1) * workers_per_core)), ncand, keep)
            for i in range(cores)]


def oracle_baseline(workers_per_core=4, ncand=32768, cores=None, keep=False):
    """Oracle evaluations/sec: each process scores all pairs of its own workers
    against the first `ncand` candidates; throughput = pairs / wall time of
    the parallel scoring (the slowest process). keep: also return the
    sample's oracle flags and near measures (worker ids, flags [ncand, nw],
    near [ncand, nw]) for the parity report of the same pairs."""
    import multiprocessing as mp
    from oracle import oracle as O
    O.build()
    cores = cores or os.cpu_count() or 1
    jobs = oracle_jobs(workers_per_core, ncand, cores, keep)
    ctx = mp.get_context("spawn")
    t0 = time.perf_counter()
    with ctx.Pool(cores) as pool:
        res = pool.map(_oracle_slice, jobs)
    wall = time.perf_counter() - t0
    pairs = sum(r[0] for r in res)
    busy = max(r[1] for r in res)
    line = {"value": pairs / busy, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "%d workers x %d candidates of %s (%d pairs, %.1f s per process, %.1f s wall "
                      "with process start-up)"
                      % (cores * workers_per_core, ncand, WORKLOAD, pairs, busy, wall)}
    if not keep:
        return line
    wid = np.concatenate([r[2] for r in res])
    return line, (wid, np.concatenate([r[3] for r in res], axis=1),
                  np.concatenate([r[4] for r in res], axis=1))


def parity_report(sample, flags_dev):
    """The benchmarked call's flags on the oracle's sample pairs: mismatches
    outside the near pairs (must be 0), near pairs and near flips by
    direction (the tolerance rule of the parity tests: a pair is near when a
    constraint group's smallest relative slack is within 1e-5 of zero)."""
    import torch
    wid, oflags, onear = sample
    idx = torch.from_numpy(wid.astype(np.int64)).to(flags_dev.device)
    g = flags_dev[: oflags.shape[0]].index_select(1, idx).cpu().numpy()
    near = onear <= 1e-5
    gf, of = g == 15, oflags == 15
    return {"pairs": int(g.size), "far_mismatches": int((~near & (g != oflags)).sum()),
            "near": int(near.sum()), "near_gpu_only": int((near & gf & ~of).sum()),
            "near_oracle_only": int((near & ~gf & of).sum()),
            "sample": "the cpu_baseline sample's pairs (oracle flags vs the benchmarked call's)"}


def _oracle_config_job(job):
    """One oracle measurement of --mode configs (runs in a spawned process)."""
    kind, name = job[0], job[1]
    from oracle import oracle as O
    from paper_2405_06856_gb300 import synth
    if kind == "search":
        g, n = job[2], job[3]
        tr = synth.diurnal_trace(4, n, 2000.0, 500.0)
        t0 = time.perf_counter()
        got = O.min_workers(dict(synth.BASE_PARAMS), [g], [MW_KV_PER_GPU * g],
                            [1.0 / math.sqrt(g)], MW_B_CAP, tr, 100.0, 4096)
        return (kind, name, g, int(got[0]), time.perf_counter() - t0)
    wl = synth.config(name)
    if kind == "score":
        oc = O.Cluster.from_workload(wl)
        t0 = time.perf_counter()
        oc.score(wl.cand_in, wl.cand_pred, wl.cand_wait, want=("flags", "margin", "argbest"))
        return (kind, name, wl.n_cand * wl.n_workers, time.perf_counter() - t0)
    if kind == "sample":
        # every pair of a few random workers with the first ncand candidates
        nw, ncand = job[2], job[3]
        wid = np.sort(np.random.default_rng(17).choice(wl.n_workers, nw, replace=False))
        sub = O.Cluster(wl.params, wl.kv_capacity[wid], wl.lat_scale[wid], wl.b_cap,
                        np.concatenate([[0], np.cumsum(np.diff(wl.roff)[wid])]).astype(np.int32),
                        np.concatenate([wl.req_in[wl.roff[w]:wl.roff[w + 1]] for w in wid]),
                        np.concatenate([wl.req_gen[wl.roff[w]:wl.roff[w + 1]] for w in wid]),
                        np.concatenate([wl.req_pred[wl.roff[w]:wl.roff[w + 1]] for w in wid]))
        t0 = time.perf_counter()
        sub.score(wl.cand_in[:ncand], wl.cand_pred[:ncand], wl.cand_wait[:ncand],
                  want=("flags", "margin"))
        return (kind, name, nw * ncand, time.perf_counter() - t0)
    oc = O.Cluster.from_workload(wl)  # round
    t0 = time.perf_counter()
    oc.place_round(wl.cand_in, wl.cand_pred, wl.cand_wait)
    return (kind, name, wl.n_cand, time.perf_counter() - t0)


def run_configs(args):
    """Every workload of the scope table, on the GPU and with the oracle (one
    host core per oracle job, jobs in parallel on a spawn pool started before
    the first CUDA call): scoring evaluations/s and fraction of the HBM
    roofline (tiny, w256, w4096, w16384), one greedy round (tiny, w256; the
    16,384-worker rounds run as in the default line), and the minimum-worker
    search on a 10,000-request scale-down of the 1,000,000-request trace."""
    import multiprocessing as mp
    from oracle import oracle as O
    O.build()
    jobs = [("score", "tiny"), ("round", "tiny"), ("score", "w256"), ("round", "w256"),
            ("sample", "w4096", 8, 8192), ("sample", "w16384", 8, 8192)]
    jobs += [("search", "trace10k", g, 10_000) for g in (1, 2, 4, 8)]
    ctx = mp.get_context("spawn")
    pool = ctx.Pool(min(len(jobs), os.cpu_count() or 1))
    pending = pool.map_async(_oracle_config_job, jobs)

    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream().cuda_stream
    peak, peak_kind = read_peaks()
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    gpu = {}
    for name in ("tiny", "w256", "w4096", "w16384"):
        wl = synth.config(name)
        W, C = wl.n_workers, wl.n_cand
        cin, cpr, cw = d(wl.cand_in), d(wl.cand_pred), d(wl.cand_wait)
        f = torch.empty((C, W), dtype=torch.uint8, device=dev)
        m = torch.empty((C, W), dtype=torch.float32, device=dev)
        a = torch.empty(C, dtype=torch.int32, device=dev)
        with A.Cluster.from_workload(wl, stream=stream) as cl:
            for _ in range(3):
                A.aladdin_score(cl.handle, C, cin, cpr, cw, f, m, a)
            torch.cuda.synchronize()
            A.aladdin_cluster_timing(cl.handle, 1)
            for _ in range(10):
                flush.zero_()
                A.aladdin_score(cl.handle, C, cin, cpr, cw, f, m, a)
            kern_ms, kern_n = A.aladdin_cluster_timing(cl.handle, 0)
            feas = float((f == 15).float().mean().item())
        kern = kern_ms / max(kern_n, 1)
        nbytes = len(wl.req_in) * 12 + C * 12 + C * W * 5 + C * 4
        row = {"workers": W, "candidates": C, "k_score_ms": round(kern, 4),
               "evals_per_s": C * W / (kern / 1000.0),
               "hbm_frac": round(nbytes / (kern / 1000.0) / 1e9 / peak, 4),
               "feasible_fraction": round(feas, 4)}
        if name in ("tiny", "w256"):
            rms = []
            for _ in range(3):
                with A.Cluster.from_workload(wl, stream=stream) as c2:
                    pl = torch.empty(C, dtype=torch.int32, device=dev)
                    torch.cuda.synchronize()
                    t0 = time.perf_counter()
                    A.aladdin_place_round(c2.handle, C, cin, cpr, cw, pl)
                    rms.append((time.perf_counter() - t0) * 1000.0)
            row["round_ms"] = round(min(rms), 3)
        gpu[name] = row
        del f, m
        torch.cuda.empty_cache()
    gpu["w16384"]["rounds"] = rounds_w16384(A, synth, stream)
    tr = synth.diurnal_trace(4, 10_000, 2000.0, 500.0)
    gpus = [1, 2, 4, 8]
    got = np.zeros(4, np.int32)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    A.aladdin_min_workers(A.make_params(dict(synth.BASE_PARAMS), MW_B_CAP),
                          A.make_cfgs(gpus, [MW_KV_PER_GPU * g for g in gpus],
                                      [1.0 / math.sqrt(g) for g in gpus]),
                          A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0, 4096, got,
                          stream=stream)
    gpu["search_10k"] = {"min_workers": got.tolist(), "wall_s": round(time.perf_counter() - t0, 2)}

    res = pending.get()
    pool.close()
    orc = {}
    for r in res:
        if r[0] == "search":
            orc.setdefault("search_10k", {"min_workers": [], "s_per_option": []})
            orc["search_10k"]["min_workers"].append(r[3])
            orc["search_10k"]["s_per_option"].append(round(r[4], 2))
        elif r[0] == "round":
            orc.setdefault(r[1], {})["round_ms"] = round(r[3] * 1000.0, 2)
        else:
            orc.setdefault(r[1], {})["evals_per_s_1core"] = r[2] / r[3]
            if r[0] == "sample":
                orc[r[1]]["sample"] = ("%d pairs (8 random workers x 8,192 candidates), "
                                       "extrapolated" % r[2])
    print(json.dumps({"mode": "configs", "peak_gbs": peak, "peak_kind": peak_kind,
                      "host_cores": os.cpu_count(), "gpu": gpu, "oracle": orc}))


# ---------------------------------------------------------------------------

def run_reference(args):
    """The reference arm: the CPU oracle on the host cores (the paper ships no
    code to install). A step scores one bounded sample of the workload, the
    same sample as the cpu_baseline leg (4 workers a core x 32,768
    candidates); ms_per_step is the measured wall time of that sample, and
    the time of a full 4,096 x 32,768 step is reported separately, labelled
    as extrapolated."""
    if int(os.environ.get("WORLD_SIZE", "1")) > 1 and int(os.environ.get("RANK", "0")) != 0:
        return
    import multiprocessing as mp
    from oracle import oracle as O
    from paper_2405_06856_gb300 import synth
    O.build()
    steps, warm = args.steps, args.warmup
    cores = os.cpu_count() or 1
    wpc, ncand = 4, 32768
    jobs = oracle_jobs(wpc, ncand, cores)
    walls, pairs = [], 0
    with mp.get_context("spawn").Pool(cores) as pool:
        pool.map(_oracle_slice, jobs)  # builds each process's sub-cluster, untimed
        for i in range(warm + steps):
            t0 = time.perf_counter()
            res = pool.map(_oracle_slice, jobs)
            wall = time.perf_counter() - t0
            if i >= warm:
                walls.append(wall)
                pairs = sum(r[0] for r in res)
    wall = float(statistics.median(walls))
    v = pairs / wall
    wl = synth.config(WORKLOAD, n_cand=16)
    sample = ("%d workers x %d candidates of %s (%d pairs) on %d host processes, one step each; "
              "median wall %.3f s over %d steps" % (cores * wpc, ncand, WORKLOAD, pairs, cores,
                                                    wall, steps))
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT,
            "n_gpus": args.gpus, "steps": steps, "warmup": warm, "ms_per_step": wall * 1000.0,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_DESC, "sample": sample, "pairs_per_step": pairs,
                       "extrapolated_full_step_ms": wl.n_workers * 32768 / v * 1000.0},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def run_ours(args):
    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth

    # The oracle's process pool is started before the first CUDA call.
    cpu = sample = None
    if args.cpu_baseline and int(os.environ.get("RANK", "0")) == 0 and args.gpus == 1:
        cpu, sample = oracle_baseline(keep=True)

    dist, rank, world, local = dist_setup(args)
    dev = torch.device("cuda", local)
    wl = synth.config(WORKLOAD)
    W, C = wl.n_workers, wl.n_cand
    Bq = int(np.diff(wl.roff).max())
    stream = torch.cuda.current_stream().cuda_stream

    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    roff, rin, rgen, rpred = d(wl.roff), d(wl.req_in), d(wl.req_gen), d(wl.req_pred)
    cin, cpr, cw = d(wl.cand_in), d(wl.cand_pred), d(wl.cand_wait)
    flags = torch.empty((C, W), dtype=torch.uint8, device=dev)
    margin = torch.empty((C, W), dtype=torch.float32, device=dev)
    arg = torch.empty(C, dtype=torch.int32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    cl = A.Cluster.from_workload(wl, stream=stream)

    def step():  # the new state, then the candidates scored against it
        A.aladdin_cluster_load_score(cl.handle, roff, rin, rgen, rpred, None, C, cin, cpr, cw,
                                     flags, margin, arg)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    assert cl.status() == A.OK
    frac_feasible = float((flags == 15).float().mean().item())

    # timed region: per-step CUDA events, L2 flushed (256 MiB write) between steps
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(local)
    barrier(dist)
    # The clock samples (200 ms apart) cover the same step load for
    # CLOCK_WINDOW_S of untimed steps ending right where the timed steps begin,
    # so that a timed region of a few milliseconds still has samples under load.
    sampler.start()
    sampler.wait_first()
    t0 = time.time()
    while time.time() - t0 < CLOCK_WINDOW_S:
        for _ in range(32):
            flush.zero_()
            step()
        torch.cuda.synchronize()
    A.aladdin_cluster_timing(cl.handle, 1)
    barrier(dist)
    for i in range(args.steps):
        flush.zero_()
        starts[i].record()
        step()
        ends[i].record()
    barrier(dist)
    clocks = sampler.stop()
    if clocks is not None:
        clocks["window"] = "%.1f s of the same steps (untimed), then the timed steps" % CLOCK_WINDOW_S
    kern_ms, kern_n = A.aladdin_cluster_timing(cl.handle, 0)
    step_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / args.steps
    parity = parity_report(sample, flags) if sample is not None else None
    step_ms = barrier_max(dist, step_ms)
    value = whole_job_value(world, C * W, step_ms)

    # end to end through the same API with pinned host buffers
    pin = lambda x: torch.from_numpy(np.ascontiguousarray(x)).pin_memory()
    h_roff, h_rin, h_rgen, h_rpred = pin(wl.roff), pin(wl.req_in), pin(wl.req_gen), pin(wl.req_pred)
    h_cin, h_cpr, h_cw = pin(wl.cand_in), pin(wl.cand_pred), pin(wl.cand_wait)
    h_flags = torch.empty((C, W), dtype=torch.uint8).pin_memory()
    h_margin = torch.empty((C, W), dtype=torch.float32).pin_memory()
    h_arg = torch.empty(C, dtype=torch.int32).pin_memory()

    def step_host():
        A.aladdin_cluster_load_score(cl.handle, h_roff, h_rin, h_rgen, h_rpred, None, C, h_cin,
                                     h_cpr, h_cw, h_flags, h_margin, h_arg)

    for _ in range(2):
        step_host()
    torch.cuda.synchronize()
    e2e_steps = max(3, min(args.steps, 10))
    barrier(dist)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        step_host()
    torch.cuda.synchronize()
    e2e_ms = barrier_max(dist, (time.perf_counter() - t0) * 1000.0 / e2e_steps)
    assert np.array_equal(h_arg.numpy(), arg.cpu().numpy())
    h2d = wl.roff.nbytes + wl.req_in.nbytes + wl.req_gen.nbytes + wl.req_pred.nbytes + \
        wl.cand_in.nbytes + wl.cand_pred.nbytes + wl.cand_wait.nbytes
    d2h = C * W * 5 + C * 4

    # round latency on the 256-worker workload (one greedy round of 2,048 candidates)
    w2 = synth.config("w256", b_cap=128)
    rounds = []
    for _ in range(3):
        with A.Cluster.from_workload(w2, stream=stream) as c2:
            pl = torch.empty(w2.n_cand, dtype=torch.int32, device=dev)
            t_in, t_pr, t_w = d(w2.cand_in), d(w2.cand_pred), d(w2.cand_wait)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            A.aladdin_place_round(c2.handle, w2.n_cand, t_in, t_pr, t_w, pl)
            rounds.append((time.perf_counter() - t0) * 1000.0)
    round_ms = min(rounds)
    r16k = rounds_w16384(A, synth, stream)
    # group counts coprime with the workload's 1/2/4/8-GPU cycle of workers,
    # so that every group holds all four worker sizes
    r16k_grp = {"G%d" % G: rounds_w16384(A, synth, stream, groups=G) for G in (7, 63)}
    apx = approx_mode(A, synth, dev, stream, flush)
    mixed = mixed_mask(A, synth, dev, stream, flush)
    pol = policy_compare(A, synth, stream, 20_000, [1, 2])
    wmod = worker_model(A, synth, stream, fit_n=0)
    search = min_workers_1m(A, synth, stream) if args.search else None

    peak, peak_kind = read_peaks()
    kern_avg = kern_ms / max(kern_n, 1)
    abytes = algorithmic_bytes(W, Bq, C)
    achieved = abytes / (kern_avg / 1000.0) / 1e9
    traffic = profiled_traffic()

    # load: two-level table build (requests packed by the first level), ranks
    # and order; score: count, scan, scatter, score, finalize
    launches_per_step = 3 + 5
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_DESC, "n_workers": W, "requests_per_worker": Bq,
                       "n_cand": C, "l2": "flushed between steps (256 MiB write)",
                       "outputs": "flags u8 + margin f32 per pair, argbest per candidate",
                       "parallelism": "replicas" if world > 1 else "single GPU",
                       "feasible_fraction": round(frac_feasible, 4)},
            "e2e": {"value": whole_job_value(world, C * W, e2e_ms), "unit": UNIT,
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms},
            "gpu_launches": launches_per_step * args.steps,
            "roofline": {"bound": "hbm", "kernel": "k_score", "achieved": achieved, "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "algorithmic_bytes_per_launch": abytes,
                         "kernel_ms": kern_avg, "launches": kern_n},
            "round_latency_ms": {"workload": "256 workers x 64 requests, 2,048 candidates, one "
                                             "greedy round", "value": round_ms},
            "rounds_w16384": r16k,
            "rounds_w16384_grouped": r16k_grp,
            "approx_mode": apx,
            "mixed_mask": mixed,
            "policies": pol,
            "worker_config": wmod,
            "min_workers_1m": search,
            "clocks": clocks}
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if parity is not None:
        line["parity_sample"] = parity
    if rank == 0:
        print(json.dumps(line))
    cl.close()
    if dist is not None:
        dist.destroy_process_group()


def rounds_w16384(A, synth, stream, n_rounds=10, dt_ms=100.0, groups=1):
    """Ten consecutive greedy rounds on the 16,384-worker workload (1/2/4/8-GPU
    workers, 256 requests each): the 131,072 candidates arrive over ten
    heartbeats, each round placing its share, then every worker executes
    100 ms. Round time is the synchronous aladdin_place_round call with host
    arrays (upload, the round, the capacity_norm ranking and the download).
    groups > 1: grouped scheduling (Appendix A), the groups' rounds in
    parallel."""
    wl = synth.config("w16384", params=dict(groups=groups))
    bounds = np.linspace(0, wl.n_cand, n_rounds + 1).astype(int)
    rounds, advances, placed = [], [], 0
    with A.Cluster.from_workload(wl, stream=stream) as cl:
        for k in range(n_rounds):
            a, b = int(bounds[k]), int(bounds[k + 1])
            t0 = time.perf_counter()
            pl = cl.place_round(wl.cand_in[a:b], wl.cand_pred[a:b], wl.cand_wait[a:b])
            rounds.append((time.perf_counter() - t0) * 1000.0)
            placed += int((pl >= 0).sum())
            t0 = time.perf_counter()
            cl.advance(dt_ms)
            advances.append((time.perf_counter() - t0) * 1000.0)
        assert cl.status() == A.OK
    return {"workload": "16,384 workers of 1/2/4/8 GPUs (KV 131,072 per GPU, latency x 1/sqrt(GPUs)), "
                        "256 requests each; 131,072 candidates over 10 greedy rounds of 13,107, "
                        "100 ms of execution between rounds; seed 3"
                        + ("; %d scheduling groups" % groups if groups > 1 else ""),
            "rounds": n_rounds, "candidates_per_round": int(bounds[1] - bounds[0]),
            "ms_per_round": statistics.mean(rounds), "ms_max_round": max(rounds),
            "ms_per_advance": statistics.mean(advances),
            "placed_fraction": placed / float(wl.n_cand)}


def approx_mode(A, synth, dev, stream, flush, launches=10):
    """The approximate mode (the placement MIP's constraints (b), with Eq.
    input limit, and (d)): scoring-kernel time on the 4,096-worker workload
    (theta 0.9), and on the 256-worker workload with a decode history how its
    flags differ from the exact projection's."""
    import torch
    wl = synth.config(WORKLOAD, params=dict(theta=0.9, mode=1))
    W, C = wl.n_workers, wl.n_cand
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    cin, cpr, cw = d(wl.cand_in), d(wl.cand_pred), d(wl.cand_wait)
    f = torch.empty((C, W), dtype=torch.uint8, device=dev)
    m = torch.empty((C, W), dtype=torch.float32, device=dev)
    a = torch.empty(C, dtype=torch.int32, device=dev)
    with A.Cluster.from_workload(wl, stream=stream) as cl:
        for _ in range(3):
            A.aladdin_score(cl.handle, C, cin, cpr, cw, f, m, a)
        torch.cuda.synchronize()
        A.aladdin_cluster_timing(cl.handle, 1)
        for _ in range(launches):
            flush.zero_()
            A.aladdin_score(cl.handle, C, cin, cpr, cw, f, m, a)
        kern_ms, kern_n = A.aladdin_cluster_timing(cl.handle, 0)
        feas4096 = float((f == 15).float().mean().item())
    kern = kern_ms / max(kern_n, 1)
    # flags of both modes on the 256-worker workload with a decode history
    gen = synth.config("w256").req_gen
    tdec = (gen * np.random.default_rng(7).uniform(10.0, 50.0, len(gen))).astype(np.float32)
    out = {}
    for mode in (0, 1):
        w2 = synth.config("w256", params=dict(theta=0.9, mode=mode))
        with A.Cluster.from_workload(w2, tdec_ms=tdec, stream=stream) as c2:
            out[mode] = c2.score(w2.cand_in, w2.cand_pred, w2.cand_wait)["flags"]
    ex, ap = out[0] == 15, out[1] == 15
    return {"workload": "4,096-worker workload with theta 0.9 (scoring time); 256-worker workload "
                        "with theta 0.9 and decode histories of 10-50 ms a token (flag gap)",
            "k_score_us": kern * 1000.0,
            "evals_per_s_kernel": C * W / (kern / 1000.0),
            "feasible_fraction_w4096": round(feas4096, 4),
            "w256_feasible_exact": round(float(ex.mean()), 4),
            "w256_feasible_approx": round(float(ap.mean()), 4),
            "w256_approx_feasible_exact_infeasible": round(float((ap & ~ex).mean()), 4),
            "w256_exact_feasible_approx_infeasible": round(float((ex & ~ap).mean()), 4)}


def mixed_mask(A, synth, dev, stream, flush, launches=10):
    """The benchmarked step on the 4,096-worker workload with tighter limits
    and a decode history (w4096_mixed: about half of the pairs feasible,
    every constraint group binding): its scoring-kernel time and HBM fraction
    against the all-feasible workload's."""
    import torch
    wl = synth.config("w4096_mixed")
    tdec = synth.decode_history(wl, 18.0, 26.0, synth.MIXED_HISTORY_SEED)
    W, C = wl.n_workers, wl.n_cand
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    roff, rin, rgen, rpred, rt = d(wl.roff), d(wl.req_in), d(wl.req_gen), d(wl.req_pred), d(tdec)
    cin, cpr, cw = d(wl.cand_in), d(wl.cand_pred), d(wl.cand_wait)
    f = torch.empty((C, W), dtype=torch.uint8, device=dev)
    m = torch.empty((C, W), dtype=torch.float32, device=dev)
    a = torch.empty(C, dtype=torch.int32, device=dev)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(launches)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(launches)]
    with A.Cluster.from_workload(wl, tdec_ms=tdec, stream=stream) as cl:
        step = lambda: A.aladdin_cluster_load_score(cl.handle, roff, rin, rgen, rpred, rt, C, cin,
                                                    cpr, cw, f, m, a)
        for _ in range(3):
            step()
        torch.cuda.synchronize()
        A.aladdin_cluster_timing(cl.handle, 1)
        for i in range(launches):
            flush.zero_()
            starts[i].record()
            step()
            ends[i].record()
        torch.cuda.synchronize()
        kern_ms, kern_n = A.aladdin_cluster_timing(cl.handle, 0)
        assert cl.status() == A.OK
        feas = float((f == 15).float().mean().item())
        cleared = [round(float(((f >> b) & 1 == 0).float().mean().item()), 4) for b in range(4)]
    kern = kern_ms / max(kern_n, 1)
    step_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends)) / launches
    peak, _ = read_peaks()
    achieved = algorithmic_bytes(W, int(np.diff(wl.roff).max()), C) / (kern / 1000.0) / 1e9
    return {"workload": "w4096 sizes and draws with KV 90,000 tokens, TTFT 95 ms, ATGT 30 ms and "
                        "decode histories of 18-26 ms a token (exact mode)",
            "k_score_us": kern * 1000.0, "hbm_gbs": achieved, "hbm_frac": achieved / peak,
            "ms_per_step": step_ms, "evals_per_s": C * W / (step_ms / 1000.0),
            "feasible_fraction": round(feas, 4),
            "cleared_fraction_by_group": dict(zip(("kv", "ttft", "ongoing_atgt", "new_atgt"),
                                                  cleared))}


def min_workers_config(synth):
    """The minimum-worker search workload: a 1,000,000-request diurnal trace
    (peak 2,000 req/s, peak:trough 4:1) and 1/2/4/8-GPU worker options."""
    tr = synth.diurnal_trace(4, 1_000_000, 2000.0, 500.0)
    gpus = [1, 2, 4, 8]
    kv = [MW_KV_PER_GPU * g for g in gpus]
    scale = [1.0 / math.sqrt(g) for g in gpus]
    return tr, gpus, kv, scale


POLICIES = (("best_fit", 0), ("jsq", 1), ("power_of_two", 2))
PHASES = (("mixed", 0), ("decode", 1))


def policy_compare(A, synth, stream, n_requests, gpus, seed=4):
    """GPUs each placement policy needs to serve a diurnal trace with every
    SLO met (P100), in the mixed setting and on the decode instances of
    split-phase inference (the comparison of Sec. 6.4): the minimum-worker
    search per worker option, on the device, for best-fit (Algorithm 1), JSQ
    and the power of two choices."""
    tr = synth.diurnal_trace(seed, n_requests, 2000.0, 500.0)
    kv = [MW_KV_PER_GPU * g for g in gpus]
    scale = [1.0 / math.sqrt(g) for g in gpus]
    trace = A.make_trace(tr.t_arr, tr.req_in, tr.req_pred)
    out = {"workload": "diurnal trace of %d requests (peak 2,000 req/s, peak:trough 4:1, %.0f s), "
                       "%s-GPU workers of %d KV tokens per GPU, latency x 1/sqrt(GPUs); "
                       "P100: no failed request and no realized TTFT, ATGT or KV violation"
                       % (n_requests, tr.t_arr[-1] / 1000.0, "/".join(map(str, gpus)),
                          MW_KV_PER_GPU)}
    for pname, phase in PHASES:
        res = {}
        for name, policy in POLICIES:
            p = dict(synth.BASE_PARAMS, phase=phase, policy=policy, seed=12345)
            got = np.zeros(len(gpus), np.int32)
            t0 = time.perf_counter()
            best, total = A.aladdin_min_workers(A.make_params(p, MW_B_CAP),
                                                A.make_cfgs(gpus, kv, scale), trace, 100.0, 4096,
                                                got, stream=stream)
            res[name] = {"min_workers": got.tolist(), "total_gpus": int(total),
                         "best_gpus_per_worker": gpus[best] if best >= 0 else None,
                         "search_s": round(time.perf_counter() - t0, 2)}
        bf = res["best_fit"]["total_gpus"]
        for name in ("jsq", "power_of_two"):
            o = res[name]["total_gpus"]
            res["gpus_saved_vs_" + name] = round(1.0 - bf / o, 4) if bf > 0 and o > 0 else None
        out[pname] = res
    return out


def worker_model(A, synth, stream, trace_n=100_000, fit_n=20_000,
                 fit_rates=(250.0, 500.0, 1000.0, 1500.0, 2000.0)):
    """The worker-configuration model of Sec. 4.1 (Eq. max throughput of each
    1/2/4/8-GPU option from the diurnal trace's demand, the optimal option)
    and Eq. total_worker_pre fitted to best-fit minimum-worker searches of
    that option at constant arrival rates (Sec. 5.2)."""
    tr = synth.diurnal_trace(4, trace_n, 2000.0, 500.0)
    gpus = [1, 2, 4, 8]
    kv = [MW_KV_PER_GPU * g for g in gpus]
    scale = [1.0 / math.sqrt(g) for g in gpus]
    p = dict(synth.BASE_PARAMS)
    prm = A.make_params(p, MW_B_CAP)
    trace = A.make_trace(tr.t_arr, tr.req_in, tr.req_pred)
    m_r, l_ave = A.aladdin_trace_demand(prm, trace, stream=stream)
    tmax = np.zeros(len(gpus))
    best = A.aladdin_pick_config(prm, A.make_cfgs(gpus, kv, scale), trace, tmax, stream=stream)
    out = {"demand": {"m_r": round(m_r, 3), "l_ave": round(l_ave, 3)},
           "t_max_tokens_per_ms_per_gpu": [round(float(v), 4) for v in tmax],
           "picked_gpus_per_worker": gpus[best]}
    if fit_n:
        trs = [synth.diurnal_trace(40 + k, fit_n, r, r) for k, r in enumerate(fit_rates)]
        nw = np.zeros(len(trs), np.int32)
        t0 = time.perf_counter()
        k5, c5 = A.aladdin_fit_workers(prm, A.make_cfgs([gpus[best]], [kv[best]],
                                                        [scale[best]])[0],
                                       [A.make_trace(t.t_arr, t.req_in, t.req_pred) for t in trs],
                                       list(fit_rates), 0.0, 100.0, 4096, nw, stream=stream)
        pred = [A.aladdin_predict_workers(k5, c5, r) for r in fit_rates]
        out["n_w_model"] = {"workload": "constant-rate Poisson traces of %d requests, %d-GPU "
                                        "workers, best-fit" % (fit_n, gpus[best]),
                            "rates_req_s": list(fit_rates), "min_workers": nw.tolist(),
                            "k5": k5, "c5": c5, "predicted": pred,
                            "fit_s": round(time.perf_counter() - t0, 2)}
    return out


def prediction_errors(A, synth, stream, n_requests=100_000, n_workers=133,
                      sigmas=(0.3, 0.6)):
    """Algorithm 2 under prediction errors (Sec. 4.3): the diurnal trace with
    predictions off by a lognormal factor exp(N(0, sigma)), served by best-fit
    on a fixed fleet of 1-GPU workers (the count the exact-prediction search
    needs) with and without re-balancing; realized violations (ATGT above
    T_dec, KV above capacity, TTFT above T_pre) and requests moved."""
    tr = synth.diurnal_trace(4, n_requests, 2000.0, 500.0)
    out = {"workload": "diurnal trace of %d requests, %d 1-GPU workers (%d KV tokens), "
                       "best-fit" % (n_requests, n_workers, MW_KV_PER_GPU)}
    cfg = A.make_cfgs([1], [MW_KV_PER_GPU], [1.0])[0]
    for sigma in sigmas:
        te = synth.with_prediction_error(tr, sigma, 7)
        row = {}
        for rb in (0, 1):
            p = dict(synth.BASE_PARAMS, rebalance=rb)
            res = np.zeros(A.SIMULATE_OUT)
            t0 = time.perf_counter()
            A.aladdin_simulate(A.make_params(p, MW_B_CAP), cfg, n_workers, A.trace_of(te), 100.0,
                               0, 1, res, stream=stream)
            row["rebalance" if rb else "no_rebalance"] = {
                "failed": int(res[0]), "violations": int(res[5]), "max_atgt_ms": round(res[4], 3),
                "repredictions": int(res[6]), "early_finishes": int(res[7]),
                "moved": int(res[8]), "sim_s": round(time.perf_counter() - t0, 2)}
        out["sigma_%g" % sigma] = row
    return out


def grouped_scheduling(A, synth, stream, n_requests=100_000, groups=(1, 2, 4, 8)):
    """Distributed grouped scheduling (Appendix A): requests dealt round-robin
    to G groups, each placing on its own workers; the workers the search
    needs for each G (1-GPU workers, best-fit) against the central
    scheduler's."""
    tr = synth.diurnal_trace(4, n_requests, 2000.0, 500.0)
    trace = A.make_trace(tr.t_arr, tr.req_in, tr.req_pred)
    out = {"workload": "diurnal trace of %d requests, 1-GPU workers (%d KV tokens), best-fit"
                       % (n_requests, MW_KV_PER_GPU)}
    base = None
    for G in groups:
        p = dict(synth.BASE_PARAMS, groups=G)
        got = np.zeros(1, np.int32)
        t0 = time.perf_counter()
        A.aladdin_min_workers(A.make_params(p, MW_B_CAP),
                              A.make_cfgs([1], [MW_KV_PER_GPU], [1.0]), trace, 100.0, 4096, got,
                              stream=stream)
        n = int(got[0])
        base = n if G == 1 else base
        out["G%d" % G] = {"min_workers": n, "workers_per_group": round(n / G, 1),
                          "extra_vs_central": round(n / base - 1.0, 4) if base else None,
                          "search_s": round(time.perf_counter() - t0, 2)}
    return out


def run_policies(args):
    """Best-fit against JSQ and the power of two choices (Sec. 6.4): GPUs each
    needs, mixed setting and decode instances, on a 100,000-request trace; the
    worker-configuration picker and the fitted worker-count model; Algorithm 2
    under prediction errors; grouped scheduling."""
    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth
    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream().cuda_stream
    t0 = time.perf_counter()
    res = policy_compare(A, synth, stream, 100_000, [1, 2, 4, 8])
    res["worker_model"] = worker_model(A, synth, stream)
    res["prediction_errors"] = prediction_errors(A, synth, stream)
    res["grouped_scheduling"] = grouped_scheduling(A, synth, stream)
    res["mode"] = "policies"
    res["wall_s"] = round(time.perf_counter() - t0, 1)
    print(json.dumps(res))


def run_min_workers(args):
    """Minimum-worker search (binary search over the worker count for each
    worker option, every probe a fleet simulation on the device)."""
    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth
    torch.cuda.set_device(0)
    tr, gpus, kv, scale = min_workers_config(synth)
    p = dict(synth.BASE_PARAMS)
    got = np.zeros(len(gpus), np.int32)
    stream = torch.cuda.current_stream().cuda_stream
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    best, total = A.aladdin_min_workers(A.make_params(p, MW_B_CAP), A.make_cfgs(gpus, kv, scale),
                                        A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0,
                                        4096, got, stream=stream)
    wall = time.perf_counter() - t0
    print(json.dumps({"mode": "min_workers", "requests": len(tr.t_arr),
                      "trace_span_s": float(tr.t_arr[-1] / 1000.0),
                      "gpus_per_worker": gpus, "kv_per_worker": kv,
                      "min_workers": got.tolist(), "best_gpus_per_worker": gpus[best],
                      "total_gpus": int(total), "wall_s": wall}))


def min_workers_1m(A, synth, stream):
    """The minimum-worker search on the 1,000,000-request diurnal trace (Sec.
    6.4's large-scale simulation): per worker option the fewest workers that
    serve every request within its SLOs, the fewest GPUs over the options,
    and the search's wall time."""
    import torch
    tr, gpus, kv, scale = min_workers_config(synth)
    got = np.zeros(len(gpus), np.int32)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    best, total = A.aladdin_min_workers(A.make_params(dict(synth.BASE_PARAMS), MW_B_CAP),
                                        A.make_cfgs(gpus, kv, scale),
                                        A.make_trace(tr.t_arr, tr.req_in, tr.req_pred), 100.0,
                                        4096, got, stream=stream)
    wall = time.perf_counter() - t0
    return {"workload": "diurnal Poisson trace of %d requests over %.0f s (peak 2,000 req/s, "
                        "peak:trough 4:1), %d KV tokens per GPU, latency x 1/sqrt(GPUs), %d request "
                        "slots a worker, heartbeat 100 ms" % (len(tr.t_arr), tr.t_arr[-1] / 1000.0,
                                                              MW_KV_PER_GPU, MW_B_CAP),
            "gpus_per_worker": list(gpus), "min_workers": got.tolist(),
            "gpus_per_option": [int(g * n) if n > 0 else None for g, n in zip(gpus, got.tolist())],
            "best_gpus_per_worker": int(gpus[best]), "total_gpus": int(total), "wall_s": wall}


def run_aux(args):
    """Small runs of the auxiliary kernels, each warm-up + steps times on the
    256-worker workload: a grouped best-fit round (k_round_grp, 7 groups), a
    JSQ round (k_round_queue), the 100 ms execution step (k_advance) and
    Algorithm 2's re-balancing of a round (k_rebalance). The command the
    profiles of those kernels capture."""
    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth
    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream().cuda_stream
    rng = np.random.default_rng(5)
    out = {}
    for _ in range(args.warmup + args.steps):
        for name, over in (("grouped", dict(groups=7)), ("jsq", dict(policy=A.POLICY_JSQ)),
                           ("bestfit", {})):
            w2 = synth.config("w256", b_cap=128, params=over)
            with A.Cluster.from_workload(w2, stream=stream) as cl:
                t0 = time.perf_counter()
                pl = cl.place_round(w2.cand_in, w2.cand_pred, w2.cand_wait)
                out.setdefault(name + "_round_ms", []).append((time.perf_counter() - t0) * 1e3)
                if name == "bestfit":
                    le = rng.integers(-4000, 4000, w2.n_workers)
                    be = rng.integers(-8, 8, w2.n_workers)
                    t0 = time.perf_counter()
                    cl.rebalance(w2.cand_in, w2.cand_pred, w2.cand_wait, pl, le, be)
                    out.setdefault("rebalance_ms", []).append((time.perf_counter() - t0) * 1e3)
                t0 = time.perf_counter()
                cl.advance(100.0)
                out.setdefault(name + "_advance_ms", []).append((time.perf_counter() - t0) * 1e3)
    print(json.dumps({"mode": "aux", **{k: round(min(v), 3) for k, v in out.items()}}))


def run_kernel_only(args):
    """The device-resident step only (warm-up + steps), nothing else: the
    command profiled by ncu."""
    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    wl = synth.config(WORKLOAD)
    W, C = wl.n_workers, wl.n_cand
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    roff, rin, rgen, rpred = d(wl.roff), d(wl.req_in), d(wl.req_gen), d(wl.req_pred)
    cin, cpr, cw = d(wl.cand_in), d(wl.cand_pred), d(wl.cand_wait)
    flags = torch.empty((C, W), dtype=torch.uint8, device=dev)
    margin = torch.empty((C, W), dtype=torch.float32, device=dev)
    arg = torch.empty(C, dtype=torch.int32, device=dev)
    cl = A.Cluster.from_workload(wl, stream=torch.cuda.current_stream().cuda_stream)
    for _ in range(args.warmup + args.steps):
        A.aladdin_cluster_load_score(cl.handle, roff, rin, rgen, rpred, None, C, cin, cpr, cw,
                                     flags, margin, arg)
    torch.cuda.synchronize()
    assert cl.status() == A.OK
    cl.close()
    print("kernel mode ok: %d steps" % (args.warmup + args.steps))


def run_round_only(args):
    """Greedy rounds on the 256-worker workload only (warm-up + steps rounds,
    each on a fresh cluster): the command profiled for the round kernel."""
    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    w2 = synth.config("w256", b_cap=128)
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    t_in, t_pr, t_w = d(w2.cand_in), d(w2.cand_pred), d(w2.cand_wait)
    times = []
    for _ in range(args.warmup + args.steps):
        with A.Cluster.from_workload(w2, stream=torch.cuda.current_stream().cuda_stream) as c2:
            pl = torch.empty(w2.n_cand, dtype=torch.int32, device=dev)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            A.aladdin_place_round(c2.handle, w2.n_cand, t_in, t_pr, t_w, pl)
            times.append((time.perf_counter() - t0) * 1000.0)
    print("round mode ok: %d rounds, best %.2f ms" % (len(times), min(times)))


def run_sim_only(args):
    """One fleet simulation of the minimum-worker search's workload, alone:
    147 one-GPU workers of 1,024 request slots over the first 12,500 requests
    (about 10 s, 100 heartbeats) of the 1,000,000-request diurnal trace. The
    command profiled for the simulation's launch list."""
    import torch
    from paper_2405_06856_gb300 import build as B
    B.build()
    from paper_2405_06856_gb300 import aladdin as A
    from paper_2405_06856_gb300 import synth
    torch.cuda.set_device(0)
    tr, gpus, kv, scale = min_workers_config(synth)
    k = 12_500
    trace = A.make_trace(tr.t_arr[:k], tr.req_in[:k], tr.req_pred[:k])
    cfg = A.make_cfgs(gpus[:1], kv[:1], scale[:1])[0]
    out = np.zeros(A.SIMULATE_OUT)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    A.aladdin_simulate(A.make_params(dict(synth.BASE_PARAMS), MW_B_CAP), cfg, 147, trace, 100.0,
                       1, 0, out)
    wall = time.perf_counter() - t0
    print(json.dumps({"mode": "sim", "workers": 147, "requests": k, "failed": int(out[0]),
                      "placed": int(out[1]), "heartbeats": int(out[2]), "wall_s": wall,
                      "ms_per_heartbeat": 1000.0 * wall / max(out[2], 1.0)}))


def profiled_traffic():
    """DRAM bytes per launch of the scoring kernel from the committed ncu
    summary, or None if the kernel source changed since it was taken."""
    import re
    path = os.path.join(ROOT, "profiles", "k_score_w4096.md")
    try:
        txt = open(path).read()
        t = re.search(r"traffic_bytes_per_launch:\s*(\d+)", txt)
        h = re.search(r"source_hash:\s*(\w+)", txt)
        if t and h and h.group(1) == kernel_source_hash():
            return int(t.group(1))
    except OSError:
        pass
    return None


def kernel_source_hash():
    import hashlib
    h = hashlib.sha256()
    for f in ("aladdin_dev.cuh", "score.cu"):
        h.update(open(os.path.join(ROOT, "paper_2405_06856_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", dest="cpu_baseline", action="store_false")
    ap.add_argument("--no-search", dest="search", action="store_false",
                    help="leave the 1,000,000-request minimum-worker search (about 95 s) out")
    ap.add_argument("--mode", default="full",
                    choices=["full", "kernel", "round", "sim", "minworkers", "policies", "configs",
                             "aux"],
                    help="kernel: only warm-up + steps of the device-resident step (for profilers)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.mode == "kernel":
        run_kernel_only(args)
    elif args.mode == "round":
        run_round_only(args)
    elif args.mode == "sim":
        run_sim_only(args)
    elif args.mode == "minworkers":
        run_min_workers(args)
    elif args.mode == "policies":
        run_policies(args)
    elif args.mode == "configs":
        run_configs(args)
    elif args.mode == "aux":
        run_aux(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
