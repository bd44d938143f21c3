"""Host-side logic of bench.py's multi-GPU path (one process per GPU, replicas
of the workload, max over ranks) on CPU: two gloo ranks on 127.0.0.1."""
import contextlib
import io
import os
import socket
import sys


ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        step_ms = [3.0, 5.0][rank]          # the slower rank decides
        m = bench.barrier_max(dist, step_ms, device="cpu")
        v = bench.whole_job_value(world, 1000, m)
        q.put((rank, m, v))
    finally:
        dist.destroy_process_group()


def test_two_rank_max_and_whole_job_value():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [5.0, 5.0]
    assert [r[2] for r in res] == [2 * 1000 / 0.005] * 2


def test_single_process_value():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.barrier_max(None, 7.5) == 7.5
    assert bench.whole_job_value(1, 4096 * 32768, 0.25) == 4096 * 32768 / 0.00025


def test_reference_arm_runs_on_rank0_only(monkeypatch):
    """Under torchrun only rank 0 runs the oracle and prints its line; the
    other ranks exit without work."""
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    out = io.StringIO()
    with contextlib.redirect_stdout(out):
        bench.run_reference(type("Args", (), dict(steps=1, warmup=3, gpus=2))())
    assert out.getvalue() == ""
