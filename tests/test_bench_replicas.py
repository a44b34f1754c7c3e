"""Multi-GPU bench path on the CPU: replicas under a gloo process group.

The verify step does not shard, so N > 1 runs N independent replicas; the only
cross-rank operation is the maximum of the per-rank step times.
"""

import contextlib
import io
import os
import socket
import sys

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, step_ms, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.reduce_step_time(step_ms[rank], world, dist, "cpu")
        q.put((rank, ms, bench.job_throughput(64, ms, world)))
    finally:
        dist.destroy_process_group()


def test_replica_step_time_is_max_over_ranks():
    world = 2
    step_ms = [5.0, 7.5]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, step_ms, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs)
    got = sorted(q.get(timeout=5) for _ in range(world))
    for rank, ms, value in got:
        assert ms == max(step_ms)
        assert value == pytest.approx(world * 64 / (max(step_ms) * 1e-3))


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.reduce_step_time(3.25, 1) == 3.25
    assert bench.job_throughput(128, 2.0, 1) == pytest.approx(64000.0)


def test_reference_arm_prints_only_on_rank_zero(monkeypatch):
    """Under torchrun every rank but 0 exits without work or output."""
    import bench
    monkeypatch.setenv("RANK", "1")

    class A:
        workload, steps, warmup, gpus = "qwen3-8b", 1, 1, 2

    out = io.StringIO()
    with contextlib.redirect_stdout(out):
        bench.run_reference(A())
    assert out.getvalue() == ""
