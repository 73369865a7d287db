"""bench.py's N > 1 path on CPU: two gloo ranks, as torchrun would start them.

The path has no data-path collective (replicas only); what the ranks share is the timing
protocol: every rank reports its own step time and work, and the line carries the slowest
rank's time and the work of all ranks.  These tests run that host logic with world size 2
on the gloo backend, and check that the reference arm does its work on rank 0 only.
"""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        # rank r was slower by r ms and processed (r + 1) units
        ms, units = bench.job_totals(dist, 2.0 + rank, 100.0 * (rank + 1))
        single = bench.job_totals(None, 2.0 + rank, 100.0 * (rank + 1))
        q.put((rank, ms, units, single))
    finally:
        dist.destroy_process_group()


def test_job_totals_two_gloo_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, units, single in out:
        assert ms == 3.0            # the slowest rank's time
        assert units == 300.0       # the work of both ranks
        assert single == (2.0 + rank, 100.0 * (rank + 1))


def _reference_rank(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import io
    from contextlib import redirect_stdout
    import bench
    a = bench.parse(["--impl", "reference", "--workload", "tiny_v2", "--steps", "1", "--warmup", "0",
                     "--gpus", str(world)])
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.run_reference(a, bench.workload(a))
    q.put((rank, buf.getvalue()))


def test_reference_arm_prints_on_rank0_only():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_reference_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=300) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    import json
    assert out[1] == ""
    line = json.loads(out[0].strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == world and line["value"] > 0
