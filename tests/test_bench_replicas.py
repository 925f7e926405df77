"""The multi-GPU path of bench.py is replicas only (every rank runs the whole round
on its own GPU, no collective on the data path): its host logic -- the job's time is
the slowest rank's, the value counts every rank's rounds, and only rank 0 of the
reference arm does work -- checked with two gloo processes on the CPU."""

import io
import contextlib
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        per_rank_ms = [3.0, 5.5][rank]
        ms = bench.max_over_ranks(per_rank_ms)
        value = bench.job_throughput(world, 1000, ms / 1e3)
        out = io.StringIO()
        with contextlib.redirect_stdout(out):
            if rank == 1:  # the reference arm: ranks other than 0 print nothing
                bench.run_reference(bench.parse_args(["--impl", "reference", "--gpus", "2"]))
        q.put((rank, ms, value, out.getvalue()))
    finally:
        dist.destroy_process_group()


def test_replicas_take_the_slowest_rank_and_count_every_rank():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, value, printed in res:
        assert ms == 5.5                         # every rank sees the slowest time
        assert value == pytest.approx(2 * 1000 / 5.5e-3)
    assert res[1][3] == ""                       # rank 1 of the reference arm is silent


def test_single_process_is_its_own_job():
    import bench
    assert bench.max_over_ranks(4.25) == 4.25
    assert bench.job_throughput(1, 200, 0.5) == 400.0
