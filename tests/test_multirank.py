"""The N > 1 host logic of bench.py on CPU ranks (gloo, world size 2): each
replica runs the whole workload, the job time is the slowest rank's, and the
value counts the units of every rank."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = [120.0, 150.0][rank]
    worst = bench.max_over_ranks(ms)
    value = bench.job_value(1_000_000_000, world, 10, worst)
    dist.barrier()
    q.put((rank, worst, value))
    dist.destroy_process_group()


def test_two_rank_replicas_report_max_time_and_job_value():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, worst, value in res:
        assert worst == 150.0
        assert value == pytest.approx(2 * 1e9 * 10 / 0.150 / 1e12)


def test_single_process_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_value(10 ** 12, 1, 1, 1000.0) == pytest.approx(1.0)
