"""The multi-rank bookkeeping of bench.py on CPU (gloo, world size 2).

On N GPUs every rank decodes its own batch (weak scaling, no collective on
the data path); the job time is the slowest rank's and the throughput counts
every rank's bytes.
"""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = 100.0 + 50.0 * rank  # rank 1 is slower
    slowest = bench.slowest_rank_ms(ms, torch.device("cpu"))
    results[rank] = (slowest, bench.job_throughput(1_000_000_000, 10, world, slowest))
    dist.barrier()
    dist.destroy_process_group()


def test_slowest_rank_and_job_throughput_gloo_world2():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    results = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, results)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    for r in range(2):
        slowest, gbps = results[r]
        assert slowest == pytest.approx(150.0)
        assert gbps == pytest.approx(2 * 10 * 1e9 / 0.150 / 1e9)


def test_single_process_is_identity():
    import bench
    assert bench.slowest_rank_ms(12.5, torch.device("cpu")) == 12.5
    assert bench.job_throughput(10**9, 1, 1, 1000.0) == pytest.approx(1.0)
