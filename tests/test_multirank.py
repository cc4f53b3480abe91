"""The multi-process path of bench.py on CPU: two gloo ranks (one process each, as torchrun
launches them) read their rank from the environment, take the maximum of their step times and
turn it into the whole-job rate, exactly as the GPU run does over NCCL. The method itself has no
data-path collective (replicas only)."""
import os
import socket
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    r, w, local = bench.rank_env()
    ms = 10.0 + 5.0 * r                              # rank r's step time
    worst = bench.max_over_ranks(ms, w, torch.device("cpu"))
    results[r] = (r, w, local, worst, bench.job_rate(1000, w, worst))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_ranks_take_the_slowest_time(world):
    mgr = mp.get_context("spawn").Manager()       # no fork of a multi-threaded parent
    results = mgr.dict()
    mp.spawn(_worker, args=(world, _free_port(), results), nprocs=world, join=True)
    assert sorted(results.keys()) == list(range(world))
    slowest = 10.0 + 5.0 * (world - 1)
    for r in range(world):
        rank, w, local, worst, rate = results[r]
        assert (rank, w, local) == (r, world, r)
        assert worst == slowest                      # every rank sees the job's time
        assert rate == pytest.approx(world * 1000 / (slowest * 1e-3))


def test_single_process_needs_no_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1, torch.device("cpu")) == 3.5
    assert bench.job_rate(16384, 1, 0.1) == pytest.approx(16384 / 1e-4)
