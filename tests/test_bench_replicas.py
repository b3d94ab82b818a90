"""The multi-replica path of bench.py on CPU: two gloo ranks (world size 2) agree on the slowest
replica's step time, and the job's throughput counts every replica's tokens.  No GPU."""
from __future__ import annotations

import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank: int, world: int, port: int, values, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    out[rank] = bench.max_over_ranks(values[rank])
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_step():
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    values = [4310.5, 4402.25]
    mp.spawn(_worker, args=(2, _free_port(), values, out), nprocs=2, join=True)
    assert out[0] == out[1] == max(values)


def test_single_process_and_throughput():
    import bench

    assert bench.max_over_ranks(123.0) == 123.0  # no process group: unchanged
    assert bench.job_tokens_per_s(64, 4000.0, 1) == pytest.approx(16000.0)
    assert bench.job_tokens_per_s(64, 4000.0, 8) == pytest.approx(128000.0)  # replicas add up
