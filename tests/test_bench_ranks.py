"""bench.py's multi-rank logic on the CPU: world_size-2 gloo ranks run their
own replicas (no data-path collective); the timing reduction takes the max over
ranks and the job throughput counts every replica."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    local_ms = 100.0 + 50.0 * rank                 # rank 1 is the slowest replica
    ms = bench.max_over_ranks(local_ms, dist, torch.device("cpu"))
    out[rank] = (ms, bench.job_throughput(1e12, world, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_weak_scaling_gloo():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        ms, tf = res[rank]
        assert ms == 150.0                           # the max over ranks, seen by every rank
        assert abs(tf - 2 * 1e12 / 0.150 / 1e12) < 1e-9


def test_single_process_paths():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, None, None) == 3.5
    assert abs(bench.attn_flops(32768, 32768, 48) - 5.278e14) / 5.278e14 < 1e-3
    assert abs(bench.attn_flops(34816, 64, 48) - 2.19e12) / 2.19e12 < 1e-2
