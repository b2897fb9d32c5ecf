"""Host logic of the multi-GPU bench (replicas, weak scaling) with world_size 2 gloo
ranks on CPU: per-rank streams differ, and the reported time is the slowest rank's."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2607_12287_gb300 import synth
    wl = bench.replica_workload(synth.WORKLOADS["so400m_224_1view"], rank)
    first = next(wl.frames(1))
    slowest = bench.max_over_ranks(10.0 + rank, dist, "cpu")
    out[rank] = (slowest, wl.seed, int(first.sum()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks():
    world = 2
    out = mp.Manager().dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    assert out[0][0] == out[1][0] == 11.0
    assert out[0][1] != out[1][1]
    assert out[0][2] != out[1][2]  # different camera streams per replica


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(3.5, None) == 3.5
    from paper_2607_12287_gb300 import synth
    wl = synth.WORKLOADS["so400m_224_1view"]
    assert bench.replica_workload(wl, 0) is wl
