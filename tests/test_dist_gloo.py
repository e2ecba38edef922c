"""The multi-process measurement path (max over ranks, weak-scaling aggregate, sharding) with two
gloo ranks on CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2002_09049_gb300 import dist as dh


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        step_ms = [3.0, 5.0][rank]
        ms = dh.max_over_ranks(step_ms)
        dist.barrier()
        out[rank] = (ms, dh.aggregate_throughput(1e9, ms, world), dh.shard(21, world, rank))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for r in range(world):
        ms, value, sh = out[r]
        assert ms == 5.0                            # the slowest rank sets the time
        assert value == pytest.approx(2e9 / 5e-3)  # both replicas' units / slowest time
    assert out[0][2] == (0, 11) and out[1][2] == (11, 21)


def test_single_process_identity():
    assert dh.max_over_ranks(4.5) == 4.5
    assert dh.shard(5, 1, 0) == (0, 5)
    assert dh.world_from_env()[0] >= 1
