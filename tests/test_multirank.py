"""Sharding by image across ranks: two gloo ranks on the CPU (no GPU involved)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2608_06411_gb300.sharding import image_range, max_over_ranks


def test_image_range_partitions_exactly():
    for total in (0, 1, 7, 64, 65):
        for ws in (1, 2, 3, 8):
            seen = []
            for r in range(ws):
                first, n = image_range(total, ws, r)
                seen.extend(range(first, first + n))
            assert seen == list(range(total))
    with pytest.raises(ValueError):
        image_range(10, 2, 2)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    first, n = image_range(128, world, rank)
    got = [None] * world
    dist.all_gather_object(got, (first, n))
    t = max_over_ranks(1.5 + rank)
    out[rank] = (got, t)
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_and_reduce():
    world = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, _free_port(), out), nprocs=world, start_method="spawn", join=True)
    for r in range(world):
        got, t = out[r]
        assert got == [(0, 64), (64, 64)]
        assert t == 2.5
