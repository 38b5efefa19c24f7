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


def _grad_worker(rank, world, port, out):
    import numpy as np
    from oracle import distill_oracle as DO
    from paper_2608_06411_gb300.sharding import allreduce_mean_grads
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    W, texts, visions, teachers = _tiny_problem()
    first, n = image_range(len(texts), world, rank)           # 3 samples: 2 on rank 0, 1 on rank 1
    loss, g = DO.loss_and_grads(texts[first:first + n], visions[first:first + n], teachers[first:first + n], W)
    grads = {k: torch.tensor(v) for k, v in g.items()}
    lt = torch.tensor([loss], dtype=torch.float64)
    total = allreduce_mean_grads(grads, n, lt)
    out[rank] = (total, float(lt.item()), {k: v.numpy() for k, v in grads.items()})
    dist.barrier()
    dist.destroy_process_group()


def _tiny_problem():
    import numpy as np
    rng = np.random.default_rng(21)
    D, Dh, dp, N = 8, 6, 4, 5
    W = {"wT1": rng.standard_normal((Dh, D)), "bT1": rng.standard_normal(Dh), "wT2": rng.standard_normal((Dh, Dh)),
         "bT2": rng.standard_normal(Dh), "wQ": rng.standard_normal((dp, Dh)), "wV1": rng.standard_normal((Dh, D)),
         "bV1": rng.standard_normal(Dh), "wV2": rng.standard_normal((Dh, Dh)), "bV2": rng.standard_normal(Dh),
         "wK": rng.standard_normal((dp, Dh))}
    W = {k: v / 3.0 for k, v in W.items()}
    texts = [rng.standard_normal((m, D)) for m in (3, 2, 4)]
    visions = [rng.standard_normal((N, D)) for _ in range(3)]
    teachers = [t / t.sum() for t in (rng.gamma(1.0, size=N) for _ in range(3))]
    return W, texts, visions, teachers


def test_two_gloo_ranks_average_distillation_gradients():
    import numpy as np
    from oracle import distill_oracle as DO
    world = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_grad_worker, args=(world, _free_port(), out), nprocs=world, start_method="spawn", join=True)
    W, texts, visions, teachers = _tiny_problem()
    loss, g = DO.loss_and_grads(texts, visions, teachers, W)   # the whole batch on one process
    for r in range(world):
        total, lr, gr = out[r]
        assert total == 3
        assert lr == pytest.approx(loss, rel=1e-12)
        for k in g:
            np.testing.assert_allclose(gr[k], g[k], rtol=1e-10, atol=1e-14)


def _leaving_rank_worker(rank, world, port, out):
    import datetime
    import time
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=5))
    dist.barrier()                              # both ranks are up
    if rank == 1:
        out[1] = "left"
        os._exit(0)                             # leaves between steps, without joining the next collective
    t0 = time.monotonic()
    try:
        max_over_ranks(1.0)
        out[0] = ("no error", time.monotonic() - t0)
    except Exception as e:                      # the collective's error is the failure signal
        out[0] = (type(e).__name__, time.monotonic() - t0)
    os._exit(0)                                 # the group is broken: skip its teardown


def test_a_rank_that_leaves_is_reported_not_waited_for():
    """A rank that leaves between steps: the other rank's next collective (the max over ranks
    that the benchmark takes) ends with an error within the process group's timeout."""
    import time
    world = 2
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    ctx = mp.start_processes(_leaving_rank_worker, args=(world, _free_port(), out), nprocs=world,
                             start_method="spawn", join=False)
    deadline = time.monotonic() + 120
    while not ctx.join(timeout=5):
        if time.monotonic() > deadline:
            for p in ctx.processes:
                p.kill()
            pytest.fail("ranks did not finish")
    assert out[1] == "left"
    name, waited = out[0]
    assert name != "no error"
    assert waited < 60
