"""Image sharding across ranks (one process per GPU).

Images are independent units of the pruning path, so a batch is split into contiguous
blocks of images, one block per rank, and nothing is exchanged on the data path.  The
only collective there is the max over ranks of a scalar (elapsed time) for reporting.
Data-parallel training of the predictor (the distillation step) has a real exchange: the
gradients of every rank's samples are averaged over all ranks (allreduce_mean_grads).
"""
from __future__ import annotations


def image_range(total_images: int, world_size: int, rank: int) -> tuple:
    """(first image, number of images) of `rank`'s contiguous block; the blocks of all
    ranks cover 0..total_images-1 exactly once, sizes differing by at most one."""
    if world_size < 1 or not 0 <= rank < world_size or total_images < 0:
        raise ValueError("bad shard request")
    base, extra = divmod(total_images, world_size)
    first = rank * base + min(rank, extra)
    return first, base + (1 if rank < extra else 0)


def max_over_ranks(value: float, device=None) -> float:
    """Max of a scalar over all ranks of the default process group (the value itself when
    torch.distributed is not initialised)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def allreduce_mean_grads(grads: dict, local_samples: int, loss=None) -> int:
    """Data-parallel distillation step (the one place where ranks exchange data): each rank
    holds the loss and gradients of the mean over its own samples (map_distill_grad); after
    this call every rank holds those of the mean over all ranks' samples.  Each rank's
    tensors are weighted by its share of the samples, then summed over ranks: one all-reduce
    per tensor, in a fixed name order, in place.  Returns the total number of samples."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return int(local_samples)
    names = sorted(grads)
    dev = grads[names[0]].device if names else None
    n = torch.tensor([float(local_samples)], dtype=torch.float64, device=dev)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    total = int(n.item())
    if total == 0:
        return 0
    share = float(local_samples) / total
    for name in names:
        grads[name].mul_(share)
        dist.all_reduce(grads[name], op=dist.ReduceOp.SUM)
    if loss is not None:
        loss.mul_(share)
        dist.all_reduce(loss, op=dist.ReduceOp.SUM)
    return total
