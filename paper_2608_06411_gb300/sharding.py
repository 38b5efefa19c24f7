"""Image sharding across ranks (one process per GPU).

Images are independent units of the pruning path, so a batch is split into contiguous
blocks of images, one block per rank, and nothing is exchanged on the data path.  The
only collective is the max over ranks of a scalar (elapsed time) for reporting.
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
