"""Host logic of running the hot path on several GPUs as independent replicas.

Every step of the path (score, split, pack, block, unpack) works on one image
at a time: the split ranks an image's own tokens (Sec. 2.3), the packed rows
of an image attend only to that image's joint text + image sequence, and
unpack writes back that image's grid. So the path shards by image with no
exchange step. N processes (one per GPU, launched by torchrun) each take a
contiguous slice of the global batch; the only cross-rank operations are a
barrier and the maximum of the timed region, both outside the data path.

Nothing here touches a GPU: the same functions run under gloo on the CPU.
"""
from __future__ import annotations

import os


def env_rank_world() -> tuple[int, int, int]:
    """(rank, world size, local rank) from the torchrun environment (1 process when unset)."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def image_slice(n_images: int, rank: int, world: int) -> tuple[int, int]:
    """The contiguous images [b0, b1) of the global batch that `rank` processes.

    Slices of neighbouring ranks abut, cover the batch exactly once and differ
    in size by at most one image.
    """
    if world < 1 or not 0 <= rank < world or n_images < 0:
        raise ValueError(f"image_slice: n_images={n_images} rank={rank} world={world}")
    return n_images * rank // world, n_images * (rank + 1) // world


def max_over_ranks(value: float, device: str = "cpu") -> float:
    """The largest `value` over all ranks (the value itself with one process).

    `device` is where the reduction tensor lives: "cuda" under NCCL, "cpu"
    under gloo.
    """
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_throughput(units_per_rank: float, world: int, ms_max: float) -> float:
    """Units per second of the whole job: all ranks' units over the slowest rank's time."""
    if ms_max <= 0:
        raise ValueError("whole_job_throughput: the time must be positive")
    return units_per_rank * world / (ms_max * 1e-3)
