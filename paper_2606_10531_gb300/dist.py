"""Multi-rank plumbing for runs with one process per GPU (torchrun).

The LC-VQ layer step partitions into independent problems (one decoder layer, or one linear,
per unit), so ranks shard the units and never exchange data on the hot path; the only
communication is a barrier around the timed region and the maximum of the per-rank times.
"""
from __future__ import annotations

import os


def rank_world():
    """(rank, local_rank, world_size) from the torchrun environment; (0, 0, 1) without it."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def shard(n_units: int, rank: int, world: int) -> range:
    """Contiguous, balanced block of unit indices owned by `rank` (sizes differ by at most one)."""
    if world < 1 or not 0 <= rank < world or n_units < 0:
        raise ValueError("bad shard arguments")
    base, extra = divmod(n_units, world)
    start = rank * base + min(rank, extra)
    return range(start, start + base + (1 if rank < extra else 0))


def init(backend: str, device=None):
    """Initialise the default process group when WORLD_SIZE > 1 (127.0.0.1 rendezvous from the env)."""
    import torch.distributed as dist
    _, _, world = rank_world()
    if world > 1 and not dist.is_initialized():
        kw = {"device_id": device} if (backend == "nccl" and device is not None) else {}
        dist.init_process_group(backend, **kw)
    return world


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


def max_over_ranks(value: float, device="cpu") -> float:
    """Maximum of a per-rank float over all ranks (identity on one rank)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def finalize():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.destroy_process_group()
