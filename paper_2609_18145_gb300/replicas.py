"""Host-side logic of running the mixing stack as independent replicas, one
process per GPU.

Samples of the rotated-hypercube stack never exchange data (every link stays
inside its sample), so N GPUs run N independent batches: no collective is on
the data path.  torch.distributed is used only to line the ranks up before
and after a timed region and to take the slowest rank's time.
"""
from __future__ import annotations

import os

import torch
import torch.distributed as dist


def env_world():
    """(rank, local_rank, world_size) from the torchrun environment."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def init(backend: str) -> None:
    """Join the process group when launched with more than one rank."""
    _, _, world = env_world()
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)


def barrier() -> None:
    if dist.is_initialized():
        dist.barrier()


def max_over_ranks(value: float, device=None) -> float:
    """Largest value over all ranks (the slowest rank's time)."""
    if not dist.is_initialized():
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, device=None) -> float:
    if not dist.is_initialized():
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def batch_seed(base: int, rank: int) -> int:
    """Seed of this rank's activations: every replica draws its own batch
    (weights are shared and drawn from `base`)."""
    return base + 1000003 * (rank + 1)


def finish() -> None:
    if dist.is_initialized():
        dist.destroy_process_group()
