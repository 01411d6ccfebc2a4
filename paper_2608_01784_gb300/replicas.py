"""Host logic of multi-GPU runs on one node: one process per GPU, each a
replica with its own seeded batch (the path shards by sequence and by token,
so ranks exchange no data); a barrier around the timed region and a
max-reduce of the timed durations are the only collectives.

Rank identity comes from the torchrun environment (RANK, WORLD_SIZE,
LOCAL_RANK).  The reductions run on whatever backend the caller initialised
(NCCL for the GPU arm, gloo for the host-only reference arm and the tests).
"""
from __future__ import annotations

import os
from dataclasses import dataclass


@dataclass(frozen=True)
class RankInfo:
    rank: int
    world: int
    local_rank: int


def rank_info(env=None) -> RankInfo:
    env = os.environ if env is None else env
    return RankInfo(rank=int(env.get("RANK", "0")),
                    world=int(env.get("WORLD_SIZE", "1")),
                    local_rank=int(env.get("LOCAL_RANK", "0")))


def rank_seed(seed: int, rank: int) -> int:
    """Seed of a replica's batch: distinct per rank, equal to `seed` on rank 0
    (so a 1-GPU run and rank 0 of an N-GPU run time the same batch)."""
    return seed + rank


def init(world: int, backend: str, device_index: int | None = None) -> None:
    if world <= 1:
        return
    import torch
    import torch.distributed as dist
    if backend == "nccl" and device_index is not None:
        torch.cuda.set_device(device_index)
    dist.init_process_group(backend=backend)


def finalize(world: int) -> None:
    if world <= 1:
        return
    import torch.distributed as dist
    if dist.is_initialized():
        dist.destroy_process_group()


def barrier(world: int, device=None) -> None:
    """All ranks reach this point (and, with a CUDA device, all their queued
    work has finished)."""
    import torch
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    if device is not None and getattr(device, "type", "cpu") == "cuda":
        torch.cuda.synchronize(device)


def max_over_ranks(x: float, world: int, device=None) -> float:
    """The largest value of x over all ranks (every rank gets it)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, world: int, ms: float) -> float:
    """Units per second of the whole job: every rank processed
    `units_per_rank` units within the slowest rank's `ms` milliseconds."""
    return units_per_rank * world / (ms * 1e-3)
