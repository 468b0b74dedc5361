"""Data-parallel replicas of the drafting hot path: one process per GPU.

Algorithm 1 drafts and verifies every request's block on its own: no value
crosses from one request to another. N GPUs therefore run N independent
replicas of the whole path, each on its own requests, with no collective on
the data path. The only cross-rank communication is in the launcher: a
barrier around the timed region and a max-reduction of the per-rank times.

This module is that launcher logic, shared by ``bench.py`` and the tests:
which requests a rank owns, the per-rank seed of its synthetic inputs, and
how per-rank timings combine into one whole-job throughput. It is pure host
code; the ranks talk through ``torch.distributed`` (NCCL on GPUs, gloo on the
CPU test path).
"""
from __future__ import annotations

import os
from typing import List, Tuple

__all__ = ["RankInfo", "rank_info", "request_range", "replica_seed", "max_over_ranks", "job_throughput",
           "barrier"]

# Distance between the input seeds of consecutive ranks; larger than any seed
# offset the workloads use, so no two ranks draw the same inputs.
SEED_STRIDE = 1000


class RankInfo(Tuple[int, int, int]):
    """(world, rank, local_rank) as read from the launcher's environment."""

    @property
    def world(self) -> int:
        return self[0]

    @property
    def rank(self) -> int:
        return self[1]

    @property
    def local(self) -> int:
        return self[2]


def rank_info() -> RankInfo:
    """World size, global rank and local rank from the environment torchrun
    sets (a single process when they are absent)."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    if world < 1 or not (0 <= rank < world):
        raise ValueError(f"bad rank {rank} for world size {world}")
    return RankInfo((world, rank, local))


def request_range(total: int, world: int, rank: int) -> Tuple[int, int]:
    """[start, stop) of the requests rank ``rank`` owns when ``total`` requests
    are split over ``world`` replicas (strong scaling). Shards are contiguous,
    disjoint, cover every request and differ in size by at most one."""
    if total < 0 or world < 1 or not (0 <= rank < world):
        raise ValueError("bad request split")
    base, extra = divmod(total, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)


def replica_seed(seed: int, rank: int) -> int:
    """Seed of rank ``rank``'s synthetic inputs (weak scaling: every replica
    drafts its own batch of the same shape). Rank 0 keeps the base seed, so a
    one-GPU run and rank 0 of an N-GPU run see the same inputs."""
    return seed + SEED_STRIDE * rank


def max_over_ranks(value: float, device=None) -> float:
    """The maximum of ``value`` over all ranks (``value`` itself when no
    process group is up). ``device`` is where the reduction tensor lives:
    a CUDA device under NCCL, the CPU under gloo."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier() -> None:
    """A barrier over all ranks, a no-op for a single process."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()


def job_throughput(units_per_rank: List[float], ms_max: float) -> float:
    """Whole-job units per second: all the units every rank processed over the
    slowest rank's wall time (the job is done when the last replica is)."""
    if ms_max <= 0:
        raise ValueError("non-positive time")
    return float(sum(units_per_rank)) / (ms_max * 1e-3)
