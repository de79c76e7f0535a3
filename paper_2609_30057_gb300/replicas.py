"""Replica bookkeeping for multi-GPU benchmarking.

The paper's unit of parallelism is independent benchmarking commands
(command concurrency per GPU, Section 6.1); a command never spans GPUs, and
multi-GPU candidates are future work (Section 7).  So N GPUs run N
independent replicas: no collective sits on the data path.  The only
cross-rank operations are control: a barrier around the timed region and the
maximum of the per-rank elapsed times, so the reported throughput is the
units all ranks processed divided by the slowest rank's time.

Works with any torch.distributed backend (NCCL on GPUs, gloo on CPU tests).
"""
from __future__ import annotations


def rank_world() -> tuple[int, int, int]:
    """(rank, world_size, local_rank) from the torchrun environment (1 rank if absent)."""
    import os
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def barrier(dist) -> None:
    if dist is not None and dist.is_initialized():
        dist.barrier()


def max_over_ranks(dist, value: float, device=None) -> float:
    """Largest `value` over all ranks (the slowest replica's time)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(dist, value: float, device=None) -> float:
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def aggregate_throughput(units_per_rank: float, world: int, slowest_elapsed_s: float) -> float:
    """Whole-job throughput: units processed by all ranks over the slowest rank's time."""
    if slowest_elapsed_s <= 0:
        raise ValueError("elapsed time must be positive")
    return units_per_rank * world / slowest_elapsed_s
