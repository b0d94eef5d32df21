"""Host side of multi-GPU runs: one process per GPU, each over its own
heads (weak scaling, heads are independent), no collective on the data path.

Only the timing uses the process group: a barrier around the timed region
and the maximum of the ranks' times. These helpers are backend-agnostic
(NCCL on GPUs, gloo in the CPU tests).
"""
from __future__ import annotations

import torch

from .workloads import Workload


def rank_workload(wl: Workload, rank: int) -> Workload:
    """Each rank draws its own inputs (seed offset by rank): the job is
    world_size independent copies of the workload."""
    return wl.with_(seed=wl.seed + 100 * rank)


def world_size() -> int:
    d = torch.distributed
    return d.get_world_size() if d.is_available() and d.is_initialized() else 1


def barrier():
    if world_size() > 1:
        torch.distributed.barrier()


def max_over_ranks(value: float, device=None) -> float:
    """The slowest rank's value (the job ends when the last rank ends)."""
    if world_size() <= 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, tokens_per_rank: int, ms_per_step: float):
    """Whole-job tokens/s: every rank's tokens over the slowest rank's time."""
    return world * tokens_per_rank / (ms_per_step / 1e3)
