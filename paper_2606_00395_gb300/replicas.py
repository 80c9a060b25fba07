"""Replica bookkeeping for multi-GPU runs of the layer benchmark (host logic only).

The layer is per-token data parallel and this library runs one process per GPU, each on its own
batch, with no collective on the data path (replicas, weak scaling).  What the ranks share is
the measurement: the job time is the slowest rank's time, and the whole-job throughput is all
ranks' tokens over that time.  The only collectives are a barrier and one max-reduction of a
scalar, on whatever process group the caller set up (NCCL on GPUs, gloo on the CPU)."""
from __future__ import annotations

import os
from typing import Optional, Tuple

import torch


def rank_env() -> Tuple[int, int, int]:
    """(RANK, WORLD_SIZE, LOCAL_RANK) from the launcher's environment; (0, 1, 0) without one."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def job_time_ms(local_ms: float, dist=None, device: Optional[torch.device] = None) -> float:
    """The job's time: the maximum of every rank's ``local_ms`` (itself without a group)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(local_ms)
    t = torch.tensor([float(local_ms)], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: int, world: int, job_ms: float) -> float:
    """Whole-job units per second: every rank's units over the slowest rank's time."""
    if job_ms <= 0:
        raise ValueError("job time must be positive")
    return units_per_rank * world / (job_ms / 1e3)
