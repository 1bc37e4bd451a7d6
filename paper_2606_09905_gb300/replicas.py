"""Host logic of the multi-GPU benchmark path: independent replicas.

The paper's method is single-device; its GEMM, conv and attention shard into
independent problems with no exchange step, so running on N GPUs means N
replicas of the same step (one process per GPU, launched by
torch.distributed.run) and no data-path collective.  The only communication
is for measurement: a barrier around the timed region and the maximum of the
per-rank times, from which the whole-job rate is computed.  The functions
here take the process group as given, so the same code runs over NCCL on
GPUs and over gloo in the CPU tests.
"""
from __future__ import annotations

import os


def env_int(name: str, default: int) -> int:
    try:
        return int(os.environ.get(name, default))
    except ValueError:
        return default


def rank_world_local() -> tuple[int, int, int]:
    """(RANK, WORLD_SIZE, LOCAL_RANK) from the launcher's environment."""
    return env_int("RANK", 0), env_int("WORLD_SIZE", 1), env_int("LOCAL_RANK", 0)


def replica_seed(rank: int) -> int:
    """Each replica draws its own synthetic inputs."""
    return int(rank)


def max_over_ranks(value: float, device=None) -> float:
    """The maximum of `value` over all ranks (the value itself without a
    process group).  `device` is where the reduction tensor lives (a CUDA
    device for NCCL, None for gloo)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, seconds_max: float, world: int) -> float:
    """Units per second of the whole job: every rank processes
    `units_per_rank` units, and the slowest rank's time bounds the job."""
    if seconds_max <= 0:
        raise ValueError("timed region must be positive")
    return world * units_per_rank / seconds_max


def barrier() -> None:
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()
