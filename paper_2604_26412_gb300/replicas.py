"""Replica bookkeeping for multi-GPU runs of the hot path.

The draft-attention path has no exchange step (caches, KV heads and
sequences are independent), so N GPUs run N independent replicas.  The only
cross-rank traffic is harness bookkeeping: a barrier and the maximum of the
ranks' timed durations, from which the whole-job rate is computed.  Works
with the gloo (CPU tensors) and nccl (CUDA tensors) backends.
"""
from __future__ import annotations

import torch


def _dist():
    import torch.distributed as dist
    return dist if dist.is_available() and dist.is_initialized() else None


def barrier() -> None:
    dist = _dist()
    if dist is not None:
        dist.barrier()


def max_over_ranks(x: float) -> float:
    dist = _dist()
    if dist is None or dist.get_world_size() == 1:
        return float(x)
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_step_per_rank: float, steps: int, world: int, max_ms: float) -> float:
    """Units processed by all ranks divided by the slowest rank's time (units/s)."""
    return units_per_step_per_rank * world * steps / (max_ms / 1e3)
