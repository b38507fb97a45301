"""Host-side logic of the N-GPU run: one replica of the hot path per rank.

Token rows are independent on every step of the path (per-token rotation and
quantization, a GEMM whose rows depend only on their own codes, per-(token,
head) KV quantization), so N GPUs run N replicas, each on its own tokens,
with the weights replicated and no collective on the data path.  The only
communication is for measurement: a barrier around the timed region and the
maximum of the per-rank times.  The whole-job throughput is the units all
ranks processed divided by that maximum ("weak" scaling: the work per rank is
fixed as N grows).

Everything here runs on the process-group backend the caller initialised:
NCCL with CUDA tensors in bench.py, gloo with CPU tensors in the tests.
"""
from __future__ import annotations

from typing import Optional


def input_seed(base: int, rank: int) -> int:
    """Seed of rank `rank`'s synthetic inputs: distinct per rank, fixed per run."""
    return base + rank


def max_over_ranks(value: float, world: int, device: Optional[str] = None) -> float:
    """The maximum of `value` over all ranks (the value itself when world == 1)."""
    if world <= 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int) -> None:
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def whole_job_rate(units_per_rank: float, seconds_max: float, world: int) -> float:
    """Units per second of the whole job: every rank processed `units_per_rank`
    in at most `seconds_max` (the slowest rank sets the job's time)."""
    if seconds_max <= 0:
        raise ValueError("seconds_max must be positive")
    return world * units_per_rank / seconds_max
