"""Replica bookkeeping for runs of the pruned prefill on several GPUs.

The forward of one sequence never reads another sequence (the pruning of
Sec. 3 keeps or drops positions within a sequence), so N GPUs run N
independent replicas: each rank prefills its own batch of B sequences, with
no collective on the data path.  What the ranks share is host-side
bookkeeping: which tokens each rank draws, the barrier around the timed
region, the step time (the slowest rank's) and the job throughput (every
rank's tokens).  `dist` is torch.distributed (any backend) or None for one
process.
"""
from __future__ import annotations


def rank_token_seed(base_seed: int, rank: int) -> int:
    """Seed of rank `rank`'s token batch: distinct per rank, fixed per run."""
    return base_seed + rank


def barrier(dist=None, sync=None) -> None:
    """Every rank reaches this point before any goes on (device work drained
    first and after, when `sync` is given)."""
    if sync is not None:
        sync()
    if dist is not None:
        dist.barrier()
    if sync is not None:
        sync()


def max_over_ranks(x: float, dist=None, device="cpu") -> float:
    """The largest `x` over all ranks (the step time of the slowest replica)."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(world: int, B: int, L: int, ms_per_step: float) -> float:
    """Prefill throughput of the whole job: world * B * L tokens per step."""
    return world * B * L / (ms_per_step / 1e3)
