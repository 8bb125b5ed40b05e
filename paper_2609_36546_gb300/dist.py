"""Request-level data parallelism across GPUs (host side).

The verify step is independent per request (Sec. 3.2.3: requests only share
the two models), so ranks take disjoint request ranges and run the step with
no exchange on the data path.  The only cross-rank step is the batch mean of
the source-split objective, which needs the numerators and denominators of
every shard: ``combine_loss`` all-reduces them (six scalars) after the step.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def shard_range(n: int, rank: int, world: int) -> range:
    """Contiguous block of ``n`` items owned by ``rank`` (sizes differ by <= 1)."""
    base, extra = divmod(n, world)
    lo = rank * base + min(rank, extra)
    return range(lo, lo + base + (1 if rank < extra else 0))


def combine_loss(out8: torch.Tensor, group=None) -> torch.Tensor:
    """All-reduce the per-shard loss record of ipd_split_loss.

    out8 = [loss, sum_on, sum_off, n_on, n_off, intervention_ratio, numer,
    denom]; the combined record has loss = sum(numer) / sum(denom) and the
    intervention ratio of all shards together."""
    v = out8.detach().to(torch.float64).clone()
    part = torch.stack([v[1], v[2], v[3], v[4], v[6], v[7]])
    dist.all_reduce(part, op=dist.ReduceOp.SUM, group=group)
    sum_on, sum_off, n_on, n_off, numer, denom = part.tolist()
    nt = n_on + n_off
    return torch.tensor([numer / denom if denom > 0 else 0.0, sum_on, sum_off, n_on, n_off,
                         n_off / nt if nt > 0 else 0.0, numer, denom], dtype=torch.float64)
