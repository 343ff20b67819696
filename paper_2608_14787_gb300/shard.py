"""Multi-rank host logic of the path.

Draft blocks (batch rows) are independent units -- the staleness counter D is
per row -- so the path shards by block with no data-path collective: each
rank (one process per GPU) runs whole rounds on its own contiguous range of
blocks.  The only cross-rank exchanges are host-side aggregates: the
agreement counters of Sec. 3.2 (the numerators and denominators of
StrictToken, Eq. 1, and FullPrefix, Eq. 2, per threshold pair) and timings.
They go through torch.distributed (gloo on CPU, NCCL between GPUs).
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def block_range(n_blocks: int, rank: int, world: int) -> tuple[int, int]:
    """The contiguous, balanced range [start, end) of blocks owned by `rank`."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside a world of {world}")
    if n_blocks < 0:
        raise ValueError("n_blocks < 0")
    return n_blocks * rank // world, n_blocks * (rank + 1) // world


def max_over_ranks(value: float, device=None) -> float:
    """The maximum of a per-rank float (e.g. a step time) over all ranks."""
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_counters(acc: torch.Tensor) -> torch.Tensor:
    """Agreement counters [n_tau, 4] (int64: sum min(K, L), sum K, count of
    K <= L, count of skipped blocks) summed over all ranks; returns a new tensor."""
    out = acc.clone()
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(out, op=dist.ReduceOp.SUM)
    return out


def agreement_rates(acc: torch.Tensor) -> list[tuple[float, float, int]]:
    """Per threshold pair: (StrictToken, FullPrefix, skipped blocks) from the
    summed counters -- the fraction of skipped tokens the shadow strict verifier
    also accepted (Eq. 1) and the fraction of skipped blocks whose whole prefix
    it accepted (Eq. 2); NaN where nothing was skipped."""
    rows = []
    for a0, a1, a2, a3 in acc.to(torch.int64).tolist():
        st = a0 / a1 if a1 > 0 else float("nan")
        fp = a2 / a3 if a3 > 0 else float("nan")
        rows.append((st, fp, int(a3)))
    return rows
