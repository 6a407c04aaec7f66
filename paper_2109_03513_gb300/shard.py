"""DDA calibration of a tensor split across ranks (Sec. III-D statistics,
data-parallel).

Each rank calibrates its own shard (esb_calibrate_dda's stats_out: mean,
spread, n).  The ranks exchange those three numbers (one all-gather), and
every rank combines all of them with libesb's esb_dda_combine (law of total
variance in fp64, then alpha = fl32(alpha* (spread + 1e-7))), so every rank
gets the same alpha.  This module only moves the numbers; the arithmetic is
in the library.  It is the path's one collective: the contraction itself
shards by batch with no exchange.
"""
from __future__ import annotations

from typing import Iterable

from . import esb


def combine_dda_stats(shards: Iterable, f: esb.Fmt) -> tuple[float, float, float, float]:
    """(alpha, mean, spread, n) of the union of shards given per-shard
    (mean, spread, n) triples."""
    return esb.esb_dda_combine(shards, f)


def allreduce_dda_alpha(stats, f: esb.Fmt, group=None) -> tuple[float, float, float]:
    """alpha, mean and spread of the whole tensor from this rank's shard
    statistics (mean, spread, n): all-gather the triples with
    torch.distributed (any backend), then combine them on the host.  Returns
    (alpha, mean, spread); every rank gets the same values."""
    import torch
    import torch.distributed as dist

    mine = torch.tensor([float(stats[0]), float(stats[1]), float(stats[2])], dtype=torch.float64)
    parts = [torch.zeros(3, dtype=torch.float64) for _ in range(dist.get_world_size(group))]
    dist.all_gather(parts, mine, group=group)
    a, mean, spread, _ = esb.esb_dda_combine([p.tolist() for p in parts], f)
    return a, mean, spread


def shard_bounds(n: int, world: int, rank: int) -> tuple[int, int]:
    """Contiguous split of n values over world ranks (sizes differ by at most 1)."""
    return n * rank // world, n * (rank + 1) // world


__all__ = ["combine_dda_stats", "allreduce_dda_alpha", "shard_bounds"]
