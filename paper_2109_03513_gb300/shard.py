"""DDA calibration of a tensor split across ranks (Sec. III-D statistics,
data-parallel).

Each rank calibrates its own shard (esb_calibrate_dda's stats_out: mean,
spread, n -- the spread is the standard deviation for the symmetric set
and the root mean square for the non-negative one).  The whole tensor's
alpha follows from the shards' statistics by the law of total variance:

  mean = sum n_i mean_i / n
  symmetric:    n sigma^2 = sum n_i sigma_i^2 + sum n_i (mean_i - mean)^2
  non-negative: n rms^2   = sum n_i rms_i^2

and alpha = fl32(alpha* (spread + 1e-7)), the same on every rank.  The
exchange is two all-reduces of fp64 scalars (the mean first, so the second
sum has no cancellation).  This is the path's one collective; the
contraction itself shards by batch with no exchange.
"""
from __future__ import annotations

import math
from typing import Iterable

import numpy as np


def combine_dda_stats(shards: Iterable, signed: bool) -> tuple[float, float, float]:
    """(n, mean, spread) of the union of shards given per-shard
    (mean, spread, n) triples."""
    st = [(float(m), float(s), float(n)) for m, s, n in shards]
    n = sum(t[2] for t in st)
    if n <= 0:
        raise ValueError("no values in any shard")
    mean = sum(t[2] * t[0] for t in st) / n
    if signed:
        m2 = sum(t[2] * t[1] * t[1] + t[2] * (t[0] - mean) ** 2 for t in st)
    else:
        m2 = sum(t[2] * t[1] * t[1] for t in st)
    return n, mean, math.sqrt(max(m2, 0.0) / n)


def dda_alpha(alpha_star: float, spread: float) -> float:
    """alpha = fl32(alpha* (spread + 1e-7)) (Sec. III-D)."""
    return float(np.float32(alpha_star * (spread + 1e-7)))


def allreduce_dda_alpha(stats, alpha_star: float, signed: bool, group=None) -> tuple[float, float, float]:
    """alpha, mean and spread of the whole tensor from this rank's shard
    statistics (mean, spread, n), with torch.distributed all-reduces (any
    backend; fp64 on the host).  Returns (alpha, mean, spread); every rank
    gets the same values."""
    import torch
    import torch.distributed as dist

    m, s, n = (float(v) for v in (stats[0], stats[1], stats[2]))
    t = torch.tensor([n, n * m], dtype=torch.float64)
    dist.all_reduce(t, group=group)
    n_all, mean = float(t[0]), float(t[1]) / float(t[0])
    if signed:
        t2 = torch.tensor([n * s * s + n * (m - mean) ** 2], dtype=torch.float64)
    else:
        t2 = torch.tensor([n * s * s], dtype=torch.float64)
    dist.all_reduce(t2, group=group)
    spread = math.sqrt(max(float(t2[0]), 0.0) / n_all)
    return dda_alpha(alpha_star, spread), mean, spread


def shard_bounds(n: int, world: int, rank: int) -> tuple[int, int]:
    """Contiguous split of n values over world ranks (sizes differ by at most 1)."""
    return n * rank // world, n * (rank + 1) // world


def local_alpha_star(b: int, k: int) -> float:
    """alpha*(b, k) from libesb (host computation, no device needed)."""
    from . import esb
    return esb.esb_alpha_star(b, k)[0]


__all__ = ["combine_dda_stats", "dda_alpha", "allreduce_dda_alpha", "shard_bounds", "local_alpha_star"]
