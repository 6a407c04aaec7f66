"""Seeded synthetic inputs shared by the tests, bench.py and the oracle side.

Random numbers only -- this module holds none of the ESB arithmetic.  Every
generator runs on the CPU with an explicit torch.Generator seed, so the same
call yields the same bytes on any machine; callers copy to the device.
Shapes and distributions follow the paper's workloads (Sec. V-A): N(0,1)
stands in for mean-subtracted images and normalised weights, |N(0,1)| for
post-ReLU activations, Laplace(0,1) for heavy-tailed data, and He-initialised
weights N(0, sqrt(2/fan_in)) for random networks.
"""
from __future__ import annotations

import numpy as np
import torch


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator()
    g.manual_seed(int(seed))
    return g


def normal(shape, seed: int, std: float = 1.0, mean: float = 0.0) -> torch.Tensor:
    t = torch.randn(*shape, generator=_gen(seed), dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    if mean != 0.0:
        t.add_(mean)
    return t


def half_normal(shape, seed: int, std: float = 1.0) -> torch.Tensor:
    return normal(shape, seed, std).abs_()


def laplace(shape, seed: int, scale: float = 1.0) -> torch.Tensor:
    # inverse CDF of Laplace(0, scale) from U(-1/2, 1/2)
    u = torch.rand(*shape, generator=_gen(seed), dtype=torch.float64) - 0.5
    u = u.clamp(-0.5 + 1e-16, 0.5 - 1e-16)
    x = -scale * torch.sign(u) * torch.log1p(-2.0 * u.abs())
    return x.to(torch.float32)


def he_normal(shape, fan_in: int, seed: int) -> torch.Tensor:
    return normal(shape, seed, std=float(np.sqrt(2.0 / fan_in)))


def uniform_ints(shape, low: int, high: int, seed: int) -> np.ndarray:
    """Integers in [low, high) (numpy uint32), e.g. raw b-bit code patterns."""
    t = torch.randint(low, high, tuple(shape), generator=_gen(seed), dtype=torch.int64)
    return t.numpy().astype(np.uint32)


def distribution(name: str, shape, seed: int) -> torch.Tensor:
    if name == "normal":
        return normal(shape, seed)
    if name == "laplace":
        return laplace(shape, seed)
    if name == "half_normal":
        return half_normal(shape, seed)
    raise ValueError(name)
