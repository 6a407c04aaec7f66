"""The seeded input generators (CPU): same seed, same bytes; the moments of
each distribution the workloads use (N(0,1), |N(0,1)|, Laplace(0,1), He
initialisation) within sampling error at 2^20 values."""
import math

import numpy as np
import pytest

from paper_2109_03513_gb300 import synth

N = 1 << 20


def test_same_seed_same_bytes():
    for name in ("normal", "half_normal", "laplace"):
        a = synth.distribution(name, (N,), seed=7).numpy()
        b = synth.distribution(name, (N,), seed=7).numpy()
        c = synth.distribution(name, (N,), seed=8).numpy()
        assert a.dtype == np.float32 and a.shape == (N,)
        assert np.array_equal(a.view(np.uint32), b.view(np.uint32))
        assert not np.array_equal(a, c)
    u = synth.uniform_ints((64, 33), 0, 16, seed=3)
    assert u.dtype == np.uint32 and u.shape == (64, 33) and u.min() >= 0 and u.max() < 16
    assert np.array_equal(u, synth.uniform_ints((64, 33), 0, 16, seed=3))


@pytest.mark.parametrize("name,mean,std,mean_abs", [
    ("normal", 0.0, 1.0, math.sqrt(2 / math.pi)),
    ("half_normal", math.sqrt(2 / math.pi), math.sqrt(1 - 2 / math.pi), math.sqrt(2 / math.pi)),
    ("laplace", 0.0, math.sqrt(2.0), 1.0),
])
def test_moments(name, mean, std, mean_abs):
    x = synth.distribution(name, (N,), seed=11).numpy().astype(np.float64)
    se = std / math.sqrt(N)
    assert abs(x.mean() - mean) < 6 * se
    assert abs(x.std() - std) < 0.01 * std
    assert abs(np.abs(x).mean() - mean_abs) < 0.01 * mean_abs
    if name == "half_normal":
        assert x.min() >= 0.0


def test_he_normal_scale():
    fan_in = 576
    w = synth.he_normal((N,), fan_in=fan_in, seed=2).numpy().astype(np.float64)
    assert abs(w.std() - math.sqrt(2.0 / fan_in)) < 0.01 * math.sqrt(2.0 / fan_in)
    assert abs(w.mean()) < 6 * math.sqrt(2.0 / fan_in) / math.sqrt(N)
