import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libesb.so")


def pytest_collection_modifyitems(config, items):
    try:
        import torch
        have_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        have_gpu = False
    if have_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


def read_golden(name):
    """Parse a whitespace fixture: '#' comments; returns a list of token lists."""
    rows = []
    with open(os.path.join(GOLDEN, name)) as fh:
        for line in fh:
            line = line.split("#", 1)[0].strip()
            if line:
                rows.append(line.split())
    return rows


def oracle_step_function(alpha, b, k, signed, rounding):
    """The projection of every fp32 value as a step function, from the oracle
    alone.  For x >= 0 the projected value is non-decreasing in x, so it is
    fixed by the bit patterns T[j] of the smallest x >= 0 whose projection
    reaches the (j+1)-th non-negative set element (bisection over fp32 bit
    patterns with the oracle's projection), plus the oracle's code of one
    value of each bucket for positive and for negative x, and of NaN.
    Returns (T int64 [L-1], pos codes [L], neg codes [L], NaN code)."""
    import numpy as np

    import oracle as o

    q = o.set_nonneg(b, k)
    L = len(q)
    lo = np.zeros(L - 1, np.int64)
    hi = np.full(L - 1, 0x7F800000, np.int64)
    while (hi - lo > 1).any():
        act = hi - lo > 1
        mid = (lo + hi) // 2
        v = o.project_values(mid.astype(np.uint32).view(np.float32), alpha, b, k, True, rounding)
        up = v >= q[1:]
        hi = np.where(act & up, mid, hi)
        lo = np.where(act & ~up, mid, lo)
    reps = np.concatenate([np.zeros(1, np.uint32), hi.astype(np.uint32)]).view(np.float32)
    pos = o.project_codes(reps, alpha, b, k, signed, rounding).astype(np.int64)
    neg = o.project_codes(-reps, alpha, b, k, signed, rounding).astype(np.int64)
    nan = int(o.project_codes(np.array([np.nan], np.float32), alpha, b, k, signed, rounding)[0])
    return hi, pos, neg, nan


def step_function_codes(bits, step):
    """Codes of the fp32 values with bit patterns `bits` (int64 tensor, 0 ..
    2^32 - 1, any device) by the step function of oracle_step_function."""
    import torch

    T, pos, neg, nan = step
    dev = bits.device
    T = torch.as_tensor(T, device=dev)
    pos = torch.as_tensor(pos, device=dev)
    neg = torch.as_tensor(neg, device=dev)
    a = bits & 0x7FFFFFFF
    j = torch.searchsorted(T, a, right=True)
    e = torch.where(((bits >> 31) & 1).bool(), neg[j], pos[j])
    return torch.where(a > 0x7F800000, torch.full_like(e, nan), e)
