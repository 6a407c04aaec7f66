"""Sharded DDA calibration on CPU ranks (gloo, world size 2): each rank
calibrates its shard with the oracle, the shards' statistics are combined
with one torch.distributed all-gather and libesb's esb_dda_combine, and
every rank must get the alpha the oracle computes on the whole tensor
(Sec. III-D)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle as o
from paper_2109_03513_gb300 import esb, shard, synth

CASES = [
    # (dist, n, b, k, signed)
    ("normal_offset", 100003, 4, 2, True),     # odd n: uneven split; |mean| = 3 sigma
    ("half_normal", 65536, 4, 2, False),
    ("laplace", 40001, 6, 3, True),
]


def _data(name, n):
    if name == "normal_offset":
        return (synth.normal((n,), seed=11).numpy() + 3.0).astype(np.float32)
    if name == "half_normal":
        return synth.half_normal((n,), seed=12).numpy()
    return synth.laplace((n,), seed=13).numpy()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, case, out_path):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    name, n, b, k, signed = case
    x = _data(name, n)
    lo, hi = shard.shard_bounds(n, world, rank)
    _, st = o.calibrate(x[lo:hi], b, k, signed)
    a, mean, spread = shard.allreduce_dda_alpha(st, esb.Fmt(b, k, signed))
    np.save(f"{out_path}.{rank}.npy", np.array([a, mean, spread], dtype=np.float64))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("case", CASES)
def test_sharded_dda_matches_whole_tensor(case, tmp_path):
    world = 2
    out = str(tmp_path / "res")
    mp.spawn(_rank, args=(world, _free_port(), case, out), nprocs=world, join=True)
    name, n, b, k, signed = case
    a_ref, st_ref = o.calibrate(_data(name, n), b, k, signed)
    res = [np.load(f"{out}.{r}.npy") for r in range(world)]
    assert res[0][0] == res[1][0]                         # identical alpha on every rank
    for a, mean, spread in res:
        assert abs(a - a_ref) <= 1e-6 * a_ref
        assert abs(mean - st_ref[0]) <= 1e-9 * max(abs(st_ref[0]), st_ref[1])
        assert abs(spread - st_ref[1]) <= 1e-9 * st_ref[1]


def test_combine_is_exact_on_host():
    # three uneven shards, no process group: the host-side combine alone
    x = _data("normal_offset", 30011)
    cuts = [0, 7000, 7001, 30011]
    stats = [o.calibrate(x[cuts[i]:cuts[i + 1]], 4, 2, True)[1] for i in range(3)]
    a, mean, spread, n = shard.combine_dda_stats(stats, esb.Fmt(4, 2, True))
    a_ref, st_ref = o.calibrate(x, 4, 2, True)
    assert n == x.size
    assert abs(a - a_ref) <= 1e-6 * a_ref
    assert abs(mean - st_ref[0]) <= 1e-9 * abs(st_ref[0])
    assert abs(spread - st_ref[1]) <= 1e-9 * st_ref[1]
