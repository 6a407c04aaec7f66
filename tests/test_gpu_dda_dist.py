"""GPU parity of the DDA for other data densities: the histogram of the
normalised magnitudes (bit-exact counts against the oracle), the Laplace
alpha* calibration and the empirical (histogram) calibration (alpha within
1e-6 of the oracle's chain on the same statistics)."""
import numpy as np
import pytest
import torch

import oracle as o
from paper_2109_03513_gb300 import esb, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


CASES = [
    # (dist, n, signed, (b, k), nbins, t_max)
    ("normal", (1 << 20) + 3, True, (4, 2), 8192, 16.0),
    ("laplace", 1 << 21, True, (5, 2), 4096, 24.0),
    ("half_normal", 300001, False, (4, 2), 8192, 16.0),
    ("normal_offset", 65536, True, (6, 3), 2048, 8.0),
]


def data(dist, n, seed):
    if dist == "normal_offset":
        return synth.normal((n,), seed=seed, mean=5.0, std=0.5)
    return synth.distribution(dist, (n,), seed=seed)


@pytest.mark.parametrize("dist,n,signed,bk,nbins,tmax", CASES)
def test_histogram_matches_oracle(dist, n, signed, bk, nbins, tmax):
    x = data(dist, n, seed=n % 101)
    f = esb.Fmt(bk[0], bk[1], signed)
    st = torch.zeros(3, dtype=torch.float64, device="cuda")
    esb.esb_calibrate_dda(x.cuda(), f, stats_out=st)
    x[7] = float("nan")                       # skipped
    x[11] = float("inf")                      # last bin
    counts = esb.esb_dda_histogram(x.cuda(), f, st, nbins=nbins, t_max=tmax)
    s = st.cpu().numpy()
    exp = o.histogram_abs(x.numpy(), signed, s[0], s[1], nbins, tmax)
    assert np.array_equal(counts.cpu().numpy().astype(np.uint64), exp)
    assert esb.esb_get_status() == 0


@pytest.mark.parametrize("dist,n,signed,bk,nbins,tmax", CASES)
def test_empirical_calibration_matches_oracle(dist, n, signed, bk, nbins, tmax):
    x = data(dist, n, seed=n % 97)
    f = esb.Fmt(bk[0], bk[1], signed)
    a, st, astar = esb.esb_calibrate_dda_empirical(x.cuda(), f, nbins=nbins, t_max=tmax)
    s = st.cpu().numpy()
    _, so = o.calibrate(x.numpy(), bk[0], bk[1], signed)
    assert abs(s[1] - so[1]) <= 1e-6 * so[1]
    # the oracle's chain on the device statistics: histogram, alpha*, alpha
    c = o.histogram_abs(x.numpy(), signed, s[0], s[1], nbins, tmax)
    ao, _ = o.alpha_star_hist(c, tmax, *bk)
    assert abs(astar - ao) <= 1e-6 * ao
    alpha_o = float(np.float32(ao * (s[1] + 1e-7)))
    assert abs(float(a.item()) - alpha_o) <= 1e-6 * alpha_o


@pytest.mark.parametrize("bk", [(3, 1), (4, 2), (6, 3)])
def test_laplace_calibration_matches_oracle(bk):
    x = synth.laplace((1 << 20,), seed=bk[0])
    f = esb.Fmt(bk[0], bk[1], True)
    a, _ = esb.esb_calibrate_dda_dist(x.cuda(), f, esb.ESB_DIST_LAPLACE)
    _, so = o.calibrate(x.numpy(), bk[0], bk[1], True)
    ao, _ = o.alpha_star_laplace(*bk)
    alpha_o = float(np.float32(ao * (so[1] + 1e-7)))
    assert abs(float(a.item()) - alpha_o) <= 1e-6 * alpha_o
