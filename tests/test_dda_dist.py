"""DDA for data densities other than N(0,1) (the paper's Sec. III-D assumes
the standard normal): the library's host solvers against the oracle's
(Laplace with unit variance; the empirical density of a histogram of the
normalised data).  CPU only: these entry points are host functions."""
import numpy as np
import pytest

import oracle as o
from paper_2109_03513_gb300 import esb, synth

FMTS = [(2, 0), (3, 1), (3, 2), (4, 0), (4, 1), (4, 2), (5, 1), (5, 2), (5, 3), (6, 2), (6, 3), (6, 4)]


@pytest.mark.parametrize("b,k", FMTS)
def test_laplace_alpha_star_matches_oracle(b, k):
    a, dda = esb.esb_alpha_star_dist(b, k, esb.ESB_DIST_LAPLACE)
    ao, ddao = o.alpha_star_laplace(b, k)
    assert abs(a - ao) <= 1e-6 * ao
    assert abs(dda - ddao) <= 1e-7 * ddao          # the oracle integrates numerically
    assert esb.esb_alpha_star_dist(b, k, esb.ESB_DIST_GAUSSIAN) == esb.esb_alpha_star(b, k)


@pytest.mark.parametrize("dist,signed", [("normal", True), ("laplace", True), ("half_normal", False)])
@pytest.mark.parametrize("b,k", [(3, 1), (4, 2), (5, 2), (6, 3), (4, 0)])
def test_histogram_alpha_star_matches_oracle(dist, signed, b, k):
    x = synth.distribution(dist, (1 << 20,), seed=b * 7 + k).numpy()
    _, st = o.calibrate(x, b, k, signed)
    c = o.histogram_abs(x, signed, st[0], st[1], 4096, 16.0)
    a, dda = esb.esb_alpha_star_hist(c, 16.0, b, k)
    ao, ddao = o.alpha_star_hist(c, 16.0, b, k)
    assert abs(a - ao) <= 1e-6 * ao
    assert abs(dda - ddao) <= 1e-9 * ddao


def test_histogram_of_laplace_data_finds_the_laplace_alpha_star():
    x = synth.laplace((1 << 22,), seed=9).numpy()
    _, st = o.calibrate(x, 4, 2, True)
    c = o.histogram_abs(x, True, st[0], st[1], 8192, 24.0)
    a, _ = esb.esb_alpha_star_hist(c, 24.0, 4, 2)
    assert abs(a - esb.esb_alpha_star_dist(4, 2, esb.ESB_DIST_LAPLACE)[0]) <= 0.01 * a


def test_dda_dist_host_validation():
    with pytest.raises(esb.EsbError):
        esb.esb_alpha_star_dist(4, 2, 7)
    with pytest.raises(esb.EsbError):
        esb.esb_alpha_star_hist(np.zeros(16), 8.0, 4, 2)          # no mass
    with pytest.raises(esb.EsbError):
        esb.esb_alpha_star_hist(np.ones(16), 0.0, 4, 2)
