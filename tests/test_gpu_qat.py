"""GPU parity of the quantisation-aware training kernels (Algorithm 1 with
the DN and EMA of Sec. III-D) against the CPU oracle: DN + projection
(bit-exact codes and fake-quantised values), the straight-through + DN
backward (1e-6 relative), and the moving average of the statistics."""
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


def u32(t):
    return t.cpu().numpy().view(np.uint32)


@pytest.mark.parametrize("shape,fmt,rounding", [((1000, 64), (4, 2, True), 0), ((333, 70), (6, 3, True), 1),
                                                ((1, 5), (3, 1, True), 0), ((256, 128), (5, 2, False), 0)])
def test_dn_project_matches_oracle(shape, fmt, rounding):
    x = synth.normal(shape, seed=shape[0], mean=0.8, std=2.2)
    xd = x.cuda()
    st = torch.zeros(3, dtype=torch.float64, device="cuda")
    esb.esb_calibrate_dda(xd, esb.Fmt(fmt[0], fmt[1], True), stats_out=st)    # mean and sigma
    codes, xq = esb.esb_dn_project(xd, st, esb.Fmt(*fmt), rounding=rounding)
    s = st.cpu().numpy()
    a = float(np.float32(esb.esb_alpha_star(fmt[0], fmt[1])[0]))
    co, xqo = o.dn_project(x.numpy(), s[0], s[1], a, *fmt, rounding=rounding)
    assert np.array_equal(u32(codes), o.pack(co.reshape(shape), fmt[0], fmt[1], ld_words=codes.shape[1]))
    assert np.array_equal(xq.cpu().numpy().ravel(), xqo)


@pytest.mark.parametrize("n", [1, 1000, 1 << 20, (1 << 20) + 77])
def test_dn_backward_matches_oracle(n):
    x = synth.normal((n,), seed=n % 31, mean=-0.4, std=1.3)
    g = synth.normal((n,), seed=n % 29 + 1)
    xd, gd = x.cuda(), g.cuda()
    st = torch.zeros(3, dtype=torch.float64, device="cuda")
    esb.esb_calibrate_dda(xd, esb.Fmt(4, 2, True), stats_out=st)
    gx = esb.esb_dn_backward(gd, xd, st)
    s = st.cpu().numpy()
    exp = o.dn_backward(g.numpy(), x.numpy(), s[0], s[1])
    got = gx.cpu().numpy()
    scale = np.abs(exp).max() if n > 1 else 1.0
    assert np.all(np.abs(got - exp) <= 1e-6 * np.maximum(np.abs(exp), 1e-3 * scale))


def test_ema_update_matches_oracle():
    run = torch.tensor([0.5, 2.0], dtype=torch.float64, device="cuda")
    r = np.array([0.5, 2.0])
    for i in range(20):
        b = torch.tensor([0.1 * i, 1.0 + 0.05 * i, 7.0], dtype=torch.float64, device="cuda")
        esb.esb_ema_update(b, run, 0.9)
        r = o.ema(b.cpu().numpy(), r, 0.9)
    assert np.array_equal(run.cpu().numpy(), r)


def test_qat_step_through_the_c_abi():
    # one training step of a layer's activation (Algorithm 1): batch
    # statistics, DN + projection, gradient back through STE + DN, moving
    # averages updated; then the test-phase forward with the moving averages
    f = esb.Fmt(4, 2, True)
    x = synth.normal((4096, 64), seed=3, mean=0.2, std=1.7).cuda()
    st = torch.zeros(3, dtype=torch.float64, device="cuda")
    esb.esb_calibrate_dda(x, f, stats_out=st)
    codes, xq = esb.esb_dn_project(x, st, f)
    g = torch.ones_like(xq)
    gx = esb.esb_dn_backward(g, x, st)
    assert float(gx.abs().max()) < 1e-5          # a constant gradient has no effect through DN
    run = torch.tensor([0.0, 1.0], dtype=torch.float64, device="cuda")
    esb.esb_ema_update(st, run, 0.99)
    codes_t, _ = esb.esb_dn_project(x, run, f, want_xq=False)
    assert esb.esb_get_status() == 0
    assert codes_t.shape == codes.shape
