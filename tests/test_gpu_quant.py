"""GPU parity of projection, dequantisation and DDA calibration against the
CPU oracle, through the C ABI (libesb.so)."""
import numpy as np
import pytest
import torch

import oracle as o
from conftest import oracle_step_function, step_function_codes
from paper_2109_03513_gb300 import esb, synth

pytestmark = pytest.mark.gpu

FORMATS = [(b, k) for b in range(2, 9) for k in range(0, b)]


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def u32(t: torch.Tensor) -> np.ndarray:
    return t.cpu().numpy().view(np.uint32)


def probe_values(b, k):
    s = o.set_nonneg(b, k)
    mids = 0.5 * (s[1:] + s[:-1])
    pts = np.concatenate([s, mids, [o.C_of(b, k) * 1.5, 1e30, 1e-40, 3e-39]]).astype(np.float32)
    out = [pts]
    cur = pts
    for _ in range(2):
        out.append(np.nextafter(cur, np.float32(np.inf)))
        out.append(np.nextafter(cur, np.float32(-np.inf)))
        cur = out[-1]
    v = np.concatenate(out)
    return np.concatenate([v, -v, np.array([0.0, -0.0, np.inf, -np.inf, np.nan], np.float32)])


@pytest.mark.parametrize("b,k", FORMATS)
@pytest.mark.parametrize("signed", [True, False])
@pytest.mark.parametrize("rounding", [0, 1])
def test_project_matches_oracle(b, k, signed, rounding):
    f = esb.Fmt(b, k, signed)
    C = o.C_of(b, k)
    x = np.concatenate([probe_values(b, k),
                        synth.normal((6000,), seed=b * 100 + k).numpy() * np.float32(C),
                        synth.laplace((2000,), seed=b * 100 + k + 1).numpy()]).astype(np.float32)
    for alpha in (1.0, 0.7310585, 3.0):
        # 1-D (vector path) and a ragged 2-D view (general path)
        for shape in ((x.size,), (7, x.size // 7)):
            xs = x[: int(np.prod(shape))].reshape(shape)
            codes = esb.esb_project(torch.from_numpy(xs).cuda(), f, alpha=alpha, rounding=rounding)
            exp = o.project_packed(xs.reshape(-1, shape[-1]), alpha, b, k, signed, rounding,
                                   ld_words=codes.shape[-1])
            assert np.array_equal(u32(codes), exp), (shape, alpha)


@pytest.mark.parametrize("k", [0, 1, 2, 3])
@pytest.mark.parametrize("signed", [True, False])
def test_project_b4_flat_probes(k, signed):
    # 4-bit codes of flat tensors take the warp-tile path; probes on
    # and next to every threshold, binade edges, subnormals, infinities and
    # NaN, for alphas whose thresholds span many binades, and alphas so small
    # or large that the kernel keeps the compare-based search
    f = esb.Fmt(4, k, signed)
    C = o.C_of(4, k)
    base = np.concatenate([probe_values(4, k), synth.normal((4000,), seed=40 + k).numpy() * np.float32(C)])
    for alpha in (1.0, 0.7310585, 3.0, 2.0 ** -20, 1e-35, 1e35, 6.0e-8):
        with np.errstate(over="ignore"):                # alpha = 1e35 sends probes to infinity on purpose
            pts = np.concatenate([base * np.float32(alpha), base]).astype(np.float32)
        pts = pts[: pts.size // 64 * 64]
        for shape in ((1, pts.size), (pts.size // 64, 64)):
            xs = pts.reshape(shape)
            codes = esb.esb_project(torch.from_numpy(xs).cuda(), f, alpha=alpha)
            exp = o.project_packed(xs, alpha, 4, k, signed, 0, ld_words=codes.shape[-1])
            assert np.array_equal(u32(codes), exp), (shape, alpha)


CELL_FORMATS = ([(3, k) for k in range(3)] + [(5, k) for k in range(5)] + [(6, k) for k in range(6)]
                + [(7, 0), (7, 3), (7, 5), (7, 6), (8, 0), (8, 4), (8, 6), (8, 7)])


@pytest.mark.parametrize("b,k", CELL_FORMATS)
@pytest.mark.parametrize("signed", [True, False])
def test_project_cell_table_probes(b, k, signed):
    # b = 3 and b >= 5 project through the per-block cell table (at most one
    # threshold per cell of 2^(21-k) fp32 patterns); probes on and next to
    # every threshold, for alphas that keep the table, and for alphas whose
    # thresholds overflow or run subnormal (or whose table is over capacity,
    # (8, 7)), where the block keeps the bisection; both tie rules
    f = esb.Fmt(b, k, signed)
    C = o.C_of(b, k)
    base = np.concatenate([probe_values(b, k), synth.normal((3000,), seed=50 + 8 * b + k).numpy() * np.float32(C)])
    for alpha in (1.0, 0.7310585, 3.0, 2.0 ** -20, 1e-35, 1e35, 6.0e-8):
        with np.errstate(over="ignore"):                # alpha = 1e35 sends probes to infinity on purpose
            pts = np.concatenate([base * np.float32(alpha), base]).astype(np.float32)
        for rounding in (0, 1):
            for shape in ((1, pts.size), (pts.size // 96, 96)):
                xs = np.ascontiguousarray(pts[: int(np.prod(shape))].reshape(shape))
                codes = esb.esb_project(torch.from_numpy(xs).cuda(), f, alpha=alpha, rounding=rounding)
                exp = o.project_packed(xs, alpha, b, k, signed, rounding, ld_words=codes.shape[-1])
                assert np.array_equal(u32(codes), exp), (shape, alpha, rounding)


EVERY_FP32_CASES = [(2, 0, True, 0, 1.0), (3, 1, True, 0, 3.0), (4, 2, True, 0, 0.7310585), (4, 2, False, 1, 1.0),
                    (5, 2, False, 0, 0.7310585), (6, 3, True, 1, 0.7310585), (8, 4, True, 0, 0.37), (8, 7, True, 0, 1.0)]


@pytest.mark.parametrize("b,k,signed,rounding,alpha", EVERY_FP32_CASES)
def test_project_every_fp32_pattern(b, k, signed, rounding, alpha):
    # All 2^32 fp32 bit patterns, projected as flat tensors of 2^26 values
    # (b = 4: the warp-tile path; b = 3, 5, 6, 8: the cell table; (8, 7) and
    # (2, 0): the bisection), against the oracle's step function (breakpoints
    # and bucket codes computed by the oracle alone, see conftest)
    step = oracle_step_function(alpha, b, k, signed, rounding)
    f = esb.Fmt(b, k, signed)
    cpw = 32 // b
    n = 1 << 26
    shifts = torch.arange(cpw, device="cuda", dtype=torch.int64) * b
    codes = torch.empty((1, esb.esb_row_words(n, b)), dtype=torch.int32, device="cuda")
    for c in range((1 << 32) // n):
        bits = torch.arange(c * n, (c + 1) * n, dtype=torch.int64, device="cuda")
        x = torch.where(bits >= (1 << 31), bits - (1 << 32), bits).to(torch.int32).view(torch.float32)
        esb.esb_project(x, f, alpha=alpha, rounding=rounding, codes=codes)
        w = codes[0].to(torch.int64) & 0xFFFFFFFF
        got = ((w[:, None] >> shifts[None, :]) & ((1 << b) - 1)).reshape(-1)[:n]
        exp = step_function_codes(bits, step)
        if not torch.equal(got, exp):
            i = int(torch.nonzero(got != exp)[0, 0])
            raise AssertionError((hex(c * n + i), int(exp[i]), int(got[i])))
    assert esb.esb_get_status() == 0


def test_project_edge_shapes_and_device_alpha():
    f = esb.Fmt(4, 2, True)
    for rows, cols in [(1, 1), (1, 7), (3, 8), (5, 33), (2, 64), (130, 576)]:
        x = synth.normal((rows, cols), seed=rows * 1000 + cols)
        a = torch.tensor([0.41], dtype=torch.float32, device="cuda")
        codes = esb.esb_project(x.cuda(), f, alpha=a)
        exp = o.project_packed(x.numpy(), 0.41, 4, 2, True, 0, ld_words=codes.shape[-1])
        assert np.array_equal(u32(codes), exp), (rows, cols)
    # explicit wider row stride: padding words hold zero codes
    x = synth.normal((4, 10), seed=3)
    codes = esb.esb_project(x.cuda(), f, alpha=0.5, ldc=12)
    assert np.array_equal(u32(codes), o.project_packed(x.numpy(), 0.5, 4, 2, ld_words=12))


def test_project_full_size_sampled():
    # 2^28 values, the size the projection sweep runs; check sampled words.
    n = 1 << 28
    f = esb.Fmt(4, 2, True)
    x = torch.randn(n, generator=torch.Generator(device="cuda").manual_seed(5), device="cuda")
    codes = esb.esb_project(x, f, alpha=0.37)
    torch.cuda.synchronize()
    cpw = 8
    idx = np.unique(np.concatenate([np.arange(64), np.arange(codes.shape[1] - 64, codes.shape[1]),
                                    np.random.default_rng(1).integers(0, codes.shape[1], 4000)]))
    ti = torch.from_numpy(idx).cuda()
    got = u32(codes[0, ti])
    xs = x.view(-1, cpw)[ti].cpu().numpy()
    exp = o.project_packed(xs, 0.37, 4, 2, True, 0, ld_words=1)[:, 0]
    assert np.array_equal(got, exp)
    del x, codes


@pytest.mark.parametrize("b,k", [(2, 0), (3, 1), (4, 2), (5, 1), (6, 3), (8, 4), (8, 0)])
def test_dequant_matches_oracle(b, k):
    f = esb.Fmt(b, k, True)
    rows, cols = 5, 77
    codes = synth.uniform_ints((rows, cols), 0, 2 ** b, seed=b * 10 + k)
    packed = o.pack(codes, b, k, ld_words=esb.esb_row_words(cols, b))
    y = esb.esb_dequant(torch.from_numpy(packed.view(np.int32)).cuda(), cols, f, 0.8125)
    vals = np.vectorize(lambda c: o.decode(int(c), b, k))(codes)
    exp = (np.float32(0.8125) * vals.astype(np.float32)).astype(np.float32)
    assert np.array_equal(y.cpu().numpy(), exp)


CAL_CASES = [
    ("normal", 1 << 20, True), ("half_normal", 1 << 20, False), ("laplace", 1 << 20, True),
    ("normal", 1, True), ("normal", 31, True), ("normal", 33, True), ("normal", 1000003, True),
    ("half_normal", 4097, False),
]


@pytest.mark.parametrize("dist,n,signed", CAL_CASES)
@pytest.mark.parametrize("bk", [(4, 2), (6, 3)])
def test_calibrate_matches_oracle(dist, n, signed, bk):
    b, k = bk
    x = synth.distribution(dist, (n,), seed=n % 1000 + b)
    f = esb.Fmt(b, k, signed)
    stats = torch.zeros(3, dtype=torch.float64, device="cuda")
    a, _ = esb.esb_calibrate_dda(x.cuda(), f, stats_out=stats)
    ao, so = o.calibrate(x.numpy(), b, k, signed)
    ag = float(a.item())
    st = stats.cpu().numpy()
    assert abs(ag - ao) <= 1e-6 * ao, (ag, ao)
    assert st[2] == n
    assert abs(st[1] - so[1]) <= 1e-6 * max(so[1], 1e-30) + 1e-12
    assert abs(st[0] - so[0]) <= 1e-6 * max(so[1], 1e-30) + 1e-12


def test_calibrate_offset_constant_and_determinism():
    f = esb.Fmt(4, 2, True)
    x = synth.normal((1 << 18,), seed=9, mean=100.0)
    a1, _ = esb.esb_calibrate_dda(x.cuda(), f)
    a2, _ = esb.esb_calibrate_dda(x.cuda(), f)
    ao, _ = o.calibrate(x.numpy(), 4, 2)
    assert abs(a1.item() - ao) <= 1e-6 * ao
    assert a1.item() == a2.item()
    c = torch.full((1000,), 2.5, dtype=torch.float32)
    ac, _ = esb.esb_calibrate_dda(c.cuda(), f)
    assert ac.item() == np.float32(o.alpha_star(4, 2)[0] * 1e-7)
    # unaligned base pointer takes the scalar path
    xu = synth.normal(((1 << 12) + 1,), seed=4)
    xd = xu.cuda()[1:]
    au, _ = esb.esb_calibrate_dda(xd, f)
    ao2, _ = o.calibrate(xu.numpy()[1:], 4, 2)
    assert abs(au.item() - ao2) <= 1e-6 * ao2


def test_calibrate_then_project_on_device():
    # alpha stays on the device between the two calls (no host round trip)
    f = esb.Fmt(5, 2, True)
    x = synth.laplace((3, 1000), seed=12)
    xd = x.cuda()
    a, _ = esb.esb_calibrate_dda(xd, f)
    codes = esb.esb_project(xd, f, alpha=a)
    ah = float(a.item())
    assert np.array_equal(u32(codes), o.project_packed(x.numpy(), ah, 5, 2, ld_words=codes.shape[-1]))


PD_CASES = [
    ("half_normal", (200704, 64), (4, 2, False)),      # the bench layer's activations (6.4 M values)
    ("normal", (1000, 96), (4, 2, True)),
    ("laplace", (333, 40), (6, 3, True)),
    ("normal", (7, 37), (5, 2, True)),                  # ragged: cols % 4 != 0 takes the two-launch form
    ("half_normal", (1, 8), (3, 1, False)),
    ("normal", (4096, 128), (4, 1, True)),
]


@pytest.mark.parametrize("dist,shape,fmt", PD_CASES)
@pytest.mark.parametrize("rounding", [0, 1])
def test_project_dda_matches_oracle(dist, shape, fmt, rounding):
    b, k, signed = fmt
    f = esb.Fmt(b, k, signed)
    x = synth.distribution(dist, shape, seed=shape[0] + b)
    stats = torch.zeros(3, dtype=torch.float64, device="cuda")
    codes, a = esb.esb_project_dda(x.cuda(), f, rounding=rounding, stats_out=stats)
    ag = float(a.item())
    ao, so = o.calibrate(x.numpy(), b, k, signed)
    assert abs(ag - ao) <= 1e-6 * ao, (ag, ao)
    st = stats.cpu().numpy()
    assert st[2] == x.numel() and abs(st[1] - so[1]) <= 1e-6 * so[1]
    if x.numel() > 100000:   # full-size case: sampled rows
        idx = np.unique(np.concatenate([np.arange(16), np.arange(shape[0] - 16, shape[0]),
                                        np.random.default_rng(3).integers(0, shape[0], 2000)]))
        got = u32(codes)[idx]
        exp = o.project_packed(x.numpy()[idx], ag, b, k, signed, rounding, ld_words=codes.shape[1])
    else:
        got = u32(codes)
        exp = o.project_packed(x.numpy(), ag, b, k, signed, rounding, ld_words=codes.shape[1])
    assert np.array_equal(got, exp)
    assert esb.esb_get_status() == 0


def test_workspace_left_zero_and_reusable():
    # the calibration workspace is zero-filled once; every call leaves its
    # 32-byte head record zero again, so one workspace serves any sequence
    # of calibrations and fused projections
    f = esb.Fmt(4, 2, False)
    xa = synth.half_normal((3000, 64), seed=41).cuda()
    xb = synth.half_normal((777, 64), seed=42).cuda()
    nb = max(esb.esb_calibrate_dda_workspace_bytes(xa.numel()), esb.esb_calibrate_dda_workspace_bytes(xb.numel()))
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    alphas = []
    for x, fused in [(xa, True), (xb, False), (xa, False), (xb, True), (xa, True)]:
        if fused:
            _, a = esb.esb_project_dda(x, f, workspace=ws)
        else:
            a, _ = esb.esb_calibrate_dda(x, f, workspace=ws)
        assert esb.esb_get_status() == 0
        assert int(ws[:32].cpu().sum()) == 0
        alphas.append(float(a.item()))
    fresh_a = float(esb.esb_calibrate_dda(xa, f)[0].item())
    fresh_b = float(esb.esb_calibrate_dda(xb, f)[0].item())
    for a, ref in zip(alphas, [fresh_a, fresh_b, fresh_a, fresh_b, fresh_a]):
        assert abs(a - ref) <= 1e-6 * ref


def test_sharded_calibration_from_device_statistics():
    # per-shard statistics from the device (esb_calibrate_dda stats_out),
    # combined on the host (esb_dda_combine), against the oracle on
    # the whole tensor
    from paper_2109_03513_gb300 import shard
    for signed, x in [(True, synth.normal((200003,), seed=21, mean=2.0)), (False, synth.half_normal((131072,), seed=22))]:
        f = esb.Fmt(4, 2, signed)
        cuts = [0, 50000, 50001, x.numel()]
        stats = []
        for i in range(3):
            st = torch.zeros(3, dtype=torch.float64, device="cuda")
            esb.esb_calibrate_dda(x[cuts[i]:cuts[i + 1]].contiguous().cuda(), f, stats_out=st)
            stats.append(st.cpu().numpy())
        a, mean, spread, n = shard.combine_dda_stats(stats, f)
        a_ref, st_ref = o.calibrate(x.numpy(), 4, 2, signed)
        assert n == x.numel()
        assert abs(a - a_ref) <= 1e-6 * a_ref


def test_barrier_wait_runs_out_and_recovers(monkeypatch):
    # The fused projection's grid-barrier wait is bounded.  With its limit cut
    # to 1 ns (ESB_BARRIER_WAIT_NS, a test aid that can only shorten it),
    # blocks that arrive before the last one give up after their first
    # bounded poll: the device status reports ESB_ERR_TIMEOUT and the kernel
    # returns (no hang, the context stays usable).  After the workspace is
    # zero-filled again the next call matches the oracle.  The wait sits
    # after the block's bulk copies have landed, so nothing is in flight.
    f = esb.Fmt(4, 2, False)
    x = synth.half_normal((1 << 16, 64), seed=51)
    xd = x.cuda()
    ws = torch.zeros(esb.esb_calibrate_dda_workspace_bytes(xd.numel()), dtype=torch.uint8, device="cuda")
    assert esb.esb_get_status() == 0
    seen = []
    monkeypatch.setenv("ESB_BARRIER_WAIT_NS", "1")
    for _ in range(5):
        esb.esb_project_dda(xd, f, workspace=ws)
        seen.append(esb.esb_get_status())
        ws.zero_()
        if seen[-1] == esb.ESB_ERR_TIMEOUT:
            break
    monkeypatch.delenv("ESB_BARRIER_WAIT_NS")
    assert esb.ESB_ERR_TIMEOUT in seen, seen
    assert set(seen) <= {esb.ESB_OK, esb.ESB_ERR_TIMEOUT}
    codes, a = esb.esb_project_dda(xd, f, workspace=ws)
    assert esb.esb_get_status() == 0
    assert int(ws[:32].cpu().sum()) == 0
    ag = float(a.item())
    ao, _ = o.calibrate(x.numpy(), 4, 2, False)
    assert abs(ag - ao) <= 1e-6 * ao
    idx = np.unique(np.concatenate([np.arange(8), np.arange(x.shape[0] - 8, x.shape[0]),
                                    np.random.default_rng(5).integers(0, x.shape[0], 1000)]))
    exp = o.project_packed(x.numpy()[idx], ag, 4, 2, False, ld_words=codes.shape[1])
    assert np.array_equal(u32(codes)[idx], exp)
