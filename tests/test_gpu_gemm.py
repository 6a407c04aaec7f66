"""GPU parity of the ESB GEMM and implicit-GEMM convolution (tcgen05 path)
against the CPU oracle: exact int32 accumulators, bit-exact fp32 epilogue
outputs and requantised codes."""
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


def dev_i32(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()


def random_packed(rows, cols, fmt, seed):
    b, k = fmt[0], fmt[1]
    codes = synth.uniform_ints((rows, cols), 0, 2 ** b, seed)
    if len(fmt) > 2 and not fmt[2]:
        codes &= np.uint32((1 << (b - 1)) - 1)        # unsigned: sign bit 0
    return o.pack(codes, b, k, ld_words=esb.esb_row_words(cols, b))


def projected_packed(x: np.ndarray, fmt, seed_alpha):
    b, k, s = fmt
    a, _ = o.calibrate(x, b, k, s)
    return o.project_packed(x, a, b, k, s, ld_words=esb.esb_row_words(x.shape[1], b)), a


GEMM_CASES = [
    # (M, N, K, fa, fb)
    (64, 64, 576, (4, 2, False), (4, 2, True)),     # a 3x3x64 conv tile
    (128, 128, 128, (4, 2, True), (4, 2, True)),
    (130, 70, 200, (4, 2, True), (4, 1, True)),     # ragged M, N, K
    (257, 33, 1000, (3, 1, True), (6, 3, True)),
    (300, 96, 515, (5, 2, True), (5, 2, True)),
    (64, 48, 4096, (6, 3, True), (6, 3, True)),
    (100, 200, 64, (4, 3, True), (5, 1, True)),
    (1, 1, 1, (4, 2, True), (4, 2, True)),
    (33, 17, 15, (2, 0, True), (3, 0, True)),
    (256, 256, 1024, (4, 0, True), (4, 2, True)),
]


@pytest.mark.parametrize("M,N,K,fa,fb", GEMM_CASES)
def test_gemm_acc_matches_oracle(M, N, K, fa, fb):
    A = random_packed(M, K, fa, seed=M * 7 + K)
    B = random_packed(N, K, fb, seed=N * 11 + K)
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa[:2]), dev_i32(B), esb.Fmt(*fb[:2]), K)
    exp = o.gemm_i64(A, fa[:2], B, fb[:2], M, N, K)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), exp)


def test_gemm_k_zero_and_empty():
    A = np.zeros((5, 4), np.uint32)
    B = np.zeros((3, 4), np.uint32)
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(4, 2), dev_i32(B), esb.Fmt(4, 2), 0)
    assert np.array_equal(acc.cpu().numpy(), np.zeros((5, 3), np.int32))


@pytest.mark.parametrize("fmt,K", [((4, 2), 16384), ((6, 3), 4600), ((5, 1), 450), ((3, 1), 262144)])
def test_gemm_exact_near_the_accumulation_bound(fmt, K):
    # Adversarial sums: A rows all at the largest image, B rows mixing the
    # largest image with +-1 so partial sums grow towards 2^24 while small
    # terms keep arriving; any loss of low bits in the fp32 TMEM
    # accumulation shows up as an integer mismatch.
    b, k = fmt
    maxc = o.encode(o.C_of(b, k), b, k)
    onep = o.encode(1.0 / 2 ** k, b, k)
    onen = o.encode(-1.0 / 2 ** k, b, k)
    M, N = 128, 64
    ca = np.full((M, K), maxc, np.uint32)
    rng = np.random.default_rng(K)
    cb = np.where(rng.random((N, K)) < 0.7, maxc, np.where(rng.random((N, K)) < 0.5, onep, onen)).astype(np.uint32)
    cb[0, :] = maxc
    A = o.pack(ca, b, k, ld_words=esb.esb_row_words(K, b))
    B = o.pack(cb, b, k, ld_words=esb.esb_row_words(K, b))
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(b, k), dev_i32(B), esb.Fmt(b, k), K)
    exp = o.gemm_i64(A, fmt, B, fmt, M, N, K)
    assert exp.max() < 2 ** 24
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), exp)


def test_gemm_range_error():
    A = np.zeros((128, esb.esb_row_words(8192, 6)), np.uint32)
    with pytest.raises(esb.EsbError) as e:
        esb.esb_gemm(dev_i32(A), esb.Fmt(6, 3), dev_i32(A), esb.Fmt(6, 3), 8192)
    assert e.value.status == esb.ESB_ERR_RANGE


EPI_CASES = [
    # (M, N, K, act, fmt_out, rounding, per_channel, residual)
    (64, 64, 576, esb.ESB_ACT_RELU, (4, 2, False), 0, False, False),
    (200, 128, 300, esb.ESB_ACT_NONE, (4, 2, True), 1, True, False),
    (150, 80, 256, esb.ESB_ACT_RELU6, (6, 3, False), 0, True, True),     # 5 codes per word -> BN = 80
    (129, 96, 640, esb.ESB_ACT_RELU, (5, 2, False), 0, False, True),     # 6 codes per word
    (70, 60, 100, esb.ESB_ACT_NONE, (3, 1, True), 0, True, False),      # 10 codes per word
]


@pytest.mark.parametrize("M,N,K,act,fo,rnd,per_channel,residual", EPI_CASES)
def test_gemm_fused_epilogue_matches_oracle(M, N, K, act, fo, rnd, per_channel, residual):
    fa, fb = (4, 2, False), (4, 2, True)
    xa = synth.half_normal((M, K), seed=M + 1).numpy()
    xb = synth.he_normal((N, K), fan_in=K, seed=N + 2).numpy()
    A, aa = projected_packed(xa, fa, 0)
    B, ab = projected_packed(xb, fb, 0)
    s0 = esb.esb_dequant_scale(aa, esb.Fmt(4, 2), ab, esb.Fmt(4, 2))
    if per_channel:
        scale = (np.float32(s0) * synth.normal((N,), seed=3).numpy().__abs__() + np.float32(1e-3)).astype(np.float32)
        bias = (0.1 * synth.normal((N,), seed=4).numpy()).astype(np.float32)
    else:
        scale = np.full(N, s0, np.float32)
        bias = np.full(N, 0.05, np.float32)
    res_fmt = (4, 2, True)
    res_codes = random_packed(M, N, res_fmt, seed=77) if residual else None
    ep = esb.Epilogue(scale=torch.from_numpy(scale).cuda() if per_channel else None,
                      bias=torch.from_numpy(bias).cuda() if per_channel else None,
                      scale0=float(s0), bias0=0.05, act=act,
                      residual=dev_i32(res_codes) if residual else None, res_fmt=esb.Fmt(*res_fmt),
                      res_scale=0.03125, alpha_out=0.173, fmt_out=esb.Fmt(*fo), rounding_out=rnd)
    acc, y, codes = esb.esb_gemm(dev_i32(A), esb.Fmt(4, 2, False), dev_i32(B), esb.Fmt(4, 2), K, ep=ep,
                                 want_acc=True, want_y=True, want_codes=True)
    acc_o = o.gemm_i64(A, fa[:2], B, fb[:2], M, N, K)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    res_img = None
    if residual:
        rc = o.unpack(res_codes, N, 4)
        res_img = np.vectorize(lambda c: o.image(int(c), 4, 2))(rc)
    yo, co = o.epilogue(acc_o, scale, bias, act, 0.173, fo, rnd, res_images=res_img, res_scale=0.03125)
    yg = y.cpu().numpy()
    # pinned fp32 op order on both sides: identical bits (tolerance 1e-6 rel)
    assert np.array_equal(yg, yo) or np.max(np.abs(yg - yo) / np.maximum(np.abs(yo), 1e-30)) <= 1e-6
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


LEAN_CASES = [
    # (act, fmt_out, bias0, scale factor): codes-only outputs with a scalar
    # scale and bias -- the epilogue's requantisation-only path
    (esb.ESB_ACT_RELU, (4, 2, False), 0.05, 1.0),
    (esb.ESB_ACT_RELU, (4, 2, False), -0.3, 3.7),
    (esb.ESB_ACT_NONE, (4, 2, False), 0.2, 1.0),
    (esb.ESB_ACT_NONE, (4, 2, True), -0.1, 2.0),       # signed, no activation: sign per element
    (esb.ESB_ACT_RELU6, (4, 0, False), 0.0, 40.0),      # thresholds above 6 are never reached
    (esb.ESB_ACT_RELU6, (4, 1, True), 0.5, 9.0),
    (esb.ESB_ACT_RELU, (4, 3, True), 0.0, 0.01),
    (esb.ESB_ACT_RELU, (4, 2, False), 0.1, -1.0),      # negative scale
    (esb.ESB_ACT_NONE, (4, 2, True), 0.0, 0.0),        # zero scale: every output is the bias
]


def lean_epilogue(fo, act, bias0, s):
    return esb.Epilogue(scale0=float(s), bias0=bias0, act=act, alpha_out=0.173, fmt_out=esb.Fmt(*fo))


@pytest.mark.parametrize("act,fo,bias0,sf", LEAN_CASES)
def test_gemm_codes_only_epilogue(act, fo, bias0, sf):
    M, N, K = 300, 64, 576
    fa, fb = (4, 2, False), (4, 2, True)
    A, aa = projected_packed(synth.half_normal((M, K), seed=M + 5).numpy(), fa, 0)
    B, ab = projected_packed(synth.he_normal((N, K), fan_in=K, seed=N + 6).numpy(), fb, 0)
    s = np.float32(esb.esb_dequant_scale(aa, esb.Fmt(4, 2), ab, esb.Fmt(4, 2)) * sf)
    _, _, codes = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K, ep=lean_epilogue(fo, act, bias0, s),
                               want_acc=False, want_y=False, want_codes=True)
    acc_o = o.gemm_i64(A, fa[:2], B, fb[:2], M, N, K)
    _, co = o.epilogue(acc_o, np.full(N, s, np.float32), np.full(N, bias0, np.float32), act, 0.173, fo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("M,N,K,fab", [(200, 64, 4096, (6, 3)), (130, 96, 2000, (5, 2))])
@pytest.mark.parametrize("act", [esb.ESB_ACT_RELU, esb.ESB_ACT_NONE])
def test_gemm_codes_only_epilogue_large_accumulators(M, N, K, fab, act):
    # K max|I_A| max|I_B| above 2^20: the requantisation compares raw
    # accumulators on the ALU pipe instead of the FMA-pipe form
    fa, fb = (fab[0], fab[1], False), (fab[0], fab[1], True)
    A, aa = projected_packed(synth.half_normal((M, K), seed=K + 1).numpy(), fa, 0)
    B, ab = projected_packed(synth.he_normal((N, K), fan_in=K, seed=K + 2).numpy(), fb, 0)
    s = np.float32(esb.esb_dequant_scale(aa, esb.Fmt(*fab), ab, esb.Fmt(*fab)))
    fo = (4, 2, False)
    _, _, codes = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K,
                               ep=lean_epilogue(fo, act, -0.02, s), want_acc=False, want_codes=True)
    acc_o = o.gemm_i64(A, fa[:2], B, fb[:2], M, N, K)
    _, co = o.epilogue(acc_o, np.full(N, s, np.float32), np.full(N, -0.02, np.float32), act, 0.173, fo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("shape", [(2, 56, 56, 64, 64, 1), (2, 9, 7, 64, 64, 1), (2, 14, 14, 128, 256, 2)])
@pytest.mark.parametrize("act,fo,bias0,sf", LEAN_CASES[:6])
def test_conv_codes_only_epilogue(shape, act, fo, bias0, sf):
    n, h, w, c, cout, stride = shape
    fx, fw = (4, 2, False), (4, 2, True)
    X, ax = projected_packed(synth.half_normal((n * h * w, c), seed=h + c).numpy(), fx, 0)
    W, aw = projected_packed(synth.he_normal((cout * 9, c), fan_in=9 * c, seed=cout).numpy(), fw, 0)
    s = np.float32(esb.esb_dequant_scale(ax, esb.Fmt(4, 2), aw, esb.Fmt(4, 2)) * sf)
    _, _, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, 3, 3,
                                      stride, 1, ep=lean_epilogue(fo, act, bias0, s), want_acc=False,
                                      want_codes=True)
    ldx = X.shape[1]
    acc_o = o.conv2d_i64(X.reshape(n, h, w, ldx), fx[:2], W.reshape(cout, 3, 3, ldx), fw[:2], n, h, w, c, cout, 3, 3,
                         stride, 1).reshape(-1, cout)
    _, co = o.epilogue(acc_o, np.full(cout, s, np.float32), np.full(cout, bias0, np.float32), act, 0.173, fo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("ldo_extra,offset_words", [(1, 0), (2, 1), (3, 2), (0, 1)])
def test_codes_store_alignment(ldo_extra, offset_words):
    # output rows at any word stride and start (no 8/16-byte alignment)
    n, h, w, c, cout = 2, 20, 24, 64, 64
    fx, fw = (4, 2, False), (4, 2, True)
    X, ax = projected_packed(synth.half_normal((n * h * w, c), seed=31).numpy(), fx, 0)
    W, aw = projected_packed(synth.he_normal((cout * 9, c), fan_in=576, seed=32).numpy(), fw, 0)
    s = np.float32(esb.esb_dequant_scale(ax, esb.Fmt(4, 2), aw, esb.Fmt(4, 2)))
    ldo = esb.esb_row_words(cout, 4) + ldo_extra
    M = n * h * w
    buf = torch.full((M * ldo + offset_words + 8,), -1, dtype=torch.int32, device="cuda")
    out = buf[offset_words:offset_words + M * ldo].view(M, ldo)
    esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, 3, 3, 1, 1,
                        ep=lean_epilogue((4, 2, False), esb.ESB_ACT_RELU, 0.0, s), want_acc=False, out_codes=out)
    acc_o = o.conv2d_i64(X.reshape(n, h, w, -1), fx[:2], W.reshape(cout, 3, 3, -1), fw[:2], n, h, w, c, cout, 3, 3,
                         1, 1).reshape(-1, cout)
    _, co = o.epilogue(acc_o, np.full(cout, s, np.float32), np.zeros(cout, np.float32), 1, 0.173, (4, 2, False))
    got = u32(out)
    assert np.array_equal(got[:, :8], o.pack(co, 4, 2, ld_words=8))
    b = u32(buf)
    assert (b[:offset_words] == 0xFFFFFFFF).all() and (b[offset_words + M * ldo:] == 0xFFFFFFFF).all()


CONV_CASES = [
    # n, h, w, c, cout, r, s, stride, pad, fx, fw
    (2, 9, 7, 64, 64, 3, 3, 1, 1, (4, 2, False), (4, 2, True)),
    (2, 56, 56, 64, 64, 3, 3, 1, 1, (4, 2, False), (4, 2, True)),     # ResNet18 3x3 layer shape, batch 2
    (2, 14, 14, 128, 256, 3, 3, 2, 1, (4, 2, False), (4, 2, True)),
    (3, 8, 8, 64, 128, 1, 1, 2, 0, (4, 2, False), (4, 2, True)),
    (1, 23, 19, 3, 64, 7, 7, 2, 3, (4, 2, True), (4, 2, True)),       # first layer: c = 3
    (2, 10, 10, 64, 64, 3, 3, 1, 1, (6, 3, False), (6, 3, True)),
    (2, 10, 10, 40, 48, 3, 3, 1, 1, (5, 2, False), (5, 2, True)),
    (2, 10, 10, 30, 32, 3, 3, 1, 1, (3, 1, False), (3, 1, True)),
]


def check_conv(n, h, w, c, cout, r, s, stride, pad, fx, fw):
    x = synth.half_normal((n * h * w, c), seed=h * 3 + c).numpy() if not fx[2] else \
        synth.normal((n * h * w, c), seed=h * 3 + c).numpy()
    wt = synth.he_normal((cout * r * s, c), fan_in=r * s * c, seed=cout + r).numpy()
    ldx = esb.esb_row_words(c, fx[0])
    X, ax = projected_packed(x, fx, 0)
    W, aw = projected_packed(wt, fw, 0)
    assert X.shape[1] == ldx and W.shape[1] == ldx
    fo = (fx[0], fx[1], False)
    s0 = esb.esb_dequant_scale(ax, esb.Fmt(*fx[:2]), aw, esb.Fmt(*fw[:2]))
    ep = esb.Epilogue(scale0=s0, bias0=0.0, act=esb.ESB_ACT_RELU, alpha_out=0.7, fmt_out=esb.Fmt(*fo))
    acc, y, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, r, s,
                                        stride, pad, ep=ep, want_acc=True, want_y=True, want_codes=True)
    acc_o = o.conv2d_i64(X.reshape(n, h, w, ldx), fx[:2], W.reshape(cout, r, s, ldx), fw[:2],
                         n, h, w, c, cout, r, s, stride, pad).reshape(-1, cout)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    yo, co = o.epilogue(acc_o, np.full(cout, s0, np.float32), np.zeros(cout, np.float32), 1, 0.7, fo)
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("n,h,w,c,cout,r,s,stride,pad,fx,fw", CONV_CASES)
def test_conv_matches_oracle(n, h, w, c, cout, r, s, stride, pad, fx, fw):
    check_conv(n, h, w, c, cout, r, s, stride, pad, fx, fw)


HALO_CASES = [
    # n, h, w, c, cout, r, s, pad, fx, fw  (stride 1, 4-bit activations)
    (2, 56, 56, 64, 64, 3, 3, 1, (4, 2, False), (4, 2, True)),        # ResNet18 layer-1 3x3 shape
    (2, 28, 28, 128, 128, 3, 3, 1, (4, 2, False), (4, 2, True)),      # layer-2 shape: 4 pieces per pixel
    (2, 14, 14, 256, 256, 3, 3, 1, (4, 2, False), (4, 2, True)),      # layer-3 shape: 2 channel blocks, 2 N-tiles
    (3, 15, 30, 40, 48, 3, 3, 1, (4, 2, False), (4, 2, True)),        # channel padding codes, last tile ragged
    (2, 12, 28, 64, 32, 5, 5, 2, (4, 1, False), (4, 1, True)),        # 5x5, pad 2
    (2, 16, 31, 96, 80, 1, 1, 0, (4, 2, False), (4, 2, True)),        # 1x1: 3 pieces per pixel, N tail
    (2, 18, 60, 64, 64, 3, 3, 0, (4, 2, False), (4, 2, True)),        # no padding: Q = w - 2
    (2, 20, 24, 64, 64, 3, 3, 1, (4, 2, True), (4, 1, True)),         # signed activations
    (1, 14, 14, 320, 64, 3, 3, 1, (4, 2, False), (4, 2, True)),       # partial last channel block
    (1, 6, 63, 64, 64, 3, 3, 1, (4, 3, False), (4, 3, True)),         # w + pad = slot pitch
    (1, 5, 100, 32, 64, 3, 3, 1, (4, 0, False), (4, 0, True)),        # pitch 128: one output row per tile
]


@pytest.mark.parametrize("n,h,w,c,cout,r,s,pad,fx,fw", HALO_CASES)
def test_conv_halo_matches_oracle(n, h, w, c, cout, r, s, pad, fx, fw):
    assert esb.esb_conv2d_kernel(n, h, w, c, cout, r, s, 1, pad, esb.Fmt(*fx), esb.Fmt(*fw),
                                 out_b=fx[0]) == esb.ESB_CONV_KERNEL_HALO
    check_conv(n, h, w, c, cout, r, s, 1, pad, fx, fw)


def test_conv_kernel_choice():
    f4, f6 = esb.Fmt(4, 2), esb.Fmt(6, 3)
    k = esb.esb_conv2d_kernel
    assert k(32, 56, 56, 64, 64, 3, 3, 1, 1, f4, f4) == esb.ESB_CONV_KERNEL_HALO
    assert k(2, 7, 7, 512, 512, 3, 3, 1, 1, f4, f4) != esb.ESB_CONV_KERNEL_HALO      # 38 % of a tile used
    assert k(2, 56, 56, 64, 128, 3, 3, 2, 1, f4, f4) != esb.ESB_CONV_KERNEL_HALO     # stride 2
    assert k(2, 10, 10, 64, 64, 3, 3, 1, 1, f6, f6) != esb.ESB_CONV_KERNEL_HALO      # 6-bit activations
    assert k(2, 10, 10, 64, 64, 3, 3, 1, 1, f4, f4, groups=64) == esb.ESB_CONV_KERNEL_DEPTHWISE


def test_conv_full_size_sampled_rows():
    # The timed workload at full size (batch 32, 56x56x64 -> 64, 3x3), in
    # the launch configuration the benchmark times; output rows of a few
    # images checked against the oracle.
    n, h, w, c, cout = 32, 56, 56, 64, 64
    fu, fs = (4, 2, False), (4, 2, True)
    x = synth.half_normal((n * h * w, c), seed=7).numpy()
    wt = synth.he_normal((cout * 9, c), fan_in=576, seed=8).numpy()
    X, ax = projected_packed(x, fu, 0)
    W, aw = projected_packed(wt, fs, 0)
    s0 = esb.esb_dequant_scale(ax, esb.Fmt(4, 2), aw, esb.Fmt(4, 2))
    ep = esb.Epilogue(scale0=s0, act=esb.ESB_ACT_RELU, alpha_out=0.7, fmt_out=esb.Fmt(4, 2, False))
    acc, _, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fu), dev_i32(W), esb.Fmt(*fs), n, h, w, c, cout, 3, 3,
                                        1, 1, ep=ep, want_acc=True, want_codes=True)
    acc = acc.cpu().numpy().astype(np.int64).reshape(n, h, w, cout)
    codes = u32(codes).reshape(n, h, w, -1)
    for img in (0, 13, 31):
        for (p0, p1) in ((0, 3), (27, 29), (53, 56)):
            ao = o.conv2d_rows_i64(X.reshape(n, h, w, -1)[img:img + 1], fu[:2], W.reshape(cout, 3, 3, -1), fs[:2],
                                   1, h, w, c, cout, 3, 3, 1, 1, p0, p1)[0]
            assert np.array_equal(acc[img, p0:p1], ao)
            _, co = o.epilogue(ao.reshape(-1, cout), np.full(cout, s0, np.float32), np.zeros(cout, np.float32), 1,
                               0.7, (4, 2, False))
            assert np.array_equal(codes[img, p0:p1].reshape(-1, codes.shape[-1]),
                                  o.pack(co, 4, 2, ld_words=codes.shape[-1]))


def test_conv_dequant_scale_from_device_alphas():
    # calibrate -> project -> conv with the "Scale" stage taken from the two
    # device alphas (no host round trip), as bench.py runs it.
    n, h, w, c, cout = 2, 12, 12, 64, 64
    fu, fs = esb.Fmt(4, 2, False), esb.Fmt(4, 2, True)
    x = synth.half_normal((n * h * w, c), seed=21)
    wt = synth.he_normal((cout * 9, c), fan_in=576, seed=22)
    xd, wd = x.cuda(), wt.cuda()
    ax, _ = esb.esb_calibrate_dda(xd, fu)
    aw, _ = esb.esb_calibrate_dda(wd, fs)
    Xc = esb.esb_project(xd, fu, alpha=ax)
    Wc = esb.esb_project(wd, fs, alpha=aw)
    ep = esb.Epilogue(scale0=1.0, alpha_a_dev=ax, alpha_b_dev=aw, bias0=-0.01, act=esb.ESB_ACT_RELU,
                      alpha_out=0.3, fmt_out=fu)
    acc, y, codes = esb.esb_conv2d_nhwc(Xc, fu, Wc, fs, n, h, w, c, cout, 3, 3, 1, 1, ep=ep, want_acc=True,
                                        want_y=True, want_codes=True)
    axh, awh = np.float32(ax.item()), np.float32(aw.item())
    dq = np.float32(np.float32(axh * awh) * np.float32(2.0 ** -4))
    sc = np.float32(np.float32(1.0) * dq)
    Xo = o.project_packed(x.numpy(), float(axh), 4, 2, False, ld_words=Xc.shape[1])
    Wo = o.project_packed(wt.numpy(), float(awh), 4, 2, True, ld_words=Wc.shape[1])
    acc_o = o.conv2d_i64(Xo.reshape(n, h, w, -1), (4, 2), Wo.reshape(cout, 3, 3, -1), (4, 2),
                         n, h, w, c, cout, 3, 3, 1, 1).reshape(-1, cout)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    yo, co = o.epilogue(acc_o, np.full(cout, sc, np.float32), np.full(cout, -0.01, np.float32), 1, 0.3, (4, 2, False))
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, 4, 2, ld_words=codes.shape[1]))


@pytest.mark.parametrize("alpha_scale", [1.0, 0.0])
def test_conv_codes_only_from_device_alphas(alpha_scale):
    # The timed layer's call (codes only, scale from the two device alphas)
    # through the specialised halo instance; with a zero activation alpha the
    # folded scale is 0 and the kernel takes its per-word path (every output
    # is act(bias) requantised).
    n, h, w, c, cout = 2, 28, 28, 64, 64
    fu, fs = esb.Fmt(4, 2, False), esb.Fmt(4, 2, True)
    assert esb.esb_conv2d_kernel(n, h, w, c, cout, 3, 3, 1, 1, fu, fs, out_b=4) == esb.ESB_CONV_KERNEL_HALO
    x = synth.half_normal((n * h * w, c), seed=31)
    wt = synth.he_normal((cout * 9, c), fan_in=576, seed=32)
    xd, wd = x.cuda(), wt.cuda()
    ax, _ = esb.esb_calibrate_dda(xd, fu)
    aw, _ = esb.esb_calibrate_dda(wd, fs)
    Xc = esb.esb_project(xd, fu, alpha=ax)
    Wc = esb.esb_project(wd, fs, alpha=aw)
    axe = ax * alpha_scale
    ep = esb.Epilogue(scale0=1.0, alpha_a_dev=axe, alpha_b_dev=aw, bias0=0.02, act=esb.ESB_ACT_RELU,
                      alpha_out=0.3, fmt_out=fu)
    _, _, codes = esb.esb_conv2d_nhwc(Xc, fu, Wc, fs, n, h, w, c, cout, 3, 3, 1, 1, ep=ep, want_acc=False,
                                      want_codes=True)
    axh, awh = np.float32(ax.item()), np.float32(aw.item())
    dq = np.float32(np.float32(np.float32(axh * np.float32(alpha_scale)) * awh) * np.float32(2.0 ** -4))
    sc = np.float32(np.float32(1.0) * dq)
    Xo = o.project_packed(x.numpy(), float(axh), 4, 2, False, ld_words=Xc.shape[1])
    Wo = o.project_packed(wt.numpy(), float(awh), 4, 2, True, ld_words=Wc.shape[1])
    acc_o = o.conv2d_i64(Xo.reshape(n, h, w, -1), (4, 2), Wo.reshape(cout, 3, 3, -1), (4, 2),
                         n, h, w, c, cout, 3, 3, 1, 1).reshape(-1, cout)
    _, co = o.epilogue(acc_o, np.full(cout, sc, np.float32), np.full(cout, 0.02, np.float32), 1, 0.3, (4, 2, False))
    assert np.array_equal(u32(codes), o.pack(co, 4, 2, ld_words=codes.shape[1]))


TILED_CASES = [
    # (M, N, K, fa, fb): the tiled large-operand path (esb_gemm_tiled)
    (300, 512, 1000, (4, 2, False), (4, 2, True)),    # ragged M and K tail, two N-tiles
    (257, 300, 515, (4, 1, True), (4, 2, True)),      # ragged N (last N-tile partly past N)
    (130, 256, 2000, (6, 3, True), (6, 3, True)),     # 6-bit codes: the general tile decode
    (520, 768, 128, (3, 1, True), (3, 1, True)),      # one K-block
    (128, 1024, 4608, (4, 2, False), (4, 2, True)),   # deep K, four N-tiles
]


@pytest.fixture
def tiled_always(monkeypatch):
    # every shape the tiled kernel takes goes to it (not only the large ones)
    monkeypatch.setenv("ESB_GEMM_TILED_MIN_MACS", "0")


def tiled_ws(M, N, K):
    nb = esb.esb_gemm_tiled_workspace_bytes(M, N, K)
    # garbage in the workspace: the tile pass overwrites every byte it uses
    return torch.full((max(nb, 16),), 0xA5, dtype=torch.uint8, device="cuda")


@pytest.mark.parametrize("M,N,K,fa,fb", TILED_CASES)
def test_gemm_tiled_matches_oracle(M, N, K, fa, fb, tiled_always):
    A = random_packed(M, K, fa, seed=M * 5 + K)
    B = random_packed(N, K, fb, seed=N * 3 + K)
    fo = (4, 2, False)
    s0 = np.float32(3e-4)
    ep = esb.Epilogue(scale0=float(s0), bias0=0.01, act=esb.ESB_ACT_RELU, alpha_out=0.41, fmt_out=esb.Fmt(*fo))
    acc, y, codes = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa[:2]), dev_i32(B), esb.Fmt(*fb[:2]), K, ep=ep,
                                 want_acc=True, want_y=True, want_codes=True, workspace=tiled_ws(M, N, K))
    exp = o.gemm_i64(A, fa[:2], B, fb[:2], M, N, K)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), exp)
    yo, co = o.epilogue(exp, np.full(N, s0, np.float32), np.full(N, 0.01, np.float32), 1, 0.41, fo)
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))
    assert esb.esb_get_status() == 0


@pytest.mark.parametrize("act,fo,bias0,sf", LEAN_CASES[:6])
def test_gemm_tiled_codes_only(act, fo, bias0, sf, tiled_always):
    # codes as the only output in whole N-tiles: the specialised epilogue
    M, N, K = 300, 512, 576
    fa, fb = (4, 2, False), (4, 2, True)
    A, aa = projected_packed(synth.half_normal((M, K), seed=M + 9).numpy(), fa, 0)
    B, ab = projected_packed(synth.he_normal((N, K), fan_in=K, seed=N + 8).numpy(), fb, 0)
    s = np.float32(esb.esb_dequant_scale(aa, esb.Fmt(4, 2), ab, esb.Fmt(4, 2)) * sf)
    _, _, codes = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K,
                               ep=lean_epilogue(fo, act, bias0, s), want_acc=False, want_codes=True,
                               workspace=tiled_ws(M, N, K))
    acc_o = o.gemm_i64(A, fa[:2], B, fb[:2], M, N, K)
    _, co = o.epilogue(acc_o, np.full(N, s, np.float32), np.full(N, bias0, np.float32), act, 0.173, fo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


def test_gemm_tiled_small_n_falls_back(tiled_always):
    # N < 256: esb_gemm_tiled runs esb_gemm's kernels and leaves the workspace alone
    M, N, K = 200, 96, 300
    A = random_packed(M, K, (4, 2, True), seed=1)
    B = random_packed(N, K, (4, 2, True), seed=2)
    ws = torch.zeros(16, dtype=torch.uint8, device="cuda")
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(4, 2), dev_i32(B), esb.Fmt(4, 2), K, workspace=ws)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), o.gemm_i64(A, (4, 2), B, (4, 2), M, N, K))
    assert int(ws.sum()) == 0


def test_gemm_tiled_full_size_sampled_rows():
    # the square 4096^3 sweep size in (4,2): int32 accumulators of sampled
    # rows against the oracle
    n = 4096
    A = random_packed(n, n, (4, 2, False), seed=41)
    B = random_packed(n, n, (4, 2, True), seed=42)
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(4, 2), dev_i32(B), esb.Fmt(4, 2), n, workspace=tiled_ws(n, n, n))
    rows = np.array([0, 1, 127, 128, 2047, 4094, 4095] + list(np.random.default_rng(5).integers(0, n, 9)))
    exp = o.gemm_i64(A[rows], (4, 2), B, (4, 2), len(rows), n, n)
    assert np.array_equal(acc.cpu().numpy()[rows].astype(np.int64), exp)
    assert esb.esb_get_status() == 0


@pytest.mark.parametrize("M,N,K", [(200, 256, 6000), (130, 300, 16384)])
def test_gemm_tiled_chunked_k(M, N, K, tiled_always):
    # K max|I_A| max|I_B| past 2^24 with 6-bit codes: the K chunks of the
    # tiled kernel (two, then four with 128-column N-tiles), added as exact
    # integers; y and codes from float(acc) rounded to nearest
    f = (6, 3, True)
    # random codes, except that a band of rows of A and of B holds the code
    # of the largest image (positive in A, both signs in B): their sums reach
    # K max|I|^2 > 2^24, the others stay small
    cmax = max(range(2 ** 6), key=lambda c: o.image(c, 6, 3))
    cneg = min(range(2 ** 6), key=lambda c: o.image(c, 6, 3))
    ca = synth.uniform_ints((M, K), 0, 2 ** 6, K + 1)
    cb = synth.uniform_ints((N, K), 0, 2 ** 6, K + 2)
    ca[:20] = cmax
    cb[:10] = cmax
    cb[10:20] = cneg
    A = o.pack(ca, 6, 3, ld_words=esb.esb_row_words(K, 6))
    B = o.pack(cb, 6, 3, ld_words=esb.esb_row_words(K, 6))
    s0 = np.float32(2e-6)
    fo = (4, 2, True)
    ep = esb.Epilogue(scale0=float(s0), bias0=-0.03, act=esb.ESB_ACT_NONE, alpha_out=0.2, fmt_out=esb.Fmt(*fo))
    with pytest.raises(RuntimeError):           # one fp32 accumulation cannot hold it
        esb.esb_gemm(dev_i32(A), esb.Fmt(6, 3), dev_i32(B), esb.Fmt(6, 3), K)
    acc, y, codes = esb.esb_gemm(dev_i32(A), esb.Fmt(6, 3), dev_i32(B), esb.Fmt(6, 3), K, ep=ep, want_acc=True,
                                 want_y=True, want_codes=True, workspace=tiled_ws(M, N, K))
    exp = o.gemm_i64(A, (6, 3), B, (6, 3), M, N, K)
    assert np.abs(exp).max() >= 2 ** 24            # the case needs the chunks
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), exp)
    yo, co = o.epilogue(exp, np.full(N, s0, np.float32), np.full(N, -0.03, np.float32), 0, 0.2, fo)
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))
    assert esb.esb_get_status() == 0
