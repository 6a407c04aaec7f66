"""GPU parity of the specialised fast paths against the CPU oracle, at
shapes chosen to reach their edge cases:

* the word-slot K layout of 2/3/5/6/7/8-bit operands (codes of a row past
  K must not enter the sums; a K-block is a whole number of words);
* the general-width epilogue (6/5/3-bit output codes, only the chunks
  inside N are computed, the rest of the row is zero codes);
* the 4-bit epilogue with a 4-bit residual (ResNet's second conv of a
  block), including N not a multiple of 16 (codes past N masked);
* the depthwise kernel's requantisation on the integer accumulator
  (codes only, scalar scale), with ragged channels and odd sizes;
* im2col filter rows walked tap by tap (first layers: 3 channels in a
  4-word pixel row)."""
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


def dev_i32(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()


def random_codes(rows, cols, b, seed, signed=True):
    codes = synth.uniform_ints((rows, cols), 0, 2 ** b, seed)
    if not signed:
        codes &= np.uint32((1 << (b - 1)) - 1)
    return codes


@pytest.mark.parametrize("fa,fb,K,extra", [((3, 1), (3, 1), 77, 3), ((5, 2), (5, 2), 131, 5), ((6, 3), (6, 3), 259, 4),
                                           ((7, 3), (7, 3), 15, 2), ((8, 4), (7, 3), 8, 3), ((2, 0), (2, 0), 515, 9), ((6, 2), (6, 3), 129, 1)])
def test_gemm_word_slots_ignore_codes_past_k(fa, fb, K, extra):
    """Rows hold K + extra random codes; the contraction takes the first K."""
    M, N = 150, 70
    cols = K + extra
    ca = random_codes(M, cols, fa[0], seed=K)
    cb = random_codes(N, cols, fb[0], seed=K + 1)
    A = o.pack(ca, fa[0], fa[1], ld_words=esb.esb_row_words(cols, fa[0]))
    B = o.pack(cb, fb[0], fb[1], ld_words=esb.esb_row_words(cols, fb[0]))
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K, want_acc=True)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), o.gemm_i64(A, fa, B, fb, M, N, K))


@pytest.mark.parametrize("N,fo,act", [(16, (6, 3, False), esb.ESB_ACT_RELU), (24, (5, 2, True), esb.ESB_ACT_NONE),
                                      (70, (3, 1, False), esb.ESB_ACT_RELU6), (260, (6, 2, False), esb.ESB_ACT_RELU)])
@pytest.mark.parametrize("ldo_extra", [0, 3])
def test_general_width_codes_only(N, fo, act, ldo_extra):
    """Codes-only epilogue for output widths other than 4, scalar scale and
    bias, row strides with extra words (they must hold zero codes)."""
    M, K = 300, 192
    fa, fb = (4, 2), (4, 2)
    A = o.pack(random_codes(M, K, 4, seed=1, signed=False), 4, 2, ld_words=esb.esb_row_words(K, 4))
    B = o.pack(random_codes(N, K, 4, seed=2), 4, 2, ld_words=esb.esb_row_words(K, 4))
    ldo = esb.esb_row_words(N, fo[0]) + ldo_extra
    out = torch.full((M, ldo), -1, dtype=torch.int32, device="cuda")
    ep = esb.Epilogue(scale0=0.0123, bias0=-0.02, act=act, alpha_out=0.31, fmt_out=esb.Fmt(fo[0], fo[1], fo[2]))
    esb.esb_gemm(dev_i32(A), esb.Fmt(4, 2, False), dev_i32(B), esb.Fmt(4, 2), K, ep=ep, want_acc=False,
                 out_codes=out)
    acc_o = o.gemm_i64(A, fa, B, fb, M, N, K)
    _, co = o.epilogue(acc_o, np.full(N, 0.0123, np.float32), np.full(N, -0.02, np.float32), act, 0.31, fo)
    assert np.array_equal(u32(out), o.pack(co, fo[0], fo[1], ld_words=ldo))


@pytest.mark.parametrize("n,h,w,c,cout,stride,fo", [
    (2, 14, 14, 64, 64, 1, (4, 2, False)),          # halo kernel, unsigned output
    (2, 14, 14, 64, 24, 1, (4, 2, True)),           # N = 24: second chunk half past N, signed output
    (2, 15, 13, 32, 40, 2, (4, 1, False)),          # im2col kernel, odd sizes
    (1, 9, 9, 128, 128, 1, (4, 2, True)),
])
def test_conv_with_4bit_residual_codes_only(n, h, w, c, cout, stride, fo):
    r = s = 3
    pad = 1
    fx, fw = (4, 2, False), (4, 2, True)
    x = synth.half_normal((n * h * w, c), seed=h + c).numpy()
    wt = synth.he_normal((cout * r * s, c), fan_in=r * s * c, seed=cout).numpy()
    ldx = esb.esb_row_words(c, 4)
    ax, _ = o.calibrate(x, 4, 2, False)
    aw, _ = o.calibrate(wt, 4, 2, True)
    X = o.project_packed(x, ax, 4, 2, False, ld_words=ldx)
    W = o.project_packed(wt, aw, 4, 2, True, ld_words=ldx)
    P = (h + 2 * pad - r) // stride + 1
    Q = (w + 2 * pad - s) // stride + 1
    res = o.pack(random_codes(n * P * Q, cout, 4, seed=9), 4, 2, ld_words=esb.esb_row_words(cout, 4))
    s0 = esb.esb_dequant_scale(ax, esb.Fmt(4, 2), aw, esb.Fmt(4, 2))
    act = esb.ESB_ACT_RELU if not fo[2] else esb.ESB_ACT_NONE
    ep = esb.Epilogue(scale0=s0, bias0=0.01, act=act, residual=dev_i32(res), res_fmt=esb.Fmt(4, 2, True),
                      res_scale=0.0625, alpha_out=0.8, fmt_out=esb.Fmt(*fo))
    _, _, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, r, s,
                                      stride, pad, ep=ep, want_acc=False, want_codes=True)
    acc_o = o.conv2d_i64(X.reshape(n, h, w, ldx), (4, 2), W.reshape(cout, r, s, ldx), (4, 2),
                         n, h, w, c, cout, r, s, stride, pad).reshape(-1, cout)
    img = np.vectorize(lambda cc: o.image(int(cc), 4, 2))(o.unpack(res, cout, 4))
    _, co = o.epilogue(acc_o, np.full(cout, s0, np.float32), np.full(cout, 0.01, np.float32), act, 0.8, fo,
                       res_images=img, res_scale=0.0625)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("n,h,w,c,stride,fo,act,bias0", [
    (2, 15, 17, 40, 1, (4, 2, False), esb.ESB_ACT_RELU6, 0.0),     # ragged channels: padding slots of the last word
    (2, 15, 17, 96, 2, (4, 2, False), esb.ESB_ACT_RELU6, 0.3),     # stride 2, odd sizes, bias above zero
    (1, 7, 7, 960, 1, (4, 1, False), esb.ESB_ACT_RELU, -0.1),
    (3, 9, 9, 24, 1, (4, 2, True), esb.ESB_ACT_RELU, 0.05),        # signed set, non-negative outputs
])
def test_depthwise_codes_only_scalar_scale(n, h, w, c, stride, fo, act, bias0):
    r = s = 3
    pad = 1
    x = synth.half_normal((n * h * w, c), seed=c + w).numpy()
    wt = synth.he_normal((r * s, c), fan_in=9, seed=c + 7).numpy()
    ldx = esb.esb_row_words(c, 4)
    ax, _ = o.calibrate(x, 4, fo[1], False)
    aw, _ = o.calibrate(wt, 4, 2, True)
    X = o.project_packed(x, ax, 4, fo[1], False, ld_words=ldx)
    W = o.project_packed(wt, aw, 4, 2, True, ld_words=ldx)
    s0 = esb.esb_dequant_scale(ax, esb.Fmt(4, fo[1]), aw, esb.Fmt(4, 2))
    ep = esb.Epilogue(scale0=s0, bias0=bias0, act=act, alpha_out=0.45, fmt_out=esb.Fmt(*fo))
    _, _, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(4, fo[1], False), dev_i32(W), esb.Fmt(4, 2, True), n, h, w,
                                      c, c, r, s, stride, pad, groups=c, ep=ep, want_acc=False, want_codes=True)
    acc_o = o.dwconv_i64(X.reshape(n, h, w, ldx), (4, fo[1]), W.reshape(r, s, -1), (4, 2), n, h, w, c, r, s, stride,
                         pad).reshape(-1, c)
    _, co = o.epilogue(acc_o, np.full(c, s0, np.float32), np.full(c, bias0, np.float32), act, 0.45, fo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("c,fmt,r,stride", [(3, (4, 2), 7, 2), (3, (6, 3), 3, 2), (16, (4, 2), 1, 1), (8, (5, 2), 3, 1)])
def test_conv_filter_rows_walked_by_tap(c, fmt, r, stride):
    """Few channels per pixel (K takes only the words holding channels)."""
    n, h, w, cout = 2, 23, 21, 40
    pad = r // 2
    fx, fw = (fmt[0], fmt[1], True), (fmt[0], fmt[1], True)
    x = synth.normal((n * h * w, c), seed=c + r).numpy()
    wt = synth.he_normal((cout * r * r, c), fan_in=r * r * c, seed=r).numpy()
    ldx = esb.esb_row_words(c, fmt[0])
    ax, _ = o.calibrate(x, *fx)
    aw, _ = o.calibrate(wt, *fw)
    X = o.project_packed(x, ax, *fx, ld_words=ldx)
    W = o.project_packed(wt, aw, *fw, ld_words=ldx)
    acc, _, _ = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, r, r, stride,
                                    pad, want_acc=True)
    acc_o = o.conv2d_i64(X.reshape(n, h, w, ldx), fmt, W.reshape(cout, r, r, ldx), fmt, n, h, w, c, cout, r, r,
                         stride, pad).reshape(-1, cout)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)


@pytest.mark.parametrize("n,h,w,c,cout,r,pad,fmt", [
    (2, 14, 14, 64, 64, 3, 1, (6, 3)),            # ResNet18 layer shape, one channel block
    (2, 28, 28, 128, 96, 3, 1, (5, 2)),           # two channel blocks (register fill path)
    (1, 14, 14, 128, 64, 3, 1, (6, 3)),           # two channel blocks, 6-bit
    (2, 15, 30, 40, 48, 5, 2, (5, 2)),            # ragged channels, 5x5
    (2, 16, 31, 96, 80, 1, 0, (6, 3)),            # 1x1
    (2, 14, 14, 64, 64, 3, 1, (3, 1)),            # 3-bit: 16 K slots per word, one plane per word
    (2, 14, 14, 96, 32, 3, 1, (3, 1)),            # 3-bit, 12-word pixels
    (2, 15, 30, 40, 48, 3, 1, (2, 0)),            # 2-bit
])
def test_conv_halo_word_slots(n, h, w, c, cout, r, pad, fmt):
    """Stride-1 convolution of 5/6-bit codes on the halo kernel (word-slot K)."""
    fx, fw = (fmt[0], fmt[1], False), (fmt[0], fmt[1], True)
    assert esb.esb_conv2d_kernel(n, h, w, c, cout, r, r, 1, pad, esb.Fmt(*fx), esb.Fmt(*fw),
                                 out_b=fmt[0]) == esb.ESB_CONV_KERNEL_HALO
    x = synth.half_normal((n * h * w, c), seed=c + h).numpy()
    wt = synth.he_normal((cout * r * r, c), fan_in=r * r * c, seed=cout + r).numpy()
    ldx = esb.esb_row_words(c, fmt[0])
    ax, _ = o.calibrate(x, *fx)
    aw, _ = o.calibrate(wt, *fw)
    X = o.project_packed(x, ax, *fx, ld_words=ldx)
    W = o.project_packed(wt, aw, *fw, ld_words=ldx)
    s0 = esb.esb_dequant_scale(ax, esb.Fmt(*fmt), aw, esb.Fmt(*fmt))
    fo = (fmt[0], fmt[1], False)
    ep = esb.Epilogue(scale0=s0, bias0=0.0, act=esb.ESB_ACT_RELU, alpha_out=0.6, fmt_out=esb.Fmt(*fo))
    acc, _, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, r, r,
                                        1, pad, ep=ep, want_acc=True, want_codes=True)
    acc_o = o.conv2d_i64(X.reshape(n, h, w, ldx), fmt, W.reshape(cout, r, r, ldx), fmt, n, h, w, c, cout, r, r,
                         1, pad).reshape(-1, cout)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    _, co = o.epilogue(acc_o, np.full(cout, s0, np.float32), np.zeros(cout, np.float32), esb.ESB_ACT_RELU, 0.6, fo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))
