"""GPU parity of the CUDA-core kernels (depthwise conv, max pool, global
average pool) against the CPU oracle, through the C ABI."""
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


DW_CASES = [
    # n, h, w, c, stride, fx, fw, act
    (2, 14, 14, 96, 1, (4, 2, False), (4, 2, True), esb.ESB_ACT_RELU6),    # MobileNetV2 block shapes
    (2, 14, 14, 144, 2, (4, 2, False), (4, 2, True), esb.ESB_ACT_RELU6),
    (1, 7, 7, 960, 1, (4, 2, False), (4, 2, True), esb.ESB_ACT_RELU6),
    (2, 9, 11, 40, 1, (4, 2, True), (4, 1, True), esb.ESB_ACT_NONE),      # ragged channels (padding words)
    (2, 8, 8, 30, 2, (3, 1, False), (3, 1, True), esb.ESB_ACT_RELU),
    (2, 8, 8, 50, 1, (5, 2, False), (5, 2, True), esb.ESB_ACT_RELU),
    (2, 8, 8, 64, 1, (6, 3, False), (6, 3, True), esb.ESB_ACT_RELU6),
]


@pytest.mark.parametrize("n,h,w,c,stride,fx,fw,act", DW_CASES)
def test_depthwise_matches_oracle(n, h, w, c, stride, fx, fw, act):
    r = s = 3
    pad = 1
    x = synth.half_normal((n * h * w, c), seed=c + h).numpy() if not fx[2] else \
        synth.normal((n * h * w, c), seed=c + h).numpy()
    wt = synth.he_normal((r * s, c), fan_in=9, seed=c + 1).numpy()
    ldx = esb.esb_row_words(c, fx[0])
    ax, _ = o.calibrate(x, fx[0], fx[1], fx[2])
    aw, _ = o.calibrate(wt, fw[0], fw[1], fw[2])
    X = o.project_packed(x, ax, fx[0], fx[1], fx[2], ld_words=ldx)
    W = o.project_packed(wt, aw, fw[0], fw[1], fw[2], ld_words=esb.esb_row_words(c, fw[0]))
    scale = (np.float32(ax * aw / 2 ** (fx[1] + fw[1])) * (1 + 0.1 * synth.normal((c,), seed=5).numpy())).astype(np.float32)
    bias = (0.05 * synth.normal((c,), seed=6).numpy()).astype(np.float32)
    fo = (fx[0], fx[1], act == esb.ESB_ACT_NONE)          # ReLU/ReLU6 outputs use the unsigned set
    ep = esb.Epilogue(scale=torch.from_numpy(scale).cuda(), bias=torch.from_numpy(bias).cuda(), act=act,
                      alpha_out=0.29, fmt_out=esb.Fmt(fo[0], fo[1], bool(fo[2])))
    acc, y, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, c, r, s,
                                        stride, pad, groups=c, ep=ep, want_acc=True, want_y=True, want_codes=True)
    acc_o = o.dwconv_i64(X.reshape(n, h, w, ldx), fx[:2], W.reshape(r, s, -1), fw[:2], n, h, w, c, r, s, stride,
                         pad).reshape(-1, c)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    yo, co = o.epilogue(acc_o, scale, bias, act, 0.29, (fo[0], fo[1], bool(fo[2])))
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("n,h,w,c,stride,fo,act", [
    (2, 14, 14, 96, 1, (4, 2, False), esb.ESB_ACT_RELU6),      # MobileNetV2: per-channel BN fold, ReLU6
    (2, 13, 15, 44, 2, (4, 2, False), esb.ESB_ACT_RELU6),      # stride 2, ragged channels
    (2, 9, 11, 40, 1, (4, 1, True), esb.ESB_ACT_NONE),         # signed outputs: sign bits, negative zero buckets
    (2, 9, 10, 24, 1, (4, 3, False), esb.ESB_ACT_NONE),        # unsigned outputs of negative values: the zero code
    (1, 7, 7, 960, 1, (4, 2, False), esb.ESB_ACT_RELU),
])
def test_depthwise_codes_only_per_channel(n, h, w, c, stride, fo, act):
    """4-bit codes out with per-channel scale and bias and no other output:
    the word-at-a-time requantisation (buckets of |y| packed into a word)."""
    r = s = 3
    pad = 1
    x = synth.normal((n * h * w, c), seed=c + h + 1).numpy()
    wt = synth.he_normal((r * s, c), fan_in=9, seed=c + 3).numpy()
    fx, fw = (4, 2, True), (4, 2, True)
    ldx = esb.esb_row_words(c, 4)
    ax, _ = o.calibrate(x, *fx)
    aw, _ = o.calibrate(wt, *fw)
    X = o.project_packed(x, ax, *fx, ld_words=ldx)
    W = o.project_packed(wt, aw, *fw, ld_words=ldx)
    scale = (np.float32(ax * aw / 16) * (1 + 0.2 * synth.normal((c,), seed=7).numpy())).astype(np.float32)
    bias = (0.1 * synth.normal((c,), seed=8).numpy()).astype(np.float32)
    ep = esb.Epilogue(scale=torch.from_numpy(scale).cuda(), bias=torch.from_numpy(bias).cuda(), act=act,
                      alpha_out=0.31, fmt_out=esb.Fmt(*fo))
    _, _, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, c, r, s,
                                      stride, pad, groups=c, ep=ep, want_acc=False, want_codes=True)
    acc_o = o.dwconv_i64(X.reshape(n, h, w, ldx), fx[:2], W.reshape(r, s, -1), fw[:2], n, h, w, c, r, s, stride,
                         pad).reshape(-1, c)
    _, co = o.epilogue(acc_o, scale, bias, act, 0.31, fo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


@pytest.mark.parametrize("stride", [1, 2])
def test_depthwise_b4_largest_sums(stride):
    """4-bit (4,1) images reach 12 in magnitude, so 3x3 sums reach 9 * 144 =
    1296: the bound under which 4-bit depthwise sums are exact in fp16.
    Image 0 holds the largest positive image in half the channels, against
    filters of the largest positive and negative images; the rest is every
    code pattern drawn uniformly (negative zero and subnormal codes too)."""
    n, h, w, c = 2, 10, 13, 72
    r = s = 3
    pad = 1
    ldx = esb.esb_row_words(c, 4)
    xc = synth.uniform_ints((n * h * w, c), 0, 16, seed=11 + stride)
    wc = synth.uniform_ints((r * s, c), 0, 16, seed=12 + stride)
    xc[:h * w, :c // 2] = 5                       # code 0101 of (4,1): image +12
    wc[:, :c // 4] = 5
    wc[:, c // 4:c // 2] = 13                     # code 1101: image -12
    X = o.pack(xc, 4, 1, ld_words=ldx)
    W = o.pack(wc, 4, 1, ld_words=ldx)
    scale = np.full(c, 1e-3, np.float32)
    bias = np.zeros(c, np.float32)
    fo = (4, 1, True)
    ep = esb.Epilogue(scale=torch.from_numpy(scale).cuda(), bias=torch.from_numpy(bias).cuda(),
                      act=esb.ESB_ACT_NONE, alpha_out=0.5, fmt_out=esb.Fmt(*fo))
    acc, y, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fo), dev_i32(W), esb.Fmt(*fo), n, h, w, c, c, r, s,
                                        stride, pad, groups=c, ep=ep, want_acc=True, want_y=True, want_codes=True)
    acc_o = o.dwconv_i64(X.reshape(n, h, w, ldx), (4, 1), W.reshape(r, s, -1), (4, 1), n, h, w, c, r, s, stride,
                         pad).reshape(-1, c)
    assert acc_o.max() == 1296 and acc_o.min() == -1296
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    yo, co = o.epilogue(acc_o, scale, bias, esb.ESB_ACT_NONE, 0.5, fo)
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


POOL_CASES = [
    # n, h, w, c, win, stride, pad, fmt
    (2, 112, 112, 64, 3, 2, 1, (4, 2)),     # ResNet18 stem pool
    (2, 7, 6, 9, 3, 2, 1, (4, 2)),          # ragged: odd sizes, channel padding
    (1, 10, 10, 33, 2, 2, 0, (5, 1)),
    (1, 9, 9, 70, 3, 1, 1, (3, 1)),
]


@pytest.mark.parametrize("n,h,w,c,win,stride,pad,fmt", POOL_CASES)
def test_maxpool_matches_oracle(n, h, w, c, win, stride, pad, fmt):
    b, k = fmt
    codes = synth.uniform_ints((n * h * w, c), 0, 2 ** b, seed=h * c)
    X = o.pack(codes, b, k, ld_words=esb.esb_row_words(c, b))
    Y = esb.esb_maxpool_nhwc(dev_i32(X), esb.Fmt(b, k), n, h, w, c, win, stride, pad)
    exp = o.maxpool_codes(X.reshape(n, h, w, -1), b, k, n, h, w, c, win, stride, pad).reshape(Y.shape[0], -1)
    assert np.array_equal(u32(Y), exp)


@pytest.mark.parametrize("n,h,w,c,win,stride,pad,k", [(2, 112, 112, 64, 3, 2, 1, 2), (2, 7, 6, 9, 3, 2, 1, 2),
                                                      (1, 11, 13, 21, 3, 2, 1, 1), (1, 9, 8, 16, 2, 2, 0, 0),
                                                      (1, 6, 7, 5, 3, 1, 1, 3)])
def test_maxpool_unsigned_4bit_matches_oracle(n, h, w, c, win, stride, pad, k):
    # the decode-free path: unsigned 4-bit codes (post-ReLU activations),
    # window maxima taken on the rotated code ranks
    codes = synth.uniform_ints((n * h * w, c), 0, 8, seed=h * c + k)
    X = o.pack(codes, 4, k, ld_words=esb.esb_row_words(c, 4))
    Y = esb.esb_maxpool_nhwc(dev_i32(X), esb.Fmt(4, k, False), n, h, w, c, win, stride, pad)
    exp = o.maxpool_codes(X.reshape(n, h, w, -1), 4, k, n, h, w, c, win, stride, pad).reshape(Y.shape[0], -1)
    assert np.array_equal(u32(Y), exp)


@pytest.mark.parametrize("n,h,w,c,win,stride,pad,fmt", [(2, 56, 56, 64, 3, 2, 1, (3, 1)), (1, 11, 13, 23, 3, 2, 1, (5, 2)),
                                                        (1, 9, 8, 16, 2, 2, 0, (6, 3)), (1, 6, 7, 5, 3, 1, 1, (2, 0)),
                                                        (1, 7, 9, 30, 3, 2, 1, (7, 2)), (1, 5, 6, 9, 3, 1, 1, (8, 4))])
def test_maxpool_unsigned_rank_matches_oracle(n, h, w, c, win, stride, pad, fmt):
    # unsigned codes of widths other than 4: window maxima on the rotated ranks
    b, k = fmt
    codes = synth.uniform_ints((n * h * w, c), 0, 2 ** (b - 1), seed=h * c + b)
    X = o.pack(codes, b, k, ld_words=esb.esb_row_words(c, b))
    Y = esb.esb_maxpool_nhwc(dev_i32(X), esb.Fmt(b, k, False), n, h, w, c, win, stride, pad)
    exp = o.maxpool_codes(X.reshape(n, h, w, -1), b, k, n, h, w, c, win, stride, pad).reshape(Y.shape[0], -1)
    assert np.array_equal(u32(Y), exp)


@pytest.mark.parametrize("n,hw,c,fmt", [(4, 49, 512, (4, 2)), (3, 49, 1280, (4, 2)), (2, 16, 37, (6, 3)),
                                        (2, 1, 5, (3, 1)), (3, 25, 530, (2, 0)), (2, 100, 300, (5, 2))])
def test_avgpool_matches_oracle(n, hw, c, fmt):
    b, k = fmt
    x = synth.half_normal((n * hw, c), seed=c).numpy()
    ax, _ = o.calibrate(x, b, k, False)
    X = o.project_packed(x, ax, b, k, False, ld_words=esb.esb_row_words(c, b))
    scale = float(np.float32(ax * 2.0 ** -k / hw))
    y, codes = esb.esb_avgpool_nhwc(dev_i32(X), esb.Fmt(b, k, False), n, hw, c, scale, 0.21, esb.Fmt(b, k, False),
                                    want_y=True)
    sums = o.avgpool_sum_i64(X.reshape(n, hw, -1), b, k, n, hw, c)
    yo = (np.float32(scale) * sums.astype(np.float32)).astype(np.float32)
    assert np.array_equal(y.cpu().numpy(), yo)
    co = o.project_codes(yo, 0.21, b, k, False)
    assert np.array_equal(u32(codes), o.pack(co, b, k, ld_words=codes.shape[1]))
