"""GPU parity of the significand-split contraction (formats with k >= 4,
whose integer images have 5 to 8 significant bits and are no E4M3 number)
and of convolutions whose input and filter codes differ in width, against
the CPU oracle: exact int32 accumulators, bit-exact fp32 epilogue outputs
and requantised codes (Sec. III-B products of set elements; Table 1's
(6,4), (7,5), (8,5) and (8,6) formats)."""
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
        codes &= np.uint32((1 << (b - 1)) - 1)
    return o.pack(codes, b, k, ld_words=esb.esb_row_words(cols, b))


def max_image(b, k):
    return o.C_of(b, k) * 2 ** k


SPLIT_GEMM = [
    # (M, N, K, fa, fb): one or both operands split, ragged shapes, K tails
    (128, 64, 512, (6, 4), (6, 4)),
    (130, 70, 333, (6, 4), (4, 2)),
    (100, 96, 200, (4, 2), (6, 5)),
    (257, 48, 1000, (5, 4), (5, 4)),
    (64, 80, 260, (7, 5), (3, 1)),
    (96, 64, 1000, (8, 6), (8, 7)),
    (33, 17, 1000, (7, 4), (7, 6)),
    (40, 24, 4, (8, 4), (4, 1)),
    (300, 256, 777, (6, 4), (5, 2)),
    (1, 1, 1, (8, 5), (6, 4)),
]


@pytest.mark.parametrize("M,N,K,fa,fb", SPLIT_GEMM)
def test_split_gemm_acc_matches_oracle(M, N, K, fa, fb):
    assert K * max_image(*fa) * max_image(*fb) < 2 ** 24
    A = random_packed(M, K, fa, seed=M * 5 + K)
    B = random_packed(N, K, fb, seed=N * 13 + K)
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K)
    exp = o.gemm_i64(A, fa, B, fb, M, N, K)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), exp)
    assert esb.esb_get_status() == 0


@pytest.mark.parametrize("fmt,K", [((6, 4), 17000), ((8, 6), 1000), ((5, 4), 70000)])
def test_split_gemm_exact_near_the_accumulation_bound(fmt, K):
    # partial sums grow to just under 2^24 while +-1 terms keep arriving:
    # a lost low bit in the fp32 accumulation of the planes is an integer
    # mismatch
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
    assert exp.max() < 2 ** 24 and exp.max() > 2 ** 23
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), exp)


def test_split_gemm_fused_epilogue_matches_oracle():
    # projected data (DDA alpha of each operand), per-channel scale and bias,
    # ReLU6, requantised to a split format as well
    M, N, K = 200, 96, 300
    fa, fb, fo = (6, 4, False), (6, 4, True), (6, 4, False)
    xa = synth.half_normal((M, K), seed=3).numpy()
    xb = synth.he_normal((N, K), fan_in=K, seed=4).numpy()
    aa, _ = o.calibrate(xa, *fa)
    ab, _ = o.calibrate(xb, *fb)
    A = o.project_packed(xa, aa, *fa, ld_words=esb.esb_row_words(K, 6))
    B = o.project_packed(xb, ab, *fb, ld_words=esb.esb_row_words(K, 6))
    s0 = esb.esb_dequant_scale(aa, esb.Fmt(6, 4), ab, esb.Fmt(6, 4))
    rng = np.random.default_rng(8)
    scale = (s0 * rng.uniform(0.5, 2.0, N)).astype(np.float32)
    bias = rng.normal(0.0, 0.3, N).astype(np.float32)
    ep = esb.Epilogue(scale=torch.from_numpy(scale).cuda(), bias=torch.from_numpy(bias).cuda(),
                      act=esb.ESB_ACT_RELU6, alpha_out=0.61, fmt_out=esb.Fmt(*fo))
    acc, y, codes = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K, ep=ep,
                                 want_acc=True, want_y=True, want_codes=True)
    acc_o = o.gemm_i64(A, fa[:2], B, fb[:2], M, N, K)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    yo, co = o.epilogue(acc_o, scale, bias, esb.ESB_ACT_RELU6, 0.61, fo)
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, 6, 4, ld_words=codes.shape[1]))


def test_split_gemm_tiled_entry_point_takes_the_split_path():
    # esb_gemm_tiled hands significand-split operands to esb_gemm's kernels
    M, N, K = 512, 512, 2048
    fa, fb = (6, 4), (6, 5)
    A = random_packed(M, K, fa, seed=1)
    B = random_packed(N, K, fb, seed=2)
    ws = torch.empty(esb.esb_gemm_tiled_workspace_bytes(M, N, K), dtype=torch.uint8, device="cuda")
    acc, _, _ = esb.esb_gemm(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K, workspace=ws)
    rows = np.r_[0:8, 250:260, M - 8:M]
    exp = o.gemm_i64(A[rows], fa, B, fb, len(rows), N, K)
    assert np.array_equal(acc.cpu().numpy()[rows].astype(np.int64), exp)


def test_split_range_error():
    # (6,4) x (6,4): K max|I|^2 >= 2^24 beyond K = 17459
    K = 17472
    A = np.zeros((128, esb.esb_row_words(K, 6)), np.uint32)
    with pytest.raises(esb.EsbError) as e:
        esb.esb_gemm(dev_i32(A), esb.Fmt(6, 4), dev_i32(A), esb.Fmt(6, 4), K)
    assert e.value.status == esb.ESB_ERR_RANGE


CONV_MIXED = [
    # n, h, w, c, cout, r, s, stride, pad, fx, fw
    (2, 10, 10, 64, 64, 3, 3, 1, 1, (6, 4, False), (6, 4, True)),     # both split
    (2, 9, 11, 40, 48, 3, 3, 1, 1, (5, 4, False), (4, 2, True)),      # split input, mixed widths
    (2, 12, 12, 64, 32, 3, 3, 2, 1, (4, 2, False), (6, 3, True)),     # mixed widths, no split
    (1, 15, 13, 30, 64, 5, 5, 1, 2, (3, 1, False), (5, 2, True)),     # 10 vs 6 codes per word
    (2, 8, 8, 96, 80, 1, 1, 1, 0, (4, 2, False), (8, 6, True)),       # 1x1, split filters
    (1, 19, 23, 3, 64, 7, 7, 2, 3, (6, 4, True), (6, 5, True)),       # first-layer shape, c = 3
]


@pytest.mark.parametrize("n,h,w,c,cout,r,s,stride,pad,fx,fw", CONV_MIXED)
def test_split_and_mixed_width_conv_matches_oracle(n, h, w, c, cout, r, s, stride, pad, fx, fw):
    x = synth.half_normal((n * h * w, c), seed=h + c).numpy() if not fx[2] else \
        synth.normal((n * h * w, c), seed=h + c).numpy()
    wt = synth.he_normal((cout * r * s, c), fan_in=r * s * c, seed=cout + r).numpy()
    ax, _ = o.calibrate(x, *fx)
    aw, _ = o.calibrate(wt, *fw)
    ldx, ldw = esb.esb_row_words(c, fx[0]), esb.esb_row_words(c, fw[0])
    X = o.project_packed(x, ax, *fx, ld_words=ldx)
    W = o.project_packed(wt, aw, *fw, ld_words=ldw)
    kern = esb.esb_conv2d_kernel(n, h, w, c, cout, r, s, stride, pad, esb.Fmt(*fx), esb.Fmt(*fw), out_b=fx[0])
    assert kern in (esb.ESB_CONV_KERNEL_IM2COL, esb.ESB_CONV_KERNEL_STREAMED)
    fo = (fx[0], fx[1], False)
    s0 = esb.esb_dequant_scale(ax, esb.Fmt(*fx[:2]), aw, esb.Fmt(*fw[:2]))
    ep = esb.Epilogue(scale0=s0, bias0=0.01, act=esb.ESB_ACT_RELU, alpha_out=0.7, fmt_out=esb.Fmt(*fo))
    acc, y, codes = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, r, s,
                                        stride, pad, ep=ep, want_acc=True, want_y=True, want_codes=True)
    acc_o = o.conv2d_i64(X.reshape(n, h, w, ldx), fx[:2], W.reshape(cout, r, s, ldw), fw[:2],
                         n, h, w, c, cout, r, s, stride, pad).reshape(-1, cout)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
    yo, co = o.epilogue(acc_o, np.full(cout, s0, np.float32), np.full(cout, 0.01, np.float32), 1, 0.7, fo)
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))
    assert esb.esb_get_status() == 0


def test_same_width_conv_with_a_wider_filter_stride():
    # filter rows padded beyond the input's stride (ldw > ldx, same width)
    n, h, w, c, cout = 2, 9, 9, 40, 32
    fx, fw = (4, 2, False), (4, 2, True)
    x = synth.half_normal((n * h * w, c), seed=5).numpy()
    wt = synth.he_normal((cout * 9, c), fan_in=9 * c, seed=6).numpy()
    ax, _ = o.calibrate(x, *fx)
    aw, _ = o.calibrate(wt, *fw)
    ldx = esb.esb_row_words(c, 4)
    X = o.project_packed(x, ax, *fx, ld_words=ldx)
    W = o.project_packed(wt, aw, *fw, ld_words=ldx + 4)
    acc, _, _ = esb.esb_conv2d_nhwc(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, 3, 3, 1, 1)
    acc_o = o.conv2d_i64(X.reshape(n, h, w, ldx), fx[:2], W.reshape(cout, 3, 3, ldx + 4), fw[:2],
                         n, h, w, c, cout, 3, 3, 1, 1).reshape(-1, cout)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o)
