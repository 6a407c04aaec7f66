"""GPU parity of the CUDA-core ESB contraction with int64 accumulators
(Eq. esb_multiplication: significand product and shift) against the CPU
oracle, for formats and sums outside the tensor-core path's int32 / 2^24
range: (5,0), (6,1), (6,0) and K past 2^24.  Exact accumulators, bit-exact
epilogue outputs."""
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


def random_packed(rows, cols, fmt, seed, ld=None):
    b, k = fmt[0], fmt[1]
    codes = synth.uniform_ints((rows, cols), 0, 2 ** b, seed)
    return o.pack(codes, b, k, ld_words=ld if ld is not None else esb.esb_row_words(cols, b))


I64_GEMM = [
    # (M, N, K, fa, fb)
    (70, 65, 300, (6, 1), (6, 1)),          # images up to 3 * 2^14: sums far past 2^31
    (64, 60, 129, (5, 0), (4, 2)),          # PoT-like set up to 2^14
    (33, 17, 5, (6, 0), (3, 1)),            # images up to 2^30
    (130, 70, 1000, (4, 2), (6, 3)),        # an ordinary pair on this path
    (1, 1, 1, (7, 2), (7, 2)),
    (5, 3, 0, (6, 1), (6, 1)),              # K = 0: zero sums
]


@pytest.mark.parametrize("M,N,K,fa,fb", I64_GEMM)
def test_gemm_i64_matches_oracle(M, N, K, fa, fb):
    A = random_packed(M, max(K, 1), fa, seed=M + K)
    B = random_packed(N, max(K, 1), fb, seed=N + 3 * K)
    acc, _, _ = esb.esb_gemm_i64(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K)
    exp = o.gemm_i64(A, fa, B, fb, M, N, K)
    assert np.array_equal(acc.cpu().numpy(), exp)
    assert esb.esb_get_status() == 0


def test_gemm_i64_sum_past_two_to_the_24():
    # (4,2) at the largest image: K * 7 * 7 passes 2^24, where the tensor
    # path reports RANGE
    K = 400000
    b, k = 4, 2
    maxc = o.encode(o.C_of(b, k), b, k)
    rng = np.random.default_rng(1)
    ca = np.where(rng.random((4, K)) < 0.9, maxc, o.encode(-0.25, b, k)).astype(np.uint32)
    A = o.pack(ca, b, k, ld_words=esb.esb_row_words(K, b))
    acc, _, _ = esb.esb_gemm_i64(dev_i32(A), esb.Fmt(b, k), dev_i32(A), esb.Fmt(b, k), K)
    exp = o.gemm_i64(A, (b, k), A, (b, k), 4, 4, K)
    assert exp.max() > 2 ** 24
    assert np.array_equal(acc.cpu().numpy(), exp)
    with pytest.raises(esb.EsbError) as e:
        esb.esb_gemm(dev_i32(A), esb.Fmt(b, k), dev_i32(A), esb.Fmt(b, k), K)
    assert e.value.status == esb.ESB_ERR_RANGE


@pytest.mark.parametrize("fo", [(4, 2, False), (6, 3, True), (3, 1, True)])
def test_gemm_i64_epilogue_matches_oracle(fo):
    M, N, K = 150, 90, 200
    fa, fb = (6, 1), (5, 0)
    A = random_packed(M, K, fa, seed=11)
    B = random_packed(N, K, fb, seed=12)
    exp = o.gemm_i64(A, fa, B, fb, M, N, K)
    rng = np.random.default_rng(2)
    scale = (rng.uniform(0.5, 2.0, N) / np.abs(exp).max()).astype(np.float32)
    bias = rng.normal(0.0, 0.2, N).astype(np.float32)
    ep = esb.Epilogue(scale=torch.from_numpy(scale).cuda(), bias=torch.from_numpy(bias).cuda(),
                      act=esb.ESB_ACT_RELU if not fo[2] else esb.ESB_ACT_NONE, alpha_out=0.37, fmt_out=esb.Fmt(*fo))
    acc, y, codes = esb.esb_gemm_i64(dev_i32(A), esb.Fmt(*fa), dev_i32(B), esb.Fmt(*fb), K, ep=ep,
                                     want_acc=True, want_y=True, want_codes=True)
    assert np.array_equal(acc.cpu().numpy(), exp)
    yo, co = o.epilogue(exp, scale, bias, ep.act, 0.37, fo)
    assert np.array_equal(y.cpu().numpy(), yo)
    assert np.array_equal(u32(codes), o.pack(co, fo[0], fo[1], ld_words=codes.shape[1]))


I64_CONV = [
    # n, h, w, c, cout, r, s, stride, pad, fx, fw
    (2, 9, 7, 24, 32, 3, 3, 1, 1, (6, 1), (6, 1)),
    (1, 11, 12, 40, 48, 3, 3, 2, 1, (5, 0), (6, 3)),       # mixed widths
    (1, 15, 13, 3, 16, 7, 7, 2, 3, (4, 2), (6, 0)),        # first-layer shape
]


@pytest.mark.parametrize("n,h,w,c,cout,r,s,stride,pad,fx,fw", I64_CONV)
def test_conv_i64_matches_oracle(n, h, w, c, cout, r, s, stride, pad, fx, fw):
    ldx, ldw = esb.esb_row_words(c, fx[0]), esb.esb_row_words(c, fw[0]) + 1
    X = random_packed(n * h * w, c, fx, seed=h + c, ld=ldx)
    W = random_packed(cout * r * s, c, fw, seed=cout + r, ld=ldw)
    acc, _, _ = esb.esb_conv2d_nhwc_i64(dev_i32(X), esb.Fmt(*fx), dev_i32(W), esb.Fmt(*fw), n, h, w, c, cout, r, s,
                                        stride, pad)
    exp = o.conv2d_i64(X.reshape(n, h, w, ldx), fx, W.reshape(cout, r, s, ldw), fw, n, h, w, c, cout, r, s,
                       stride, pad).reshape(-1, cout)
    assert np.array_equal(acc.cpu().numpy(), exp)


def test_i64_range_error():
    f = esb.Fmt(7, 1)                  # images up to 3 * 2^30: products pass 2^62
    A = torch.zeros((4, 8), dtype=torch.int32, device="cuda")
    with pytest.raises(esb.EsbError) as e:
        esb.esb_gemm_i64(A, f, A, f, 8)
    assert e.value.status == esb.ESB_ERR_RANGE
