"""Whole-network parity: every layer of a ResNet18-shaped forward (stem to
classifier), of MobileNetV2-shaped inverted-residual blocks and of the
AlexNet-shaped classifier chain, run through the C ABI layer by layer and
checked against the CPU oracle: exact int32 accumulators, fp32 epilogue
outputs and requantised codes at every layer, DDA alphas within 1e-6.

Each layer is calibrated as a deployed network would be: the fp32 output of a
first pass gives the layer's output alpha (DDA), and the second pass emits the
requantised codes the next layer reads.  The oracle chain takes the GPU's
alphas (each checked against the oracle's own calibration of the same fp32
tensor) so that every layer compares codes bit for bit.  Random He-init
weights, batch 1-8 synthetic inputs N(0,1) (the configurations' shapes at a
batch the oracle finishes in seconds)."""
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


def images(codes, cols, b, k):
    c = o.unpack(codes, cols, b)
    lut = np.array([o.image(v, b, k) for v in range(2 ** b)], np.int64)
    return lut[c]


class Act:
    """A quantised activation: packed codes on the device and on the host,
    its format and alpha, its NHWC geometry."""

    def __init__(self, codes_dev, codes_np, fmt, alpha, n, h, w, c):
        self.d, self.np, self.f, self.a = codes_dev, codes_np, fmt, alpha
        self.n, self.h, self.w, self.c = n, h, w, c


class Net:
    def __init__(self, fmt, seed):
        self.b, self.k = fmt
        self.seed = seed
        self.layers = 0

    def fa(self, signed=False):
        return (self.b, self.k, signed)

    def weights(self, rows, c, fan_in):
        """He-init fp32 weights -> signed codes (GPU DDA alpha, checked against the oracle)."""
        self.seed += 1
        wt = synth.he_normal((rows, c), fan_in=fan_in, seed=self.seed)
        f = esb.Fmt(self.b, self.k, True)
        a, _ = esb.esb_calibrate_dda(wt.cuda(), f)
        ag = float(a.item())
        ao, _ = o.calibrate(wt.numpy(), self.b, self.k, True)
        assert abs(ag - ao) <= 1e-6 * ao
        Wd = esb.esb_project(wt.cuda(), f, alpha=ag)
        Wn = o.project_packed(wt.numpy(), ag, self.b, self.k, True, ld_words=Wd.shape[1])
        assert np.array_equal(u32(Wd), Wn)
        return Wd, Wn, ag

    def input(self, n, h, w, c):
        self.seed += 1
        x = synth.normal((n * h * w, c), seed=self.seed)
        f = esb.Fmt(self.b, self.k, True)
        a, _ = esb.esb_calibrate_dda(x.cuda(), f)
        ag = float(a.item())
        Xd = esb.esb_project(x.cuda(), f, alpha=ag)
        Xn = o.project_packed(x.numpy(), ag, self.b, self.k, True, ld_words=Xd.shape[1])
        assert np.array_equal(u32(Xd), Xn)
        return Act(Xd, Xn, self.fa(True), ag, n, h, w, c)

    def out_alpha(self, y, signed):
        """DDA alpha of a layer's fp32 output, GPU and oracle."""
        a, _ = esb.esb_calibrate_dda(y, esb.Fmt(self.b, self.k, signed))
        ag = float(a.item())
        ao, _ = o.calibrate(y.cpu().numpy().reshape(-1), self.b, self.k, signed)
        assert abs(ag - ao) <= 1e-6 * ao, (self.layers, ag, ao)
        return ag

    def conv(self, x: Act, cout, r, s, stride, pad, act=esb.ESB_ACT_RELU, res: Act = None, groups=1):
        """One conv layer (dense or depthwise) with the fused epilogue: scale
        alpha_x alpha_w 2^-(kx+kw), optional residual (its integer image times
        its alpha 2^-k), activation, requantisation with the layer's DDA alpha."""
        self.layers += 1
        dw = groups == x.c
        c = x.c
        Wd, Wn, aw = self.weights((r * s) if dw else cout * r * s, c, r * s if dw else r * s * c)
        fx, fw = esb.Fmt(*x.f), esb.Fmt(self.b, self.k, True)
        s0 = esb.esb_dequant_scale(x.a, fx, aw, fw)
        signed_out = act == esb.ESB_ACT_NONE
        fo = (self.b, self.k, signed_out)
        res_scale = float(np.float32(res.a) * np.float32(2.0 ** -res.f[1])) if res is not None else 0.0
        kw = dict(stride=stride, pad=pad, groups=groups)
        ep = dict(scale0=s0, bias0=0.0, act=act, residual=res.d if res is not None else None,
                  res_fmt=esb.Fmt(*res.f) if res is not None else None, res_scale=res_scale)
        acc, y, _ = esb.esb_conv2d_nhwc(x.d, fx, Wd, fw, x.n, x.h, x.w, c, cout, r, s, **kw,
                                        ep=esb.Epilogue(**ep, alpha_out=1.0, fmt_out=esb.Fmt(*fo)),
                                        want_acc=True, want_y=True)
        a_out = self.out_alpha(y, signed_out)
        _, _, codes = esb.esb_conv2d_nhwc(x.d, fx, Wd, fw, x.n, x.h, x.w, c, cout, r, s, **kw,
                                          ep=esb.Epilogue(**ep, alpha_out=a_out, fmt_out=esb.Fmt(*fo)),
                                          want_acc=False, want_codes=True)
        P, Q = esb.conv_out_hw(x.h, x.w, r, s, stride, pad)
        ldx = x.np.shape[1]
        if dw:
            acc_o = o.dwconv_i64(x.np.reshape(x.n, x.h, x.w, ldx), x.f[:2], Wn.reshape(r, s, -1), (self.b, self.k),
                                 x.n, x.h, x.w, c, r, s, stride, pad).reshape(-1, c)
        else:
            acc_o = o.conv2d_i64(x.np.reshape(x.n, x.h, x.w, ldx), x.f[:2], Wn.reshape(cout, r, s, -1),
                                 (self.b, self.k), x.n, x.h, x.w, c, cout, r, s, stride, pad).reshape(-1, cout)
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o), ("acc", self.layers)
        res_img = images(res.np, cout, res.f[0], res.f[1]) if res is not None else None
        yo, _ = o.epilogue(acc_o, np.full(cout, s0, np.float32), np.zeros(cout, np.float32), act, 1.0, fo,
                           res_images=res_img, res_scale=res_scale)
        assert np.array_equal(y.cpu().numpy(), yo), ("y", self.layers)
        _, co = o.epilogue(acc_o, np.full(cout, s0, np.float32), np.zeros(cout, np.float32), act, a_out, fo,
                           res_images=res_img, res_scale=res_scale)
        cn = o.pack(co, fo[0], fo[1], ld_words=codes.shape[1])
        assert np.array_equal(u32(codes), cn), ("codes", self.layers)
        return Act(codes, cn, fo, a_out, x.n, P, Q, cout)

    def maxpool(self, x: Act, win=3, stride=2, pad=1):
        Y = esb.esb_maxpool_nhwc(x.d, esb.Fmt(*x.f), x.n, x.h, x.w, x.c, win, stride, pad)
        P, Q = esb.conv_out_hw(x.h, x.w, win, win, stride, pad)
        Yn = o.maxpool_codes(x.np.reshape(x.n, x.h, x.w, -1), x.f[0], x.f[1], x.n, x.h, x.w, x.c, win, stride, pad,
                             ld_out=Y.shape[1]).reshape(Y.shape[0], -1)
        assert np.array_equal(u32(Y), Yn)
        return Act(Y, Yn, x.f, x.a, x.n, P, Q, x.c)

    def avgpool(self, x: Act):
        hw = x.h * x.w
        scale = float(np.float32(x.a * 2.0 ** -x.f[1] / hw))
        y, _ = esb.esb_avgpool_nhwc(x.d, esb.Fmt(*x.f), x.n, hw, x.c, scale, 1.0, esb.Fmt(*x.f), want_y=True)
        a_out = self.out_alpha(y, x.f[2])
        _, codes = esb.esb_avgpool_nhwc(x.d, esb.Fmt(*x.f), x.n, hw, x.c, scale, a_out, esb.Fmt(*x.f))
        sums = o.avgpool_sum_i64(x.np.reshape(x.n, hw, -1), x.f[0], x.f[1], x.n, hw, x.c)
        yo = (np.float32(scale) * sums.astype(np.float32)).astype(np.float32)
        assert np.array_equal(y.cpu().numpy(), yo)
        cn = o.pack(o.project_codes(yo, a_out, x.f[0], x.f[1], x.f[2]), x.f[0], x.f[1], ld_words=codes.shape[1])
        assert np.array_equal(u32(codes), cn)
        return Act(codes, cn, x.f, a_out, x.n, 1, 1, x.c)

    def fc(self, x: Act, nout, act=esb.ESB_ACT_NONE, workspace=False):
        """Fully connected layer: GEMM over the flattened codes (M = batch)."""
        self.layers += 1
        Wd, Wn, aw = self.weights(nout, x.c, x.c)
        fx, fw = esb.Fmt(*x.f), esb.Fmt(self.b, self.k, True)
        s0 = esb.esb_dequant_scale(x.a, fx, aw, fw)
        signed_out = act == esb.ESB_ACT_NONE
        fo = (self.b, self.k, signed_out)
        M, K = x.n, x.c
        ws = None
        if workspace:
            ws = torch.empty(max(16, esb.esb_gemm_tiled_workspace_bytes(M, nout, K)), dtype=torch.uint8, device="cuda")
        acc, y, _ = esb.esb_gemm(x.d, fx, Wd, fw, K, ep=esb.Epilogue(scale0=s0, act=act, fmt_out=esb.Fmt(*fo)),
                                 want_acc=True, want_y=True, workspace=ws)
        a_out = self.out_alpha(y, signed_out)
        _, _, codes = esb.esb_gemm(x.d, fx, Wd, fw, K, workspace=ws,
                                   ep=esb.Epilogue(scale0=s0, act=act, alpha_out=a_out, fmt_out=esb.Fmt(*fo)),
                                   want_acc=False, want_codes=True)
        acc_o = o.gemm_i64(x.np, x.f[:2], Wn, (self.b, self.k), M, nout, K)
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), acc_o), ("acc", self.layers)
        yo, co = o.epilogue(acc_o, np.full(nout, s0, np.float32), np.zeros(nout, np.float32), act, a_out, fo)
        assert np.array_equal(y.cpu().numpy(), yo), ("y", self.layers)
        cn = o.pack(co, fo[0], fo[1], ld_words=codes.shape[1])
        assert np.array_equal(u32(codes), cn), ("codes", self.layers)
        return Act(codes, cn, fo, a_out, x.n, 1, 1, nout)


def basic_block(net, x, cout, stride):
    h = net.conv(x, cout, 3, 3, stride, 1)
    short = x if (stride == 1 and x.c == cout) else net.conv(x, cout, 1, 1, stride, 0, act=esb.ESB_ACT_NONE)
    return net.conv(h, cout, 3, 3, 1, 1, res=short)


@pytest.mark.parametrize("fmt", [(3, 1), (4, 2), (5, 2), (6, 3)])
def test_resnet18_forward_matches_oracle(fmt):
    # ResNet18 (BN folded to identity): 7x7/2 stem, 3x3/2 max pool, four
    # stages of two basic blocks (1x1/2 projection shortcuts), global average
    # pool, 512 -> 1000 classifier; batch 1 at 224 x 224
    net = Net(fmt, seed=100 * fmt[0] + fmt[1])
    x = net.input(1, 224, 224, 3)
    x = net.conv(x, 64, 7, 7, 2, 3)
    x = net.maxpool(x)
    for cout, stride in [(64, 1), (64, 1), (128, 2), (128, 1), (256, 2), (256, 1), (512, 2), (512, 1)]:
        x = basic_block(net, x, cout, stride)
    assert (x.h, x.w, x.c) == (7, 7, 512)
    x = net.avgpool(x)
    net.fc(x, 1000)
    assert net.layers == 21
    assert esb.esb_get_status() == 0


def test_mobilenetv2_blocks_match_oracle():
    # MobileNetV2 (width 1.0, ReLU6): the 3x3/2 stem, the first bottleneck,
    # a stride-2 inverted-residual block and a stride-1 one with its
    # residual (1x1 expand -> depthwise 3x3 -> 1x1 linear projection)
    net = Net((4, 2), seed=7)
    r6 = esb.ESB_ACT_RELU6
    x = net.input(1, 112, 112, 3)
    x = net.conv(x, 32, 3, 3, 2, 1, act=r6)                          # 56 x 56 x 32
    h = net.conv(x, 32, 3, 3, 1, 1, act=r6, groups=32)               # t = 1: depthwise, then project
    x = net.conv(h, 16, 1, 1, 1, 0, act=esb.ESB_ACT_NONE)
    h = net.conv(x, 96, 1, 1, 1, 0, act=r6)                          # t = 6, stride 2
    h = net.conv(h, 96, 3, 3, 2, 1, act=r6, groups=96)
    x = net.conv(h, 24, 1, 1, 1, 0, act=esb.ESB_ACT_NONE)            # 28 x 28 x 24
    h = net.conv(x, 144, 1, 1, 1, 0, act=r6)                         # t = 6, stride 1, residual
    h = net.conv(h, 144, 3, 3, 1, 1, act=r6, groups=144)
    y = net.conv(h, 24, 1, 1, 1, 0, act=esb.ESB_ACT_NONE, res=x)
    assert (y.h, y.w, y.c) == (28, 28, 24)
    assert esb.esb_get_status() == 0


# MobileNetV2 (width 1.0) inverted-residual settings: expansion t, output
# channels c, repeats n, first stride s
MBV2 = [(1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2), (6, 96, 3, 1), (6, 160, 3, 2), (6, 320, 1, 1)]


def test_mobilenetv2_forward_matches_oracle():
    # the whole MobileNetV2 at 224 x 224, batch 1: 3x3/2 stem, all 17
    # bottlenecks (1x1 expand, depthwise 3x3, 1x1 linear projection, residual
    # where stride 1 and widths match), the 320 -> 1280 1x1 conv, global
    # average pool and the 1280 -> 1000 classifier, every layer checked
    net = Net((4, 2), seed=21)
    r6 = esb.ESB_ACT_RELU6
    x = net.input(1, 224, 224, 3)
    x = net.conv(x, 32, 3, 3, 2, 1, act=r6)
    blocks = 0
    for t, c, n, s in MBV2:
        for i in range(n):
            stride = s if i == 0 else 1
            h = x if t == 1 else net.conv(x, x.c * t, 1, 1, 1, 0, act=r6)
            h = net.conv(h, h.c, 3, 3, stride, 1, act=r6, groups=h.c)
            res = x if (stride == 1 and x.c == c) else None
            x = net.conv(h, c, 1, 1, 1, 0, act=esb.ESB_ACT_NONE, res=res)
            blocks += 1
    assert blocks == 17 and (x.h, x.w, x.c) == (7, 7, 320)
    x = net.conv(x, 1280, 1, 1, 1, 0, act=r6)
    x = net.avgpool(x)
    net.fc(x, 1000)
    assert net.layers == 1 + 17 * 3 - 1 + 1 + 1
    assert esb.esb_get_status() == 0


def test_alexnet_classifier_matches_oracle(monkeypatch):
    # AlexNet's classifier 9216 -> 4096 -> 4096 -> 1000 (ReLU between), batch
    # 8, through the tiled large-operand GEMM (workspace; every shape to it)
    monkeypatch.setenv("ESB_GEMM_TILED_MIN_MACS", "0")
    net = Net((4, 2), seed=11)
    x = net.input(8, 1, 1, 9216)
    x = net.fc(x, 4096, act=esb.ESB_ACT_RELU, workspace=True)
    x = net.fc(x, 4096, act=esb.ESB_ACT_RELU, workspace=True)
    net.fc(x, 1000, workspace=True)
    assert esb.esb_get_status() == 0
