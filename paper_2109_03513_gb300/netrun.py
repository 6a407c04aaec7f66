"""Whole-network forward passes through the C ABI, for the paper's workload
shapes (Sec. V-A): ResNet18, MobileNetV2 (width 1.0, ReLU6) and AlexNet's
classifier, every conv/FC layer ESB-coded.

A network is a Python function over a Runner; the runner only sequences
libesb calls and keeps their buffers (all arithmetic runs in the library).
The first pass ("calibrate") creates random He-init weights, calibrates and
projects them once, and takes each layer's output alpha from the DDA of its
fp32 output on a calibration batch.  Later passes ("infer") emit only the
packed codes of every layer with those fixed alphas, so a pass is a fixed
sequence of launches that a CUDA graph can replay.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import torch

from . import esb, synth


@dataclass
class DAct:
    """A quantised activation on the device: packed NHWC codes."""
    codes: torch.Tensor
    fmt: esb.Fmt
    alpha: float
    n: int
    h: int
    w: int
    c: int


@dataclass
class LayerInfo:
    kind: str
    macs: int
    shape: str


class Runner:
    def __init__(self, b: int, k: int, seed: int = 0, device="cuda"):
        self.b, self.k = b, k
        self.seed = seed
        self.dev = torch.device(device)
        self.mode = "calibrate"
        self.params: list[dict] = []
        self.idx = 0
        self.info: list[LayerInfo] = []
        self.marks: Optional[list] = None            # per-layer CUDA events of a timed pass

    # ------------------------------------------------------------ helpers
    def _layer(self):
        i = self.idx
        self.idx += 1
        if self.mode == "calibrate":
            self.params.append({})
        return i, self.params[i]

    def _mark(self):
        if self.marks is not None:
            e = torch.cuda.Event(enable_timing=True)
            e.record()
            self.marks.append(e)

    def _weights(self, p, rows, c, fan_in):
        self.seed += 1
        wt = synth.he_normal((rows, c), fan_in=fan_in, seed=self.seed).to(self.dev)
        f = esb.Fmt(self.b, self.k, True)
        a, _ = esb.esb_calibrate_dda(wt, f)
        p["aw"] = float(a.item())
        p["W"] = esb.esb_project(wt, f, alpha=p["aw"])

    def _out_alpha(self, y, signed):
        a, _ = esb.esb_calibrate_dda(y, esb.Fmt(self.b, self.k, signed))
        return float(a.item())

    def begin(self, mode):
        self.mode = mode
        self.idx = 0
        if mode == "calibrate":
            self.info = []

    # ------------------------------------------------------------- layers
    def input(self, x: torch.Tensor, n, h, w, c) -> DAct:
        """fp32 NHWC images -> signed codes with the calibrated input alpha."""
        _, p = self._layer()
        f = esb.Fmt(self.b, self.k, True)
        if self.mode == "calibrate":
            a, _ = esb.esb_calibrate_dda(x, f)
            p["a"] = float(a.item())
        codes = esb.esb_project(x.reshape(-1, c), f, alpha=p["a"])
        self._mark()
        return DAct(codes, f, p["a"], n, h, w, c)

    def conv(self, x: DAct, cout, r, s, stride, pad, act=esb.ESB_ACT_RELU, res: Optional[DAct] = None,
             groups=1) -> DAct:
        _, p = self._layer()
        dw = groups == x.c and x.c > 1
        if self.mode == "calibrate":
            self._weights(p, (r * s) if dw else cout * r * s, x.c, r * s if dw else r * s * x.c)
        fw = esb.Fmt(self.b, self.k, True)
        signed_out = act == esb.ESB_ACT_NONE
        fo = esb.Fmt(self.b, self.k, signed_out)
        s0 = esb.esb_dequant_scale(x.alpha, x.fmt, p["aw"], fw)
        res_scale = esb.esb_dequant_scale(res.alpha, res.fmt, 1.0, esb.Fmt(8, 0)) if res is not None else 0.0
        ep = dict(scale0=s0, act=act, residual=res.codes if res is not None else None,
                  res_fmt=res.fmt if res is not None else None, res_scale=res_scale)
        geo = (x.n, x.h, x.w, x.c, cout, r, s, stride, pad)
        if self.mode == "calibrate":
            _, y, _ = esb.esb_conv2d_nhwc(x.codes, x.fmt, p["W"], fw, *geo, groups=groups,
                                          ep=esb.Epilogue(**ep, alpha_out=1.0, fmt_out=fo),
                                          want_acc=False, want_y=True)
            p["a_out"] = self._out_alpha(y, signed_out)
            del y
            P, Q = esb.conv_out_hw(x.h, x.w, r, s, stride, pad)
            macs = x.n * P * Q * cout * r * s * (1 if dw else x.c)
            self.info.append(LayerInfo("dwconv" if dw else "conv", macs,
                                       f"{x.h}x{x.w}x{x.c}->{cout} {r}x{s}/{stride}"))
        _, _, codes = esb.esb_conv2d_nhwc(x.codes, x.fmt, p["W"], fw, *geo, groups=groups,
                                          ep=esb.Epilogue(**ep, alpha_out=p["a_out"], fmt_out=fo),
                                          want_acc=False, want_codes=True)
        self._mark()
        P, Q = esb.conv_out_hw(x.h, x.w, r, s, stride, pad)
        return DAct(codes, fo, p["a_out"], x.n, P, Q, cout)

    def maxpool(self, x: DAct, win=3, stride=2, pad=1) -> DAct:
        _, p = self._layer()
        Y = esb.esb_maxpool_nhwc(x.codes, x.fmt, x.n, x.h, x.w, x.c, win, stride, pad)
        if self.mode == "calibrate":
            self.info.append(LayerInfo("maxpool", 0, f"{x.h}x{x.w}x{x.c} {win}x{win}/{stride}"))
        self._mark()
        P, Q = esb.conv_out_hw(x.h, x.w, win, win, stride, pad)
        return DAct(Y, x.fmt, x.alpha, x.n, P, Q, x.c)

    def avgpool(self, x: DAct) -> DAct:
        _, p = self._layer()
        hw = x.h * x.w
        scale = esb.esb_dequant_scale(x.alpha, x.fmt, 1.0 / hw, esb.Fmt(8, 0))
        if self.mode == "calibrate":
            y, _ = esb.esb_avgpool_nhwc(x.codes, x.fmt, x.n, hw, x.c, scale, 1.0, x.fmt, want_y=True)
            p["a_out"] = self._out_alpha(y, x.fmt.signed)
            self.info.append(LayerInfo("avgpool", 0, f"{x.h}x{x.w}x{x.c}"))
        _, codes = esb.esb_avgpool_nhwc(x.codes, x.fmt, x.n, hw, x.c, scale, p["a_out"], x.fmt)
        self._mark()
        return DAct(codes, x.fmt, p["a_out"], x.n, 1, 1, x.c)

    def fc(self, x: DAct, nout, act=esb.ESB_ACT_NONE, workspace: bool = False) -> DAct:
        _, p = self._layer()
        if self.mode == "calibrate":
            self._weights(p, nout, x.c, x.c)
            M = x.n
            p["ws"] = (torch.empty(max(16, esb.esb_gemm_tiled_workspace_bytes(M, nout, x.c)), dtype=torch.uint8,
                                   device=self.dev) if workspace else None)
        fw = esb.Fmt(self.b, self.k, True)
        signed_out = act == esb.ESB_ACT_NONE
        fo = esb.Fmt(self.b, self.k, signed_out)
        s0 = esb.esb_dequant_scale(x.alpha, x.fmt, p["aw"], fw)
        if self.mode == "calibrate":
            _, y, _ = esb.esb_gemm(x.codes, x.fmt, p["W"], fw, x.c, ep=esb.Epilogue(scale0=s0, act=act, fmt_out=fo),
                                   want_acc=False, want_y=True, workspace=p["ws"])
            p["a_out"] = self._out_alpha(y, signed_out)
            self.info.append(LayerInfo("fc", x.n * nout * x.c, f"{x.c}->{nout}"))
        _, _, codes = esb.esb_gemm(x.codes, x.fmt, p["W"], fw, x.c, workspace=p["ws"],
                                   ep=esb.Epilogue(scale0=s0, act=act, alpha_out=p["a_out"], fmt_out=fo),
                                   want_acc=False, want_codes=True)
        self._mark()
        return DAct(codes, fo, p["a_out"], x.n, 1, 1, nout)


# ----------------------------------------------------------- networks

def resnet18(rn: Runner, x: torch.Tensor, n: int) -> DAct:
    """ResNet18 (BN folded to identity): 7x7/2 stem, 3x3/2 max pool, four
    stages of two basic blocks (1x1/2 projection shortcuts), global average
    pool, 512 -> 1000 classifier; x is n x 224 x 224 x 3 fp32 NHWC."""
    a = rn.input(x, n, 224, 224, 3)
    a = rn.conv(a, 64, 7, 7, 2, 3)
    a = rn.maxpool(a)
    for cout, stride in [(64, 1), (64, 1), (128, 2), (128, 1), (256, 2), (256, 1), (512, 2), (512, 1)]:
        h = rn.conv(a, cout, 3, 3, stride, 1)
        short = a if (stride == 1 and a.c == cout) else rn.conv(a, cout, 1, 1, stride, 0, act=esb.ESB_ACT_NONE)
        a = rn.conv(h, cout, 3, 3, 1, 1, res=short)
    a = rn.avgpool(a)
    return rn.fc(a, 1000)


# MobileNetV2 (width 1.0) inverted-residual settings: expansion t, output
# channels c, repeats n, first stride s
MBV2 = [(1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2), (6, 96, 3, 1), (6, 160, 3, 2), (6, 320, 1, 1)]


def mobilenetv2(rn: Runner, x: torch.Tensor, n: int) -> DAct:
    """MobileNetV2 (ReLU6): 3x3/2 stem, 17 bottlenecks (1x1 expand,
    depthwise 3x3, 1x1 linear projection, residual where stride 1 and widths
    match), 320 -> 1280 1x1 conv, global average pool, 1280 -> 1000."""
    r6 = esb.ESB_ACT_RELU6
    a = rn.input(x, n, 224, 224, 3)
    a = rn.conv(a, 32, 3, 3, 2, 1, act=r6)
    for t, c, reps, s in MBV2:
        for i in range(reps):
            stride = s if i == 0 else 1
            h = a if t == 1 else rn.conv(a, a.c * t, 1, 1, 1, 0, act=r6)
            h = rn.conv(h, h.c, 3, 3, stride, 1, act=r6, groups=h.c)
            res = a if (stride == 1 and a.c == c) else None
            a = rn.conv(h, c, 1, 1, 1, 0, act=esb.ESB_ACT_NONE, res=res)
    a = rn.conv(a, 1280, 1, 1, 1, 0, act=r6)
    a = rn.avgpool(a)
    return rn.fc(a, 1000)


def alexnet_fc(rn: Runner, x: torch.Tensor, n: int) -> DAct:
    """AlexNet's classifier 9216 -> 4096 -> 4096 -> 1000 (ReLU between) on
    the tiled large-operand GEMM; x is n x 9216 fp32."""
    a = rn.input(x, n, 1, 1, 9216)
    a = rn.fc(a, 4096, act=esb.ESB_ACT_RELU, workspace=True)
    a = rn.fc(a, 4096, act=esb.ESB_ACT_RELU, workspace=True)
    return rn.fc(a, 1000, workspace=True)


NETWORKS = {"resnet18": (resnet18, (224, 224, 3)), "mobilenetv2": (mobilenetv2, (224, 224, 3)),
            "alexnet_fc": (alexnet_fc, (1, 1, 9216))}
