"""ctypes binding of libesb.so -- the C ABI declared in include/esb.h.

Argument marshalling only: every step of the ESB path runs in the library's
CUDA kernels.  PyTorch supplies device memory and streams.  Packed code
tensors are torch.int32 tensors whose bits are the uint32 code words.
If the library is missing this module raises; there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libesb.so")

ESB_OK = 0
ESB_ERR_INVALID_ARG = 1
ESB_ERR_UNSUPPORTED = 2
ESB_ERR_RANGE = 3
ESB_ERR_ALIGN = 4
ESB_ERR_CUDA = 5
ESB_ERR_TIMEOUT = 6
ESB_ERR_INTERNAL = 7

ESB_ROUND_HALF_AWAY = 0
ESB_ROUND_HALF_EVEN = 1
ESB_ACT_NONE = 0
ESB_ACT_RELU = 1
ESB_ACT_RELU6 = 2


class EsbError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: esb_status {status}")


class esb_format(ctypes.Structure):
    _fields_ = [("b", ctypes.c_int32), ("k", ctypes.c_int32), ("is_signed", ctypes.c_int32)]


class esb_epilogue(ctypes.Structure):
    _fields_ = [
        ("scale", ctypes.c_void_p), ("alpha_a_dev", ctypes.c_void_p), ("alpha_b_dev", ctypes.c_void_p),
        ("bias", ctypes.c_void_p),
        ("scale0", ctypes.c_float), ("bias0", ctypes.c_float),
        ("act", ctypes.c_int32),
        ("residual", ctypes.c_void_p), ("res_ld", ctypes.c_int64), ("res_fmt", esb_format),
        ("res_scale", ctypes.c_float),
        ("alpha_out", ctypes.c_float), ("alpha_out_dev", ctypes.c_void_p),
        ("fmt_out", esb_format), ("rounding_out", ctypes.c_int32),
    ]


class esb_conv_desc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("n", "h", "w", "c", "cout", "r", "s", "stride", "pad", "groups")]


@dataclass(frozen=True)
class Fmt:
    """ESB format: b total bits, k fraction bits (k+1 significant bits)."""
    b: int
    k: int
    signed: bool = True

    def c(self) -> esb_format:
        return esb_format(self.b, self.k, 1 if self.signed else 0)


_lib = None

# (name, restype, argtypes) of every exported symbol of include/esb.h.
_P, _I32, _I64, _F32, _SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
SIGNATURES = {
    "esb_version": (_I32, []),
    "esb_status_string": (ctypes.c_char_p, [_I32]),
    "esb_format_check": (_I32, [esb_format]),
    "esb_codes_per_word": (_I32, [_I32]),
    "esb_row_words": (_I64, [_I64, _I32]),
    "esb_zero_code": (ctypes.c_uint32, [esb_format]),
    "esb_alpha_star": (_I32, [_I32, _I32, _P, _P]),
    "esb_calibrate_dda_workspace_bytes": (_SZ, [_I64]),
    "esb_calibrate_dda": (_I32, [_P, _I64, esb_format, _P, _SZ, _P, _P, _P]),
    "esb_calibrate_dda_noalloc": (_I32, [_P, _I64, esb_format, _P, _P, _P]),
    "esb_dda_combine": (_I32, [_P, _I64, esb_format, _P, _P]),
    "esb_dn_project": (_I32, [_P, _I64, _I64, _P, esb_format, _I32, _P, _I64, _P, _P]),
    "esb_dn_backward_workspace_bytes": (_SZ, [_I64]),
    "esb_dn_backward": (_I32, [_P, _P, _I64, _P, _P, _SZ, _P, _P]),
    "esb_ema_update": (_I32, [_P, _P, ctypes.c_double, _P]),
    "esb_alpha_star_dist": (_I32, [_I32, _I32, _I32, _P, _P]),
    "esb_calibrate_dda_dist": (_I32, [_P, _I64, esb_format, _I32, _P, _SZ, _P, _P, _P]),
    "esb_dda_histogram": (_I32, [_P, _I64, esb_format, _P, _I32, _F32, _P, _P]),
    "esb_alpha_star_hist": (_I32, [_P, _I32, _F32, _I32, _I32, _P, _P]),
    "esb_calibrate_dda_empirical": (_I32, [_P, _I64, esb_format, _P, _SZ, _I32, _F32, _P, _P, _P, _P, _P]),
    "esb_dequant_scale": (_I32, [_F32, esb_format, _F32, esb_format, _P]),
    "esb_fold_bn_dn": (_I32, [_F32, esb_format, _F32, esb_format, _P, _P, _P, _P, _I64, ctypes.c_double,
                              ctypes.c_double, _P, _P]),
    "esb_project": (_I32, [_P, _I64, _I64, _I64, _F32, _P, esb_format, _I32, _P, _I64, _P]),
    "esb_project_dda": (_I32, [_P, _I64, _I64, esb_format, _I32, _P, _SZ, _P, _P, _P, _I64, _P]),
    "esb_dequant": (_I32, [_P, _I64, _I64, _I64, _F32, _P, esb_format, _P, _I64, _P]),
    "esb_gemm": (_I32, [_I64, _I64, _I64, _P, _I64, esb_format, _P, _I64, esb_format, _P, _P, _P, _P, _I64, _P]),
    "esb_gemm_tiled_workspace_bytes": (_SZ, [_I64, _I64, _I64]),
    "esb_gemm_tiled": (_I32, [_I64, _I64, _I64, _P, _I64, esb_format, _P, _I64, esb_format, _P, _P, _P, _P, _I64,
                              _P, _SZ, _P]),
    "esb_conv2d_nhwc": (_I32, [_P, _P, _I64, esb_format, _P, _I64, esb_format, _P, _P, _P, _P, _I64, _P]),
    "esb_conv2d_kernel": (_I32, [_P, _I64, esb_format, esb_format, _I32, _P]),
    "esb_gemm_i64": (_I32, [_I64, _I64, _I64, _P, _I64, esb_format, _P, _I64, esb_format, _P, _P, _P, _P, _I64,
                            _P]),
    "esb_conv2d_nhwc_i64": (_I32, [_P, _P, _I64, esb_format, _P, _I64, esb_format, _P, _P, _P, _P, _I64, _P]),
    "esb_maxpool_nhwc": (_I32, [_P, _I64, esb_format] + [_I32] * 7 + [_P, _I64, _P]),
    "esb_avgpool_nhwc": (_I32, [_P, _I64, esb_format, _I32, _I32, _I32, _F32, _F32, esb_format, _I32, _P, _P, _I64,
                                _P]),
    "esb_get_status": (_I32, [_P, _P]),
    "esb_peak_launch": (_I32, [_I32, _I64, _P, _P]),
}


def lib():
    """Load libesb.so (built by __graft_entry__.build()).  Raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libesb.so not built ({LIB_PATH}); run __graft_entry__.build()")
        l = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(l, name)
            fn.restype = res
            fn.argtypes = args
        _lib = l
    return _lib


def _check(st: int, where: str):
    if st != ESB_OK:
        raise EsbError(st, where)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t: torch.Tensor, name: str):
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


# ------------------------------------------------------------------ info

def esb_version() -> int:
    return int(lib().esb_version())


def esb_codes_per_word(b: int) -> int:
    return int(lib().esb_codes_per_word(b))


def esb_row_words(cols: int, b: int) -> int:
    return int(lib().esb_row_words(cols, b))


def esb_zero_code(f: Fmt) -> int:
    return int(lib().esb_zero_code(f.c()))


def esb_alpha_star(b: int, k: int) -> tuple[float, float]:
    a = ctypes.c_double(0.0)
    d = ctypes.c_double(0.0)
    _check(lib().esb_alpha_star(b, k, ctypes.byref(a), ctypes.byref(d)), "esb_alpha_star")
    return a.value, d.value


# ------------------------------------------------------------- calibrate

def esb_calibrate_dda(x: torch.Tensor, f: Fmt, alpha_out: Optional[torch.Tensor] = None,
                      stats_out: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                      stream=None) -> tuple[torch.Tensor, Optional[torch.Tensor]]:
    """Device alpha (1 float) and stats {mean, spread, n} of x (Sec. III-D)."""
    _dev(x, "x")
    assert x.dtype == torch.float32
    n = x.numel()
    if alpha_out is None:
        alpha_out = torch.empty(1, dtype=torch.float32, device=x.device)
    if workspace is None:
        nb = int(lib().esb_calibrate_dda_workspace_bytes(n))
        workspace = torch.zeros(max(nb, 16), dtype=torch.uint8, device=x.device)
    _check(lib().esb_calibrate_dda(_ptr(x), n, f.c(), _ptr(workspace), workspace.numel(), _ptr(alpha_out),
                                   _ptr(stats_out), _stream(stream)), "esb_calibrate_dda")
    return alpha_out, stats_out


def esb_calibrate_dda_noalloc(x: torch.Tensor, f: Fmt, alpha_out: Optional[torch.Tensor] = None,
                              stats_out: Optional[torch.Tensor] = None,
                              stream=None) -> tuple[torch.Tensor, Optional[torch.Tensor]]:
    """esb_calibrate_dda for callers that cannot allocate device memory: the
    scratch is a fixed array inside libesb.so, so no workspace is passed (the
    caller still supplies x, alpha_out and stats_out).  Calls that overlap on
    the GPU share that array and must be serialised."""
    _dev(x, "x")
    assert x.dtype == torch.float32
    if alpha_out is None:
        alpha_out = torch.empty(1, dtype=torch.float32, device=x.device)
    _check(lib().esb_calibrate_dda_noalloc(_ptr(x), x.numel(), f.c(), _ptr(alpha_out), _ptr(stats_out),
                                           _stream(stream)), "esb_calibrate_dda_noalloc")
    return alpha_out, stats_out


ESB_DIST_GAUSSIAN = 0
ESB_DIST_LAPLACE = 1


def esb_alpha_star_dist(b: int, k: int, dist: int) -> tuple[float, float]:
    a = ctypes.c_double(0.0)
    d = ctypes.c_double(0.0)
    _check(lib().esb_alpha_star_dist(b, k, dist, ctypes.byref(a), ctypes.byref(d)), "esb_alpha_star_dist")
    return a.value, d.value


def esb_calibrate_dda_dist(x: torch.Tensor, f: Fmt, dist: int, alpha_out: Optional[torch.Tensor] = None,
                           stats_out: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                           stream=None) -> tuple[torch.Tensor, Optional[torch.Tensor]]:
    """esb_calibrate_dda with the alpha* of another data density (ESB_DIST_*)."""
    _dev(x, "x")
    assert x.dtype == torch.float32
    n = x.numel()
    if alpha_out is None:
        alpha_out = torch.empty(1, dtype=torch.float32, device=x.device)
    if workspace is None:
        workspace = torch.zeros(max(int(lib().esb_calibrate_dda_workspace_bytes(n)), 16), dtype=torch.uint8,
                                device=x.device)
    _check(lib().esb_calibrate_dda_dist(_ptr(x), n, f.c(), dist, _ptr(workspace), workspace.numel(),
                                        _ptr(alpha_out), _ptr(stats_out), _stream(stream)), "esb_calibrate_dda_dist")
    return alpha_out, stats_out


def esb_dda_histogram(x: torch.Tensor, f: Fmt, stats: torch.Tensor, nbins: int = 8192, t_max: float = 16.0,
                      counts: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Histogram (int64 CUDA tensor of nbins counts) of the normalised |t| of x."""
    _dev(x, "x"); _dev(stats, "stats")
    if counts is None:
        counts = torch.empty(nbins, dtype=torch.int64, device=x.device)
    _check(lib().esb_dda_histogram(_ptr(x), x.numel(), f.c(), _ptr(stats), nbins, t_max, _ptr(counts),
                                   _stream(stream)), "esb_dda_histogram")
    return counts


def esb_alpha_star_hist(counts, t_max: float, b: int, k: int) -> tuple[float, float]:
    """alpha* and 2 D(alpha*) of a histogram of |t| (host counts, any int array)."""
    import numpy as np
    c = np.ascontiguousarray(np.asarray(counts, dtype=np.uint64))
    a = ctypes.c_double(0.0)
    d = ctypes.c_double(0.0)
    _check(lib().esb_alpha_star_hist(c.ctypes.data, c.size, t_max, b, k, ctypes.byref(a), ctypes.byref(d)),
           "esb_alpha_star_hist")
    return a.value, d.value


def esb_calibrate_dda_empirical(x: torch.Tensor, f: Fmt, nbins: int = 8192, t_max: float = 16.0,
                                alpha_out: Optional[torch.Tensor] = None, stats_out: Optional[torch.Tensor] = None,
                                workspace: Optional[torch.Tensor] = None, counts: Optional[torch.Tensor] = None,
                                stream=None) -> tuple[torch.Tensor, torch.Tensor, float]:
    """DDA calibration with the data's own density -> (alpha (1,), stats (3,), alpha*).  Synchronises."""
    _dev(x, "x")
    n = x.numel()
    dev = x.device
    if alpha_out is None:
        alpha_out = torch.empty(1, dtype=torch.float32, device=dev)
    if stats_out is None:
        stats_out = torch.empty(3, dtype=torch.float64, device=dev)
    if workspace is None:
        workspace = torch.zeros(max(int(lib().esb_calibrate_dda_workspace_bytes(n)), 16), dtype=torch.uint8,
                                device=dev)
    if counts is None:
        counts = torch.empty(nbins, dtype=torch.int64, device=dev)
    a = ctypes.c_double(0.0)
    _check(lib().esb_calibrate_dda_empirical(_ptr(x), n, f.c(), _ptr(workspace), workspace.numel(), nbins, t_max,
                                             _ptr(counts), _ptr(alpha_out), _ptr(stats_out), ctypes.byref(a),
                                             _stream(stream)), "esb_calibrate_dda_empirical")
    return alpha_out, stats_out, a.value


def esb_calibrate_dda_workspace_bytes(n: int) -> int:
    return int(lib().esb_calibrate_dda_workspace_bytes(n))


# --------------------------------------------------------------- project

def esb_project(x: torch.Tensor, f: Fmt, alpha=None, rounding: int = ESB_ROUND_HALF_AWAY,
                codes: Optional[torch.Tensor] = None, ldc: Optional[int] = None, stream=None) -> torch.Tensor:
    """Project a (rows, cols) or 1-D fp32 tensor to packed codes (rows, ldc) int32.
    alpha: python float or a 1-element CUDA float tensor (read on the device)."""
    _dev(x, "x")
    assert x.dtype == torch.float32
    x2 = x.reshape(1, -1) if x.dim() == 1 else x.reshape(-1, x.shape[-1])
    rows, cols = x2.shape
    if ldc is None:
        ldc = esb_row_words(cols, f.b)
    if codes is None:
        codes = torch.empty((rows, ldc), dtype=torch.int32, device=x.device)
    a_host, a_dev = (float(alpha), None) if not isinstance(alpha, torch.Tensor) else (0.0, alpha)
    _check(lib().esb_project(_ptr(x2), rows, cols, cols, a_host, _ptr(a_dev), f.c(), rounding, _ptr(codes), ldc,
                             _stream(stream)), "esb_project")
    return codes


def esb_project_dda(x: torch.Tensor, f: Fmt, rounding: int = ESB_ROUND_HALF_AWAY,
                    alpha_out: Optional[torch.Tensor] = None, stats_out: Optional[torch.Tensor] = None,
                    workspace: Optional[torch.Tensor] = None, codes: Optional[torch.Tensor] = None,
                    ldc: Optional[int] = None, stream=None) -> tuple[torch.Tensor, torch.Tensor]:
    """DDA calibration and projection of x in one launch -> (codes (rows, ldc) int32, alpha (1,) float)."""
    _dev(x, "x")
    assert x.dtype == torch.float32
    x2 = x.reshape(1, -1) if x.dim() == 1 else x.reshape(-1, x.shape[-1])
    rows, cols = x2.shape
    if ldc is None:
        ldc = esb_row_words(cols, f.b)
    if codes is None:
        codes = torch.empty((rows, ldc), dtype=torch.int32, device=x.device)
    if alpha_out is None:
        alpha_out = torch.empty(1, dtype=torch.float32, device=x.device)
    if workspace is None:
        nb = int(lib().esb_calibrate_dda_workspace_bytes(rows * cols))
        workspace = torch.zeros(max(nb, 16), dtype=torch.uint8, device=x.device)
    _check(lib().esb_project_dda(_ptr(x2), rows, cols, f.c(), rounding, _ptr(workspace), workspace.numel(),
                                 _ptr(alpha_out), _ptr(stats_out), _ptr(codes), ldc, _stream(stream)),
           "esb_project_dda")
    return codes, alpha_out


def esb_dn_project(x: torch.Tensor, stats: torch.Tensor, f: Fmt, rounding: int = ESB_ROUND_HALF_AWAY,
                   want_xq: bool = True, stream=None) -> tuple[torch.Tensor, Optional[torch.Tensor]]:
    """DN then ESB projection with alpha* -> (codes (rows, ldc) int32, fake-quantised values | None)."""
    _dev(x, "x"); _dev(stats, "stats")
    x2 = x.reshape(1, -1) if x.dim() == 1 else x.reshape(-1, x.shape[-1])
    rows, cols = x2.shape
    ldc = esb_row_words(cols, f.b)
    codes = torch.empty((rows, ldc), dtype=torch.int32, device=x.device)
    xq = torch.empty_like(x2) if want_xq else None
    _check(lib().esb_dn_project(_ptr(x2), rows, cols, _ptr(stats), f.c(), rounding, _ptr(codes), ldc, _ptr(xq),
                                _stream(stream)), "esb_dn_project")
    return codes, xq


def esb_dn_backward(grad: torch.Tensor, x: torch.Tensor, stats: torch.Tensor,
                    workspace: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Straight-through + DN backward -> dL/dx (fp32, shape of x)."""
    _dev(grad, "grad"); _dev(x, "x"); _dev(stats, "stats")
    n = x.numel()
    if workspace is None:
        workspace = torch.empty(max(int(lib().esb_dn_backward_workspace_bytes(n)), 16), dtype=torch.uint8,
                                device=x.device)
    gx = torch.empty_like(x)
    _check(lib().esb_dn_backward(_ptr(grad), _ptr(x), n, _ptr(stats), _ptr(workspace), workspace.numel(), _ptr(gx),
                                 _stream(stream)), "esb_dn_backward")
    return gx


def esb_ema_update(batch_stats: torch.Tensor, running_stats: torch.Tensor, gamma: float, stream=None) -> None:
    _dev(batch_stats, "batch_stats"); _dev(running_stats, "running_stats")
    _check(lib().esb_ema_update(_ptr(batch_stats), _ptr(running_stats), gamma, _stream(stream)), "esb_ema_update")


def esb_dequant(codes: torch.Tensor, cols: int, f: Fmt, alpha, stream=None) -> torch.Tensor:
    _dev(codes, "codes")
    c2 = codes.reshape(-1, codes.shape[-1])
    rows, ldc = c2.shape
    y = torch.empty((rows, cols), dtype=torch.float32, device=codes.device)
    a_host, a_dev = (float(alpha), None) if not isinstance(alpha, torch.Tensor) else (0.0, alpha)
    _check(lib().esb_dequant(_ptr(c2), rows, cols, ldc, a_host, _ptr(a_dev), f.c(), _ptr(y), cols, _stream(stream)),
           "esb_dequant")
    return y


# ------------------------------------------------------------------ gemm

@dataclass
class Epilogue:
    """Fused post-processing (include/esb.h, esb_epilogue)."""
    scale: Optional[torch.Tensor] = None
    bias: Optional[torch.Tensor] = None
    alpha_a_dev: Optional[torch.Tensor] = None
    alpha_b_dev: Optional[torch.Tensor] = None
    scale0: float = 1.0
    bias0: float = 0.0
    act: int = ESB_ACT_NONE
    residual: Optional[torch.Tensor] = None
    res_fmt: Optional[Fmt] = None
    res_scale: float = 0.0
    alpha_out: float = 1.0
    alpha_out_dev: Optional[torch.Tensor] = None
    fmt_out: Fmt = Fmt(4, 2, True)
    rounding_out: int = ESB_ROUND_HALF_AWAY

    def c(self) -> esb_epilogue:
        e = esb_epilogue()
        e.scale = None if self.scale is None else self.scale.data_ptr()
        e.bias = None if self.bias is None else self.bias.data_ptr()
        e.alpha_a_dev = None if self.alpha_a_dev is None else self.alpha_a_dev.data_ptr()
        e.alpha_b_dev = None if self.alpha_b_dev is None else self.alpha_b_dev.data_ptr()
        e.scale0 = self.scale0
        e.bias0 = self.bias0
        e.act = self.act
        if self.residual is not None:
            e.residual = self.residual.data_ptr()
            e.res_ld = self.residual.shape[-1]
            e.res_fmt = self.res_fmt.c()
        e.res_scale = self.res_scale
        e.alpha_out = self.alpha_out
        e.alpha_out_dev = None if self.alpha_out_dev is None else self.alpha_out_dev.data_ptr()
        e.fmt_out = self.fmt_out.c()
        e.rounding_out = self.rounding_out
        return e


def esb_gemm_tiled_workspace_bytes(M: int, N: int, K: int) -> int:
    return int(lib().esb_gemm_tiled_workspace_bytes(M, N, K))


def esb_gemm(A: torch.Tensor, fa: Fmt, B: torch.Tensor, fb: Fmt, K: int, ep: Optional[Epilogue] = None,
             want_acc: bool = True, want_y: bool = False, want_codes: bool = False,
             out_acc: Optional[torch.Tensor] = None, out_y: Optional[torch.Tensor] = None,
             out_codes: Optional[torch.Tensor] = None, stream=None, workspace: Optional[torch.Tensor] = None):
    """(acc int32 (M,N) | None, y fp32 (M,N) | None, codes int32 (M, ldo) | None).
    With a workspace (a CUDA uint8 tensor of at least
    esb_gemm_tiled_workspace_bytes(M, N, K) bytes) the call is esb_gemm_tiled."""
    _dev(A, "A"); _dev(B, "B")
    M, lda = A.shape
    N, ldb = B.shape
    dev = A.device
    acc = out_acc if out_acc is not None else (torch.empty((M, N), dtype=torch.int32, device=dev) if want_acc else None)
    y = out_y if out_y is not None else (torch.empty((M, N), dtype=torch.float32, device=dev) if want_y else None)
    codes = out_codes
    if codes is None and want_codes:
        codes = torch.empty((M, esb_row_words(N, ep.fmt_out.b)), dtype=torch.int32, device=dev)
    ldo = codes.shape[-1] if codes is not None else 0
    epc = ep.c() if ep is not None else None
    if workspace is not None:
        _dev(workspace, "workspace")
        _check(lib().esb_gemm_tiled(M, N, K, _ptr(A), lda, fa.c(), _ptr(B), ldb, fb.c(),
                                    ctypes.byref(epc) if epc is not None else None,
                                    _ptr(acc), _ptr(y), _ptr(codes), ldo, _ptr(workspace),
                                    workspace.numel() * workspace.element_size(), _stream(stream)), "esb_gemm_tiled")
        return acc, y, codes
    _check(lib().esb_gemm(M, N, K, _ptr(A), lda, fa.c(), _ptr(B), ldb, fb.c(),
                          ctypes.byref(epc) if epc is not None else None,
                          _ptr(acc), _ptr(y), _ptr(codes), ldo, _stream(stream)), "esb_gemm")
    return acc, y, codes


def esb_gemm_i64(A: torch.Tensor, fa: Fmt, B: torch.Tensor, fb: Fmt, K: int, ep: Optional[Epilogue] = None,
                 want_acc: bool = True, want_y: bool = False, want_codes: bool = False, stream=None):
    """CUDA-core contraction with int64 accumulators -> (acc int64 (M,N) | None,
    y fp32 (M,N) | None, codes int32 (M, ldo) | None)."""
    _dev(A, "A"); _dev(B, "B")
    M, lda = A.shape
    N, ldb = B.shape
    dev = A.device
    acc = torch.empty((M, N), dtype=torch.int64, device=dev) if want_acc else None
    y = torch.empty((M, N), dtype=torch.float32, device=dev) if want_y else None
    codes = torch.empty((M, esb_row_words(N, ep.fmt_out.b)), dtype=torch.int32, device=dev) if want_codes else None
    ldo = codes.shape[-1] if codes is not None else 0
    epc = ep.c() if ep is not None else None
    _check(lib().esb_gemm_i64(M, N, K, _ptr(A), lda, fa.c(), _ptr(B), ldb, fb.c(),
                              ctypes.byref(epc) if epc is not None else None, _ptr(acc), _ptr(y), _ptr(codes), ldo,
                              _stream(stream)), "esb_gemm_i64")
    return acc, y, codes


def esb_conv2d_nhwc_i64(X: torch.Tensor, fx: Fmt, W: torch.Tensor, fw: Fmt, n: int, h: int, w: int, c: int,
                        cout: int, r: int, s: int, stride: int, pad: int, ep: Optional[Epilogue] = None,
                        want_acc: bool = True, want_y: bool = False, want_codes: bool = False, stream=None):
    """esb_conv2d_nhwc on the int64 CUDA-core path; outputs (n*P*Q, cout)-shaped."""
    _dev(X, "X"); _dev(W, "W")
    P, Q = conv_out_hw(h, w, r, s, stride, pad)
    M = n * P * Q
    dev = X.device
    acc = torch.empty((M, cout), dtype=torch.int64, device=dev) if want_acc else None
    y = torch.empty((M, cout), dtype=torch.float32, device=dev) if want_y else None
    codes = torch.empty((M, esb_row_words(cout, ep.fmt_out.b)), dtype=torch.int32, device=dev) if want_codes else None
    ldo = codes.shape[-1] if codes is not None else 0
    d = esb_conv_desc(n, h, w, c, cout, r, s, stride, pad, 1)
    epc = ep.c() if ep is not None else None
    _check(lib().esb_conv2d_nhwc_i64(ctypes.byref(d), _ptr(X), X.shape[-1], fx.c(), _ptr(W), W.shape[-1], fw.c(),
                                     ctypes.byref(epc) if epc is not None else None, _ptr(acc), _ptr(y), _ptr(codes),
                                     ldo, _stream(stream)), "esb_conv2d_nhwc_i64")
    return acc, y, codes


def conv_out_hw(h: int, w: int, r: int, s: int, stride: int, pad: int) -> tuple[int, int]:
    return (h + 2 * pad - r) // stride + 1, (w + 2 * pad - s) // stride + 1


def esb_conv2d_nhwc(X: torch.Tensor, fx: Fmt, W: torch.Tensor, fw: Fmt, n: int, h: int, w: int, c: int, cout: int,
                    r: int, s: int, stride: int, pad: int, groups: int = 1, ep: Optional[Epilogue] = None,
                    want_acc: bool = True, want_y: bool = False, want_codes: bool = False,
                    out_acc: Optional[torch.Tensor] = None, out_y: Optional[torch.Tensor] = None,
                    out_codes: Optional[torch.Tensor] = None, stream=None):
    """NHWC conv on packed codes.  X: (n*h*w, ldx) int32; W: (cout*r*s, ldx) int32
    (depthwise: (r*s, ldx)).  Outputs are (n*P*Q, cout)-shaped."""
    _dev(X, "X"); _dev(W, "W")
    ldx = X.shape[-1]
    ldw = W.shape[-1]
    P, Q = conv_out_hw(h, w, r, s, stride, pad)
    M = n * P * Q
    dev = X.device
    acc = out_acc if out_acc is not None else (torch.empty((M, cout), dtype=torch.int32, device=dev) if want_acc else None)
    y = out_y if out_y is not None else (torch.empty((M, cout), dtype=torch.float32, device=dev) if want_y else None)
    codes = out_codes
    if codes is None and want_codes:
        codes = torch.empty((M, esb_row_words(cout, ep.fmt_out.b)), dtype=torch.int32, device=dev)
    ldo = codes.shape[-1] if codes is not None else 0
    d = esb_conv_desc(n, h, w, c, cout, r, s, stride, pad, groups)
    epc = ep.c() if ep is not None else None
    _check(lib().esb_conv2d_nhwc(ctypes.byref(d), _ptr(X), ldx, fx.c(), _ptr(W), ldw, fw.c(),
                                 ctypes.byref(epc) if epc is not None else None,
                                 _ptr(acc), _ptr(y), _ptr(codes), ldo, _stream(stream)), "esb_conv2d_nhwc")
    return acc, y, codes


ESB_CONV_KERNEL_HALO, ESB_CONV_KERNEL_IM2COL, ESB_CONV_KERNEL_STREAMED, ESB_CONV_KERNEL_DEPTHWISE = 1, 2, 3, 4


def esb_conv2d_kernel(n: int, h: int, w: int, c: int, cout: int, r: int, s: int, stride: int, pad: int,
                      fx: Fmt, fw: Fmt, out_b: int = 4, groups: int = 1, ldx: Optional[int] = None) -> int:
    """Which kernel esb_conv2d_nhwc runs for this convolution (ESB_CONV_KERNEL_*)."""
    d = esb_conv_desc(n, h, w, c, cout, r, s, stride, pad, groups)
    out = ctypes.c_int32(0)
    _check(lib().esb_conv2d_kernel(ctypes.byref(d), esb_row_words(c, fx.b) if ldx is None else ldx, fx.c(), fw.c(),
                                   out_b, ctypes.byref(out)), "esb_conv2d_kernel")
    return int(out.value)


def esb_maxpool_nhwc(X: torch.Tensor, f: Fmt, n: int, h: int, w: int, c: int, win: int = 3, stride: int = 2,
                     pad: int = 1, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Max pooling of NHWC codes; returns (n*P*Q, ldx) int32 codes."""
    _dev(X, "X")
    ldx = X.shape[-1]
    P, Q = conv_out_hw(h, w, win, win, stride, pad)
    Y = out if out is not None else torch.empty((n * P * Q, ldx), dtype=torch.int32, device=X.device)
    _check(lib().esb_maxpool_nhwc(_ptr(X), ldx, f.c(), n, h, w, c, win, stride, pad, _ptr(Y), Y.shape[-1],
                                  _stream(stream)), "esb_maxpool_nhwc")
    return Y


def esb_avgpool_nhwc(X: torch.Tensor, f: Fmt, n: int, hw: int, c: int, scale: float, alpha_out: float, fmt_out: Fmt,
                     rounding: int = ESB_ROUND_HALF_AWAY, want_y: bool = False, stream=None):
    """Global average pooling of NHWC codes -> (y (n, c) fp32 | None, codes (n, ldo) int32)."""
    _dev(X, "X")
    ldx = X.shape[-1]
    y = torch.empty((n, c), dtype=torch.float32, device=X.device) if want_y else None
    ldo = esb_row_words(c, fmt_out.b)
    codes = torch.empty((n, ldo), dtype=torch.int32, device=X.device)
    _check(lib().esb_avgpool_nhwc(_ptr(X), ldx, f.c(), n, hw, c, scale, alpha_out, fmt_out.c(), rounding, _ptr(y),
                                  _ptr(codes), ldo, _stream(stream)), "esb_avgpool_nhwc")
    return y, codes


ESB_PEAK_TCGEN05_F8F6F4 = 0
ESB_PEAK_MMA_SYNC_S8 = 1


def esb_peak_launch(kind: int, iters: int, stream=None) -> int:
    """Launch a tensor-pipe peak microbenchmark; returns its operation count."""
    ops = ctypes.c_int64(0)
    _check(lib().esb_peak_launch(kind, iters, ctypes.byref(ops), _stream(stream)), "esb_peak_launch")
    return int(ops.value)


def esb_get_status(stream=None) -> int:
    v = ctypes.c_int32(0)
    _check(lib().esb_get_status(_stream(stream), ctypes.byref(v)), "esb_get_status")
    return int(v.value)


# ------------------------------------------------------------ host helpers

def esb_dda_combine(stats, f: Fmt) -> tuple[float, float, float, float]:
    """(alpha, mean, spread, n) of a tensor from its parts' statistics
    (an iterable of {mean, spread, n} triples, e.g. esb_calibrate_dda's
    stats_out of each part)."""
    import numpy as np
    st = np.ascontiguousarray(np.asarray([[float(v) for v in t] for t in stats], dtype=np.float64).reshape(-1, 3))
    out = np.zeros(3, dtype=np.float64)
    a = ctypes.c_float(0.0)
    _check(lib().esb_dda_combine(st.ctypes.data, st.shape[0], f.c(), out.ctypes.data, ctypes.byref(a)),
           "esb_dda_combine")
    return float(a.value), float(out[0]), float(out[1]), float(out[2])


def esb_dequant_scale(alpha_a: float, fa: Fmt, alpha_b: float, fb: Fmt) -> float:
    """fp32 factor turning the integer accumulator into the product of the values."""
    s = ctypes.c_float(0.0)
    _check(lib().esb_dequant_scale(alpha_a, fa.c(), alpha_b, fb.c(), ctypes.byref(s)), "esb_dequant_scale")
    return float(s.value)


def esb_fold_bn_dn(alpha_a: float, fa: Fmt, alpha_w: float, fw: Fmt, bn_mean, bn_std, bn_gamma, bn_beta,
                   dn_mean: float, dn_std: float):
    """Sec. IV-C "BN and DN" fold -> (scale, bias) float64 numpy arrays of the epilogue."""
    import numpy as np
    arrs = [np.ascontiguousarray(np.asarray(v, dtype=np.float64).ravel()) for v in (bn_mean, bn_std, bn_gamma, bn_beta)]
    n = arrs[0].size
    if any(a.size != n for a in arrs):
        raise ValueError("bn_mean, bn_std, bn_gamma and bn_beta must have the same length")
    scale = np.zeros(n, dtype=np.float64)
    bias = np.zeros(n, dtype=np.float64)
    _check(lib().esb_fold_bn_dn(alpha_a, fa.c(), alpha_w, fw.c(), *[a.ctypes.data for a in arrs], n, dn_mean, dn_std,
                                scale.ctypes.data, bias.ctypes.data), "esb_fold_bn_dn")
    return scale, bias
