"""CPU oracle for ESB quantization (arXiv 2109.03513) -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this package.  It is a thin ctypes/numpy marshalling layer over
``esb_oracle.c`` (plain C, fp64, written from the paper section by section);
it shares no code with the CUDA library and never imports it.

Parity status of each function (what pins it, see ``tests/test_oracle_pins.py``):

* set enumeration, C, encode/decode -- pinned (set sizes, the five-bit
  two-significant-bit example set of Sec. I, the 1-sign/2-exponent/1-fraction
  set of Fig. 10, linear/PoT/ternary special cases of Sec. III-B, the
  multiplication identity Eq. esb_multiplication over all code pairs).
* projection -- pinned (worked example of Sec. III-C, equality of the two
  formulations Eq. thresholing_func / Eq. fast_projection on a strided sweep
  of the fp32 patterns of small formats' ranges plus every midpoint and its
  neighbours, idempotence, symmetry, monotonicity, brute-force nearest
  search with numpy, and the step-function form the GPU's projection of all
  2^32 patterns is compared with).
* alpha*, D -- pinned (all 18 alpha* and DDA values of Table 1; the 3-level
  Lloyd-Max quantizer of N(0,1); the scale identity alpha*(b,b-1) = 2 alpha*(b,b-2)).
* calibration -- pinned (closed-form moments of constructed inputs).
* GEMM / conv / depthwise / pooling -- pinned (numpy integer matmul and
  scipy-free direct sums on tiny inputs, symmetry/linearity properties).
* epilogue -- pinned (fmaf op order checked against numpy float32 and the
  BN/DN fold identity of Sec. IV-C in fp64).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "esb_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

_CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def build(force: bool = False) -> str:
    """Compile esb_oracle.c into liboracle.so (gcc), if missing or stale."""
    with _lock:
        stale = (not os.path.exists(_LIB_PATH)
                 or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
        if force or stale:
            tmp = _LIB_PATH + f".tmp{os.getpid()}"
            subprocess.check_call(["gcc", *_CFLAGS, "-o", tmp, _SRC, "-lm"])
            os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    i32, i64, f32, f64 = ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_double
    p = ctypes.c_void_p
    sig = {
        "oracle_N": (i32, [i32, i32]),
        "oracle_set_nonneg": (i32, [i32, i32, p]),
        "oracle_set_full": (i32, [i32, i32, p]),
        "oracle_C": (f64, [i32, i32]),
        "oracle_project_value": (f64, [f32, f32, i32, i32, i32, i32]),
        "oracle_project_value_shift": (f64, [f32, f32, i32, i32, i32, i32]),
        "oracle_project_values_shift": (None, [p, i64, f32, i32, i32, i32, i32, p]),
        "oracle_project_values": (None, [p, i64, f32, i32, i32, i32, i32, p]),
        "oracle_encode": (ctypes.c_uint32, [f64, i32, i32, i32]),
        "oracle_decode": (f64, [ctypes.c_uint32, i32, i32]),
        "oracle_zero_code": (ctypes.c_uint32, [i32, i32]),
        "oracle_project_codes": (None, [p, i64, f32, i32, i32, i32, i32, p]),
        "oracle_pack": (None, [p, i64, i64, i32, i32, i64, p]),
        "oracle_unpack": (None, [p, i64, i64, i32, i64, p]),
        "oracle_D": (f64, [f64, i32, i32]),
        "oracle_alpha_star": (f64, [i32, i32, p]),
        "oracle_dD": (f64, [f64, i32, i32]),
        "oracle_calibrate_with": (f32, [p, i64, f64, i32, p]),
        "oracle_D_laplace": (f64, [f64, i32, i32]),
        "oracle_dn_project": (None, [p, i64, f64, f64, f32, i32, i32, i32, i32, p, p]),
        "oracle_dn_backward": (None, [p, p, i64, f64, f64, p]),
        "oracle_ema": (None, [p, p, f64]),
        "oracle_alpha_star_laplace": (f64, [i32, i32, p]),
        "oracle_histogram_abs": (None, [p, i64, i32, f64, f64, i32, f32, p]),
        "oracle_D_hist": (f64, [f64, p, i32, f64, i32, i32]),
        "oracle_alpha_star_hist": (f64, [p, i32, f64, i32, i32, p]),
        "oracle_gemm_i64": (None, [p, i64, i32, i32, p, i64, i32, i32, i64, i64, i64, p]),
        "oracle_gemm_entry": (i64, [p, i64, i32, i32, p, i64, i32, i32, i64, i64, i64]),
        "oracle_epilogue_one": (f32, [i64, f32, f32, i32, i64, f32, i32, f32, i32, i32, i32, i32, p]),
        "oracle_epilogue_array": (None, [p, i64, i64, p, p, p, f32, i32, f32, i32, i32, i32, i32, p, p]),
        "oracle_conv2d_i64": (None, [p, i64, i32, i32, p, i64, i32, i32] + [i32] * 11 + [p]),
        "oracle_conv2d_rows_i64": (None, [p, i64, i32, i32, p, i64, i32, i32] + [i32] * 13 + [p]),
        "oracle_dwconv_i64": (None, [p, i64, i32, i32, p, i64, i32, i32] + [i32] * 10 + [p]),
        "oracle_maxpool_codes": (None, [p, i64, i32, i32] + [i32] * 9 + [i64, p]),
        "oracle_avgpool_sum_i64": (None, [p, i64, i32, i32, i32, i32, i32, p]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data)


# ---------------------------------------------------------------- format ---

def N_of(b: int, k: int) -> int:
    return _load().oracle_N(b, k)


def codes_per_word(b: int) -> int:
    return 32 // b


def words_for(cols: int, b: int) -> int:
    return -(-cols // (32 // b))


def set_nonneg(b: int, k: int) -> np.ndarray:
    out = np.zeros(1 << (b - 1), dtype=np.float64)
    n = _load().oracle_set_nonneg(b, k, _ptr(out))
    return out[:n]


def set_full(b: int, k: int) -> np.ndarray:
    out = np.zeros((1 << b), dtype=np.float64)
    n = _load().oracle_set_full(b, k, _ptr(out))
    return out[:n]


def C_of(b: int, k: int) -> float:
    return _load().oracle_C(b, k)


def encode(q: float, b: int, k: int, signed: bool = True) -> int:
    return int(_load().oracle_encode(float(q), b, k, int(signed)))


def decode(code: int, b: int, k: int) -> float:
    return _load().oracle_decode(int(code), b, k)


def zero_code(b: int, k: int) -> int:
    return int(_load().oracle_zero_code(b, k))


def image(code: int, b: int, k: int) -> int:
    """Integer image I = q * 2^k of a code."""
    return int(round(decode(code, b, k) * (1 << k)))


# ------------------------------------------------------------ projection ---

def project_value(x: float, alpha: float, b: int, k: int, signed: bool = True,
                  rounding: int = 0) -> float:
    return _load().oracle_project_value(x, alpha, b, k, int(signed), rounding)


def project_value_shift(x: float, alpha: float, b: int, k: int, signed: bool = True,
                        rounding: int = 0) -> float:
    return _load().oracle_project_value_shift(x, alpha, b, k, int(signed), rounding)


def project_values(x: np.ndarray, alpha: float, b: int, k: int, signed: bool = True,
                   rounding: int = 0) -> np.ndarray:
    """Projected values (units of alpha) by the look-up form, Eq. thresholing_func."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.zeros(x.shape, dtype=np.float64)
    _load().oracle_project_values(_ptr(x), x.size, float(alpha), b, k, int(signed), rounding, _ptr(out))
    return out


def project_values_shift(x: np.ndarray, alpha: float, b: int, k: int, signed: bool = True,
                         rounding: int = 0) -> np.ndarray:
    """Projected values (units of alpha) by the shift-and-round form, Eq. fast_projection."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.zeros(x.shape, dtype=np.float64)
    _load().oracle_project_values_shift(_ptr(x), x.size, float(alpha), b, k, int(signed), rounding,
                                        _ptr(out))
    return out


def project_codes(x: np.ndarray, alpha: float, b: int, k: int, signed: bool = True,
                  rounding: int = 0) -> np.ndarray:
    """Unpacked codes (uint32, same shape as x) of Eq. cheap_projection."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.zeros(x.shape, dtype=np.uint32)
    _load().oracle_project_codes(_ptr(x), x.size, float(alpha), b, k, int(signed), rounding, _ptr(out))
    return out


def pack(codes: np.ndarray, b: int, k: int, ld_words: int | None = None) -> np.ndarray:
    """Pack a (rows, cols) array of codes into (rows, ld_words) uint32 words."""
    codes = np.ascontiguousarray(codes, dtype=np.uint32)
    if codes.ndim == 1:
        codes = codes.reshape(1, -1)
    rows, cols = codes.shape
    ld = words_for(cols, b) if ld_words is None else ld_words
    out = np.zeros((rows, ld), dtype=np.uint32)
    _load().oracle_pack(_ptr(codes), rows, cols, b, k, ld, _ptr(out))
    return out


def unpack(words: np.ndarray, cols: int, b: int) -> np.ndarray:
    words = np.ascontiguousarray(words, dtype=np.uint32)
    if words.ndim == 1:
        words = words.reshape(1, -1)
    rows, ld = words.shape
    out = np.zeros((rows, cols), dtype=np.uint32)
    _load().oracle_unpack(_ptr(words), rows, cols, b, ld, _ptr(out))
    return out


def project_packed(x2d: np.ndarray, alpha: float, b: int, k: int, signed: bool = True,
                   rounding: int = 0, ld_words: int | None = None) -> np.ndarray:
    x2d = np.ascontiguousarray(x2d, dtype=np.float32)
    if x2d.ndim == 1:
        x2d = x2d.reshape(1, -1)
    return pack(project_codes(x2d, alpha, b, k, signed, rounding), b, k, ld_words)


# ------------------------------------------------------------------- DDA ---

def D(alpha: float, b: int, k: int) -> float:
    return _load().oracle_D(alpha, b, k)


def dD(alpha: float, b: int, k: int) -> float:
    return _load().oracle_dD(alpha, b, k)


def alpha_star(b: int, k: int) -> tuple[float, float]:
    """(alpha*, D_half(alpha*)) for N(0,1) data.  Table 1's DDA is 2 * D_half."""
    d = np.zeros(1, dtype=np.float64)
    a = _load().oracle_alpha_star(b, k, _ptr(d))
    return a, float(d[0])


_ASTAR_CACHE: dict[tuple[int, int], float] = {}


def alpha_star_cached(b: int, k: int) -> float:
    key = (b, k)
    if key not in _ASTAR_CACHE:
        _ASTAR_CACHE[key] = alpha_star(b, k)[0]
    return _ASTAR_CACHE[key]


def calibrate(x: np.ndarray, b: int, k: int, signed: bool = True) -> tuple[float, np.ndarray]:
    """(alpha, stats[mu, sigma|rms, d]) of Sec. III-D for data x."""
    x = np.ascontiguousarray(x, dtype=np.float32).ravel()
    st = np.zeros(3, dtype=np.float64)
    a = _load().oracle_calibrate_with(_ptr(x), x.size, alpha_star_cached(b, k), int(signed), _ptr(st))
    return float(np.float32(a)), st


def D_laplace(alpha: float, b: int, k: int) -> float:
    """D(alpha) of Eq. objective_function_expansion for Laplace data with unit variance."""
    return _load().oracle_D_laplace(alpha, b, k)


def alpha_star_laplace(b: int, k: int) -> tuple[float, float]:
    """(alpha*, 2 D(alpha*)) for Laplace data with unit variance."""
    d = ctypes.c_double(0.0)
    a = _load().oracle_alpha_star_laplace(b, k, ctypes.byref(d))
    return a, 2.0 * d.value


def histogram_abs(x: np.ndarray, signed: bool, mean: float, spread: float, nbins: int, t_max: float) -> np.ndarray:
    """Counts (uint64, nbins) of the normalised magnitudes of x."""
    x = np.ascontiguousarray(x, dtype=np.float32).ravel()
    out = np.zeros(nbins, dtype=np.uint64)
    _load().oracle_histogram_abs(_ptr(x), x.size, int(signed), float(mean), float(spread), nbins, float(t_max),
                                 _ptr(out))
    return out


def D_hist(alpha: float, counts: np.ndarray, t_max: float, b: int, k: int) -> float:
    c = np.ascontiguousarray(counts, dtype=np.uint64)
    return _load().oracle_D_hist(alpha, _ptr(c), c.size, float(t_max), b, k)


def alpha_star_hist(counts: np.ndarray, t_max: float, b: int, k: int) -> tuple[float, float]:
    """(alpha*, 2 D(alpha*)) of the empirical density of a histogram of |t|."""
    c = np.ascontiguousarray(counts, dtype=np.uint64)
    d = ctypes.c_double(0.0)
    a = _load().oracle_alpha_star_hist(_ptr(c), c.size, float(t_max), b, k, ctypes.byref(d))
    return a, 2.0 * d.value


def dn_project(x: np.ndarray, mu: float, sigma: float, alpha: float, b: int, k: int, signed: bool = True,
               rounding: int = 0) -> tuple[np.ndarray, np.ndarray]:
    """(unpacked codes, fake-quantised values) of DN then projection (Algorithm 1 forward)."""
    x = np.ascontiguousarray(x, dtype=np.float32).ravel()
    codes = np.zeros(x.size, dtype=np.uint32)
    xq = np.zeros(x.size, dtype=np.float32)
    _load().oracle_dn_project(_ptr(x), x.size, float(mu), float(sigma), float(alpha), b, k, int(signed), rounding,
                              _ptr(codes), _ptr(xq))
    return codes, xq


def dn_backward(g: np.ndarray, x: np.ndarray, mu: float, sigma: float) -> np.ndarray:
    g = np.ascontiguousarray(g, dtype=np.float32).ravel()
    x = np.ascontiguousarray(x, dtype=np.float32).ravel()
    out = np.zeros(x.size, dtype=np.float32)
    _load().oracle_dn_backward(_ptr(g), _ptr(x), x.size, float(mu), float(sigma), _ptr(out))
    return out


def ema(batch, running, gamma: float) -> np.ndarray:
    b = np.ascontiguousarray(np.asarray(batch, dtype=np.float64)[:2])
    r = np.ascontiguousarray(np.asarray(running, dtype=np.float64)[:2]).copy()
    _load().oracle_ema(_ptr(b), _ptr(r), float(gamma))
    return r


# --------------------------------------------------------- contraction ---

def gemm_i64(A: np.ndarray, fa: tuple, B: np.ndarray, fb: tuple, M: int, N: int, K: int) -> np.ndarray:
    """int64 accumulators of the ESB GEMM (A: M x lda words, B: N x ldb words)."""
    A = np.ascontiguousarray(A, dtype=np.uint32)
    B = np.ascontiguousarray(B, dtype=np.uint32)
    out = np.zeros((M, N), dtype=np.int64)
    _load().oracle_gemm_i64(_ptr(A), A.shape[1], fa[0], fa[1], _ptr(B), B.shape[1], fb[0], fb[1],
                            M, N, K, _ptr(out))
    return out


def gemm_entry(A: np.ndarray, fa: tuple, B: np.ndarray, fb: tuple, K: int, m: int, n: int) -> int:
    return int(_load().oracle_gemm_entry(_ptr(A), A.shape[1], fa[0], fa[1], _ptr(B), B.shape[1],
                                         fb[0], fb[1], K, m, n))


def epilogue(acc: np.ndarray, scale: np.ndarray, bias: np.ndarray, act: int, alpha_out: float,
             fo: tuple, rounding: int = 0, res_images: np.ndarray | None = None,
             res_scale: float = 0.0) -> tuple[np.ndarray, np.ndarray]:
    """Per-element post-processing of an (M, N) accumulator; scale/bias are
    per column n.  Returns (y fp32 (M,N), unpacked output codes (M,N))."""
    acc = np.ascontiguousarray(acc, dtype=np.int64)
    M, N = acc.shape
    scale = np.ascontiguousarray(scale, dtype=np.float32)
    bias = np.ascontiguousarray(bias, dtype=np.float32)
    y = np.zeros((M, N), dtype=np.float32)
    codes = np.zeros((M, N), dtype=np.uint32)
    res = None if res_images is None else np.ascontiguousarray(res_images, dtype=np.int64)
    _load().oracle_epilogue_array(_ptr(acc), M, N, _ptr(scale), _ptr(bias),
                                  None if res is None else _ptr(res), float(res_scale), act, float(alpha_out),
                                  fo[0], fo[1], int(fo[2]), rounding, _ptr(y), _ptr(codes))
    return y, codes


def conv2d_i64(X, fx, W, fw, Nb, H, Wd, C, Cout, R, S, stride, pad):
    P = (H + 2 * pad - R) // stride + 1
    Q = (Wd + 2 * pad - S) // stride + 1
    X = np.ascontiguousarray(X, dtype=np.uint32)
    W = np.ascontiguousarray(W, dtype=np.uint32)
    acc = np.zeros((Nb, P, Q, Cout), dtype=np.int64)
    _load().oracle_conv2d_i64(_ptr(X), X.shape[-1], fx[0], fx[1], _ptr(W), W.shape[-1], fw[0], fw[1],
                              Nb, H, Wd, C, Cout, R, S, stride, pad, P, Q, _ptr(acc))
    return acc


def conv2d_rows_i64(X, fx, W, fw, Nb, H, Wd, C, Cout, R, S, stride, pad, p0, p1):
    """conv2d_i64 restricted to output rows [p0, p1)."""
    P = (H + 2 * pad - R) // stride + 1
    Q = (Wd + 2 * pad - S) // stride + 1
    X = np.ascontiguousarray(X, dtype=np.uint32)
    W = np.ascontiguousarray(W, dtype=np.uint32)
    acc = np.zeros((Nb, p1 - p0, Q, Cout), dtype=np.int64)
    _load().oracle_conv2d_rows_i64(_ptr(X), X.shape[-1], fx[0], fx[1], _ptr(W), W.shape[-1], fw[0], fw[1],
                                   Nb, H, Wd, C, Cout, R, S, stride, pad, P, Q, p0, p1, _ptr(acc))
    return acc


def dwconv_i64(X, fx, W, fw, Nb, H, Wd, C, R, S, stride, pad):
    P = (H + 2 * pad - R) // stride + 1
    Q = (Wd + 2 * pad - S) // stride + 1
    X = np.ascontiguousarray(X, dtype=np.uint32)
    W = np.ascontiguousarray(W, dtype=np.uint32)
    acc = np.zeros((Nb, P, Q, C), dtype=np.int64)
    _load().oracle_dwconv_i64(_ptr(X), X.shape[-1], fx[0], fx[1], _ptr(W), W.shape[-1], fw[0], fw[1],
                              Nb, H, Wd, C, R, S, stride, pad, P, Q, _ptr(acc))
    return acc


def maxpool_codes(X, b, k, Nb, H, Wd, C, win, stride, pad, ld_out=None):
    P = (H + 2 * pad - win) // stride + 1
    Q = (Wd + 2 * pad - win) // stride + 1
    X = np.ascontiguousarray(X, dtype=np.uint32)
    ld = X.shape[-1] if ld_out is None else ld_out
    Y = np.zeros((Nb, P, Q, ld), dtype=np.uint32)
    _load().oracle_maxpool_codes(_ptr(X), X.shape[-1], b, k, Nb, H, Wd, C, win, stride, pad, P, Q,
                                 ld, _ptr(Y))
    return Y


def avgpool_sum_i64(X, b, k, Nb, HW, C):
    X = np.ascontiguousarray(X, dtype=np.uint32)
    out = np.zeros((Nb, C), dtype=np.int64)
    _load().oracle_avgpool_sum_i64(_ptr(X), X.shape[-1], b, k, Nb, HW, C, _ptr(out))
    return out
