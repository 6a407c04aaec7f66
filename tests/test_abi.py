"""C-ABI library: loads, exports every declared symbol, host-only entry
points and host-side validation (no device work; runs without a GPU)."""
import ctypes
import os
import re
from fractions import Fraction

import numpy as np
import pytest

import oracle as o
from conftest import ROOT, read_golden
from paper_2109_03513_gb300 import esb

HEADER = os.path.join(ROOT, "include", "esb.h")


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__.build()
    return esb.lib()


def declared_functions():
    txt = open(HEADER).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"^\s*[A-Za-z_][A-Za-z0-9_ ]*?[\s\*]+(esb_[a-z0-9_]+)\s*\(", txt, flags=re.M)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n
        assert n in esb.SIGNATURES, n
    assert set(esb.SIGNATURES) == set(names)


def test_info_functions(lib):
    assert esb.esb_version() >= 100
    for b in range(2, 9):
        assert esb.esb_codes_per_word(b) == 32 // b
        for k in range(0, b):
            assert esb.esb_zero_code(esb.Fmt(b, k)) == o.zero_code(b, k)
        for cols in (0, 1, 37, 64, 576):
            rw = esb.esb_row_words(cols, b)
            assert rw % 4 == 0 and rw * (32 // b) >= cols and (rw - 4) * (32 // b) < max(cols, 1)
    assert esb.esb_codes_per_word(9) == 0
    assert lib.esb_status_string(3) == b"exactness bound exceeded"


@pytest.mark.parametrize("row", read_golden("table1_alpha_dda.txt"))
def test_library_alpha_star_matches_table1(lib, row):
    b, k, dda, astar = int(row[0]), int(row[1]), float(row[2]), float(row[3])
    a, d = esb.esb_alpha_star(b, k)
    assert abs(a - astar) <= 5e-5 + 1e-12
    assert abs(d - dda) <= 5e-5 + 1e-12
    ao, _ = o.alpha_star(b, k)
    assert abs(a - ao) <= 1e-9 * ao


def test_library_alpha_star_other_formats(lib):
    for b in range(2, 8):
        for k in range(0, b):
            a, _ = esb.esb_alpha_star(b, k)
            ao, _ = o.alpha_star(b, k)
            assert abs(a - ao) <= 1e-9 * ao, (b, k, a, ao)


def test_host_validation_without_device(lib):
    f = esb.esb_format(4, 2, 1)
    bad = esb.esb_format(9, 2, 1)
    null = None
    fake = ctypes.c_void_p(4096)
    # unsupported / invalid formats and sizes are rejected before any launch
    assert lib.esb_project(fake, 1, 8, 8, 1.0, null, bad, 0, fake, 4, null) == esb.ESB_ERR_UNSUPPORTED
    assert lib.esb_project(fake, 1, 8, 8, 0.0, null, f, 0, fake, 4, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project(fake, 1, 8, 8, float("nan"), null, f, 0, fake, 4, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project(fake, 1, 8, 8, 1.0, null, f, 7, fake, 4, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project(fake, 1, 64, 64, 1.0, null, f, 0, fake, 7, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project(fake, 0, 8, 8, 1.0, null, f, 0, fake, 4, null) == esb.ESB_OK
    assert lib.esb_calibrate_dda(fake, 0, f, fake, 64, fake, null, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_calibrate_dda(fake, 100, f, ctypes.c_void_p(4097), 1 << 20, fake, null, null) == esb.ESB_ERR_ALIGN
    assert lib.esb_calibrate_dda(fake, 100, f, fake, 1, fake, null, null) == esb.ESB_ERR_INVALID_ARG
    # contraction: exactness bound and unsupported formats
    big = esb.esb_format(6, 3, 1)
    ep = esb.Epilogue().c()
    assert lib.esb_gemm(128, 64, 8192, fake, 2048, big, fake, 2048, big, ctypes.byref(ep), fake, null, null, 0,
                        null) == esb.ESB_ERR_RANGE
    f71 = esb.esb_format(7, 1, 1)     # 5-bit exponent field: no E4M3 image, no significand split
    assert lib.esb_gemm(128, 64, 64, fake, 16, f71, fake, 16, f71, ctypes.byref(ep), fake, null, null, 0,
                        null) == esb.ESB_ERR_UNSUPPORTED
    assert lib.esb_gemm(128, 64, 64, fake, 4, f, fake, 8, f, ctypes.byref(ep), fake, null, null, 0,
                        null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_gemm(128, 64, 64, ctypes.c_void_p(4100), 8, f, fake, 8, f, ctypes.byref(ep), fake, null, null, 0,
                        null) == esb.ESB_ERR_ALIGN
    assert lib.esb_gemm(0, 64, 64, fake, 8, f, fake, 8, f, ctypes.byref(ep), fake, null, null, 0,
                        null) == esb.ESB_OK
    d = esb.esb_conv_desc(1, 8, 8, 64, 64, 3, 3, 1, 1, 1)
    assert lib.esb_conv2d_nhwc(ctypes.byref(d), fake, 8, f, fake, 7, f, ctypes.byref(ep), fake, null, null, 0,
                               null) == esb.ESB_ERR_INVALID_ARG
    # filter rows of another width: stride for their own codes, 16-byte multiple
    f63 = esb.esb_format(6, 3, 1)
    assert lib.esb_conv2d_nhwc(ctypes.byref(d), fake, 8, f, fake, 12, f63, ctypes.byref(ep), fake, null, null, 0,
                               null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_conv2d_nhwc(ctypes.byref(d), fake, 8, f, fake, 14, f63, ctypes.byref(ep), fake, null, null, 0,
                               null) == esb.ESB_ERR_ALIGN
    d2 = esb.esb_conv_desc(1, 8, 8, 64, 64, 3, 3, 1, 3, 1)
    assert lib.esb_conv2d_nhwc(ctypes.byref(d2), fake, 8, f, fake, 8, f, ctypes.byref(ep), fake, null, null, 0,
                               null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_get_status(null, null) == esb.ESB_ERR_INVALID_ARG


def test_host_validation_other_entry_points(lib):
    # every check below returns before any launch or device query
    f = esb.esb_format(4, 2, 1)
    f63 = esb.esb_format(6, 3, 1)
    null = None
    fake = ctypes.c_void_p(4096)
    ep = ctypes.byref(esb.Epilogue().c())
    R = esb.ESB_ERR_RANGE
    # tiled GEMM: K max|I_A| max|I_B| < 2^31 for the chunked path ((6,3): 60 x 60)
    K = 600000                         # 600000 * 3600 >= 2^31
    ld = esb.esb_row_words(K, 6)
    assert lib.esb_gemm_tiled(256, 256, K, fake, ld, f63, fake, ld, f63, ep, fake, null, null, 0, fake, 1 << 40,
                              null) == R
    # below it the chunked path runs (K past 2^24 / 3600): it needs a workspace
    K = 8192
    ld = esb.esb_row_words(K, 6)
    ws = lib.esb_gemm_tiled_workspace_bytes(256, 256, K)
    assert ws > 0
    assert lib.esb_gemm_tiled(256, 256, K, fake, ld, f63, fake, ld, f63, ep, fake, null, null, 0, null, 0,
                              null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_gemm_tiled(256, 256, K, fake, ld, f63, fake, ld, f63, ep, fake, null, null, 0, fake, ws - 1,
                              null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_gemm_tiled(256, 256, K, fake, ld, f63, fake, ld, f63, ep, fake, null, null, 0,
                              ctypes.c_void_p(4104), ws, null) == esb.ESB_ERR_ALIGN
    # ... which esb_gemm (one fp32 accumulation, bound 2^24) refuses
    assert lib.esb_gemm(256, 256, K, fake, ld, f63, fake, ld, f63, ep, fake, null, null, 0, null) == R
    assert lib.esb_gemm_tiled_workspace_bytes(0, 256, K) == 0
    # fused calibration + projection
    wsb = lib.esb_calibrate_dda_workspace_bytes(64)
    assert lib.esb_project_dda(fake, 1, 64, f, 2, fake, wsb, fake, null, fake, 8, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project_dda(fake, 1, 64, f, 0, fake, wsb - 1, fake, null, fake, 8, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project_dda(fake, 1, 64, f, 0, ctypes.c_void_p(4100), wsb, fake, null, fake, 8,
                               null) == esb.ESB_ERR_ALIGN
    assert lib.esb_project_dda(fake, 1, 64, f, 0, fake, wsb, fake, null, fake, 7, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project_dda(fake, 0, 64, f, 0, fake, wsb, fake, null, fake, 8, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_project_dda(fake, 1, 64, esb.esb_format(4, 4, 1), 0, fake, wsb, fake, null, fake, 8,
                               null) == esb.ESB_ERR_UNSUPPORTED
    # dequantisation
    assert lib.esb_dequant(fake, 2, 64, 8, 1.0, null, f, fake, 63, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_dequant(fake, 2, 64, 7, 1.0, null, f, fake, 64, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_dequant(fake, 2, 64, 8, -1.0, null, f, fake, 64, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_dequant(fake, 0, 64, 8, 1.0, null, f, fake, 64, null) == esb.ESB_OK
    # depthwise convolution (groups = C): Cout = C, output width = input width, bound 2^31
    dw = esb.esb_conv_desc(1, 8, 8, 64, 32, 3, 3, 1, 1, 64)
    assert lib.esb_conv2d_nhwc(ctypes.byref(dw), fake, 8, f, fake, 8, f, ep, fake, null, null, 0,
                               null) == esb.ESB_ERR_INVALID_ARG
    f81 = esb.esb_format(8, 1, 1)      # max|I| = 3 * 2^62: any window exceeds 2^31
    dw = esb.esb_conv_desc(1, 8, 8, 64, 64, 3, 3, 1, 1, 64)
    assert lib.esb_conv2d_nhwc(ctypes.byref(dw), fake, 16, f81, fake, 16, f81, ep, fake, null, null, 0, null) == R
    # grouped convolution other than depthwise
    g2 = esb.esb_conv_desc(1, 8, 8, 64, 64, 3, 3, 1, 1, 2)
    assert lib.esb_conv2d_nhwc(ctypes.byref(g2), fake, 8, f, fake, 8, f, ep, fake, null, null, 0,
                               null) == esb.ESB_ERR_UNSUPPORTED
    # pooling
    assert lib.esb_maxpool_nhwc(fake, 8, f, 1, 8, 8, 64, 3, 2, 3, fake, 8, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_maxpool_nhwc(fake, 8, f, 1, 8, 8, 64, 3, 2, 1, fake, 7, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_maxpool_nhwc(fake, 8, f, 0, 8, 8, 64, 3, 2, 1, fake, 8, null) == esb.ESB_OK
    f52 = esb.esb_format(5, 2, 0)
    assert lib.esb_avgpool_nhwc(fake, 8, f, 1, 49, 64, 1.0, 0.5, f52, 0, null, fake, 8,
                                null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_avgpool_nhwc(fake, 8, f, 1, 49, 64, 1.0, 0.0, f, 0, null, fake, 8, null) == esb.ESB_ERR_INVALID_ARG
    assert lib.esb_avgpool_nhwc(fake, 16, f81, 1, 49, 64, 1.0, 0.5, f81, 0, null, fake, 16, null) == R


def test_bn_dn_fold_identity():
    # Sec. IV-C: DN(BN(Scale(x))) / alpha_{l+1} = a x + b with the printed a, b.
    rng = np.random.default_rng(4)
    aw, ka, aa, kw = np.float32(0.37), 2, np.float32(1.3), 1   # fp32 scales, as the library takes them
    aw, aa = float(aw), float(aa)
    mu_bn, sd_bn, g, beta = rng.normal(size=5), rng.uniform(0.5, 2, 5), rng.normal(size=5), rng.normal(size=5)
    mu_dn, sd_dn, a_next = 0.3, 1.7, 0.61
    scale, bias = esb.esb_fold_bn_dn(aa, esb.Fmt(8, ka), aw, esb.Fmt(8, kw), mu_bn, sd_bn, g, beta, mu_dn, sd_dn)
    acc = rng.integers(-500, 500, size=5).astype(np.float64)
    x = acc * (aw * 2.0 ** -kw) * (aa * 2.0 ** -ka)          # Scale: dequantised product
    bn = g * (x - mu_bn) / sd_bn + beta                      # BN
    dn = (bn - mu_dn) / sd_dn                                # DN
    lhs = dn / a_next
    # the paper's a and b (over the raw product x' = acc * alpha_W * alpha_A)
    a_p = (aw * aa * g) / (a_next * sd_dn * sd_bn)
    b_p = (sd_bn * beta - mu_bn * g - sd_bn * mu_dn) / (a_next * sd_dn * sd_bn)
    xr = acc * 2.0 ** -(kw + ka)
    assert np.allclose(lhs, a_p * xr + b_p, rtol=1e-12, atol=1e-12)
    assert np.allclose(lhs, (scale * acc + bias) / a_next, rtol=1e-12, atol=1e-12)


def test_dequant_scale_is_the_scale_stage():
    # Sec. IV-C "Scale": acc * alpha_a 2^-ka * alpha_b 2^-kb is the product of
    # the two values; the fp32 factor has one rounding (of alpha_a * alpha_b)
    rng = np.random.default_rng(9)
    for _ in range(200):
        aa, ab = (float(np.float32(v)) for v in rng.uniform(1e-3, 3.0, 2))
        ka, kb = (int(v) for v in rng.integers(0, 7, 2))
        s = esb.esb_dequant_scale(aa, esb.Fmt(8, ka), ab, esb.Fmt(8, kb))
        exact = Fraction(aa) * Fraction(ab) / 2 ** (ka + kb)
        assert abs(Fraction(s) - exact) <= exact * Fraction(1, 2 ** 24)      # within half an fp32 ulp
        assert s == float(np.float32(aa * ab)) / 2 ** (ka + kb)
    f = esb.Fmt(4, 2)
    with pytest.raises(esb.EsbError):
        esb.esb_dequant_scale(0.0, f, 1.0, f)
    with pytest.raises(esb.EsbError):
        esb.esb_dequant_scale(1.0, esb.Fmt(4, 4), 1.0, f)


def test_dda_combine_law_of_total_variance():
    # Sec. III-D statistics of a whole tensor from its parts: against numpy
    # fp64 two-pass moments of the concatenation, then alpha = fl32(alpha* (s + 1e-7))
    rng = np.random.default_rng(10)
    parts = [rng.normal(3.0, 0.5, 7001), rng.normal(2.5, 2.0, 1), np.abs(rng.normal(size=30000)), np.zeros(0)]
    for signed in (True, False):
        f = esb.Fmt(5, 2, signed)
        st = []
        for p in parts:
            if p.size == 0:
                st.append((0.0, 0.0, 0.0))
                continue
            m = p.mean()
            sp = np.sqrt(((p - m) ** 2).mean()) if signed else np.sqrt((p * p).mean())
            st.append((m, sp, p.size))
        a, mean, spread, n = esb.esb_dda_combine(st, f)
        x = np.concatenate(parts)
        ref_sp = np.sqrt(((x - x.mean()) ** 2).mean()) if signed else np.sqrt((x * x).mean())
        assert n == x.size
        assert abs(mean - x.mean()) <= 1e-12 * abs(x.mean())
        assert abs(spread - ref_sp) <= 1e-12 * ref_sp
        astar = esb.esb_alpha_star(5, 2)[0]
        assert a == float(np.float32(astar * (spread + 1e-7)))
    with pytest.raises(esb.EsbError):
        esb.esb_dda_combine([(0.0, 0.0, 0.0)], esb.Fmt(4, 2))
    with pytest.raises(esb.EsbError):
        esb.esb_dda_combine([(0.0, -1.0, 5.0)], esb.Fmt(4, 2))


def test_binding_refuses_host_tensors_and_missing_library(monkeypatch):
    # no CPU fallback: every compute entry point of the binding takes device
    # tensors only, and a missing libesb.so is an error, not a slower path
    import torch
    x = torch.zeros(64, dtype=torch.float32)
    codes = torch.zeros((1, 8), dtype=torch.int32)
    f = esb.Fmt(4, 2, True)
    with pytest.raises(ValueError):
        esb.esb_project(x, f, alpha=1.0)
    with pytest.raises(ValueError):
        esb.esb_calibrate_dda(x, f)
    with pytest.raises(ValueError):
        esb.esb_project_dda(x, f)
    with pytest.raises(ValueError):
        esb.esb_gemm(codes, f, codes, f, 64)
    with pytest.raises(ValueError):
        esb.esb_conv2d_nhwc(codes, f, codes, f, 1, 1, 1, 64, 64, 1, 1, 1, 0)
    monkeypatch.setattr(esb, "_lib", None)
    monkeypatch.setattr(esb, "LIB_PATH", os.path.join(ROOT, "no_such_dir", "libesb.so"))
    with pytest.raises(RuntimeError):
        esb.lib()
