// esb_cc.cu -- ESB kernels that run on CUDA cores (HBM-bound, no dense
// contraction to put on tensor cores):
//   * depthwise convolution (one r x s filter per channel, MobileNetV2's 3x3
//     layers) with the same fused epilogue as the tensor-core contraction,
//   * max pooling of codes with the intersection window of Sec. IV-B
//     (projection is monotone, so pooling codes = pooling quantised values),
//   * global average pooling: exact integer sum of the images per channel,
//     then one fp32 scale and ESB requantisation.
#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

// Integer image of a code (exact; max |I| < 2^31 for every accepted format).
__device__ __forceinline__ int32_t code_image_i(uint32_t c, int b, int k, int ew, int N)
{
    const uint32_t s = (c >> (b - 1)) & 1u;
    const uint32_t e = ew > 0 ? (c >> k) & ((1u << ew) - 1u) : 0u;
    const uint32_t f = c & ((1u << k) - 1u);
    const int32_t mag = ((int)e == N) ? (int32_t)f : (int32_t)(((1u << k) + f) << e);
    return s ? -mag : mag;
}

struct CcEpi {
    const float* scale;
    const float* bias;
    const float* alpha_a_dev;
    const float* alpha_b_dev;
    float dq_pow2;
    float scale0, bias0;
    int act;
    const uint32_t* residual;
    int64_t res_ld;
    int res_b, res_k;
    float res_scale;
    float alpha_out;
    const float* alpha_out_dev;
    ProjParams out;
    int32_t* acc_out;
    float* y_out;
    uint32_t* codes_out;
    int64_t ldo;
    int acc24;             // every accumulator below 2^24 in magnitude (exact as fp32)
};

__device__ __forceinline__ float cc_act(float y, int act)
{
    if (act == ESB_ACT_RELU) {
        y = (y > 0.0f) ? y : 0.0f;
    } else if (act == ESB_ACT_RELU6) {
        y = (y > 0.0f) ? y : 0.0f;
        y = (y < 6.0f) ? y : 6.0f;
    }
    return y;
}

// ------------------------------------------------------------ depthwise

// One thread = one output code word (cpw channels) of one output pixel.
// The r*s input words of its window and the r*s filter words are read
// through the read-only cache (neighbouring threads share the inputs), each
// code decoded to its integer image, multiplied and accumulated exactly in
// int32, then the epilogue writes the output word.
__global__ void __launch_bounds__(256)
esb_dwconv_kernel(const uint32_t* __restrict__ X, int64_t ldx, int bx, int kx,
                  const uint32_t* __restrict__ W, int64_t ldw, int bw, int kw,
                  int n, int H, int Wd, int C, int R, int S, int stride, int pad, int P, int Q, CcEpi ep)
{
    const int cpw = 32 / bx;
    const int words = (C + cpw - 1) / cpw;          // code words holding channels
    const int64_t total = (int64_t)n * P * Q * ep.ldo;
    const int ewx = bx - kx - 1, Nx = (1 << ewx) - 1;
    const int eww = bw - kw - 1, Nw = (1 << eww) - 1;
    const uint32_t mx = (1u << bx) - 1u, mw = (1u << bw) - 1u;
    const float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
    const bool dq = ep.alpha_a_dev && ep.alpha_b_dev;
    const float dqs = dq ? __fmul_rn(__ldg(ep.alpha_a_dev), __ldg(ep.alpha_b_dev)) * ep.dq_pow2 : 1.0f;
    const int rcpw = ep.residual ? 32 / ep.res_b : 1;
    const uint32_t rmask = ep.residual ? (1u << ep.res_b) - 1u : 0u;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t pix = t / ep.ldo;
        const int w = (int)(t - pix * ep.ldo);
        const int q = (int)(pix % Q);
        const int64_t np_ = pix / Q;
        const int p = (int)(np_ % P);
        const int64_t nn = np_ / P;
        if (w >= words) {                              // padding words: zero codes
            if (ep.codes_out) {
                uint32_t word = 0;
                for (int j = 0; j < cpw; j++) word |= ep.out.zero_code << (bx * j);
                ep.codes_out[pix * ep.ldo + w] = word;
            }
            continue;
        }
        int32_t acc[16];
#pragma unroll
        for (int j = 0; j < 16; j++) acc[j] = 0;
        for (int r = 0; r < R; r++) {
            const int h = p * stride - pad + r;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < S; s++) {
                const int ww = q * stride - pad + s;
                if (ww < 0 || ww >= Wd) continue;
                const uint32_t xw = __ldg(X + ((nn * H + h) * Wd + ww) * ldx + w);
                const uint32_t fw = __ldg(W + (int64_t)(r * S + s) * ldw + w);
#pragma unroll
                for (int j = 0; j < 16; j++) {
                    if (j < cpw) {
                        const int32_t ix = code_image_i((xw >> (bx * j)) & mx, bx, kx, ewx, Nx);
                        const int32_t iw = code_image_i((fw >> (bw * j)) & mw, bw, kw, eww, Nw);
                        acc[j] += ix * iw;
                    }
                }
            }
        }
        uint32_t word = 0;
#pragma unroll
        for (int j = 0; j < 16; j++) {
            if (j >= cpw) break;
            const int c = w * cpw + j;
            uint32_t code = ep.out.zero_code;
            if (c < C) {
                const int64_t o = pix * C + c;
                if (ep.acc_out) ep.acc_out[o] = acc[j];
                float sc = ep.scale ? __ldg(ep.scale + c) : ep.scale0;
                if (dq) sc = __fmul_rn(sc, dqs);
                const float bi = ep.bias ? __ldg(ep.bias + c) : ep.bias0;
                float y = __fmaf_rn(sc, (float)acc[j], bi);
                if (ep.residual) {
                    const uint32_t rc = (__ldg(ep.residual + pix * ep.res_ld + c / rcpw) >> (ep.res_b * (c % rcpw))) & rmask;
                    y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
                }
                y = cc_act(y, ep.act);
                if (ep.y_out) ep.y_out[o] = y;
                if (ep.codes_out) code = project_code(y, alpha_out, ep.out);
            }
            word |= code << (bx * j);
        }
        if (ep.codes_out) ep.codes_out[pix * ep.ldo + w] = word;
    }
}

// Depthwise 3x3 for code widths 3..6 with filters and inputs of one width
// (every MobileNetV2 layer).  Each block decodes the filters of all
// channels once into shared memory (integer images, [tap][channel]) and
// builds the table of input images and the requantisation thresholds, then
// walks work items: one item = one code word (CPW channels) of QT
// consecutive output pixels of one output row (QT = 4 at stride 1, 2 at
// stride 2).  For each filter row, the item's NIN input words are loaded
// together (independent loads in flight), each is decoded once and added
// into every output of the strip that uses it, with the row's three taps
// in registers.  Index arithmetic is 32-bit (the host checks the sizes).
// The lean epilogue (4-bit codes only, a positive scalar scale, monotone
// requantisation) compares the integer accumulator with the 7 thresholds
// moved onto it and packs a word in one step; everything else takes the
// per-element path.
template <int B, int STRIDE>
__global__ void __launch_bounds__(128)
esb_dwconv3_kernel(const uint32_t* __restrict__ X, int ldx, int kx, const uint32_t* __restrict__ W, int ldw, int kw,
                   int H, int Wd, int C, int pad, int P, int Q, int QS, int rows, CcEpi ep)
{
    constexpr int CPW = 32 / B;
    constexpr int QT = STRIDE == 1 ? 4 : 2;
    constexpr int NIN = (QT - 1) * STRIDE + 3;        // input columns of a strip
    constexpr uint32_t MASK = (1u << B) - 1u;
    extern __shared__ int32_t wtab[];                 // [9][words * CPW] filter images
    __shared__ int32_t lutx[1 << B];
    __shared__ float T[128];
    __shared__ float Rs[8];
    const int words = (C + CPW - 1) / CPW;
    const int cp = words * CPW;
    const int ewx = B - kx - 1, Nx = (1 << ewx) - 1;
    const int eww = B - kw - 1, Nw = (1 << eww) - 1;
    griddep_wait();                                   // inputs and alphas may come from the previous launch
    for (int i = threadIdx.x; i < (1 << B); i += blockDim.x) lutx[i] = code_image_i((uint32_t)i, B, kx, ewx, Nx);
    for (int i = threadIdx.x; i < 9 * words; i += blockDim.x) {
        const int t = i / words, w = i - (i / words) * words;
        const uint32_t fw = __ldg(W + t * ldw + w);
#pragma unroll
        for (int j = 0; j < CPW; j++) wtab[t * cp + w * CPW + j] = code_image_i((fw >> (B * j)) & MASK, B, kw, eww, Nw);
    }
    const float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
    if (ep.codes_out) build_thresholds(T, ep.out, alpha_out, threadIdx.x >> 5, threadIdx.x & 31, 0, blockDim.x >> 5);
    const bool dq = ep.alpha_a_dev && ep.alpha_b_dev;
    const float dqs = dq ? __fmul_rn(__ldg(ep.alpha_a_dev), __ldg(ep.alpha_b_dev)) * ep.dq_pow2 : 1.0f;
    const float sc_fixed = ep.scale ? 0.0f : (dq ? __fmul_rn(ep.scale0, dqs) : ep.scale0);
    const bool b4 = ep.out.b == 4 && ep.codes_out;
    const bool lean = b4 && ep.acc24 && !ep.scale && !ep.bias && !ep.residual && !ep.acc_out && !ep.y_out &&
                      sc_fixed > 0.0f && (!ep.out.is_signed || ep.act != ESB_ACT_NONE);
    __syncthreads();
    if (lean && threadIdx.x < 7) Rs[threadIdx.x] = acc_raw_threshold(sc_fixed, ep.bias0, T[threadIdx.x], ep.act, 1.0f);
    __syncthreads();
    Thr7 t7, r7;
#pragma unroll
    for (int i = 0; i < 7; i++) {
        t7.t[i] = b4 ? T[i] : 0.0f;
        r7.t[i] = lean ? Rs[i] : 0.0f;
    }
    const int rcpw = ep.residual ? 32 / ep.res_b : 1;
    const uint32_t rmask = ep.residual ? (1u << ep.res_b) - 1u : 0u;
    uint32_t zx = 0u, zo = 0u;                        // zero-code words of the input and output formats
#pragma unroll
    for (int j = 0; j < CPW; j++) zx |= (uint32_t)fmt_zero_code(B, kx) << (B * j);
    for (int j = 0; j < CPW; j++) zo |= ep.out.zero_code << (ep.out.b * j);
    const int ldo = (int)ep.ldo;
    const int upr = QS * ldo;
    const int total = rows * upr;
    for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < total; it += gridDim.x * blockDim.x) {
        const int row = it / upr;                     // n * P + p
        const int u = it - row * upr;
        const int qs = u / ldo;
        const int w = u - qs * ldo;
        const int nn = row / P;
        const int p = row - nn * P;
        const int q0 = qs * QT;
        const int64_t obase = ((int64_t)row * Q + q0) * ldo + w;    // output word of pixel q0
        if (w >= words) {                             // padding words of the output rows: zero codes
            if (ep.codes_out) {
#pragma unroll
                for (int uu = 0; uu < QT; uu++)
                    if (q0 + uu < Q) ep.codes_out[obase + (int64_t)uu * ldo] = zo;
            }
            continue;
        }
        int32_t acc[QT][CPW];
#pragma unroll
        for (int uu = 0; uu < QT; uu++)
#pragma unroll
            for (int j = 0; j < CPW; j++) acc[uu][j] = 0;
        const int c0 = q0 * STRIDE - pad;             // first input column of the strip
#pragma unroll 1
        for (int r = 0; r < 3; r++) {
            const int h = p * STRIDE - pad + r;
            if ((unsigned)h >= (unsigned)H) continue;
            const uint32_t* xrow = X + (int64_t)(nn * H + h) * Wd * ldx + w;
            uint32_t xw[NIN];
#pragma unroll
            for (int c = 0; c < NIN; c++) {
                const int col = c0 + c;
                xw[c] = ((unsigned)col < (unsigned)Wd) ? __ldg(xrow + (int64_t)col * ldx) : zx;
            }
            int32_t wf[3][CPW];
#pragma unroll
            for (int s2 = 0; s2 < 3; s2++)
#pragma unroll
                for (int j = 0; j < CPW; j++) wf[s2][j] = wtab[(r * 3 + s2) * cp + w * CPW + j];
#pragma unroll
            for (int c = 0; c < NIN; c++) {
                int32_t img[CPW];
#pragma unroll
                for (int j = 0; j < CPW; j++) img[j] = lutx[(xw[c] >> (B * j)) & MASK];
#pragma unroll
                for (int uu = 0; uu < QT; uu++) {
                    const int s2 = c - uu * STRIDE;
                    if (s2 >= 0 && s2 < 3) {
#pragma unroll
                        for (int j = 0; j < CPW; j++) acc[uu][j] += img[j] * wf[s2][j];
                    }
                }
            }
        }
        const int cvalid = C - w * CPW;               // channels of this word inside C
        // per-channel scale and bias of the word's channels, once per item
        float scv[CPW], biv[CPW];
        if (!lean) {
#pragma unroll
            for (int j = 0; j < CPW; j++) {
                const int c = w * CPW + j < C ? w * CPW + j : C - 1;
                float sc = ep.scale ? __ldg(ep.scale + c) : ep.scale0;
                if (dq) sc = __fmul_rn(sc, dqs);
                scv[j] = sc;
                biv[j] = ep.bias ? __ldg(ep.bias + c) : ep.bias0;
            }
        }
#pragma unroll
        for (int uu = 0; uu < QT; uu++) {
            if (q0 + uu >= Q) break;
            const int64_t ow = obase + (int64_t)uu * ldo;
            if (lean) {
                uint32_t J = 0u;
#pragma unroll
                for (int j = 0; j < CPW; j++) {
                    const float v = (float)acc[uu][j];
                    const bool b2 = v >= r7.t[3];
                    const bool b1 = v >= (b2 ? r7.t[5] : r7.t[1]);
                    const bool b0 = v >= (b2 ? (b1 ? r7.t[6] : r7.t[4]) : (b1 ? r7.t[2] : r7.t[0]));
                    const uint32_t jb = (b2 ? 4u : 0u) | (b1 ? 2u : 0u) | (b0 ? 1u : 0u);
                    J |= (j < cvalid ? jb : 0u) << (4 * j);
                }
                ep.codes_out[ow] = codes8_b4(J, 0u, ep.out.k);
                continue;
            }
            const int64_t pix = (int64_t)row * Q + q0 + uu;
            uint32_t word = 0;
#pragma unroll
            for (int j = 0; j < CPW; j++) {
                const int c = w * CPW + j;
                uint32_t code = ep.out.zero_code;
                if (c < C) {
                    const int64_t o = pix * C + c;
                    if (ep.acc_out) ep.acc_out[o] = acc[uu][j];
                    float y = __fmaf_rn(scv[j], (float)acc[uu][j], biv[j]);
                    if (ep.residual) {
                        const uint32_t rc =
                            (__ldg(ep.residual + pix * ep.res_ld + c / rcpw) >> (ep.res_b * (c % rcpw))) & rmask;
                        y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
                    }
                    y = cc_act(y, ep.act);
                    if (ep.y_out) ep.y_out[o] = y;
                    if (ep.codes_out) code = b4 ? project_by_thr7(y, t7, ep.out) : project_by_table(y, T, ep.out);
                }
                word |= code << (B * j);
            }
            if (ep.codes_out) ep.codes_out[ow] = word;
        }
    }
}

// Depthwise 3x3 of 4-bit codes on packed fp16 pairs.  Every 4-bit image is
// an integer of magnitude at most 12, so every partial sum of the 9 taps is
// an integer of magnitude at most 9 * 12 * 12 = 1296 < 2^11: fp16 holds each
// one exactly and a fused multiply-add of two such pairs never rounds (the
// host takes this kernel only when 9 * max|Ix| * max|Iw| <= 2048).  One
// half2 = the images of two neighbouring channels (one byte of a code
// word), so one instruction does two channels' multiply-adds and one table
// load decodes two codes.  The sums never take the value -0 (they start at
// +0, and an exact zero sum rounds to +0), so their conversion to float is
// the integer accumulator's.  Work items, the strip walk and the epilogues
// are those of the integer kernel above, plus a word-at-a-time one for
// codes-only outputs with per-channel scale and bias; the next filter row's
// input words are loaded while the current row is multiplied.
template <int STRIDE>
__global__ void __launch_bounds__(128, 6)
esb_dwconv3_b4h_kernel(const uint32_t* __restrict__ X, int ldx, int kx, const uint32_t* __restrict__ W, int ldw,
                       int kw, int H, int Wd, int C, int pad, int P, int Q, int QS, int rows, CcEpi ep)
{
    constexpr int QT = STRIDE == 1 ? 4 : 2;
    constexpr int NIN = (QT - 1) * STRIDE + 3;
    extern __shared__ __half2 wtab2[];                // [9][words * 4] filter images, channel pairs
    __shared__ __half2 lut2[256];                     // code byte -> (image of low nibble, image of high nibble)
    __shared__ float T[128];
    __shared__ float Rs[8];
    const int words = (C + 7) / 8;
    const int cp2 = words * 4;
    const int ewx = 3 - kx, Nx = (1 << ewx) - 1;
    const int eww = 3 - kw, Nw = (1 << eww) - 1;
    griddep_wait();
    for (int i = threadIdx.x; i < 256; i += blockDim.x)
        lut2[i] = __halves2half2(__int2half_rn(code_image_i((uint32_t)i & 15u, 4, kx, ewx, Nx)),
                                 __int2half_rn(code_image_i((uint32_t)i >> 4, 4, kx, ewx, Nx)));
    for (int i = threadIdx.x; i < 9 * words; i += blockDim.x) {
        const int t = i / words, w = i - (i / words) * words;
        const uint32_t fw = __ldg(W + t * ldw + w);
#pragma unroll
        for (int m = 0; m < 4; m++)
            wtab2[t * cp2 + w * 4 + m] =
                __halves2half2(__int2half_rn(code_image_i((fw >> (8 * m)) & 15u, 4, kw, eww, Nw)),
                               __int2half_rn(code_image_i((fw >> (8 * m + 4)) & 15u, 4, kw, eww, Nw)));
    }
    const float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
    if (ep.codes_out) build_thresholds(T, ep.out, alpha_out, threadIdx.x >> 5, threadIdx.x & 31, 0, blockDim.x >> 5);
    const bool dq = ep.alpha_a_dev && ep.alpha_b_dev;
    const float dqs = dq ? __fmul_rn(__ldg(ep.alpha_a_dev), __ldg(ep.alpha_b_dev)) * ep.dq_pow2 : 1.0f;
    const float sc_fixed = ep.scale ? 0.0f : (dq ? __fmul_rn(ep.scale0, dqs) : ep.scale0);
    const bool b4 = ep.out.b == 4 && ep.codes_out;
    const bool lean = b4 && ep.acc24 && !ep.scale && !ep.bias && !ep.residual && !ep.acc_out && !ep.y_out &&
                      sc_fixed > 0.0f && (!ep.out.is_signed || ep.act != ESB_ACT_NONE);
    // codes only, any scale and bias: the word's 8 codes from their buckets at once
    const bool words8 = b4 && !lean && !ep.residual && !ep.acc_out && !ep.y_out;
    const uint32_t sgn_out = ep.out.is_signed ? 1u : 0u;
    __syncthreads();
    if (lean && threadIdx.x < 7) Rs[threadIdx.x] = acc_raw_threshold(sc_fixed, ep.bias0, T[threadIdx.x], ep.act, 1.0f);
    __syncthreads();
    Thr7 t7, r7;
#pragma unroll
    for (int i = 0; i < 7; i++) {
        t7.t[i] = b4 ? T[i] : 0.0f;
        r7.t[i] = lean ? Rs[i] : 0.0f;
    }
    const int rcpw = ep.residual ? 32 / ep.res_b : 1;
    const uint32_t rmask = ep.residual ? (1u << ep.res_b) - 1u : 0u;
    const uint32_t zx = 0x11111111u * (uint32_t)fmt_zero_code(4, kx);
    uint32_t zo = 0u;
    for (int j = 0; j < 32 / ep.out.b; j++) zo |= ep.out.zero_code << (ep.out.b * j);
    const int ldo = (int)ep.ldo;
    const int upr = QS * ldo;
    const int total = rows * upr;
    for (int it = blockIdx.x * blockDim.x + threadIdx.x; it < total; it += gridDim.x * blockDim.x) {
        const int row = it / upr;                     // n * P + p
        const int u = it - row * upr;
        const int qs = u / ldo;
        const int w = u - qs * ldo;
        const int nn = row / P;
        const int p = row - nn * P;
        const int q0 = qs * QT;
        const int64_t obase = ((int64_t)row * Q + q0) * ldo + w;
        if (w >= words) {
            if (ep.codes_out) {
#pragma unroll
                for (int uu = 0; uu < QT; uu++)
                    if (q0 + uu < Q) ep.codes_out[obase + (int64_t)uu * ldo] = zo;
            }
            continue;
        }
        const int c0 = q0 * STRIDE - pad;
        const int h0 = p * STRIDE - pad;
        const uint32_t* xim = X + (int64_t)nn * H * Wd * ldx + w;
        // input words of filter row r (rows outside the image read as zero codes)
        auto load_row = [&](uint32_t (&xv)[NIN], int r) {
            const int h = h0 + r;
            const bool hin = (unsigned)h < (unsigned)H;
            const uint32_t* xrow = xim + (int64_t)h * Wd * ldx;
#pragma unroll
            for (int c = 0; c < NIN; c++) {
                const int col = c0 + c;
                xv[c] = (hin && (unsigned)col < (unsigned)Wd) ? __ldg(xrow + (int64_t)col * ldx) : zx;
            }
        };
        __half2 acc[QT][4];
#pragma unroll
        for (int uu = 0; uu < QT; uu++)
#pragma unroll
            for (int m = 0; m < 4; m++) acc[uu][m] = __float2half2_rn(0.0f);
        uint32_t xw[NIN], xn[NIN];
        load_row(xw, 0);
#pragma unroll 1
        for (int r = 0; r < 3; r++) {
            if (r < 2) load_row(xn, r + 1);
            __half2 wf[3][4];
#pragma unroll
            for (int s2 = 0; s2 < 3; s2++)
#pragma unroll
                for (int m = 0; m < 4; m++) wf[s2][m] = wtab2[(r * 3 + s2) * cp2 + w * 4 + m];
#pragma unroll
            for (int c = 0; c < NIN; c++) {
                __half2 img[4];
#pragma unroll
                for (int m = 0; m < 4; m++) img[m] = lut2[__byte_perm(xw[c], 0u, 0x4440u + (uint32_t)m)];
#pragma unroll
                for (int uu = 0; uu < QT; uu++) {
                    const int s2 = c - uu * STRIDE;
                    if (s2 >= 0 && s2 < 3) {
#pragma unroll
                        for (int m = 0; m < 4; m++) acc[uu][m] = __hfma2(img[m], wf[s2][m], acc[uu][m]);
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < NIN; c++) xw[c] = xn[c];
        }
        const int cvalid = C - w * 8;
        float scv[8], biv[8];
        if (!lean) {
#pragma unroll
            for (int j = 0; j < 8; j++) {
                const int c = w * 8 + j < C ? w * 8 + j : C - 1;
                float sc = ep.scale ? __ldg(ep.scale + c) : ep.scale0;
                if (dq) sc = __fmul_rn(sc, dqs);
                scv[j] = sc;
                biv[j] = ep.bias ? __ldg(ep.bias + c) : ep.bias0;
            }
        }
#pragma unroll
        for (int uu = 0; uu < QT; uu++) {
            if (q0 + uu >= Q) break;
            const int64_t ow = obase + (int64_t)uu * ldo;
            float a[8];
#pragma unroll
            for (int m = 0; m < 4; m++) {
                const float2 f2 = __half22float2(acc[uu][m]);
                a[2 * m] = f2.x;
                a[2 * m + 1] = f2.y;
            }
            if (lean) {
                uint32_t J = 0u;
#pragma unroll
                for (int j = 0; j < 8; j++) {
                    const float v = a[j];
                    const bool b2 = v >= r7.t[3];
                    const bool b1 = v >= (b2 ? r7.t[5] : r7.t[1]);
                    const bool b0 = v >= (b2 ? (b1 ? r7.t[6] : r7.t[4]) : (b1 ? r7.t[2] : r7.t[0]));
                    const uint32_t jb = (b2 ? 4u : 0u) | (b1 ? 2u : 0u) | (b0 ? 1u : 0u);
                    J |= (j < cvalid ? jb : 0u) << (4 * j);
                }
                ep.codes_out[ow] = codes8_b4(J, 0u, ep.out.k);
                continue;
            }
            if (words8) {
                // per element: y = fma(scale, acc, bias), the activation, then
                // the bucket of |y| (zero for negatives of an unsigned set);
                // codes8_b4 turns buckets and signs into the word (zero
                // buckets keep sign 0), as project_by_thr7 does per code
                uint32_t J = 0u, S = 0u;
#pragma unroll
                for (int j = 0; j < 8; j++) {
                    const uint32_t u = __float_as_uint(cc_act(__fmaf_rn(scv[j], a[j], biv[j]), ep.act));
                    const uint32_t neg = u >> 31;
                    const uint32_t jb = bucket7(__uint_as_float(u & 0x7fffffffu), t7);
                    J |= ((j < cvalid && (sgn_out | (neg ^ 1u))) ? jb : 0u) << (4 * j);
                    S |= (neg & sgn_out) << (4 * j + 3);
                }
                ep.codes_out[ow] = codes8_b4(J, S, ep.out.k);
                continue;
            }
            const int64_t pix = (int64_t)row * Q + q0 + uu;
            uint32_t word = 0;
#pragma unroll
            for (int j = 0; j < 8; j++) {
                const int c = w * 8 + j;
                uint32_t code = ep.out.zero_code;
                if (c < C) {
                    const int64_t o = pix * C + c;
                    if (ep.acc_out) ep.acc_out[o] = (int32_t)a[j];
                    float y = __fmaf_rn(scv[j], a[j], biv[j]);
                    if (ep.residual) {
                        const uint32_t rc =
                            (__ldg(ep.residual + pix * ep.res_ld + c / rcpw) >> (ep.res_b * (c % rcpw))) & rmask;
                        y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
                    }
                    y = cc_act(y, ep.act);
                    if (ep.y_out) ep.y_out[o] = y;
                    if (ep.codes_out) code = b4 ? project_by_thr7(y, t7, ep.out) : project_by_table(y, T, ep.out);
                }
                word |= code << (ep.out.b * j);
            }
            if (ep.codes_out) ep.codes_out[ow] = word;
        }
    }
}

// One resident wave of blocks (each block's set-up -- filter table,
// thresholds -- is then paid once per block and amortised over many items).
template <class Kern>
static cudaError_t launch_dw_wave(Kern kern, size_t smem, int64_t items, const esb_conv_desc& d, int P, int Q, int QS,
                                  const uint32_t* X, int64_t ldx, int kx, const uint32_t* W, int64_t ldw, int kw,
                                  const CcEpi& ep, cudaStream_t st)
{
    int64_t blocks = (items + 127) / 128;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 128, smem) != cudaSuccess || per_sm < 1)
        per_sm = 4;
    const int64_t cap = (int64_t)device_sm_count() * per_sm;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    kern<<<(unsigned)blocks, 128, smem, st>>>(X, (int)ldx, kx, W, (int)ldw, kw, d.h, d.w, d.c, d.pad, P, Q, QS,
                                              d.n * P, ep);
    return cudaGetLastError();
}

template <int B, int STRIDE>
static cudaError_t launch_dw3(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int kx,
                              const uint32_t* W, int64_t ldw, int kw, const CcEpi& ep, bool h16, cudaStream_t st)
{
    constexpr int QT = STRIDE == 1 ? 4 : 2;
    const int QS = (Q + QT - 1) / QT;
    const int64_t items = (int64_t)d.n * P * QS * ep.ldo;
    const int words = (d.c + 32 / B - 1) / (32 / B);
    if constexpr (B == 4) {
        if (h16)
            return launch_dw_wave(esb_dwconv3_b4h_kernel<STRIDE>, sizeof(__half2) * 9 * (size_t)words * 4, items, d, P,
                                  Q, QS, X, ldx, kx, W, ldw, kw, ep, st);
    }
    return launch_dw_wave(esb_dwconv3_kernel<B, STRIDE>, sizeof(int32_t) * 9 * (size_t)words * (32 / B), items, d, P,
                          Q, QS, X, ldx, kx, W, ldw, kw, ep, st);
}

static CcEpi make_cc_epi(const GemmOutputs& o, int ka, int kb)
{
    CcEpi ep;
    const esb_epilogue* e = o.ep;
    ep.scale = e ? e->scale : nullptr;
    ep.bias = e ? e->bias : nullptr;
    ep.alpha_a_dev = e ? e->alpha_a_dev : nullptr;
    ep.alpha_b_dev = e ? e->alpha_b_dev : nullptr;
    ep.dq_pow2 = ldexpf(1.0f, -(ka + kb));
    ep.scale0 = e ? e->scale0 : 1.0f;
    ep.bias0 = e ? e->bias0 : 0.0f;
    ep.act = e ? e->act : ESB_ACT_NONE;
    ep.residual = e ? e->residual : nullptr;
    ep.res_ld = e ? e->res_ld : 0;
    ep.res_b = (e && e->residual) ? e->res_fmt.b : 4;
    ep.res_k = (e && e->residual) ? e->res_fmt.k : 0;
    ep.res_scale = e ? e->res_scale : 0.0f;
    ep.alpha_out = e ? e->alpha_out : 1.0f;
    ep.alpha_out_dev = e ? e->alpha_out_dev : nullptr;
    const bool oc = e && o.codes_out;
    ep.out = make_proj_params(oc ? e->fmt_out.b : 4, oc ? e->fmt_out.k : 2, oc ? e->fmt_out.is_signed : 1,
                              oc ? e->rounding_out : 0);
    ep.acc_out = o.acc_out;
    ep.y_out = o.y_out;
    ep.codes_out = o.codes_out;
    ep.ldo = o.ldo;
    ep.acc24 = 0;
    return ep;
}

static unsigned grid_for(int64_t work)
{
    int64_t blocks = (work + 255) / 256;
    const int64_t cap = (int64_t)device_sm_count() * 16;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    return (unsigned)blocks;
}

cudaError_t launch_dwconv(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int bx, int kx,
                          const uint32_t* W, int64_t ldw, int bw, int kw, const GemmOutputs& o, cudaStream_t st)
{
    CcEpi ep = make_cc_epi(o, kx, kw);
    ep.acc24 = (double)d.r * d.s * fmt_max_image(bx, kx) * fmt_max_image(bw, kw) < 16777216.0;
    // Thread grid covers words of the output row stride: ldo words when codes
    // are written, else the input's words (acc/y only).
    if (!o.codes_out) ep.ldo = (d.c + (32 / bx) - 1) / (32 / bx);
    // filter table of the fast kernel: 9 taps x the padded channels, int32, in 48 KiB
    const int64_t tab = 9 * (int64_t)((d.c + 32 / bx - 1) / (32 / bx)) * (32 / bx) * 4;
    // the specialised kernel indexes in 32 bits: work items, input and output words of one image
    const int P1 = P, Q1 = Q;
    const int64_t items = (int64_t)d.n * P1 * ((Q1 + 1) / 2) * (o.codes_out ? o.ldo : 1);
    const bool fits32 = items < (1ll << 31) && (int64_t)d.n * d.h * d.w * ldx < (1ll << 31) && ldx < (1 << 20) &&
                        ldw < (1 << 20) && ep.ldo < (1 << 20);
    if (d.r == 3 && d.s == 3 && bw == bx && bx >= 3 && bx <= 6 && (d.stride == 1 || d.stride == 2) &&
        tab <= 48 * 1024 && fits32) {
        const bool s1 = d.stride == 1;
        // packed fp16 sums are exact while every partial sum stays below 2^11
        const bool h16 = 9.0 * fmt_max_image(bx, kx) * fmt_max_image(bw, kw) <= 2048.0;
        switch (bx) {
        case 3: return s1 ? launch_dw3<3, 1>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, false, st)
                          : launch_dw3<3, 2>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, false, st);
        case 4: return s1 ? launch_dw3<4, 1>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, h16, st)
                          : launch_dw3<4, 2>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, h16, st);
        case 5: return s1 ? launch_dw3<5, 1>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, false, st)
                          : launch_dw3<5, 2>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, false, st);
        default: return s1 ? launch_dw3<6, 1>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, false, st)
                           : launch_dw3<6, 2>(d, P, Q, X, ldx, kx, W, ldw, kw, ep, false, st);
        }
    }
    const int64_t total = (int64_t)d.n * P * Q * ep.ldo;
    esb_dwconv_kernel<<<grid_for(total), 256, 0, st>>>(X, ldx, bx, kx, W, ldw, bw, kw, d.n, d.h, d.w, d.c, d.r, d.s,
                                                        d.stride, d.pad, P, Q, ep);
    return cudaGetLastError();
}

// ------------------------------------------------------------- max pool

// One thread = one output code word: per channel slot, the code with the
// largest value over the window clipped to the image (Sec. IV-B intersection
// window); zero (sign 0) if the maximum is zero.
__global__ void __launch_bounds__(256)
esb_maxpool_kernel(const uint32_t* __restrict__ X, int64_t ldx, int b, int k, int n, int H, int Wd, int C, int win,
                   int stride, int pad, int P, int Q, uint32_t* __restrict__ Y, int64_t ldy)
{
    const int cpw = 32 / b;
    const int ew = b - k - 1, N = (1 << ew) - 1;
    const uint32_t mask = (1u << b) - 1u;
    const uint32_t zero = (uint32_t)N << k;
    const int64_t total = (int64_t)n * P * Q * ldy;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t pix = t / ldy;
        const int w = (int)(t - pix * ldy);
        const int q = (int)(pix % Q);
        const int64_t np_ = pix / Q;
        const int p = (int)(np_ % P);
        const int64_t nn = np_ / P;
        int32_t best[16];
        uint32_t bestc[16];
#pragma unroll
        for (int j = 0; j < 16; j++) { best[j] = INT32_MIN; bestc[j] = zero; }
        if (w < ldx) {
            for (int r = 0; r < win; r++) {
                const int h = p * stride - pad + r;
                if (h < 0 || h >= H) continue;
                for (int s = 0; s < win; s++) {
                    const int ww = q * stride - pad + s;
                    if (ww < 0 || ww >= Wd) continue;
                    const uint32_t xw = __ldg(X + ((nn * H + h) * Wd + ww) * ldx + w);
#pragma unroll
                    for (int j = 0; j < 16; j++) {
                        if (j < cpw) {
                            const uint32_t c = (xw >> (b * j)) & mask;
                            const int32_t v = code_image_i(c, b, k, ew, N);
                            if (v > best[j]) { best[j] = v; bestc[j] = c; }
                        }
                    }
                }
            }
        }
        uint32_t word = 0;
#pragma unroll
        for (int j = 0; j < 16; j++) {
            if (j >= cpw) break;
            const int ch = w * cpw + j;
            const uint32_t c = (ch < C && best[j] != 0) ? bestc[j] : zero;
            word |= c << (b * j);
        }
        Y[pix * ldy + w] = word;
    }
}

// Window walk of the rank max pools: calls take(word) for every input word
// of output pixel (q, p) of image nn at word w.  With WIN > 0 (the 3x3
// window of ResNet18's stem pool) all WIN*WIN loads are issued before the
// first maximum; taps outside the image read the zero-code word, whose
// ranks are all 0 (the minimum), so they change nothing.
template <int WIN, class Take>
__device__ __forceinline__ void pool_window(const uint32_t* __restrict__ X, int64_t ldx, int nn, int p, int q, int w,
                                            int H, int Wd, int win, int stride, int pad, uint32_t zw, Take take)
{
    if constexpr (WIN > 0) {
        uint32_t xv[WIN * WIN];
#pragma unroll
        for (int r = 0; r < WIN; r++) {
            const int h = p * stride - pad + r;
            const bool hin = (unsigned)h < (unsigned)H;
            const uint32_t* xr = X + ((int64_t)nn * H + (hin ? h : 0)) * Wd * ldx + w;
#pragma unroll
            for (int s2 = 0; s2 < WIN; s2++) {
                const int ww = q * stride - pad + s2;
                xv[r * WIN + s2] = (hin && (unsigned)ww < (unsigned)Wd) ? __ldg(xr + (int64_t)ww * ldx) : zw;
            }
        }
#pragma unroll
        for (int i = 0; i < WIN * WIN; i++) take(xv[i]);
    } else {
        for (int r = 0; r < win; r++) {
            const int h = p * stride - pad + r;
            if (h < 0 || h >= H) continue;
            const uint32_t* xr = X + ((int64_t)nn * H + h) * Wd * ldx + w;
            for (int s2 = 0; s2 < win; s2++) {
                const int ww = q * stride - pad + s2;
                if (ww < 0 || ww >= Wd) continue;
                take(__ldg(xr + (int64_t)ww * ldx));
            }
        }
    }
}

// Max pooling of unsigned 4-bit codes without decoding them: the value
// order of the non-negative set is the order of the rotated code
// (e + 1 mod 2^(b-1-k), then f), i.e. rank = (code + 2^k) mod 8, so the
// maximum of a window is the nibble-wise maximum of the ranks and the code
// comes back by the inverse rotation.  The eight 3-bit ranks of a word are
// compared at once: (best | 8) - rank in each nibble lies in 1..15 (no
// borrow crosses a nibble) and keeps bit 3 exactly where best >= rank,
// which selects the larger of the two.  One thread = one output word;
// blockIdx.y = image row (n, p), threads over (q, word).
template <int WIN>
__global__ void __launch_bounds__(256)
esb_maxpool_b4u_kernel(const uint32_t* __restrict__ X, int64_t ldx, int k, int H, int Wd, int C, int win, int stride,
                       int pad, int P, int Q, uint32_t* __restrict__ Y, int64_t ldy)
{
    const int np_ = blockIdx.y;
    const int nn = np_ / P, p = np_ - (np_ / P) * P;
    const int per_row = Q * (int)ldy;
    const uint32_t rot = 0x11111111u << k;            // + 2^k in every nibble
    const int words = (C + 7) / 8;
    const uint32_t zero = (uint32_t)((1 << (3 - k)) - 1) << k;   // e = N, f = 0 for b = 4
    const uint32_t zw = 0x11111111u * zero;
    for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < per_row; t += gridDim.x * blockDim.x) {
        const int q = t / (int)ldy, w = t - (t / (int)ldy) * (int)ldy;
        uint32_t best = 0u;                           // rank maxima, one per nibble (0 = the rank of zero)
        if (w < words)
            pool_window<WIN>(X, ldx, nn, p, q, w, H, Wd, win, stride, pad, zw, [&](uint32_t xw) {
                const uint32_t rk = ((xw & 0x77777777u) + rot) & 0x77777777u;
                const uint32_t ge = ((best | 0x88888888u) - rk) & 0x88888888u;   // bit 3: best >= rk
                const uint32_t keep = ge - (ge >> 3);                            // 7 where best >= rk
                best = (best & keep) | (rk & ~keep);
            });
        // inverse rotation: code = (rank - 2^k) mod 8; rank 0 is the zero code
        uint32_t word = (best + (0x88888888u - rot)) & 0x77777777u;
        // channels past C (in the last word) and padding words: the zero code
        const int c0 = w * 8;
        if (w >= words) word = zw;
        else if (c0 + 8 > C) {
            const int keep = C - c0;
            const uint32_t m = keep >= 8 ? 0xffffffffu : ((1u << (4 * keep)) - 1u);
            word = (word & m) | (zw & ~m);
        }
        Y[(((int64_t)nn * P + p) * Q + q) * ldy + w] = word;
    }
}

// Max pool of unsigned B-bit codes (B != 4) by the same rank rotation:
// rank = (code + 2^k) mod 2^(B-1) orders the non-negative set (rank 0 is
// the zero code), so each channel slot keeps the largest rank of its
// window and the code comes back by the inverse rotation.  One thread =
// one output word; blockIdx.y = image row (n, p); 32-bit indices.
template <int B, int WIN>
__global__ void __launch_bounds__(256)
esb_maxpool_rank_kernel(const uint32_t* __restrict__ X, int64_t ldx, int k, int H, int Wd, int C, int win, int stride,
                        int pad, int P, int Q, uint32_t* __restrict__ Y, int64_t ldy)
{
    constexpr int CPW = 32 / B;
    constexpr uint32_t RM = (1u << (B - 1)) - 1u;     // ranks live in B - 1 bits
    const int np_ = blockIdx.y;
    const int nn = np_ / P, p = np_ - (np_ / P) * P;
    const int per_row = Q * (int)ldy;
    const uint32_t rot = 1u << k;
    const int words = (C + CPW - 1) / CPW;
    const uint32_t zero = (uint32_t)((1 << (B - 1 - k)) - 1) << k;   // e = N, f = 0
    uint32_t zw = 0u;
#pragma unroll
    for (int j = 0; j < CPW; j++) zw |= zero << (B * j);
    for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < per_row; t += gridDim.x * blockDim.x) {
        const int q = t / (int)ldy, w = t - (t / (int)ldy) * (int)ldy;
        uint32_t best[CPW];
#pragma unroll
        for (int j = 0; j < CPW; j++) best[j] = 0u;
        if (w < words)
            pool_window<WIN>(X, ldx, nn, p, q, w, H, Wd, win, stride, pad, zw, [&](uint32_t xw) {
#pragma unroll
                for (int j = 0; j < CPW; j++) {
                    const uint32_t rk = (((xw >> (B * j)) & RM) + rot) & RM;
                    best[j] = best[j] > rk ? best[j] : rk;
                }
            });
        uint32_t word = 0u;
#pragma unroll
        for (int j = 0; j < CPW; j++) {
            const bool in = w < words && w * CPW + j < C;
            const uint32_t code = in ? ((best[j] + (RM + 1u) - rot) & RM) : zero;
            word |= code << (B * j);
        }
        Y[(((int64_t)nn * P + p) * Q + q) * ldy + w] = word;
    }
}

template <int B>
static void launch_maxpool_rank(const uint32_t* X, int64_t ldx, int k, int n, int H, int Wd, int C, int win,
                                int stride, int pad, int P, int Q, uint32_t* Y, int64_t ldy, cudaStream_t st)
{
    const int per_row = (int)(Q * ldy);
    const dim3 grid((unsigned)((per_row + 255) / 256), (unsigned)(n * P));
    if (win == 3)
        esb_maxpool_rank_kernel<B, 3><<<grid, 256, 0, st>>>(X, ldx, k, H, Wd, C, win, stride, pad, P, Q, Y, ldy);
    else
        esb_maxpool_rank_kernel<B, 0><<<grid, 256, 0, st>>>(X, ldx, k, H, Wd, C, win, stride, pad, P, Q, Y, ldy);
}

cudaError_t launch_maxpool(const uint32_t* X, int64_t ldx, int b, int k, int n, int H, int Wd, int C, int win,
                           int stride, int pad, int P, int Q, uint32_t* Y, int64_t ldy, cudaStream_t st,
                           int is_signed)
{
    if (b != 4 && !is_signed && (int64_t)n * P <= 65535 && (int64_t)Q * ldy < (1ll << 31)) {
        switch (b) {
        case 2: launch_maxpool_rank<2>(X, ldx, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy, st); break;
        case 3: launch_maxpool_rank<3>(X, ldx, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy, st); break;
        case 5: launch_maxpool_rank<5>(X, ldx, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy, st); break;
        case 6: launch_maxpool_rank<6>(X, ldx, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy, st); break;
        case 7: launch_maxpool_rank<7>(X, ldx, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy, st); break;
        default: launch_maxpool_rank<8>(X, ldx, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy, st); break;
        }
        return cudaGetLastError();
    }
    if (b == 4 && !is_signed && (int64_t)n * P <= 65535 && (int64_t)Q * ldy < (1ll << 31)) {
        const int per_row = (int)(Q * ldy);
        const dim3 grid((unsigned)((per_row + 255) / 256), (unsigned)(n * P));
        if (win == 3)
            esb_maxpool_b4u_kernel<3><<<grid, 256, 0, st>>>(X, ldx, k, H, Wd, C, win, stride, pad, P, Q, Y, ldy);
        else
            esb_maxpool_b4u_kernel<0><<<grid, 256, 0, st>>>(X, ldx, k, H, Wd, C, win, stride, pad, P, Q, Y, ldy);
        return cudaGetLastError();
    }
    const int64_t total = (int64_t)n * P * Q * ldy;
    esb_maxpool_kernel<<<grid_for(total), 256, 0, st>>>(X, ldx, b, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy);
    return cudaGetLastError();
}

// ------------------------------------------------------ global avg pool

// One block = 32 consecutive code words (lanes) of one image; its
// kPoolWarps warps split the image's pixels (warp i takes pixels i, i + 8,
// ...), so each warp load reads 128 contiguous bytes and a lane's loads are
// independent.  Codes decode through a 2^B-entry table of integer images;
// each lane sums its CPW channels exactly in int32; the partial sums of
// warps 1..7 meet warp 0's in shared memory (integer sums: the result does
// not depend on the split), and warp 0 scales and requantises each sum
// through the block's threshold table.
constexpr int kPoolWarps = 8;

template <int B>
__global__ void __launch_bounds__(kPoolWarps * 32)
esb_avgpool_kernel(const uint32_t* __restrict__ X, int64_t ldx, int k, int n, int HW, int C, int wout, float scale,
                   float alpha_out, ProjParams out, float* __restrict__ y_out, uint32_t* __restrict__ codes_out,
                   int64_t ldo)
{
    constexpr int CPW = 32 / B;
    constexpr uint32_t MASK = (1u << B) - 1u;
    __shared__ float T[128];
    __shared__ int32_t lut[1 << B];
    __shared__ int32_t part[kPoolWarps - 1][CPW][32]; // [warp - 1][channel slot][lane]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    griddep_wait();
    const int ew = B - k - 1, N = (1 << ew) - 1;
    for (int i = threadIdx.x; i < (1 << B); i += blockDim.x) lut[i] = code_image_i((uint32_t)i, B, k, ew, N);
    if (codes_out) build_thresholds(T, out, alpha_out, warp, lane, 0, kPoolWarps);
    __syncthreads();
    const int w = blockIdx.x * 32 + lane;
    const bool has = w < wout && w * CPW < C;
    for (int nn = blockIdx.y; nn < n; nn += gridDim.y) {
        int32_t acc[CPW];
#pragma unroll
        for (int j = 0; j < CPW; j++) acc[j] = 0;
        if (has) {
            const uint32_t* xp = X + (int64_t)nn * HW * ldx + w;
#pragma unroll 4
            for (int i = warp; i < HW; i += kPoolWarps) {
                const uint32_t xw = __ldg(xp + (int64_t)i * ldx);
#pragma unroll
                for (int j = 0; j < CPW; j++) acc[j] += lut[(xw >> (B * j)) & MASK];
            }
        }
        if (warp > 0) {
#pragma unroll
            for (int j = 0; j < CPW; j++) part[warp - 1][j][lane] = acc[j];
        }
        __syncthreads();                              // partial sums ready
        if (warp == 0 && w < wout) {
            uint32_t word = 0;
            if (has) {
#pragma unroll 1
                for (int j = 0; j < CPW; j++) {
                    int32_t sum = acc[j];
#pragma unroll
                    for (int v = 0; v < kPoolWarps - 1; v++) sum += part[v][j][lane];
                    const int c = w * CPW + j;
                    uint32_t code = out.zero_code;
                    if (c < C) {
                        const float y = __fmul_rn(scale, (float)sum);
                        if (y_out) y_out[(int64_t)nn * C + c] = y;
                        if (codes_out) code = project_by_table(y, T, out);
                    }
                    word |= code << (out.b * j);
                }
            } else {
                for (int j = 0; j < 32 / out.b; j++) word |= out.zero_code << (out.b * j);
            }
            if (codes_out && w < ldo) codes_out[(int64_t)nn * ldo + w] = word;
        }
        __syncthreads();                              // part is rewritten by the next image
    }
}

cudaError_t launch_avgpool(const uint32_t* X, int64_t ldx, int b, int k, int n, int HW, int C, float scale,
                           float alpha_out, int bo, int ko, int so, int rounding, float* y_out, uint32_t* codes_out,
                           int64_t ldo, cudaStream_t st)
{
    ProjParams out = make_proj_params(bo, ko, so, rounding);
    int64_t words = (C + (32 / b) - 1) / (32 / b);
    if (codes_out && ldo > words) words = ldo;          // also write the row's padding words
    const dim3 grid((unsigned)((words + 31) / 32), (unsigned)(n < 65535 ? n : 65535));
    const int wo = (int)words;
    switch (b) {
    case 2: esb_avgpool_kernel<2><<<grid, kPoolWarps * 32, 0, st>>>(X, ldx, k, n, HW, C, wo, scale, alpha_out, out,
                                                                     y_out, codes_out, ldo); break;
    case 3: esb_avgpool_kernel<3><<<grid, kPoolWarps * 32, 0, st>>>(X, ldx, k, n, HW, C, wo, scale, alpha_out, out,
                                                                     y_out, codes_out, ldo); break;
    case 4: esb_avgpool_kernel<4><<<grid, kPoolWarps * 32, 0, st>>>(X, ldx, k, n, HW, C, wo, scale, alpha_out, out,
                                                                     y_out, codes_out, ldo); break;
    case 5: esb_avgpool_kernel<5><<<grid, kPoolWarps * 32, 0, st>>>(X, ldx, k, n, HW, C, wo, scale, alpha_out, out,
                                                                     y_out, codes_out, ldo); break;
    case 6: esb_avgpool_kernel<6><<<grid, kPoolWarps * 32, 0, st>>>(X, ldx, k, n, HW, C, wo, scale, alpha_out, out,
                                                                     y_out, codes_out, ldo); break;
    case 7: esb_avgpool_kernel<7><<<grid, kPoolWarps * 32, 0, st>>>(X, ldx, k, n, HW, C, wo, scale, alpha_out, out,
                                                                     y_out, codes_out, ldo); break;
    default: esb_avgpool_kernel<8><<<grid, kPoolWarps * 32, 0, st>>>(X, ldx, k, n, HW, C, wo, scale, alpha_out, out,
                                                                      y_out, codes_out, ldo); break;
    }
    return cudaGetLastError();
}

}  // namespace esb
