// esb_cc.cu -- ESB kernels that run on CUDA cores (HBM-bound, no dense
// contraction to put on tensor cores):
//   * depthwise convolution (one r x s filter per channel, MobileNetV2's 3x3
//     layers) with the same fused epilogue as the tensor-core contraction,
//   * max pooling of codes with the intersection window of Sec. IV-B
//     (projection is monotone, so pooling codes = pooling quantised values),
//   * global average pooling: exact integer sum of the images per channel,
//     then one fp32 scale and ESB requantisation.
#include <cstdint>
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
    // Thread grid covers words of the output row stride: ldo words when codes
    // are written, else the input's words (acc/y only).
    if (!o.codes_out) ep.ldo = (d.c + (32 / bx) - 1) / (32 / bx);
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

cudaError_t launch_maxpool(const uint32_t* X, int64_t ldx, int b, int k, int n, int H, int Wd, int C, int win,
                           int stride, int pad, int P, int Q, uint32_t* Y, int64_t ldy, cudaStream_t st)
{
    const int64_t total = (int64_t)n * P * Q * ldy;
    esb_maxpool_kernel<<<grid_for(total), 256, 0, st>>>(X, ldx, b, k, n, H, Wd, C, win, stride, pad, P, Q, Y, ldy);
    return cudaGetLastError();
}

// ------------------------------------------------------ global avg pool

// One block per (image, channel word): threads stride over the HW pixels,
// per-thread int32 sums per channel slot, a shared-memory reduction, then
// y = fl32(scale * (float)sum) and the ESB projection of y with alpha_out
// (output codes use the input's b, so words line up).
__global__ void __launch_bounds__(256)
esb_avgpool_kernel(const uint32_t* __restrict__ X, int64_t ldx, int b, int k, int HW, int C, float scale,
                   float alpha_out, ProjParams out, float* __restrict__ y_out, uint32_t* __restrict__ codes_out,
                   int64_t ldo)
{
    const int cpw = 32 / b;
    const int ew = b - k - 1, N = (1 << ew) - 1;
    const uint32_t mask = (1u << b) - 1u;
    const int64_t nn = blockIdx.y;
    const int w = blockIdx.x;                           // code word of the channel group
    if (w * cpw >= C) {                                 // padding word of the output row
        if (threadIdx.x == 0 && codes_out && w < ldo) {
            uint32_t word = 0;
            for (int j = 0; j < 32 / out.b; j++) word |= out.zero_code << (out.b * j);
            codes_out[nn * ldo + w] = word;
        }
        return;
    }
    __shared__ int32_t red[256][16];
    int32_t acc[16];
#pragma unroll
    for (int j = 0; j < 16; j++) acc[j] = 0;
    for (int i = threadIdx.x; i < HW; i += blockDim.x) {
        const uint32_t xw = __ldg(X + (nn * HW + i) * ldx + w);
#pragma unroll
        for (int j = 0; j < 16; j++)
            if (j < cpw) acc[j] += code_image_i((xw >> (b * j)) & mask, b, k, ew, N);
    }
#pragma unroll
    for (int j = 0; j < 16; j++) red[threadIdx.x][j] = acc[j];
    __syncthreads();
    for (int h = blockDim.x / 2; h > 0; h >>= 1) {
        if ((int)threadIdx.x < h) {
#pragma unroll
            for (int j = 0; j < 16; j++) red[threadIdx.x][j] += red[threadIdx.x + h][j];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        uint32_t word = 0;
        for (int j = 0; j < cpw; j++) {
            const int c = w * cpw + j;
            uint32_t code = out.zero_code;
            if (c < C) {
                const float y = __fmul_rn(scale, (float)red[0][j]);
                if (y_out) y_out[nn * C + c] = y;
                code = project_code(y, alpha_out, out);
            }
            word |= code << (out.b * j);
        }
        if (codes_out && w < ldo) codes_out[nn * ldo + w] = word;
    }
}

cudaError_t launch_avgpool(const uint32_t* X, int64_t ldx, int b, int k, int n, int HW, int C, float scale,
                           float alpha_out, int bo, int ko, int so, int rounding, float* y_out, uint32_t* codes_out,
                           int64_t ldo, cudaStream_t st)
{
    ProjParams out = make_proj_params(bo, ko, so, rounding);
    int64_t words = (C + (32 / b) - 1) / (32 / b);
    if (codes_out && ldo > words) words = ldo;          // also write the row's padding words
    dim3 grid((unsigned)words, (unsigned)n);
    esb_avgpool_kernel<<<grid, 256, 0, st>>>(X, ldx, b, k, HW, C, scale, alpha_out, out, y_out, codes_out, ldo);
    return cudaGetLastError();
}

}  // namespace esb
