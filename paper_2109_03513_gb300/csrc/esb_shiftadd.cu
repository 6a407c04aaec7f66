// esb_shiftadd.cu -- ESB contraction on the CUDA cores with int64
// accumulation, for formats whose sums leave the range of the tensor-core
// path (exact fp32 TMEM sums below 2^24, int32 outputs): power-of-two-like
// sets such as (5,0), (6,1) or (6,0), and any K large enough to pass 2^24.
//
// Eq. esb_multiplication: the product of two set elements is the product
// of their significands (a small integer product: the paper's LUT fraction
// multiplier) shifted by the sum of their exponents.  Each code is decoded
// once per K-chunk into (signed significand, shift), and every
// multiply-accumulate is one 32-bit product, one 64-bit shift and one 64-bit
// add.  A block computes a 64 x TN output tile (TN = 64, or 60 when 64 is
// not a whole number of output code words), 16 x 16 threads with 4 x 4
// outputs each; the epilogue is the one of the tensor-core kernels, fed with
// float(acc) rounded to nearest.
#include <cstdint>
#include <cuda_runtime.h>

#include "esb_tc.cuh"

namespace esb {

namespace {

constexpr int kSaTileM = 64;
constexpr int kSaChunk = 32;           // codes of K per shared-memory stage
constexpr int kSaThreads = 256;

// Implicit im2col of NHWC codes with K over taps of kp codes (the input's
// codes per pixel): code kk of output pixel m is channel kk % kp of tap
// kk / kp.
struct Im2colSrc {
    const uint32_t* X;
    int64_t ldx;
    int64_t rows;
    int64_t kp;
    int H, W, P, Q, S, stride, pad;
    struct Row { int64_t pix0; int h0, w0; bool valid; };
    __device__ __forceinline__ Row row(int64_t m) const
    {
        Row x;
        x.valid = m < rows;
        const int64_t pq = (int64_t)P * Q;
        const int64_t n = x.valid ? m / pq : 0;
        const int rem = x.valid ? (int)(m - n * pq) : 0;
        const int p = rem / Q, q = rem - (rem / Q) * Q;
        x.h0 = p * stride - pad;
        x.w0 = q * stride - pad;
        x.pix0 = n * H;
        return x;
    }
    __device__ __forceinline__ const uint32_t* code_word(const Row& x, int64_t kk, int cpw, int& slot) const
    {
        const int64_t tap = kk / kp;
        const int64_t c = kk - tap * kp;
        const int r = (int)(tap / S), s = (int)(tap - (tap / S) * S);
        const int h = x.h0 + r, w = x.w0 + s;
        if (!x.valid || h < 0 || h >= H || w < 0 || w >= W) return nullptr;
        const int64_t wi = c / cpw;
        slot = (int)(c - wi * cpw);
        return X + ((x.pix0 + h) * W + w) * ldx + wi;
    }
};

struct SaFmt {
    int b, k, ew, cpw;
    uint32_t mask, zero;
};

__host__ inline SaFmt make_safmt(int b, int k)
{
    SaFmt f;
    f.b = b; f.k = k; f.ew = b - k - 1; f.cpw = 32 / b; f.mask = (1u << b) - 1u;
    f.zero = fmt_zero_code(b, k);
    return f;
}

// Code -> (signed significand m, shift sh), packed as (sh << 16) | (m & 0xffff):
// I = m << sh, with m = f for the "0.f" exponent N and 2^k + f otherwise.
__device__ __forceinline__ uint32_t sa_decode(uint32_t c, const SaFmt& f)
{
    const uint32_t s = (c >> (f.b - 1)) & 1u;
    const uint32_t N = (1u << f.ew) - 1u;
    const uint32_t e = f.ew > 0 ? (c >> f.k) & N : N;
    const uint32_t fr = c & ((1u << f.k) - 1u);
    const int m = (int)((e == N) ? fr : ((1u << f.k) | fr));
    const uint32_t sh = (e == N) ? 0u : e;
    return (sh << 16) | ((uint32_t)(s ? -m : m) & 0xffffu);
}

template <class Src>
__device__ __forceinline__ uint32_t sa_load(const Src& src, const typename Src::Row& row, int64_t kk, int64_t K,
                                            const SaFmt& f)
{
    uint32_t c = f.zero;
    if (kk < K) {
        int slot = 0;
        const uint32_t* p = src.code_word(row, kk, f.cpw, slot);
        if (p) c = (__ldg(p) >> (f.b * slot)) & f.mask;
    }
    return sa_decode(c, f);
}

template <class SrcA, class SrcB>
__global__ void __launch_bounds__(kSaThreads)
esb_shiftadd_kernel(SrcA srcA, SrcB srcB, int64_t M, int64_t N, int64_t K, SaFmt fa, SaFmt fb, int TN,
                    int64_t* __restrict__ acc64, EpiParams ep)
{
    __shared__ uint32_t sA[kSaChunk][kSaTileM];
    __shared__ uint32_t sB[kSaChunk][kSaTileM];
    __shared__ float thr[128];
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;
    const int64_t m0 = (int64_t)blockIdx.x * kSaTileM;
    const int64_t n0 = (int64_t)blockIdx.y * TN;
    griddep_wait();                                   // operands may come from the previous launch
    if (ep.codes_out) {
        const float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
        build_thresholds(thr, ep.out, alpha_out, tid >> 5, tid & 31, 0, kSaThreads / 32);
    }
    // the loader thread of element e = tid + 256 i: row e / 32, code e % 32
    const int lk = tid & 31;
    typename SrcA::Row ra[8];
    typename SrcB::Row rb[8];
#pragma unroll
    for (int i = 0; i < 8; i++) {
        const int r = (tid >> 5) + 8 * i;
        ra[i] = srcA.row(m0 + r);
        rb[i] = srcB.row(r < TN ? n0 + r : srcB.rows);
    }
    int64_t acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; i++)
#pragma unroll
        for (int j = 0; j < 4; j++) acc[i][j] = 0;
    for (int64_t k0 = 0; k0 < K; k0 += kSaChunk) {
        __syncthreads();
#pragma unroll
        for (int i = 0; i < 8; i++) {
            const int r = (tid >> 5) + 8 * i;
            sA[lk][r] = sa_load(srcA, ra[i], k0 + lk, K, fa);
            sB[lk][r] = sa_load(srcB, rb[i], k0 + lk, K, fb);
        }
        __syncthreads();
#pragma unroll 4
        for (int kk = 0; kk < kSaChunk; kk++) {
            uint32_t a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; i++) a[i] = sA[kk][ty + 16 * i];
#pragma unroll
            for (int j = 0; j < 4; j++) b[j] = sB[kk][tx + 16 * j];
#pragma unroll
            for (int i = 0; i < 4; i++)
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    // significand product (at most 17 bits), shifted by the exponent sum
                    const int prod = (int)(short)(a[i] & 0xffffu) * (int)(short)(b[j] & 0xffffu);
                    acc[i][j] += (int64_t)prod << ((a[i] >> 16) + (b[j] >> 16));
                }
        }
    }
    __syncthreads();
    // outputs: int64 accumulators, then the epilogue; codes go through a
    // shared-memory tile so that each packed word is written whole
    uint8_t* ctile = reinterpret_cast<uint8_t*>(&sA[0][0]);   // 64 x 64 bytes
    const EpiCtx cx = make_epi_ctx(ep, thr);
#pragma unroll
    for (int i = 0; i < 4; i++) {
        const int r = ty + 16 * i;
        const int64_t m = m0 + r;
#pragma unroll
        for (int j = 0; j < 4; j++) {
            const int cl = tx + 16 * j;
            const int64_t n = n0 + cl;
            if (cl >= TN) continue;
            uint32_t code = ep.out.zero_code;
            if (m < M && n < N) {
                if (acc64) acc64[m * N + n] = acc[i][j];
                if (ep.y_out || ep.codes_out) code = epi_element(ep, cx, __ll2float_rn(acc[i][j]), m, n, N);
            }
            ctile[r * kSaTileM + cl] = (uint8_t)code;
        }
    }
    if (!ep.codes_out) return;
    __syncthreads();
    const int cpw = ep.out_cpw;
    const int wpr = TN / cpw;                         // TN is a whole number of words
    const int64_t w0 = n0 / cpw;
    for (int idx = tid; idx < kSaTileM * wpr; idx += kSaThreads) {
        const int r = idx / wpr, wj = idx - (idx / wpr) * wpr;
        const int64_t m = m0 + r;
        if (m >= M || w0 + wj >= ep.ldo) continue;
        uint32_t word = 0u;
        for (int t = 0; t < cpw; t++) word |= (uint32_t)ctile[r * kSaTileM + wj * cpw + t] << (ep.out.b * t);
        ep.codes_out[m * ep.ldo + w0 + wj] = word;
    }
}

int sa_tile_n(int out_cpw) { return (64 % out_cpw == 0) ? 64 : 60; }

template <class SrcA, class SrcB>
cudaError_t launch_sa(const SrcA& a, const SrcB& b, int64_t M, int64_t N, int64_t K, const SaFmt& fa, const SaFmt& fb,
                      int64_t* acc64, const EpiParams& ep, cudaStream_t st)
{
    const int TN = sa_tile_n(ep.out_cpw);
    const dim3 grid((unsigned)((M + kSaTileM - 1) / kSaTileM), (unsigned)((N + TN - 1) / TN));
    return launch_pdl(esb_shiftadd_kernel<SrcA, SrcB>, grid, dim3(kSaThreads), 0, st, a, b, M, N, K, fa, fb, TN, acc64,
                      ep);
}

EpiParams sa_epi(const GemmOutputs& o, int ka, int kb)
{
    GemmOutputs o2 = o;
    o2.acc_out = nullptr;                             // the int64 accumulators are stored by the kernel
    EpiParams ep = make_epi(o2);
    ep.dq_pow2 = ldexpf(1.0f, -(ka + kb));
    return ep;
}

}  // namespace

bool shiftadd_grid_ok(int64_t M, int64_t N, int out_b)
{
    const int TN = sa_tile_n(32 / out_b);
    return (M + kSaTileM - 1) / kSaTileM < (1ll << 31) && (N + TN - 1) / TN <= 65535;
}

cudaError_t launch_gemm_i64(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, int ba, int ka,
                            const uint32_t* B, int64_t ldb, int bb, int kb, int64_t* acc64, const GemmOutputs& o,
                            cudaStream_t st)
{
    RowsSrc a{A, lda, M};
    RowsSrc b{B, ldb, N};
    return launch_sa(a, b, M, N, K, make_safmt(ba, ka), make_safmt(bb, kb), acc64, sa_epi(o, ka, kb), st);
}

cudaError_t launch_conv_i64(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int bx, int kx,
                            const uint32_t* W, int64_t ldw, int bw, int kw, int64_t* acc64, const GemmOutputs& o,
                            cudaStream_t st)
{
    const int64_t M = (int64_t)d.n * P * Q;
    const int64_t kp = ldx * (32 / bx);
    Im2colSrc a;
    a.X = X; a.ldx = ldx; a.rows = M; a.kp = kp; a.H = d.h; a.W = d.w; a.P = P; a.Q = Q; a.S = d.s;
    a.stride = d.stride; a.pad = d.pad;
    RowsSrc b{W, (int64_t)d.r * d.s * ldw, d.cout};
    b.kp = kp;
    b.ldt = ldw;
    const int64_t K = (int64_t)d.r * d.s * kp;
    return launch_sa(a, b, M, (int64_t)d.cout, K, make_safmt(bx, kx), make_safmt(bw, kw), acc64, sa_epi(o, kx, kw), st);
}

}  // namespace esb
