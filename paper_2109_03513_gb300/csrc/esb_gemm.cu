// esb_gemm.cu -- ESB-coded contraction on the tcgen05 tensor cores.
//
// acc[m][n] = sum_k I(A[m][k]) * I(B[n][k]) (Sec. III-B: a product of two set
// elements is a product of fraction values and a shift; Sec. IV-B: the
// convolution computing logic), followed by the post-processing of
// Sec. IV-C fused into the same kernel.
//
// Operand decode.  An ESB code (sign | e | f) with e = N meaning "0.f" is a
// floating-point number with a bias-1 exponent whose field is rotated by
// one: value = 2^(E-1) * 1.f for E = e + 1 >= 1 and 0.f for E = 0.  Scaled
// by 2^-6 this is exactly the fp8 E4M3 number with exponent field E and
// mantissa f << (3 - k), for every format with k <= 3 and b-k-1 <= 4
// (the E4M3 NaN pattern cannot occur).  So decode is a handful of bit
// operations per 8 codes, and the MMA multiplies I_A * I_B * 2^-(kA+kB+12)
// exactly.  The fp32 TMEM accumulator holds every partial sum exactly while
// K * max|I_A| * max|I_B| < 2^24 (checked on the host), and the epilogue
// scales it back to the exact int32 sum.
//
// Pipeline (per CTA, one 128 x BN output tile): all warps load packed code
// words and decode them into a kStages-deep ring of shared-memory stages in
// the 128-byte-swizzled K-major layout; one thread issues
// tcgen05.mma.kind::f8f6f4 (M = 128, N = BN, K = 32) into a TMEM
// accumulator and commits each stage to an mbarrier, which gates the reuse
// of that stage.  The MMAs of one stage run while the next stages are being
// decoded (the paper's ping-pong buffers, Sec. IV-C/IV-D).  The epilogue
// reads TMEM with tcgen05.ld and runs the fused affine / residual /
// activation / requantisation.
#include <cstdint>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

constexpr int kBM = 128;           // rows per tile (TMEM lanes)
constexpr int kBK = 128;           // codes (= E4M3 bytes) per K-block: one 128-byte swizzle row
constexpr int kStages = 4;
constexpr int kGemmThreads = 256;
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s

struct OpFmt {
    int b, k, ew, cpw;
    uint32_t mask;
};

__host__ inline OpFmt make_opfmt(int b, int k)
{
    OpFmt o;
    o.b = b; o.k = k; o.ew = b - k - 1; o.cpw = 32 / b; o.mask = (1u << b) - 1u;
    return o;
}

// Byte position of code j (0..15) of a 16-code unit.  The fast b = 4
// decode emits codes 0,2,4,6 | 1,3,5,7 of each word; every path uses the
// same order, so A and B agree on the K permutation (a contraction is
// invariant under a common permutation of K).
__device__ __forceinline__ int unit_pos(int j) { return ((j >> 3) << 3) | ((j & 1) << 2) | ((j & 7) >> 1); }

// One code -> scaled E4M3 byte.
__device__ __forceinline__ uint32_t code_to_e4m3(uint32_t c, const OpFmt& f)
{
    const uint32_t s = (c >> (f.b - 1)) & 1u;
    const uint32_t fr = c & ((1u << f.k) - 1u);
    uint32_t E = 0u;
    if (f.ew > 0) {
        const uint32_t em = (1u << f.ew) - 1u;
        E = (((c >> f.k) & em) + 1u) & em;
    }
    return (s << 7) | (E << 3) | (fr << (3 - f.k));
}

// 8 four-bit codes (one word) -> 8 scaled E4M3 bytes (lo: codes 0,2,4,6; hi: 1,3,5,7).
__device__ __forceinline__ void decode_word_b4(uint32_t w, int k, int ew, uint32_t& lo, uint32_t& hi)
{
    uint32_t u = w;
    if (ew > 0) u = (((w & 0x77777777u) + (0x11111111u << k)) & 0x77777777u) | (w & 0x88888888u);
    const uint32_t a = u & 0x0F0F0F0Fu;
    const uint32_t b = (u >> 4) & 0x0F0F0F0Fu;
    const int sh = 3 - k;
    lo = ((a & 0x07070707u) << sh) | ((a & 0x08080808u) << 4);
    hi = ((b & 0x07070707u) << sh) | ((b & 0x08080808u) << 4);
}

// ------------------------------------------------------------ row sources

// Plain K-major rows: logical word w of row r is base[r * ld + w].
struct RowsSrc {
    const uint32_t* base;
    int64_t ld;
    int64_t rows;
    struct Row { const uint32_t* p; };
    __device__ __forceinline__ Row row(int64_t r) const { Row x; x.p = (r < rows) ? base + r * ld : nullptr; return x; }
    __device__ __forceinline__ const uint32_t* words(const Row& x, int64_t w) const { return x.p ? x.p + w : nullptr; }
};

// Implicit im2col of NHWC codes: row m = (n, p, q) output pixel; logical
// word w = tap * ldx + word, tap = (r, s); out-of-image taps read as zero.
struct ConvSrc {
    const uint32_t* X;
    int64_t ldx;
    int64_t rows;                 // n * P * Q
    int H, W, P, Q, S, stride, pad;
    struct Row { int64_t pix0; int h0, w0; bool valid; };
    __device__ __forceinline__ Row row(int64_t m) const
    {
        Row x;
        x.valid = m < rows;
        const int64_t pq = (int64_t)P * Q;
        const int64_t n = x.valid ? m / pq : 0;
        const int64_t rem = x.valid ? m - n * pq : 0;
        const int p = (int)(rem / Q), q = (int)(rem - (int64_t)(rem / Q) * Q);
        x.h0 = p * stride - pad;
        x.w0 = q * stride - pad;
        x.pix0 = n * H;
        return x;
    }
    __device__ __forceinline__ const uint32_t* words(const Row& x, int64_t w) const
    {
        if (!x.valid) return nullptr;
        const int64_t tap = w / ldx;
        const int64_t word = w - tap * ldx;
        const int r = (int)(tap / S), s = (int)(tap - (int64_t)(tap / S) * S);
        const int h = x.h0 + r, ww = x.w0 + s;
        if (h < 0 || h >= H || ww < 0 || ww >= W) return nullptr;
        return X + ((x.pix0 + h) * W + ww) * ldx + word;
    }
};

// Decode the 16-code unit [k0, k0 + 16) of one row into 16 bytes.
template <class Src>
__device__ __forceinline__ uint4 decode_unit(const Src& src, const typename Src::Row& row, int64_t k0, int64_t K,
                                             const OpFmt& f)
{
    uint32_t o[4] = {0u, 0u, 0u, 0u};
    if (f.b == 4 && k0 + 16 <= K) {
        const uint32_t* p = src.words(row, k0 >> 3);
        if (p) {
            const uint2 w = __ldg(reinterpret_cast<const uint2*>(p));
            decode_word_b4(w.x, f.k, f.ew, o[0], o[1]);
            decode_word_b4(w.y, f.k, f.ew, o[2], o[3]);
        }
    } else {
        uint8_t* ob = reinterpret_cast<uint8_t*>(o);
#pragma unroll 1
        for (int j = 0; j < 16; j++) {
            const int64_t kk = k0 + j;
            if (kk >= K) break;
            const int64_t wi = kk / f.cpw;
            const int slot = (int)(kk - wi * f.cpw);
            const uint32_t* p = src.words(row, wi);
            if (!p) continue;
            const uint32_t c = (__ldg(p) >> (f.b * slot)) & f.mask;
            ob[unit_pos(j)] = (uint8_t)code_to_e4m3(c, f);
        }
    }
    return make_uint4(o[0], o[1], o[2], o[3]);
}

// ------------------------------------------------------------ epilogue

struct EpiParams {
    const float* scale;
    const float* alpha_a_dev;
    const float* alpha_b_dev;
    float dq_pow2;            // 2^-(kA+kB)
    const float* bias;
    float scale0, bias0;
    int act;
    const uint32_t* residual;
    int64_t res_ld;
    int res_b, res_k;
    float res_scale;
    float alpha_out;
    const float* alpha_out_dev;
    ProjParams out;
    int out_cpw;
    int32_t* acc_out;
    float* y_out;
    uint32_t* codes_out;
    int64_t ldo;
    int* status;
};

__device__ __forceinline__ float apply_act(float y, int act)
{
    if (act == ESB_ACT_RELU) {
        y = (y > 0.0f) ? y : 0.0f;
    } else if (act == ESB_ACT_RELU6) {
        y = (y > 0.0f) ? y : 0.0f;
        y = (y < 6.0f) ? y : 6.0f;
    }
    return y;
}

// ------------------------------------------------------------ the kernel

template <class SrcA, class SrcB>
__global__ void __launch_bounds__(kGemmThreads, 1)
esb_gemm_tc_kernel(SrcA srcA, SrcB srcB, int64_t M, int64_t N, int64_t K, OpFmt fa, OpFmt fb, int BN,
                   float acc_scale, EpiParams ep)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // 1024-byte aligned base for the swizzled stages.
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int a_bytes = kBM * kBK;
    const int b_bytes = BN * kBK;
    const int stage_bytes = a_bytes + b_bytes;
    uint64_t* mma_bar = reinterpret_cast<uint64_t*>(smem + kStages * stage_bytes);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_bar + kStages);
    volatile int* err_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int64_t m0 = (int64_t)blockIdx.x * kBM;
    const int64_t n0 = (int64_t)blockIdx.y * BN;
    uint32_t tmem_cols = 32;
    while ((int)tmem_cols < BN) tmem_cols <<= 1;

    if (tid == 0) {
        for (int s = 0; s < kStages; s++) mbar_init(&mma_bar[s], 1);
        *err_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(tmem_slot, tmem_cols);
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_d = *tmem_slot;

    const int64_t nkb = (K + kBK - 1) / kBK;
    const uint32_t idesc = idesc_e4m3_f32(BN);

    // Each thread owns fixed rows of the A and B tiles across all K-blocks.
    constexpr int kAUnits = kBM * (kBK / 16) / kGemmThreads;   // 4
    typename SrcA::Row arow[kAUnits];
#pragma unroll
    for (int i = 0; i < kAUnits; i++) arow[i] = srcA.row(m0 + (tid + i * kGemmThreads) / (kBK / 16));

    for (int64_t kb = 0; kb < nkb; kb++) {
        const int s = (int)(kb % kStages);
        if (kb >= kStages && tid == 0) {
            if (!mbar_wait_bounded(&mma_bar[s], (uint32_t)(((kb / kStages) - 1) & 1), kWaitLimitNs)) *err_flag = 1;
        }
        __syncthreads();
        if (*err_flag) break;
        uint8_t* sa = smem + s * stage_bytes;
        uint8_t* sb = sa + a_bytes;
        const int64_t kbase = kb * kBK;
#pragma unroll
        for (int i = 0; i < kAUnits; i++) {
            const int u = tid + i * kGemmThreads;
            const int r = u >> 3, g = u & 7;
            const uint4 v = decode_unit(srcA, arow[i], kbase + g * 16, K, fa);
            *reinterpret_cast<uint4*>(sa + r * 128 + ((g ^ (r & 7)) << 4)) = v;
        }
        for (int u = tid; u < BN * 8; u += kGemmThreads) {
            const int r = u >> 3, g = u & 7;
            const typename SrcB::Row brow = srcB.row(n0 + r);
            const uint4 v = decode_unit(srcB, brow, kbase + g * 16, K, fb);
            *reinterpret_cast<uint4*>(sb + r * 128 + ((g ^ (r & 7)) << 4)) = v;
        }
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == 0) {
            tc_fence_after();
            const uint32_t a0 = smem_u32(sa), b0 = smem_u32(sb);
#pragma unroll
            for (int j = 0; j < kBK / 32; j++) {
                mma_f8f6f4(tmem_d, smem_desc_sw128(a0 + j * 32), smem_desc_sw128(b0 + j * 32), idesc,
                           (kb > 0 || j > 0) ? 1u : 0u);
            }
            mma_commit(&mma_bar[s]);
        }
    }

    if (tid == 0 && !*err_flag && nkb > 0) {
        const int64_t last = nkb - 1;
        if (!mbar_wait_bounded(&mma_bar[last % kStages], (uint32_t)((last / kStages) & 1), kWaitLimitNs)) *err_flag = 1;
    }
    __syncthreads();
    tc_fence_after();
    const bool failed = *err_flag != 0;
    if (failed && tid == 0) record_status(ep.status, ESB_ERR_TIMEOUT);

    if (!failed) {
        // ---------------------------------------------------- epilogue
        const int quarter = warp & 3;              // TMEM lanes 32*quarter .. +31
        const int half = warp >> 2;                // column chunks of this warp
        const int row = quarter * 32 + lane;
        const int64_t m = m0 + row;
        const bool mrow = m < M;
        float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
        const bool dq = ep.alpha_a_dev && ep.alpha_b_dev;
        const float dqs = dq ? __fmul_rn(__ldg(ep.alpha_a_dev), __ldg(ep.alpha_b_dev)) * ep.dq_pow2 : 1.0f;
        uint8_t* stage_codes = smem;               // 128 x BN bytes, stages are free now
        const int rcpw = ep.residual ? 32 / ep.res_b : 1;
        const uint32_t rmask = ep.residual ? (1u << ep.res_b) - 1u : 0u;
        for (int c16 = half; c16 < BN / 16; c16 += 2) {
            uint32_t r[16];
            if (nkb > 0) {
                tmem_ld16(tmem_d + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(c16 * 16), r);
            } else {
#pragma unroll
                for (int j = 0; j < 16; j++) r[j] = 0u;
            }
#pragma unroll
            for (int j = 0; j < 16; j++) {
                const int col = c16 * 16 + j;
                const int64_t n = n0 + col;
                uint32_t code = ep.out.zero_code;
                if (mrow && n < N) {
                    const float af = __uint_as_float(r[j]) * acc_scale;   // exact integer
                    if (ep.acc_out) ep.acc_out[m * N + n] = __float2int_rn(af);
                    float sc = ep.scale ? __ldg(ep.scale + n) : ep.scale0;
                    if (dq) sc = __fmul_rn(sc, dqs);
                    const float bi = ep.bias ? __ldg(ep.bias + n) : ep.bias0;
                    float y = __fmaf_rn(sc, af, bi);
                    if (ep.residual) {
                        const uint32_t rc = (__ldg(ep.residual + m * ep.res_ld + n / rcpw) >> (ep.res_b * (int)(n % rcpw))) & rmask;
                        y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
                    }
                    y = apply_act(y, ep.act);
                    if (ep.y_out) ep.y_out[m * N + n] = y;
                    if (ep.codes_out) code = project_code(y, alpha_out, ep.out);
                }
                if (ep.codes_out) stage_codes[row * BN + col] = (uint8_t)code;
            }
        }
        if (ep.codes_out) {
            __syncthreads();
            const int cpw = ep.out_cpw;
            const int wpr = BN / cpw;
            const int64_t wbase = n0 / cpw;
            for (int idx = tid; idx < kBM * wpr; idx += kGemmThreads) {
                const int rr = idx / wpr, j = idx - rr * wpr;
                const int64_t mm = m0 + rr;
                const int64_t wg = wbase + j;
                if (mm < M && wg < ep.ldo) {
                    uint32_t word = 0;
                    for (int t = 0; t < cpw; t++) word |= (uint32_t)stage_codes[rr * BN + j * cpw + t] << (ep.out.b * t);
                    ep.codes_out[mm * ep.ldo + wg] = word;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem_d, tmem_cols);
    }
}

// ------------------------------------------------------------ host side

static int pick_bn(int64_t N, int out_cpw)
{
    // BN must be a multiple of 16 (MMA N step) and of the output codes per
    // word (so no packed word straddles two tiles).
    static const int cands_small[] = {64, 48, 80, 96, 32, 112, 128, 16};
    static const int cands_big[] = {128, 160, 192, 240, 256, 96, 80, 112, 64, 48, 144, 176, 208, 224};
    if (N <= 64) {
        for (int bn : cands_small)
            if (bn >= N && bn % out_cpw == 0) return bn;
    }
    for (int bn : cands_big)
        if (bn % out_cpw == 0) return bn;
    for (int bn = 16; bn <= 256; bn += 16)
        if (bn % out_cpw == 0) return bn;
    return 0;
}

static size_t gemm_smem_bytes(int BN)
{
    return 1024 + (size_t)kStages * (kBM * kBK + (size_t)BN * kBK) + kStages * 8 + 16;
}

template <class SrcA, class SrcB>
static cudaError_t launch_tc(const SrcA& a, const SrcB& b, int64_t M, int64_t N, int64_t K, const OpFmt& fa,
                             const OpFmt& fb, int BN, const EpiParams& ep, cudaStream_t st)
{
    const size_t smem = gemm_smem_bytes(BN);
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(esb_gemm_tc_kernel<SrcA, SrcB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)gemm_smem_bytes(256));
        if (e != cudaSuccess) return e;
        configured = true;
    }
    const float acc_scale = ldexpf(1.0f, fa.k + fb.k + 12);
    dim3 grid((unsigned)((M + kBM - 1) / kBM), (unsigned)((N + BN - 1) / BN));
    esb_gemm_tc_kernel<SrcA, SrcB><<<grid, kGemmThreads, smem, st>>>(a, b, M, N, K, fa, fb, BN, acc_scale, ep);
    return cudaGetLastError();
}

static EpiParams make_epi(const GemmOutputs& o)
{
    EpiParams ep;
    const esb_epilogue* e = o.ep;
    ep.scale = e ? e->scale : nullptr;
    ep.alpha_a_dev = e ? e->alpha_a_dev : nullptr;
    ep.alpha_b_dev = e ? e->alpha_b_dev : nullptr;
    ep.dq_pow2 = 1.0f;
    ep.bias = e ? e->bias : nullptr;
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
    const int ob = (e && o.codes_out) ? e->fmt_out.b : 4;
    const int ok = (e && o.codes_out) ? e->fmt_out.k : 2;
    ep.out = make_proj_params(ob, ok, (e && o.codes_out) ? e->fmt_out.is_signed : 1,
                              (e && o.codes_out) ? e->rounding_out : 0);
    ep.out_cpw = 32 / ob;
    ep.acc_out = o.acc_out;
    ep.y_out = o.y_out;
    ep.codes_out = o.codes_out;
    ep.ldo = o.ldo;
    ep.status = device_status_ptr();
    return ep;
}

cudaError_t launch_gemm(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, int ba, int ka,
                        const uint32_t* B, int64_t ldb, int bb, int kb, const GemmOutputs& o, cudaStream_t st)
{
    EpiParams ep = make_epi(o);
    ep.dq_pow2 = ldexpf(1.0f, -(ka + kb));
    const int BN = pick_bn(N, ep.out_cpw);
    RowsSrc a{A, lda, M};
    RowsSrc b{B, ldb, N};
    return launch_tc(a, b, M, N, K, make_opfmt(ba, ka), make_opfmt(bb, kb), BN, ep, st);
}

cudaError_t launch_conv_tc(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int bx, int kx,
                           const uint32_t* W, int64_t ldw, int bw, int kw, const GemmOutputs& o, cudaStream_t st)
{
    EpiParams ep = make_epi(o);
    ep.dq_pow2 = ldexpf(1.0f, -(kx + kw));
    const int64_t M = (int64_t)d.n * P * Q;
    const int64_t N = d.cout;
    const int64_t K = (int64_t)d.r * d.s * ldx * (32 / bx);
    const int BN = pick_bn(N, ep.out_cpw);
    ConvSrc a;
    a.X = X; a.ldx = ldx; a.rows = M; a.H = d.h; a.W = d.w; a.P = P; a.Q = Q; a.S = d.s;
    a.stride = d.stride; a.pad = d.pad;
    RowsSrc b{W, (int64_t)d.r * d.s * ldw, N};
    return launch_tc(a, b, M, N, K, make_opfmt(bx, kx), make_opfmt(bw, kw), BN, ep, st);
}

bool gemm_pick_ok(int64_t N, int out_b) { return pick_bn(N, 32 / out_b) != 0; }

}  // namespace esb
