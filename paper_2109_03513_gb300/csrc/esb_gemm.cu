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
// Two kernels share the decode and the epilogue:
//  * esb_gemm_ws_kernel (B resident): persistent, warp-specialised.  The
//    CTA decodes its N-tile of B once into shared memory; 8 producer warps
//    decode A tiles into an 8-deep ring of shared-memory stages; one MMA
//    warp issues tcgen05.mma (M = 128, N = BN, K = 32) into one of two TMEM
//    accumulators and commits each stage to the mbarrier that frees it;
//    4 epilogue warps drain the other accumulator with tcgen05.ld, so the
//    post-processing of tile i overlaps the MMAs of tile i+1 and the decode
//    of later tiles (the paper's ping-pong buffers and overlapped timing
//    graph, Sec. IV-C/IV-D).
//  * esb_gemm_tc_kernel (B streamed): one 128 x BN tile per CTA; all warps
//    decode A and B K-blocks into a ring of stages, one thread issues the
//    MMAs.  Used when B does not fit in shared memory.
// Every mbarrier wait is bounded (kWaitLimitNs); on expiry the kernel records
// ESB_ERR_TIMEOUT, stops issuing work, frees TMEM and returns.
#include <cstdint>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

constexpr int kBM = 128;           // rows per tile (TMEM lanes)
constexpr int kBK = 128;           // codes (= E4M3 bytes) per K-block: one 128-byte swizzle row
constexpr int kStages = 4;         // streamed kernel
constexpr int kGemmThreads = 256;  // streamed kernel
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
    struct Cursor { int64_t w; };
    __device__ __forceinline__ Row row(int64_t r) const { Row x; x.p = (r < rows) ? base + r * ld : nullptr; return x; }
    __device__ __forceinline__ const uint32_t* words(const Row& x, int64_t w) const { return x.p ? x.p + w : nullptr; }
    __device__ __forceinline__ Cursor cursor(int64_t w) const { Cursor c; c.w = w; return c; }
    __device__ __forceinline__ void advance(Cursor& c, int dw) const { c.w += dw; }
    __device__ __forceinline__ const uint32_t* at(const Row& x, const Cursor& c) const { return x.p ? x.p + c.w : nullptr; }
};

// Implicit im2col of NHWC codes: row m = (n, p, q) output pixel; logical
// word w = tap * ldx + word, tap = (r, s); out-of-image taps read as zero.
// All index arithmetic is 32-bit except the final pixel offset.
struct ConvSrc {
    const uint32_t* X;
    int ldx;
    int rows;                     // n * P * Q
    int H, W, P, Q, S, stride, pad;
    struct Row { int pix0; int h0, w0; bool valid; };
    struct Cursor { int r, s, word; };
    __device__ __forceinline__ Row row(int64_t m64) const
    {
        Row x;
        const int m = (int)m64;
        x.valid = m64 < rows;
        const int pq = P * Q;
        const int n = x.valid ? m / pq : 0;
        const int rem = x.valid ? m - n * pq : 0;
        const int p = rem / Q, q = rem - (rem / Q) * Q;
        x.h0 = p * stride - pad;
        x.w0 = q * stride - pad;
        x.pix0 = n * H;
        return x;
    }
    __device__ __forceinline__ const uint32_t* tap_ptr(const Row& x, int r, int s, int word) const
    {
        const int h = x.h0 + r, ww = x.w0 + s;
        if (!x.valid || h < 0 || h >= H || ww < 0 || ww >= W) return nullptr;
        return X + ((int64_t)(x.pix0 + h) * W + ww) * ldx + word;
    }
    __device__ __forceinline__ const uint32_t* words(const Row& x, int64_t w) const
    {
        const int tap = (int)(w / ldx);
        const int word = (int)(w - (int64_t)tap * ldx);
        return tap_ptr(x, tap / S, tap - (tap / S) * S, word);
    }
    __device__ __forceinline__ Cursor cursor(int64_t w) const
    {
        Cursor c;
        const int tap = (int)(w / ldx);
        c.word = (int)(w - (int64_t)tap * ldx);
        c.r = tap / S;
        c.s = tap - c.r * S;
        return c;
    }
    __device__ __forceinline__ void advance(Cursor& c, int dw) const
    {
        c.word += dw;
        while (c.word >= ldx) {
            c.word -= ldx;
            if (++c.s == S) { c.s = 0; ++c.r; }
        }
    }
    __device__ __forceinline__ const uint32_t* at(const Row& x, const Cursor& c) const { return tap_ptr(x, c.r, c.s, c.word); }
};

// General decode of the 16-code unit [k0, k0 + 16) of one row (any b, K tail).
template <class Src>
__device__ __noinline__ uint4 decode_unit_any(const Src& src, const typename Src::Row& row, int64_t k0, int64_t K,
                                              const OpFmt f)
{
    uint32_t o0 = 0u, o1 = 0u, o2 = 0u, o3 = 0u;
#pragma unroll 1
    for (int j = 0; j < 16; j++) {
        const int64_t kk = k0 + j;
        if (kk >= K) break;
        const int64_t wi = kk / f.cpw;
        const int slot = (int)(kk - wi * f.cpw);
        const uint32_t* p = src.words(row, wi);
        if (!p) continue;
        const uint32_t c = (__ldg(p) >> (f.b * slot)) & f.mask;
        const uint32_t byte = code_to_e4m3(c, f);
        const int pos = unit_pos(j);
        const uint32_t v = byte << (8 * (pos & 3));
        switch (pos >> 2) {
        case 0: o0 |= v; break;
        case 1: o1 |= v; break;
        case 2: o2 |= v; break;
        default: o3 |= v; break;
        }
    }
    return make_uint4(o0, o1, o2, o3);
}

// Fast decode of a full b = 4 unit (two words) at a cursor.
template <class Src>
__device__ __forceinline__ uint4 decode_unit_b4(const Src& src, const typename Src::Row& row,
                                                const typename Src::Cursor& c, const OpFmt& f)
{
    uint32_t o[4] = {0u, 0u, 0u, 0u};
    const uint32_t* p = src.at(row, c);
    if (p) {
        const uint2 w = __ldg(reinterpret_cast<const uint2*>(p));
        decode_word_b4(w.x, f.k, f.ew, o[0], o[1]);
        decode_word_b4(w.y, f.k, f.ew, o[2], o[3]);
    }
    return make_uint4(o[0], o[1], o[2], o[3]);
}

// Decode the 16-code unit [k0, k0 + 16) of one row into 16 bytes.
template <class Src>
__device__ __forceinline__ uint4 decode_unit(const Src& src, const typename Src::Row& row, int64_t k0, int64_t K,
                                             const OpFmt& f)
{
    if (f.b == 4 && k0 + 16 <= K) return decode_unit_b4(src, row, src.cursor(k0 >> 3), f);
    return decode_unit_any(src, row, k0, K, f);
}

__device__ __forceinline__ uint32_t swz(int r, int g) { return (uint32_t)(r * 128 + ((g ^ (r & 7)) << 4)); }

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

// Per-kernel constants of the epilogue.
struct EpiCtx {
    bool dq;
    float dqs;
    const float* T;     // requantisation thresholds (shared memory)
    Thr7 t7;
    bool b4;
};

__device__ __forceinline__ EpiCtx make_epi_ctx(const EpiParams& ep, const float* T)
{
    EpiCtx c;
    c.dq = ep.alpha_a_dev && ep.alpha_b_dev;
    c.dqs = c.dq ? __fmul_rn(__ldg(ep.alpha_a_dev), __ldg(ep.alpha_b_dev)) * ep.dq_pow2 : 1.0f;
    c.T = T;
    c.b4 = ep.out.b == 4;
#pragma unroll
    for (int i = 0; i < 7; i++) c.t7.t[i] = (ep.codes_out && c.b4) ? T[i] : 0.0f;
    return c;
}

// One output element: affine, residual, activation, optional stores, code.
__device__ __forceinline__ uint32_t epi_element(const EpiParams& ep, const EpiCtx& cx, float af, int64_t m, int64_t n,
                                                int64_t N)
{
    if (ep.acc_out) ep.acc_out[m * N + n] = __float2int_rn(af);
    float sc = ep.scale ? __ldg(ep.scale + n) : ep.scale0;
    if (cx.dq) sc = __fmul_rn(sc, cx.dqs);
    const float bi = ep.bias ? __ldg(ep.bias + n) : ep.bias0;
    float y = __fmaf_rn(sc, af, bi);
    if (ep.residual) {
        const int rcpw = 32 / ep.res_b;
        const uint32_t rc = (__ldg(ep.residual + m * ep.res_ld + n / rcpw) >> (ep.res_b * (int)(n % rcpw))) &
                            ((1u << ep.res_b) - 1u);
        y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
    }
    y = apply_act(y, ep.act);
    if (ep.y_out) ep.y_out[m * N + n] = y;
    if (!ep.codes_out) return 0u;
    return cx.b4 ? project_by_thr7(y, cx.t7, ep.out) : project_by_table(y, cx.T, ep.out);
}

// Wait on an mbarrier phase with a wall-clock bound and an abort flag
// raised by another role of the CTA.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* err)
{
    const uint32_t a = smem_u32(bar);
    if (mbar_try_wait(a, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(a, parity)) return true;
        if ((it & 255u) == 0u) {
            if (*err) return false;
            if (globaltimer_ns() - t0 > kWaitLimitNs) return false;
        }
    }
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// ------------------------------------------------- streamed-B kernel

template <class SrcA, class SrcB>
__global__ void __launch_bounds__(kGemmThreads, 1)
esb_gemm_tc_kernel(SrcA srcA, SrcB srcB, int64_t M, int64_t N, int64_t K, OpFmt fa, OpFmt fb, int BN,
                   float acc_scale, EpiParams ep)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int a_bytes = kBM * kBK;
    const int b_bytes = BN * kBK;
    const int stage_bytes = a_bytes + b_bytes;
    uint64_t* mma_bar = reinterpret_cast<uint64_t*>(smem + kStages * stage_bytes);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_bar + kStages);
    volatile int* err_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    float* thr = reinterpret_cast<float*>(tmem_slot + 4);

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
    if (ep.codes_out) {
        const float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
        build_thresholds(thr, ep.out, alpha_out, warp, lane, 0, kGemmThreads / 32);
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_d = *tmem_slot;

    const int64_t nkb = (K + kBK - 1) / kBK;
    const uint32_t idesc = idesc_e4m3_f32(BN);

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
            *reinterpret_cast<uint4*>(sa + swz(r, g)) = decode_unit(srcA, arow[i], kbase + g * 16, K, fa);
        }
        for (int u = tid; u < BN * 8; u += kGemmThreads) {
            const int r = u >> 3, g = u & 7;
            *reinterpret_cast<uint4*>(sb + swz(r, g)) = decode_unit(srcB, srcB.row(n0 + r), kbase + g * 16, K, fb);
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
        const int quarter = warp & 3;              // TMEM lanes 32*quarter .. +31
        const int half = warp >> 2;                // column chunks of this warp
        const int row = quarter * 32 + lane;
        const int64_t m = m0 + row;
        const bool mrow = m < M;
        const EpiCtx cx = make_epi_ctx(ep, thr);
        uint8_t* stage_codes = smem;               // 128 x BN bytes, stages are free now
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
                if (mrow && n < N) code = epi_element(ep, cx, __uint_as_float(r[j]) * acc_scale, m, n, N);
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

// ----------------------------------------- resident-B persistent kernel

constexpr int kWsEpiWarps = 8;                 // warps 0-7: epilogue (lanes 32*(w&3).., column half w>>2)
constexpr int kWsMmaWarp = 8;                  // warp 8: TMEM allocation and MMA issue
constexpr int kWsProdWarp0 = 9;                // warps 9-15: A producers, one stage at a time each
constexpr int kWsProdWarps = 7;
constexpr int kWsThreads = (kWsProdWarp0 + kWsProdWarps) * 32;   // 512: 4 warps per SM sub-partition
constexpr int kWsMaxStages = 8;

struct WsLayout {
    int nkb;          // K-blocks
    int BN;
    int stages;
    int b_bytes;      // resident B: nkb * BN * 128
    int smem_bytes;   // total dynamic shared memory incl. alignment slack
};

__host__ inline WsLayout ws_layout(int64_t K, int BN, int max_smem)
{
    WsLayout L;
    L.nkb = (int)((K + kBK - 1) / kBK);
    L.BN = BN;
    L.b_bytes = L.nkb * BN * kBK;
    const int fixed = 1024 + L.b_bytes + 4 * 128 + 512;      // slack, B, thresholds, barriers
    int st = (max_smem - fixed) / (kBM * kBK);
    if (st > kWsMaxStages) st = kWsMaxStages;
    L.stages = st;
    L.smem_bytes = fixed + st * kBM * kBK;
    return L;
}

// Byte masks of the decoded lo/hi words of one b = 4 word when only its
// first v codes (0..8) are inside K.
__device__ __forceinline__ void tail_masks(int v, uint32_t& mlo, uint32_t& mhi)
{
    const int nlo = (v + 1) >> 1, nhi = v >> 1;       // lo holds codes 0,2,4,6; hi 1,3,5,7
    mlo = nlo >= 4 ? 0xffffffffu : ((1u << (8 * nlo)) - 1u);
    mhi = nhi >= 4 ? 0xffffffffu : ((1u << (8 * nhi)) - 1u);
}

// Decode one 128-code K-block slice (16 words, four 16-byte pieces) of a
// b = 4 row and store its 8 units to a swizzled stage row.  The loads of
// all four pieces are issued before any decode.
// Pieces outside the operand (rows past M or N, out-of-image taps, words
// past K) are filled with the zero code -- the all-zero bit pattern is not
// zero in this format (it is the value 1).
template <class Src>
__device__ __forceinline__ void load_row_b4(const Src& src, const typename Src::Row& row,
                                            const typename Src::Cursor (&cur)[4], int64_t kw0, int64_t K,
                                            uint32_t zero_word, uint4 (&v)[4])
{
#pragma unroll
    for (int pc = 0; pc < 4; pc++) {
        const int64_t kk0 = (kw0 + 4 * pc) * 8;       // first code of the piece
        const uint32_t* p = (kk0 < K) ? src.at(row, cur[pc]) : nullptr;
        v[pc] = p ? __ldg(reinterpret_cast<const uint4*>(p)) : make_uint4(zero_word, zero_word, zero_word, zero_word);
    }
}

__device__ __forceinline__ void store_row_b4(uint8_t* stage, int r, const uint4 (&v)[4], int64_t kw0, int64_t K,
                                             const OpFmt& f)
{
    const bool tail = (kw0 + 16) * 8 > K;             // only the last K-block can reach past K
#pragma unroll
    for (int pc = 0; pc < 4; pc++) {
        const uint32_t w[4] = {v[pc].x, v[pc].y, v[pc].z, v[pc].w};
#pragma unroll
        for (int h = 0; h < 2; h++) {
            uint32_t o0, o1, o2, o3;
            decode_word_b4(w[2 * h], f.k, f.ew, o0, o1);
            decode_word_b4(w[2 * h + 1], f.k, f.ew, o2, o3);
            const int64_t wi = kw0 + 4 * pc + 2 * h;  // word index of w[2h]
            if (tail && (wi + 2) * 8 > K) {           // K tail: zero the codes past K
                uint32_t ml, mh;
                int va = (int)(K - wi * 8);
                va = va < 0 ? 0 : (va > 8 ? 8 : va);
                tail_masks(va, ml, mh);
                o0 &= ml; o1 &= mh;
                int vb = (int)(K - (wi + 1) * 8);
                vb = vb < 0 ? 0 : (vb > 8 ? 8 : vb);
                tail_masks(vb, ml, mh);
                o2 &= ml; o3 &= mh;
            }
            *reinterpret_cast<uint4*>(stage + swz(r, 2 * pc + h)) = make_uint4(o0, o1, o2, o3);
        }
    }
}

// Stage fill for formats other than b = 4 (general decode, out of line to
// keep the hot b = 4 loop small; takes scalars only, so no register array of
// the caller has to live in memory).
template <class Src>
__device__ __noinline__ void fill_stage_any(const Src src, int64_t m0, uint8_t* st, int lane, int64_t k0, int64_t K,
                                            const OpFmt f)
{
#pragma unroll 1
    for (int q = 0; q < 4; q++) {
        const typename Src::Row row = src.row(m0 + lane + 32 * q);
#pragma unroll 1
        for (int g = 0; g < 8; g++)
            *reinterpret_cast<uint4*>(st + swz(lane + 32 * q, g)) = decode_unit_any(src, row, k0 + g * 16, K, f);
    }
}

// Epilogue of one 16-column chunk for outputs other than the lean 4-bit
// path (general packing), out of line; reads its own TMEM chunk.
__device__ __noinline__ void epi_chunk_any(const EpiParams* __restrict__ sep, const EpiCtx* __restrict__ scx,
                                           uint32_t taddr, float acc_scale, int64_t m, bool mrow, int64_t n_first,
                                           int64_t N, uint32_t* word_slot_w)
{
    const EpiParams& ep = *sep;
    const EpiCtx cx = *scx;
    uint32_t r[16];
    tmem_ld16(taddr, r);
    const int cpw = ep.out_cpw;
    uint32_t word = word_slot_w[0];
    int slot = (int)word_slot_w[1];
    int64_t wcol = (int64_t)word_slot_w[2] | ((int64_t)word_slot_w[3] << 32);
#pragma unroll
    for (int j = 0; j < 16; j++) {
        const int64_t n = n_first + j;
        uint32_t code = ep.out.zero_code;
        if (mrow && n < N) code = epi_element(ep, cx, __uint_as_float(r[j]) * acc_scale, m, n, N);
        word |= code << (ep.out.b * slot);
        if (++slot == cpw) {
            if (ep.codes_out && mrow && wcol < ep.ldo) ep.codes_out[m * ep.ldo + wcol] = word;
            word = 0;
            slot = 0;
            wcol++;
        }
    }
    word_slot_w[0] = word;
    word_slot_w[1] = (uint32_t)slot;
    word_slot_w[2] = (uint32_t)(wcol & 0xffffffff);
    word_slot_w[3] = (uint32_t)(wcol >> 32);
}

template <class SrcA>
__global__ void __launch_bounds__(kWsThreads, 1)
esb_gemm_ws_kernel(SrcA srcA, RowsSrc srcB, int64_t M, int64_t N, int64_t K, OpFmt fa, OpFmt fb, int BN, int nkb,
                   int stages, int n_tiles, int64_t m_tiles, float acc_scale, EpiParams ep)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sB = smem;                                        // nkb blocks of BN x 128 bytes
    uint8_t* sA = sB + nkb * BN * kBK;                         // stages x 16 KiB
    float* thr = reinterpret_cast<float*>(sA + stages * kBM * kBK);
    uint64_t* full = reinterpret_cast<uint64_t*>(thr + 128);
    uint64_t* empty = full + kWsMaxStages;
    uint64_t* tfull = empty + kWsMaxStages;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* err = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int n_tile = (int)(blockIdx.x % n_tiles);
    const int64_t cta_in_n = blockIdx.x / n_tiles;
    const int64_t ctas_per_n = gridDim.x / n_tiles;
    const int64_t n0 = (int64_t)n_tile * BN;
    const int64_t my_tiles = (m_tiles > cta_in_n) ? (m_tiles - cta_in_n + ctas_per_n - 1) / ctas_per_n : 0;
    uint32_t tmem_cols = 32;
    while ((int)tmem_cols < 2 * BN) tmem_cols <<= 1;
    // Epilogue column split: both halves of BN must be whole 16-column chunks
    // and whole output words; otherwise warps 0-3 take every column.
    const int half_cols = BN / 2;
    const bool split = (half_cols % 16 == 0) && (half_cols % ep.out_cpw == 0);
    const int epi_warps = split ? 8 : 4;

    if (tid == 0) {
        for (int s = 0; s < stages; s++) {
            mbar_init(&full[s], 1);                   // the producer warp that filled the stage
            mbar_init(&empty[s], 1);                  // the MMA commit that drained it
        }
        for (int a = 0; a < 2; a++) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], epi_warps);
        }
        mbar_init(drain, 1);
        *err = 0;
        fence_mbar_init();
    }
    __syncthreads();                                  // barriers initialised

    // Producers start loading A at once; meanwhile the MMA and epilogue
    // warps decode the resident B, allocate TMEM and build the
    // requantisation thresholds, then meet on named barrier 1.
    constexpr int kSetupThreads = kWsProdWarp0 * 32;  // warps 0..8
    uint32_t tmem_base = 0;
    if (warp < kWsProdWarp0) {
        if (warp == kWsMmaWarp) {
            tmem_alloc(tmem_slot, tmem_cols);
            tc_fence_before();
        }
        // Resident B: this CTA's N-tile, every K-block, decoded once.
        if (fb.b == 4) {
            for (int pr = tid; pr < nkb * BN; pr += kSetupThreads) {
                const int kb = pr / BN, r = pr - kb * BN;
                const RowsSrc::Row row = srcB.row(n0 + r);
                const int64_t kw0 = (int64_t)kb * 16;
                RowsSrc::Cursor cur[4];
#pragma unroll
                for (int pc = 0; pc < 4; pc++) cur[pc] = srcB.cursor(kw0 + 4 * pc);
                uint4 v[4];
                load_row_b4(srcB, row, cur, kw0, K, fmt_zero_code(4, fb.k) * 0x11111111u, v);
                store_row_b4(sB + kb * BN * kBK, r, v, kw0, K, fb);
            }
        } else {
            for (int u = tid; u < nkb * BN * 8; u += kSetupThreads) {
                const int kb = u / (BN * 8);
                const int rem = u - kb * BN * 8;
                const int r = rem >> 3, g = rem & 7;
                *reinterpret_cast<uint4*>(sB + kb * BN * kBK + swz(r, g)) =
                    decode_unit_any(srcB, srcB.row(n0 + r), (int64_t)kb * kBK + g * 16, K, fb);
            }
        }
        fence_proxy_async_smem();
        if (ep.codes_out) {
            const float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
            build_thresholds(thr, ep.out, alpha_out, warp, lane, 0, kWsProdWarp0);
        }
        asm volatile("bar.sync 1, %0;" ::"n"(kSetupThreads) : "memory");
        tc_fence_after();
        tmem_base = *tmem_slot;
    }

    if (warp >= kWsProdWarp0) {
        // ---------------------------------------------- A producers
        // Warp p fills the stages of iterations p, p + 7, ... of this CTA's
        // (tile, K-block) sequence, so up to 7 K-blocks are loading at once.
        // Lane l owns rows l, l + 32, l + 64, l + 96 of the tile.
        // At most `stages` producers are active: a producer then never waits
        // on a stage more than one phase ahead of the MMA's progress, which
        // is all the parity of an mbarrier can tell apart.
        const int p = warp - kWsProdWarp0;
        const int nprod = stages < kWsProdWarps ? stages : kWsProdWarps;
        const int64_t total_it = (p < nprod) ? my_tiles * nkb : 0;
        const uint32_t zwa = fmt_zero_code(4, fa.k) * 0x11111111u;
        int64_t cur_tile = -1;
        typename SrcA::Row rows[4];
        for (int64_t it = p; it < total_it && !*err; it += nprod) {
            const int64_t ti = it / nkb;
            const int kb = (int)(it - ti * nkb);
            if (ti != cur_tile) {
                cur_tile = ti;
                const int64_t m0 = (cta_in_n + ti * ctas_per_n) * kBM;
#pragma unroll
                for (int q = 0; q < 4; q++) rows[q] = srcA.row(m0 + lane + 32 * q);
            }
            const int s = (int)(it % stages);
            const uint32_t ph = (uint32_t)((it / stages) & 1);
            if (!wait_or_abort(&empty[s], ph ^ 1u, err)) { *err = 1; break; }
            uint8_t* st = sA + s * kBM * kBK;
            if (fa.b == 4) {
                const int64_t kw0 = (int64_t)kb * 16;
                typename SrcA::Cursor cur[4];
#pragma unroll
                for (int pc = 0; pc < 4; pc++) cur[pc] = srcA.cursor(kw0 + 4 * pc);
                uint4 v[4][4];
#pragma unroll
                for (int q = 0; q < 4; q++) load_row_b4(srcA, rows[q], cur, kw0, K, zwa, v[q]);
#pragma unroll
                for (int q = 0; q < 4; q++) store_row_b4(st, lane + 32 * q, v[q], kw0, K, fa);
            } else {
                fill_stage_any(srcA, (cta_in_n + ti * ctas_per_n) * kBM, st, lane, (int64_t)kb * kBK, K, fa);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&full[s]);
        }
    } else if (warp == kWsMmaWarp) {
        // ---------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = idesc_e4m3_f32(BN);
            const uint32_t b_base = smem_u32(sB), a_base = smem_u32(sA);
            int64_t it = 0;
            for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
                const int a = (int)(ti & 1);
                if (!wait_or_abort(&tempty[a], (uint32_t)((ti >> 1) & 1) ^ 1u, err)) { *err = 1; break; }
                tc_fence_after();
                const uint32_t d = tmem_base + (uint32_t)(a * BN);
                for (int kb = 0; kb < nkb; kb++, it++) {
                    const int s = (int)(it % stages);
                    if (!wait_or_abort(&full[s], (uint32_t)((it / stages) & 1), err)) { *err = 1; break; }
                    tc_fence_after();
                    const uint32_t a0 = a_base + (uint32_t)(s * kBM * kBK);
                    const uint32_t b0 = b_base + (uint32_t)(kb * BN * kBK);
#pragma unroll
                    for (int j = 0; j < kBK / 32; j++)
                        mma_f8f6f4(d, smem_desc_sw128(a0 + j * 32), smem_desc_sw128(b0 + j * 32), idesc,
                                   (kb > 0 || j > 0) ? 1u : 0u);
                    mma_commit(&empty[s]);
                }
                if (*err) break;
                mma_commit(&tfull[a]);
            }
            // Every MMA this thread issued has completed before TMEM is freed
            // (also on the abort path).
            mma_commit(drain);
            volatile int no_abort = 0;
            if (!wait_or_abort(drain, 0u, &no_abort)) *err = 1;
        }
    } else if (warp < epi_warps) {
        // ---------------------------------------------- epilogue
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;          // TMEM lane = tile row
        __shared__ EpiParams sh_ep;                   // copies for the out-of-line general path
        __shared__ EpiCtx sh_cx;
        const int c_lo = split ? (warp >> 2) * half_cols : 0;
        const int c_hi = split ? c_lo + half_cols : BN;
        const EpiCtx cx = make_epi_ctx(ep, thr);
        if (warp == 0 && lane == 0) { sh_ep = ep; sh_cx = cx; }
        asm volatile("bar.sync 2, %0;" ::"r"(epi_warps * 32) : "memory");   // exactly the epilogue warps in use
        const int cpw = ep.out_cpw;
        const bool swar = ep.codes_out && ep.out.b == 4;
        const float T0 = cx.t7.t[0], T1 = cx.t7.t[1], T2 = cx.t7.t[2], T3 = cx.t7.t[3], T4 = cx.t7.t[4],
                    T5 = cx.t7.t[5], T6 = cx.t7.t[6];
        const float sc_fixed = ep.scale ? 0.0f : (cx.dq ? __fmul_rn(ep.scale0, cx.dqs) : ep.scale0);
        const float sc_lean = sc_fixed * acc_scale;
        const bool out_signed = ep.out.is_signed != 0;
        // the lean path needs every column of the chunk inside N and a finite folded scale
        const bool lean_ok = swar && !ep.scale && !ep.bias && !ep.residual && !ep.acc_out && !ep.y_out &&
                             isfinite(sc_lean) && (sc_lean != 0.0f || sc_fixed == 0.0f);
        for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
            const int a = (int)(ti & 1);
            if (!wait_or_abort(&tfull[a], (uint32_t)((ti >> 1) & 1), err)) { *err = 1; break; }
            tc_fence_after();
            const int64_t m = (cta_in_n + ti * ctas_per_n) * kBM + row;
            const bool mrow = m < M;
            const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(a * BN);
            uint32_t wsw[4] = {0u, 0u, (uint32_t)(((n0 + c_lo) / cpw) & 0xffffffff),
                               (uint32_t)(((n0 + c_lo) / cpw) >> 32)};   // general path: word, slot, column
            for (int c = c_lo; c < c_hi; c += 16) {
                if (!swar) {
                    epi_chunk_any(&sh_ep, &sh_cx, taddr + (uint32_t)c, acc_scale, m, mrow, n0 + c, N, wsw);
                    if (c + 16 >= c_hi) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&tempty[a]);
                    }
                    continue;
                }
                uint32_t r[16];
                tmem_ld16(taddr + (uint32_t)c, r);
                const bool lean = lean_ok && (n0 + c + 16 <= N);
                if (c + 16 >= c_hi) {                 // every column of this warp is in registers
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&tempty[a]);
                }
                if (lean) {
                    // 4-bit output codes only, scalar scale/bias, no residual:
                    // y = fma(scale * 2^(kA+kB+12), raw, bias) equals
                    // fma(scale, acc, bias) exactly (power-of-two scaling),
                    // then the bucket of y among the 7 thresholds, eight codes
                    // per word at once.
                    uint32_t wds[2];
#pragma unroll
                    for (int h = 0; h < 2; h++) {
                        uint32_t J = 0u, S = 0u;
#pragma unroll
                        for (int j = 0; j < 8; j++) {
                            float y = __fmaf_rn(sc_lean, __uint_as_float(r[8 * h + j]), ep.bias0);
                            y = apply_act(y, ep.act);
                            const float a = out_signed ? fabsf(y) : y;
                            const bool b2 = a >= T3;
                            const bool b1 = a >= (b2 ? T5 : T1);
                            const bool b0 = a >= (b2 ? (b1 ? T6 : T4) : (b1 ? T2 : T0));
                            J |= ((b2 ? 4u : 0u) | (b1 ? 2u : 0u) | (b0 ? 1u : 0u)) << (4 * j);
                            if (out_signed) S |= (__float_as_uint(y) >> 31) << (4 * j + 3);
                        }
                        wds[h] = codes8_b4(J, S, ep.out.k);
                    }
                    const int64_t w0 = (n0 + c) >> 3;
                    if (mrow) {
                        if (w0 + 1 < ep.ldo) {
                            *reinterpret_cast<uint2*>(ep.codes_out + m * ep.ldo + w0) = make_uint2(wds[0], wds[1]);
                        } else if (w0 < ep.ldo) {
                            ep.codes_out[m * ep.ldo + w0] = wds[0];
                        }
                    }
                } else if (swar) {
                    // 4-bit output codes with per-channel parameters, residual or extra outputs
                    uint32_t wds[2];
#pragma unroll
                    for (int h = 0; h < 2; h++) {
                        uint32_t J = 0u, S = 0u;
#pragma unroll 1
                        for (int j = 0; j < 8; j++) {
                            const int64_t n = n0 + c + 8 * h + j;
                            const float af = __uint_as_float(r[8 * h + j]) * acc_scale;
                            if (mrow && n < N) {
                                if (ep.acc_out) ep.acc_out[m * N + n] = __float2int_rn(af);
                                float sc = sc_fixed;
                                if (ep.scale) { sc = __ldg(ep.scale + n); if (cx.dq) sc = __fmul_rn(sc, cx.dqs); }
                                const float bi = ep.bias ? __ldg(ep.bias + n) : ep.bias0;
                                float y = __fmaf_rn(sc, af, bi);
                                if (ep.residual) {
                                    const int rcpw = 32 / ep.res_b;
                                    const uint32_t rc = (__ldg(ep.residual + m * ep.res_ld + n / rcpw) >>
                                                         (ep.res_b * (int)(n % rcpw))) & ((1u << ep.res_b) - 1u);
                                    y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
                                }
                                y = apply_act(y, ep.act);
                                if (ep.y_out) ep.y_out[m * N + n] = y;
                                const uint32_t u = __float_as_uint(y);
                                J |= bucket7(ep.out.is_signed ? fabsf(y) : y, cx.t7) << (4 * j);
                                S |= ((u >> 31) & (uint32_t)ep.out.is_signed) << (4 * j + 3);
                            }
                        }
                        wds[h] = codes8_b4(J, S, ep.out.k);
                    }
                    const int64_t w0 = (n0 + c) >> 3;
                    if (mrow) {
                        if (w0 + 1 < ep.ldo) {
                            *reinterpret_cast<uint2*>(ep.codes_out + m * ep.ldo + w0) = make_uint2(wds[0], wds[1]);
                        } else if (w0 < ep.ldo) {
                            ep.codes_out[m * ep.ldo + w0] = wds[0];
                        }
                    }
                }
            }
        }
    }

    __syncthreads();
    if (*err && tid == 0) record_status(ep.status, ESB_ERR_TIMEOUT);
    if (warp == kWsMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, tmem_cols);
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
    return 1024 + (size_t)kStages * (kBM * kBK + (size_t)BN * kBK) + kStages * 8 + 16 + 512;
}

static int max_dyn_smem()
{
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 227 * 1024;
    if (!cache[dev]) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess || v <= 0)
            v = 227 * 1024;
        cache[dev] = v;
    }
    return cache[dev];
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

// Resident-B launch when B's N-tile fits in shared memory with at least
// three A stages; returns false (nothing launched) otherwise.
template <class SrcA>
static bool launch_ws(const SrcA& a, const RowsSrc& b, int64_t M, int64_t N, int64_t K, const OpFmt& fa,
                      const OpFmt& fb, int BN, const EpiParams& ep, cudaStream_t st, cudaError_t* err)
{
    // dynamic shared memory = the opt-in maximum minus the kernel's static shared memory
    static int static_smem = -1;
    if (static_smem < 0) {
        cudaFuncAttributes fa_attr;
        *err = cudaFuncGetAttributes(&fa_attr, esb_gemm_ws_kernel<SrcA>);
        if (*err != cudaSuccess) return true;
        static_smem = (int)fa_attr.sharedSizeBytes;
    }
    const int maxs = max_dyn_smem() - static_smem;
    const WsLayout L = ws_layout(K, BN, maxs);
    if (L.stages < 3) return false;
    static bool configured = false;
    if (!configured) {
        *err = cudaFuncSetAttribute(esb_gemm_ws_kernel<SrcA>, cudaFuncAttributeMaxDynamicSharedMemorySize, maxs);
        if (*err != cudaSuccess) return true;
        configured = true;
    }
    const int n_tiles = (int)((N + BN - 1) / BN);
    const int64_t m_tiles = (M + kBM - 1) / kBM;
    int64_t per_n = device_sm_count() / n_tiles;
    if (per_n < 1) per_n = 1;
    if (per_n > m_tiles) per_n = m_tiles;
    const int64_t grid = per_n * n_tiles;
    const float acc_scale = ldexpf(1.0f, fa.k + fb.k + 12);
    esb_gemm_ws_kernel<SrcA><<<(unsigned)grid, kWsThreads, L.smem_bytes, st>>>(a, b, M, N, K, fa, fb, BN, L.nkb,
                                                                               L.stages, n_tiles, m_tiles, acc_scale,
                                                                               ep);
    *err = cudaGetLastError();
    return true;
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
    const OpFmt fa = make_opfmt(ba, ka), fb = make_opfmt(bb, kb);
    if (K > 0) {
        cudaError_t e = cudaSuccess;
        if (launch_ws(a, b, M, N, K, fa, fb, BN, ep, st, &e)) return e;
    }
    return launch_tc(a, b, M, N, K, fa, fb, BN, ep, st);
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
    a.X = X; a.ldx = (int)ldx; a.rows = (int)M; a.H = d.h; a.W = d.w; a.P = P; a.Q = Q; a.S = d.s;
    a.stride = d.stride; a.pad = d.pad;
    RowsSrc b{W, (int64_t)d.r * d.s * ldw, N};
    const OpFmt fa = make_opfmt(bx, kx), fb = make_opfmt(bw, kw);
    cudaError_t e = cudaSuccess;
    if (K > 0 && launch_ws(a, b, M, N, K, fa, fb, BN, ep, st, &e)) return e;
    return launch_tc(a, b, M, N, K, fa, fb, BN, ep, st);
}

bool gemm_pick_ok(int64_t N, int out_b) { return pick_bn(N, 32 / out_b) != 0; }

}  // namespace esb
