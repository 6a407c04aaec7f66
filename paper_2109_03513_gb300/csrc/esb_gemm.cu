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
// Two kernels here share the decode and the epilogue (esb_tc.cuh) with the
// halo convolution of esb_conv_halo.cu:
//  * esb_gemm_ws_kernel: persistent, warp-specialised.  The CTA decodes
//    its N-tile of B once into shared memory when it fits beside three A
//    stages (B resident), else each stage carries the B block of its
//    K-block too (B streamed); 7 producer warps decode the stages of a ring
//    of up to 8; one MMA warp issues tcgen05.mma (M = 128, N = BN, K = 32)
//    into one of two TMEM accumulators and commits each stage to the
//    mbarrier that frees it; 8 epilogue warps drain the other accumulator
//    with tcgen05.ld, so the post-processing of tile i overlaps the MMAs of
//    tile i+1 and the decode of later tiles (the paper's ping-pong buffers
//    and overlapped timing graph, Sec. IV-C/IV-D).
//  * esb_gemm_tc_kernel (fallback): one 128 x BN tile per CTA; all warps
//    decode A and B K-blocks into a ring of stages, one thread issues the
//    MMAs.
// Every mbarrier wait is bounded (kWaitLimitNs); on expiry the kernel records
// ESB_ERR_TIMEOUT, stops issuing work, frees TMEM and returns.
#include <cstdint>
#include <cstdlib>
#include <cuda_runtime.h>

#include "esb_tc.cuh"

#include <type_traits>

namespace esb {

constexpr int kStages = 4;         // streamed kernel
constexpr int kGemmThreads = 256;  // streamed kernel

// ------------------------------------------------------------ row sources

// Implicit im2col of NHWC codes: row m = (n, p, q) output pixel; logical
// word w = tap * ldx + word, tap = (r, s); out-of-image taps read as zero.
// All index arithmetic is 32-bit except the final pixel offset.
struct ConvSrc {
    const uint32_t* X;
    int ldx;
    int rows;                     // n * P * Q
    int H, W, P, Q, S, stride, pad;
    // Words of each pixel in the logical K (<= ldx): the words that hold
    // channels, so a pixel row's padding words (e.g. the 3 of a first
    // layer's 4-word rows) take no K.  The logical word w is word w % kw of
    // tap w / kw.
    int kw = 0;
    // A row: the word offset of its tap (0, 0) (negative at the top-left
    // border) and the in-image tap ranges r in [rlo, rlo + rn), s in [slo,
    // slo + sn) (rn = 0 for rows past M).  A cursor follows the word offset
    // of its (r, s, word) incrementally, so a step costs a few adds.
    struct Row { int64_t base; int rlo, rn, slo, sn; };
    struct Cursor { int r, s, word; int64_t off; };
    __device__ __forceinline__ Row row(int64_t m64) const
    {
        Row x;
        const int m = (int)m64;
        const bool valid = m64 < rows;
        const int pq = P * Q;
        const int n = valid ? m / pq : 0;
        const int rem = valid ? m - n * pq : 0;
        const int p = rem / Q, q = rem - (rem / Q) * Q;
        const int h0 = p * stride - pad, w0 = q * stride - pad;
        x.base = ((int64_t)(n * H + h0) * W + w0) * ldx;
        x.rlo = h0 < 0 ? -h0 : 0;
        x.slo = w0 < 0 ? -w0 : 0;
        const int rn = H - h0 - x.rlo, sn = W - w0 - x.slo;
        x.rn = (valid && rn > 0) ? rn : 0;
        x.sn = sn > 0 ? sn : 0;
        return x;
    }
    __device__ __forceinline__ bool inside(const Row& x, int r, int s) const
    {
        return (unsigned)(r - x.rlo) < (unsigned)x.rn && (unsigned)(s - x.slo) < (unsigned)x.sn;
    }
    __device__ __forceinline__ const uint32_t* tap_ptr(const Row& x, int r, int s, int word) const
    {
        return inside(x, r, s) ? X + x.base + ((int64_t)r * W + s) * ldx + word : nullptr;
    }
    __device__ __forceinline__ const uint32_t* words(const Row& x, int64_t w) const
    {
        const int tap = (int)(w / kw);
        const int word = (int)(w - (int64_t)tap * kw);
        return tap_ptr(x, tap / S, tap - (tap / S) * S, word);
    }
    __device__ __forceinline__ Cursor cursor(int64_t w) const
    {
        Cursor c;
        const int tap = (int)(w / kw);
        c.word = (int)(w - (int64_t)tap * kw);
        c.r = tap / S;
        c.s = tap - c.r * S;
        c.off = ((int64_t)c.r * W + c.s) * ldx + c.word;
        return c;
    }
    __device__ __forceinline__ void advance(Cursor& c, int dw) const
    {
        c.word += dw;
        c.off += dw;
        while (c.word >= kw) {
            c.word -= kw;
            c.off += ldx - kw;
            if (++c.s == S) {
                c.s = 0;
                ++c.r;
                c.off += (int64_t)(W - S) * ldx;
            }
        }
    }
    // 16-byte pieces (4 logical words) are contiguous in memory
    __host__ __device__ __forceinline__ bool vec4() const { return (kw & 3) == 0; }
    __device__ __forceinline__ const uint32_t* at(const Row& x, const Cursor& c) const
    {
        return inside(x, c.r, c.s) ? X + x.base + c.off : nullptr;
    }
    __host__ __device__ __forceinline__ bool linear() const { return true; }
    __device__ __forceinline__ const uint32_t* code_word(const Row& x, int64_t kk, int cpw, int& slot) const
    {
        const int64_t wi = kk / cpw;
        slot = (int)(kk - wi * cpw);
        return words(x, wi);
    }
};

template <class T>
constexpr bool kIsConv = std::is_same<T, ConvSrc>::value;

// ---------------------------------------- im2col rows through a tap table
//
// The words of one K-block sit at the same taps and offsets in every row of
// the tile, so the producer warp builds a table of them once per stage
// (lane i: word w0 + i -> tap (r, s) and word offset from a row's tap-(0,0)
// base) and each row's loads then need no running cursor: independent
// address adds and loads, all in flight together.
__device__ __forceinline__ void conv_tap_table(const ConvSrc& src, int64_t w0, int n, int4* tab, int lane)
{
    __syncwarp();                                     // the previous stage's readers are done
    if (lane < n) {
        const ConvSrc::Cursor c = src.cursor(w0 + lane);
        tab[lane] = make_int4(c.r, c.s, (int)c.off, 0);
    }
    __syncwarp();
}

// 4-bit codes: the K-block's 16 words of row `row` (rows past M and taps
// outside the image give the E4M3 zero), decoded and stored to stage row r.
__device__ __forceinline__ void walk_b4_tab(const ConvSrc& src, const ConvSrc::Row& row, const int4* tab, int64_t k0,
                                            int64_t K, const OpFmt& f, uint8_t* stage, int r)
{
#pragma unroll 1
    for (int hf = 0; hf < 2; hf++) {                  // two halves of 8 words: a small loop body
        uint32_t wv[8];
        uint32_t ok = 0u;
        const int64_t kh = k0 + hf * 64;
#pragma unroll
        for (int i = 0; i < 8; i++) {
            const int4 e = tab[8 * hf + i];
            const bool in = (kh + i * 8 < K) && src.inside(row, e.x, e.y);
            wv[i] = in ? __ldg(src.X + (row.base + e.z)) : 0u;
            ok |= (in ? 1u : 0u) << i;
        }
        store_b4_words<8>(wv, ok, kh, K, f, stage, r, 4 * hf);
    }
}

// Word-slot codes (see plan_slots): the K-block's NW words, CH at a time.
template <int B>
__device__ __forceinline__ void walk_slots_tab(const ConvSrc& src, const ConvSrc::Row& row, const int4* tab,
                                               int64_t k0, const OpFmt& f, const uint8_t* lut, uint8_t* stage, int r)
{
    constexpr int CPW = 32 / B;
    constexpr int SPW = CPW > 8 ? 16 : (CPW > 4 ? 8 : 4);
    constexpr int NW = kBK / SPW;
    constexpr int CH = 8;                             // words per chunk (a small loop body)
    const int64_t w0 = k0 / SPW;
#pragma unroll 1
    for (int c0 = 0; c0 < NW; c0 += CH) {
        const int64_t left = f.korig - (w0 + c0) * CPW;
        const int lim = left < 0 ? 0 : (left > CH * CPW ? CH * CPW : (int)left);
        uint32_t wv[CH];
        uint32_t ok = 0u;
#pragma unroll
        for (int i = 0; i < CH; i++) {
            const int4 e = tab[c0 + i];
            const bool in = (i * CPW < lim) && src.inside(row, e.x, e.y);
            wv[i] = in ? __ldg(src.X + (row.base + e.z)) : 0u;
            ok |= (in ? 1u : 0u) << i;
        }
        store_slot_words<B, CH>(wv, ok, lim, lut, stage, r, c0 * SPW / 16);
    }
}

__device__ __forceinline__ void walk_row_tab(const ConvSrc& src, const ConvSrc::Row& row, const int4* tab,
                                             int64_t k0, int64_t K, const OpFmt& f, const uint8_t* lut, uint8_t* stage,
                                             int r)
{
    if (f.b == 4) { walk_b4_tab(src, row, tab, k0, K, f, stage, r); return; }
    switch (f.b) {
    case 2: walk_slots_tab<2>(src, row, tab, k0, f, lut, stage, r); return;
    case 3: walk_slots_tab<3>(src, row, tab, k0, f, lut, stage, r); return;
    case 5: walk_slots_tab<5>(src, row, tab, k0, f, lut, stage, r); return;
    case 6: walk_slots_tab<6>(src, row, tab, k0, f, lut, stage, r); return;
    case 7: walk_slots_tab<7>(src, row, tab, k0, f, lut, stage, r); return;
    default: walk_slots_tab<8>(src, row, tab, k0, f, lut, stage, r); return;
    }
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
    if (f.b == 4 && f.planes == 1 && src.linear() && src.vec4() && k0 + 16 <= K)
        return decode_unit_b4(src, row, src.cursor(k0 >> 3), f);
    return decode_unit_any(src, row, k0, K, f);
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
    // word walks (one row per thread) for widths whose 16-code units are not
    // 16-byte pieces: 3/5/6-bit codes, 4-bit rows whose words are not contiguous
    __shared__ uint8_t luta[256], lutb[256];
    const bool walk_a = fa.planes == 1 && srcA.linear() && !(fa.b == 4 && srcA.vec4());
    const bool walk_b = fb.planes == 1 && srcB.linear() && !(fb.b == 4 && srcB.vec4());
    if (walk_a) build_e4m3_lut(luta, fa, tid, kGemmThreads);
    if (walk_b) build_e4m3_lut(lutb, fb, tid, kGemmThreads);
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
        if (walk_a) {
            if (tid < kBM) walk_row_kblock(srcA, srcA.row(m0 + tid), kbase, K, fa, luta, sa, tid);
        } else {
#pragma unroll
            for (int i = 0; i < kAUnits; i++) {
                const int u = tid + i * kGemmThreads;
                const int r = u >> 3, g = u & 7;
                *reinterpret_cast<uint4*>(sa + swz(r, g)) = decode_unit(srcA, arow[i], kbase + g * 16, K, fa);
            }
        }
        if (walk_b) {
            // rows rotated by kBM so that the threads past the A rows start
            for (int r = (tid + kGemmThreads - kBM) % kGemmThreads; r < BN; r += kGemmThreads)
                walk_row_kblock(srcB, srcB.row(n0 + r), kbase, K, fb, lutb, sb, r);
        } else {
            for (int u = tid; u < BN * 8; u += kGemmThreads) {
                const int r = u >> 3, g = u & 7;
                *reinterpret_cast<uint4*>(sb + swz(r, g)) = decode_unit(srcB, srcB.row(n0 + r), kbase + g * 16, K, fb);
            }
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
            if (n0 + BN >= N) {                      // the last N-tile fills the rows' padding words
                uint32_t zw = 0u;
                for (int t = 0; t < cpw; t++) zw |= ep.out.zero_code << (ep.out.b * t);
                const int64_t w_end = (n0 + BN) / cpw;
                for (int rr = tid; rr < kBM; rr += kGemmThreads) {
                    const int64_t mm = m0 + rr;
                    if (mm < M)
                        for (int64_t wq = w_end; wq < ep.ldo; wq++) ep.codes_out[mm * ep.ldo + wq] = zw;
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

struct WsLayout {
    int nkb;          // K-blocks
    int BN;
    int stages;
    int b_bytes;      // resident B: nkb * BN * 128
    int smem_bytes;   // total dynamic shared memory incl. alignment slack
};

// The B-streamed layout: stages of one A block and one B block, no resident B.
__host__ inline WsLayout ws_layout_streamed(int64_t K, int BN, int max_smem)
{
    WsLayout L;
    L.nkb = (int)((K + kBK - 1) / kBK);
    L.BN = BN;
    L.b_bytes = 0;
    const int fixed = 1024 + 4 * 128 + 512;                      // slack, thresholds, barriers
    int st = (max_smem - fixed) / ((kBM + BN) * kBK);
    if (st > kWsMaxStages) st = kWsMaxStages;
    L.stages = st;
    L.smem_bytes = fixed + st * (kBM + BN) * kBK;
    return L;
}

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

template <class SrcA, bool GEN>
__global__ void __launch_bounds__(kWsThreads, 1)
esb_gemm_ws_kernel(SrcA srcA, RowsSrc srcB, int64_t M, int64_t N, int64_t K, OpFmt fa, OpFmt fb, int BN, int nkb,
                   int stages, int n_tiles, int64_t m_tiles, float acc_scale, EpiParams ep, int bstream)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    // B resident: nkb blocks of BN x 128 bytes, then stages of one A block.
    // B streamed (bstream, when B's N-tile does not fit): no resident B;
    // each stage holds the A block and the B block of its K-block.
    const int stage_bytes = kBM * kBK + (bstream ? BN * kBK : 0);
    uint8_t* sB = smem;
    uint8_t* sA = sB + (bstream ? 0 : nkb * BN * kBK);
    float* thr = reinterpret_cast<float*>(sA + stages * stage_bytes);
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
    // E4M3 tables of the word-walk decoder (widths other than 4)
    __shared__ uint8_t luta[256], lutb[256];
    __shared__ int4 ptab[kWsProdWarps][32];          // producers' per-stage tap tables (im2col rows)
    if (fa.planes == 1) build_e4m3_lut(luta, fa, tid, kWsThreads);
    if (fb.planes == 1 && fb.b != 4) build_e4m3_lut(lutb, fb, tid, kWsThreads);
    // Epilogue column split: both halves of BN must be whole 16-column chunks
    // and whole output words; otherwise warps 0-3 take every column.
    const int half_cols = BN / 2;
    const bool split = (half_cols % 16 == 0) && (half_cols % ep.out_cpw == 0);
    const int epi_warps = split ? 8 : 4;
    // the layout above must fit the dynamic allocation (uniform for the CTA)
    if ((uintptr_t)(reinterpret_cast<const volatile uint8_t*>(err) + 4 - smem_raw) > dynamic_smem_bytes()) {
        if (tid == 0) record_status(ep.status, ESB_ERR_INTERNAL);
        return;
    }

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
    ws_alloc(warp, tmem_slot, tmem_cols);
    __syncthreads();                                  // barriers initialised, TMEM allocated

    // Producers start loading A at once; meanwhile the MMA and epilogue
    // warps decode the resident B and build the requantisation thresholds
    // (ws_setup).
    uint32_t tmem_base = 0;
    if (warp < kWsProdWarp0)
        tmem_base = ws_setup<false>(srcB, n0, K, fb, BN, bstream ? 0 : nkb, sB, thr, ep, tmem_slot, tid, lutb);

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
        griddep_wait();                               // A may come from the previous launch
        const uint32_t zwa = fmt_zero_code(4, fa.k) * 0x11111111u;
        const uint32_t zwb = fmt_zero_code(4, fb.k) * 0x11111111u;
        const bool b_vec = fb.b == 4 && fb.planes == 1 && srcB.linear() && srcB.vec4();
        int64_t cur_tile = -1;
        typename SrcA::Row rows[4];
        // stage s and its phase ph follow it incrementally (no division in
        // the loop): it advances by nprod <= stages, so s wraps at most once
        int s = p;
        uint32_t ph = 0u;
        for (int64_t it = p; it < total_it && !*err; it += nprod) {
            const int64_t ti = it / nkb;
            const int kb = (int)(it - ti * nkb);
            if (ti != cur_tile) {
                cur_tile = ti;
                const int64_t m0 = (cta_in_n + ti * ctas_per_n) * kBM;
#pragma unroll
                for (int q = 0; q < 4; q++) rows[q] = srcA.row(m0 + lane + 32 * q);
            }
            if (!wait_or_abort(&empty[s], ph ^ 1u, err)) { *err = 1; break; }
            uint8_t* st = sA + s * stage_bytes;
            if (fa.b == 4 && fa.planes == 1 && srcA.linear() && srcA.vec4()) {
                const int64_t kw0 = (int64_t)kb * 16;
                typename SrcA::Cursor cur[4];
#pragma unroll
                for (int pc = 0; pc < 4; pc++) cur[pc] = srcA.cursor(kw0 + 4 * pc);
                // one row at a time: a rolled loop keeps the producers' code
                // small (the SM's instruction caches hold every role's loop;
                // measured faster than four rows' loads in flight unrolled)
#pragma unroll 1
                for (int q = 0; q < 4; q++) {
                    uint4 v[4];
                    load_row_b4(srcA, rows[q], cur, kw0, K, zwa, v);
                    store_row_b4(st, lane + 32 * q, v, kw0, K, fa);
                }
            } else if (fa.planes == 1 && srcA.linear()) {
                bool done = false;
                if constexpr (kIsConv<SrcA>) {
                    if (fa.b == 4 || fa.spw) {
                        // im2col rows: the K-block's words through a tap table
                        const int nw = kBK / (fa.b == 4 ? 8 : fa.spw);
                        int4* tab = ptab[p];
                        conv_tap_table(srcA, (int64_t)kb * nw, nw, tab, lane);
#pragma unroll 1
                        for (int q = 0; q < 4; q++)
                            walk_row_tab(srcA, rows[q], tab, (int64_t)kb * kBK, K, fa, luta, st, lane + 32 * q);
                        done = true;
                    }
                }
                if (!done) {
                    // other widths: one word walk per row of the K-block
#pragma unroll 1
                    for (int q = 0; q < 4; q++)
                        walk_row_kblock(srcA, rows[q], (int64_t)kb * kBK, K, fa, luta, st, lane + 32 * q);
                }
            } else {
                fill_stage_any(srcA, (cta_in_n + ti * ctas_per_n) * kBM, st, lane, (int64_t)kb * kBK, K, fa);
            }
            if (bstream) {
                // this K-block of the CTA's B rows n0 .. n0 + BN, two rows per lane in flight
                uint8_t* sb = st + kBM * kBK;
                const int64_t k0 = (int64_t)kb * kBK;
                if (b_vec) {
                    const int64_t kw0 = (int64_t)kb * 16;
                    RowsSrc::Cursor cur[4];
#pragma unroll
                    for (int pc = 0; pc < 4; pc++) cur[pc] = srcB.cursor(kw0 + 4 * pc);
#pragma unroll 1
                    for (int r = lane; r < BN; r += 64) {
                        const bool two = r + 32 < BN;
                        uint4 v0[4], v1[4];
                        load_row_b4(srcB, srcB.row(n0 + r), cur, kw0, K, zwb, v0);
                        if (two) load_row_b4(srcB, srcB.row(n0 + r + 32), cur, kw0, K, zwb, v1);
                        store_row_b4(sb, r, v0, kw0, K, fb);
                        if (two) store_row_b4(sb, r + 32, v1, kw0, K, fb);
                    }
                } else if (fb.planes == 1 && srcB.linear()) {
#pragma unroll 1
                    for (int r = lane; r < BN; r += 32) walk_row_kblock(srcB, srcB.row(n0 + r), k0, K, fb, lutb, sb, r);
                } else {
#pragma unroll 1
                    for (int u = lane; u < BN * 8; u += 32) {
                        const int r = u >> 3, g = u & 7;
                        *reinterpret_cast<uint4*>(sb + swz(r, g)) = decode_unit_any(srcB, srcB.row(n0 + r), k0 + g * 16, K, fb);
                    }
                }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&full[s]);
            s += nprod;
            if (s >= stages) { s -= stages; ph ^= 1u; }
        }
    } else if (warp == kWsMmaWarp) {
        // ---------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = idesc_e4m3_f32(BN);
            const uint32_t b_base = smem_u32(sB), a_base = smem_u32(sA);
            int s = 0;                                         // stage and phase of the next K-block
            uint32_t ph = 0u;
            for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
                const int a = (int)(ti & 1);
                if (!wait_or_abort(&tempty[a], (uint32_t)((ti >> 1) & 1) ^ 1u, err)) { *err = 1; break; }
                tc_fence_after();
                const uint32_t d = tmem_base + (uint32_t)(a * BN);
                for (int kb = 0; kb < nkb; kb++) {
                    if (!wait_or_abort(&full[s], ph, err)) { *err = 1; break; }
                    tc_fence_after();
                    const uint32_t a0 = a_base + (uint32_t)(s * stage_bytes);
                    const uint32_t b0 = bstream ? a0 + (uint32_t)(kBM * kBK) : b_base + (uint32_t)(kb * BN * kBK);
#pragma unroll
                    for (int j = 0; j < kBK / 32; j++)
                        mma_f8f6f4(d, smem_desc_sw128(a0 + j * 32), smem_desc_sw128(b0 + j * 32), idesc,
                                   (kb > 0 || j > 0) ? 1u : 0u);
                    mma_commit(&empty[s]);
                    if (++s == stages) { s = 0; ph ^= 1u; }
                }
                if (*err) break;
                mma_commit(&tfull[a]);
            }
            ws_drain(drain, err);
        }
    } else if (warp < epi_warps) {
        // ---------------------------------------------- epilogue
        const int64_t ctas = ctas_per_n, first = cta_in_n;
        auto rows = [=](int64_t ti, int row, int64_t& m) -> bool {
            m = (first + ti * ctas) * kBM + row;
            return m < M;
        };
        ws_epilogue<false, GEN>(ep, thr, rows, my_tiles, n0, N, BN, split, epi_warps, tmem_base, acc_scale, tfull, tempty, err,
                    warp, lane);
    }

    __syncthreads();
    if (*err && tid == 0) record_status(ep.status, ESB_ERR_TIMEOUT);
    if (warp == kWsMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, tmem_cols);
    }
}

// ------------------------------------------------------------ host side

int pick_bn(int64_t N, int out_cpw)
{
    // BN must be a multiple of 16 (MMA N step) and of the output codes per
    // word (so no packed word straddles two tiles).  Up to 256 columns: the
    // smallest such width that covers N (no wasted MMA columns or epilogue
    // lanes for narrow layers); wider: the width in [128, 256] that wastes
    // the fewest columns over the N-tiles, the wider on a tie.
    int best = 0;
    if (N <= 256) {
        for (int bn = 16; bn <= 256; bn += 16)
            if (bn >= N && bn % out_cpw == 0) return bn;
    }
    int64_t waste_best = -1;
    for (int bn = 256; bn >= 128; bn -= 16) {
        if (bn % out_cpw) continue;
        const int64_t waste = ((N + bn - 1) / bn) * bn - N;
        if (waste_best < 0 || waste < waste_best) { waste_best = waste; best = bn; }
    }
    if (best) return best;
    for (int bn = 16; bn <= 256; bn += 16)
        if (bn % out_cpw == 0) return bn;
    return 0;
}

// N-tile width of the streamed kernel.  Each of its CTAs decodes 128 A rows
// and BN B rows for every K-block, so a tile costs about 128 + BN row
// decodes; when M gives few row tiles, narrower N-tiles spread that work
// over more SMs.  The width (a multiple of 16 and of the output codes per
// word, at most bn0 = pick_bn's choice, at least 64) that minimises
// waves x (128 + BN), one CTA per SM; the wider on a tie.
static int streamed_bn(int64_t M, int64_t N, int out_cpw, int bn0)
{
    const int64_t sms = device_sm_count();
    const int64_t mt = (M + kBM - 1) / kBM;
    int best = bn0;
    int64_t cbest = ((mt * ((N + bn0 - 1) / bn0) + sms - 1) / sms) * (128 + bn0);
    for (int bn = bn0 - 16; bn >= 64; bn -= 16) {
        if (bn % out_cpw) continue;
        const int64_t waves = (mt * ((N + bn - 1) / bn) + sms - 1) / sms;
        const int64_t c = waves * (128 + bn);
        if (c < cbest) { cbest = c; best = bn; }
    }
    return best;
}

// N-tile width of the warp-specialised kernel with B resident when the
// tiles do not fill the SMs (small M: a classifier, the last stages of a
// network at small batch).  A CTA then decodes the A rows of its few tiles
// (128 rows each, again for every N-tile) and its BN rows of B once; the
// width (a multiple of 16 and of the output codes per word, at most bn0)
// that minimises waves x tiles per CTA x (128 + BN), the wider on a tie.
static int resident_bn(int64_t M, int64_t N, int out_cpw, int bn0)
{
    const int64_t sms = device_sm_count();
    const int64_t mt = (M + kBM - 1) / kBM;
    auto cost = [&](int bn) {
        const int64_t nt = (N + bn - 1) / bn;
        const int64_t per_n = nt >= sms ? 1 : sms / nt;
        const int64_t waves = (nt + sms - 1) / sms;
        const int64_t my = (mt + per_n - 1) / per_n;
        return waves * my * (128 + bn);
    };
    if (mt * ((N + bn0 - 1) / bn0) >= sms) return bn0;
    int best = bn0;
    int64_t cbest = cost(bn0);
    for (int bn = bn0 - 16; bn >= 16; bn -= 16) {
        if (bn % out_cpw) continue;
        const int64_t c = cost(bn);
        if (c < cbest) { cbest = c; best = bn; }
    }
    return best;
}

static size_t gemm_smem_bytes(int BN)
{
    return 1024 + (size_t)kStages * (kBM * kBK + (size_t)BN * kBK) + kStages * 8 + 16 + 512;
}

int max_dyn_smem()
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
    BN = streamed_bn(M, N, ep.out_cpw, BN);
    const size_t smem = gemm_smem_bytes(BN);
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(esb_gemm_tc_kernel<SrcA, SrcB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)gemm_smem_bytes(256));
        if (e != cudaSuccess) return e;
        configured = true;
    }
    const float acc_scale = ldexpf(1.0f, fa.csc + fb.csc);
    dim3 grid((unsigned)((M + kBM - 1) / kBM), (unsigned)((N + BN - 1) / BN));
    esb_gemm_tc_kernel<SrcA, SrcB><<<grid, kGemmThreads, smem, st>>>(a, b, M, N, K, fa, fb, BN, acc_scale, ep);
    return cudaGetLastError();
}

template <class SrcA>
static int ws_static_smem(cudaError_t* err)
{
    static int v = -1;
    if (v < 0) {
        cudaFuncAttributes a0, a1;
        *err = cudaFuncGetAttributes(&a0, esb_gemm_ws_kernel<SrcA, false>);
        if (*err != cudaSuccess) return -1;
        *err = cudaFuncGetAttributes(&a1, esb_gemm_ws_kernel<SrcA, true>);
        if (*err != cudaSuccess) return -1;
        v = (int)(a0.sharedSizeBytes > a1.sharedSizeBytes ? a0.sharedSizeBytes : a1.sharedSizeBytes);
    }
    return v;
}

// Warp-specialised launch: B resident when its N-tile fits in shared
// memory with at least three A stages, else streamed with A through the
// stages; returns false (nothing launched) when neither fits.
template <class SrcA>
static bool launch_ws(const SrcA& a, const RowsSrc& b, int64_t M, int64_t N, int64_t K, const OpFmt& fa,
                      const OpFmt& fb, int BN, const EpiParams& ep, cudaStream_t st, cudaError_t* err)
{
    // dynamic shared memory = the opt-in maximum minus the kernel's static shared memory
    const int static_smem = ws_static_smem<SrcA>(err);
    if (static_smem < 0) return true;
    const int maxs = max_dyn_smem() - static_smem;
    BN = resident_bn(M, N, ep.out_cpw, BN);
    WsLayout L = ws_layout(K, BN, maxs);
    int bstream = 0;
    if (L.stages < 3) {
        // B's N-tile does not fit beside three A stages: stream B through
        // the stages with A, at the N-tile width that suits the row tiles
        BN = streamed_bn(M, N, ep.out_cpw, BN);
        L = ws_layout_streamed(K, BN, maxs);
        if (L.stages < 3) return false;
        bstream = 1;
    }
    static bool configured = false;
    if (!configured) {
        *err = cudaFuncSetAttribute(esb_gemm_ws_kernel<SrcA, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, maxs);
        if (*err != cudaSuccess) return true;
        *err = cudaFuncSetAttribute(esb_gemm_ws_kernel<SrcA, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, maxs);
        if (*err != cudaSuccess) return true;
        configured = true;
    }
    const int n_tiles = (int)((N + BN - 1) / BN);
    const int64_t m_tiles = (M + kBM - 1) / kBM;
    int64_t per_n = device_sm_count() / n_tiles;
    if (per_n < 1) per_n = 1;
    if (per_n > m_tiles) per_n = m_tiles;
    const int64_t grid = per_n * n_tiles;
    const float acc_scale = ldexpf(1.0f, fa.csc + fb.csc);
    const bool gen = !(ep.codes_out && ep.out.b == 4);       // the general-width epilogue instance
    *err = launch_pdl(gen ? esb_gemm_ws_kernel<SrcA, true> : esb_gemm_ws_kernel<SrcA, false>, dim3((unsigned)grid), dim3(kWsThreads), (size_t)L.smem_bytes, st, a, b,
                      M, N, K, fa, fb, BN, L.nkb, L.stages, n_tiles, m_tiles, acc_scale, ep, bstream);
    return true;
}

// Bound + 2 on |acc| for the epilogue's FMA-pipe requantisation, or 0 when
// K max|I_A| max|I_B| reaches 2^20.
float acc_fma_limit(int64_t K, int ba, int ka, int bb, int kb)
{
    const double bound = (double)K * fmt_max_image(ba, ka) * fmt_max_image(bb, kb);
    return bound < 1048576.0 ? (float)(bound + 2.0) : 0.0f;
}

EpiParams make_epi(const GemmOutputs& o)
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
    {
        const uintptr_t pa = reinterpret_cast<uintptr_t>(o.codes_out);
        ep.codes_vec = ((pa & 15u) == 0 && (o.ldo & 3) == 0) ? 4 : ((pa & 7u) == 0 && (o.ldo & 1) == 0) ? 2 : 1;
    }
    ep.acc_lim = 0.0f;
    ep.status = device_status_ptr();
    return ep;
}

cudaError_t launch_gemm(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, int ba, int ka,
                        const uint32_t* B, int64_t ldb, int bb, int kb, const GemmOutputs& o, cudaStream_t st)
{
    EpiParams ep = make_epi(o);
    ep.dq_pow2 = ldexpf(1.0f, -(ka + kb));
    ep.acc_lim = acc_fma_limit(K, ba, ka, bb, kb);
    const int BN = pick_bn(N, ep.out_cpw);
    RowsSrc a{A, lda, M};
    RowsSrc b{B, ldb, N};
    OpFmt fa = make_opfmt(ba, ka), fb = make_opfmt(bb, kb);
    int64_t Kx = plan_planes(fa, fb, K);              // the kernels' K (significand planes)
    if (const int64_t Ks = plan_slots(fa, fb, K, (K + fa.cpw - 1) / fa.cpw)) Kx = Ks;
    if (Kx > 0) {
        cudaError_t e = cudaSuccess;
        if (launch_ws(a, b, M, N, Kx, fa, fb, BN, ep, st, &e)) return e;
    }
    return launch_tc(a, b, M, N, Kx, fa, fb, BN, ep, st);
}

// ESB_CONV_IM2COL=1 in the environment (read once) routes every dense
// convolution through the im2col kernels: a check of one path against the
// other on the same shapes.
static bool conv_force_im2col()
{
    static const int v = [] {
        const char* e = getenv("ESB_CONV_IM2COL");
        return (e && e[0] == '1') ? 1 : 0;
    }();
    return v != 0;
}

// Words of each pixel that enter the implicit GEMM's K: all ldx of them
// (the halo kernel and the 16-byte decode read whole 4-word pieces) unless
// at least half are padding (a first layer's 3 channels in a 4-word row),
// then only the words that hold channels.
static int conv_k_words(const esb_conv_desc& d, int64_t ldx, int bx)
{
    const int cpw = 32 / bx;
    const int used = (d.c + cpw - 1) / cpw;
    return (2 * used <= ldx) ? used : (int)ldx;
}

// Filter rows of the im2col K: plain rows when every tap's ldx input words
// enter K with filter taps of the same width and stride; otherwise taps of
// kwx input words (kwx * cpw_x codes) at a tap stride of ldw filter words,
// walkable word by word when both operands have the same width.
static RowsSrc conv_filter_rows(const esb_conv_desc& d, const uint32_t* W, int64_t ldx, int bx, int64_t ldw, int bw,
                                int kwx)
{
    RowsSrc b{W, (int64_t)d.r * d.s * ldw, d.cout};
    if (kwx != ldx || bw != bx || ldw != ldx) {
        b.kp = (int64_t)kwx * (32 / bx);
        b.ldt = ldw;
        if (bw == bx) b.kwt = kwx;
    }
    return b;
}

cudaError_t launch_conv_tc(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int bx, int kx,
                           const uint32_t* W, int64_t ldw, int bw, int kw, const GemmOutputs& o, cudaStream_t st)
{
    EpiParams ep = make_epi(o);
    ep.dq_pow2 = ldexpf(1.0f, -(kx + kw));
    ep.acc_lim = acc_fma_limit((int64_t)d.r * d.s * d.c, bx, kx, bw, kw);   // padding slots add exact zeros
    const int64_t M = (int64_t)d.n * P * Q;
    const int64_t N = d.cout;
    const int kwx = conv_k_words(d, ldx, bx);
    const int64_t K = (int64_t)d.r * d.s * kwx * (32 / bx);
    const int BN = pick_bn(N, ep.out_cpw);
    ConvSrc a;
    a.X = X; a.ldx = (int)ldx; a.rows = (int)M; a.H = d.h; a.W = d.w; a.P = P; a.Q = Q; a.S = d.s;
    a.stride = d.stride; a.pad = d.pad; a.kw = kwx;
    RowsSrc b = conv_filter_rows(d, W, ldx, bx, ldw, bw, kwx);
    OpFmt fa = make_opfmt(bx, kx), fb = make_opfmt(bw, kw);
    int64_t Kx = plan_planes(fa, fb, K);              // the kernels' K (significand planes)
    if (b.linear()) {
        const int64_t words = (int64_t)d.r * d.s * kwx;
        if (const int64_t Ks = plan_slots(fa, fb, words * fa.cpw, words)) Kx = Ks;
    }
    cudaError_t e = cudaSuccess;
    if (Kx > 0 && !conv_force_im2col() && fa.planes == 1 && b.kp == 0 &&
        launch_conv_halo(d, P, Q, X, ldx, fa, W, ldw, fb, BN, ep, st, &e))
        return e;
    if (Kx > 0 && launch_ws(a, b, M, N, Kx, fa, fb, BN, ep, st, &e)) return e;
    return launch_tc(a, b, M, N, Kx, fa, fb, BN, ep, st);
}

int conv_kernel_choice(const esb_conv_desc& d, int P, int Q, int64_t ldx, int bx, int kx, int64_t ldw, int bw,
                       int kw, int out_b)
{
    const int cpw = 32 / out_b;
    const int kwd = conv_k_words(d, ldx, bx);
    const int64_t K = (int64_t)d.r * d.s * kwd * (32 / bx);
    OpFmt fa = make_opfmt(bx, kx), fb = make_opfmt(bw, kw);
    int64_t Kx = plan_planes(fa, fb, K);
    const RowsSrc b = conv_filter_rows(d, nullptr, ldx, bx, ldw, bw, kwd);
    const bool same_layout = b.kp == 0 && fa.planes == 1;
    if (b.linear()) {                                 // as launch_conv_tc
        const int64_t words = (int64_t)d.r * d.s * kwd;
        if (const int64_t Ks = plan_slots(fa, fb, words * fa.cpw, words)) Kx = Ks;
    }
    if (Kx > 0 && !conv_force_im2col() && same_layout && conv_halo_ok(d, P, Q, ldx, bx, kx, cpw))
        return ESB_CONV_KERNEL_HALO;
    cudaError_t e = cudaSuccess;
    const int st = ws_static_smem<ConvSrc>(&e);
    if (st < 0) return -1;
    const int bn = resident_bn((int64_t)d.n * P * Q, d.cout, cpw, pick_bn(d.cout, cpw));   // as launch_ws
    if (Kx > 0 && ws_layout(Kx, bn, max_dyn_smem() - st).stages >= 3) return ESB_CONV_KERNEL_IM2COL;
    return ESB_CONV_KERNEL_STREAMED;
}

bool gemm_pick_ok(int64_t N, int out_b) { return pick_bn(N, 32 / out_b) != 0; }

}  // namespace esb
