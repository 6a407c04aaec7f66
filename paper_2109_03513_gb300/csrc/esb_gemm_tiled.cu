// ESB GEMM for large operands (Sec. III-B products, Sec. IV-B/IV-C
// computing logic): C[m, n] = sum_k I(A[m, k]) I(B[n, k]) with the fused
// epilogue, for shapes whose B does not stay resident in shared memory.
//
// Two steps on the caller's stream:
//  1. esb_tile_kernel decodes each operand once into a tiled image of E4M3
//     bytes in the caller's workspace: tile (rb, kb) holds rows
//     rb*TH .. rb*TH + TH - 1 and codes 128 kb .. 128 kb + 127 as TH x 128
//     bytes in the SW128 K-major layout of an MMA operand (row r, 16-byte
//     chunk g at r*128 + ((g ^ (r & 7)) * 16)); tiles follow in (rb, kb)
//     order, so every tile is one contiguous block.  Rows past the operand
//     and codes past K are E4M3 zeros.  HBM-bound: code bytes in, one byte
//     per code out.
//  2. esb_gemm_tiled_kernel, persistent and warp-specialised: one producer
//     thread bulk-copies whole tiles (A: 128 rows, 16 KiB; B: 256 rows,
//     32 KiB) into a ring of shared-memory stages (cp.async.bulk completing
//     on mbarriers), the MMA thread issues four 128 x 256 x 32 tcgen05.mma
//     per K-block into one of two 256-column TMEM accumulators, and eight
//     epilogue warps drain them through the epilogue of the other tcgen05
//     kernels (ws_epilogue).  Each CTA keeps one 256-column N-tile and walks
//     the M-tiles.
// The contraction is exact: fp32 TMEM accumulation of integer-valued
// products holds every partial sum exactly while it stays below 2^24, so a K
// with K max|I_A| max|I_B| >= 2^24 is split into chunks that each stay
// below it, accumulated in separate TMEM regions (up to four, with a
// 128-column N-tile beyond two) and added as integers in the epilogue
// (int32: K max|I_A| max|I_B| < 2^31).
#include <cstdint>
#include <cstdlib>
#include <cuda_runtime.h>

#include "esb_tc.cuh"
#include "esb_internal.h"

namespace esb {

namespace {

constexpr int kTiledBN = 256;                  // N-tile width (rows of a B tile); 128 with > 2 K-chunks
constexpr int kTiledThreads = 320;             // warps 0-7 epilogue, 8 MMA, 9 producer
constexpr int kTiledProdWarp = 9;
constexpr int kTileA = kBM * kBK;              // 16 KiB
constexpr int kTmemCols = 512;

}  // namespace

// One 16-byte chunk (16 codes) per thread and pass: u enumerates (tile,
// row, physical chunk), so consecutive threads write consecutive bytes.
__global__ void __launch_bounds__(256) esb_tile_kernel(RowsSrc src, int64_t K, OpFmt f, int TH, int nkb,
                                                       int64_t rblocks, uint8_t* __restrict__ out)
{
    const int64_t total = rblocks * nkb * (int64_t)TH * 8;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += (int64_t)gridDim.x * blockDim.x) {
        const int gp = (int)(u & 7);                         // physical chunk in the 128-byte row
        const int64_t rt = u >> 3;
        const int r = (int)(rt % TH);
        const int64_t t = rt / TH;                           // tile index rb * nkb + kb
        const int64_t rb = t / nkb;
        const int kb = (int)(t - rb * nkb);
        const int g = gp ^ (r & 7);                          // logical chunk: codes 16 g .. 16 g + 15
        const int64_t row = rb * TH + r;
        const int64_t k0 = (int64_t)kb * kBK + g * 16;
        uint4 o = make_uint4(0u, 0u, 0u, 0u);
        if (row < src.rows && k0 < K) {
            const RowsSrc::Row rw = src.row(row);
            if (f.b == 4) {
                // two words (16 codes) at word k0 / 8 (even: 8-byte aligned);
                // rows are padded to whole 16-byte groups, so both exist
                const uint2 w = __ldg(reinterpret_cast<const uint2*>(src.words(rw, k0 >> 3)));
                uint32_t o0, o1, o2, o3;
                decode_word_b4(w.x, f.k, f.ew, o0, o1);
                decode_word_b4(w.y, f.k, f.ew, o2, o3);
                if (k0 + 16 > K) {                           // K tail: zero the codes past K
                    uint32_t ml, mh;
                    int va = (int)(K - k0);
                    va = va < 0 ? 0 : (va > 8 ? 8 : va);
                    tail_masks(va, ml, mh);
                    o0 &= ml; o1 &= mh;
                    int vb = (int)(K - k0 - 8);
                    vb = vb < 0 ? 0 : (vb > 8 ? 8 : vb);
                    tail_masks(vb, ml, mh);
                    o2 &= ml; o3 &= mh;
                }
                o = make_uint4(o0, o1, o2, o3);
            } else {
                // any width: walk the 16 codes through their words (a code
                // never straddles two words), one load per word
                const uint32_t* p = src.words(rw, 0);
                int64_t wi = k0 / f.cpw;
                int slot = (int)(k0 - wi * f.cpw);
                uint32_t w = __ldg(p + wi);
                uint32_t ob[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                for (int j = 0; j < 16; j++) {
                    if (k0 + j >= K) break;
                    const uint32_t byte = code_to_e4m3((w >> (f.b * slot)) & f.mask, f);
                    const int pos = unit_pos(j);
                    ob[pos >> 2] |= byte << (8 * (pos & 3));
                    if (++slot == f.cpw) {
                        slot = 0;
                        ++wi;
                        if (k0 + j + 1 < K) w = __ldg(p + wi);
                    }
                }
                o = make_uint4(ob[0], ob[1], ob[2], ob[3]);
            }
        }
        reinterpret_cast<uint4*>(out + t * (int64_t)TH * kBK + (int64_t)r * kBK)[gp] = o;
    }
}

// Epilogue of a chunked accumulation: the nch chunk accumulators of a tile
// (TMEM regions (buf * nch + ch) * BN) are added as exact integers, the sum
// is stored as the int32 accumulator, and float(acc) (round to nearest, as
// the oracle converts it) goes through epi_element.  Codes of any width
// that divides 16 codes per word; padding slots past N take the zero code.
// Warps 0-7: TMEM lane quarter warp & 3, column half warp >> 2.
template <int BN>
__device__ void tiled_chunked_epilogue(const EpiParams& ep, const float* thr, int64_t M, int64_t N, int64_t n0,
                                       int64_t first, int64_t ctas, int64_t my_tiles, int nch, int nbuf,
                                       uint32_t tmem_base, float acc_scale, uint64_t* tfull, uint64_t* tempty,
                                       volatile int* err, int warp, int lane)
{
    const EpiCtx cx = make_epi_ctx(ep, thr);
    EpiParams e2 = ep;
    e2.acc_out = nullptr;                                // the exact sum is stored here instead
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const int c_lo = (warp >> 2) * (BN / 2), c_hi = c_lo + BN / 2;
    const int cpw = ep.out_cpw, ob = ep.out.b;
    const uint32_t zc = ep.codes_out ? fmt_zero_code(ep.out.b, ep.out.k) : 0u;
    for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
        const int buf = (int)(ti % nbuf);
        if (!wait_or_abort(&tfull[buf], (uint32_t)((ti / nbuf) & 1), err)) { *err = 1; break; }
        tc_fence_after();
        const int64_t m = (first + ti * ctas) * kBM + row;
        const bool mrow = m < M;
        const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16);
        for (int c = c_lo; c < c_hi; c += 16) {
            int isum[16];
#pragma unroll
            for (int j = 0; j < 16; j++) isum[j] = 0;
            for (int ch = 0; ch < nch; ch++) {
                uint32_t r[16];
                tmem_ld16(taddr + (uint32_t)((buf * nch + ch) * BN + c), r);
#pragma unroll
                for (int j = 0; j < 16; j++) isum[j] += __float2int_rn(__uint_as_float(r[j]) * acc_scale);
            }
            if (c + 16 >= c_hi) {                        // every column of this warp is in registers
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_tmem_free(&tempty[buf]);
            }
            if (!mrow) continue;
            uint32_t word = 0u;
            int slot = 0;
#pragma unroll
            for (int j = 0; j < 16; j++) {
                const int64_t n = n0 + c + j;
                uint32_t code = zc;
                if (n < N) {
                    if (ep.acc_out) ep.acc_out[m * N + n] = isum[j];
                    code = epi_element(e2, cx, __int2float_rn(isum[j]), m, n, N);
                }
                if (ep.codes_out) {
                    word |= code << (ob * slot);
                    if (++slot == cpw) {
                        const int64_t wcol = (n0 + c + j) / cpw;
                        if (wcol < ep.ldo) ep.codes_out[m * ep.ldo + wcol] = word;
                        word = 0u;
                        slot = 0;
                    }
                }
            }
        }
    }
}

template <bool LEAN4, int BN>
__global__ void __launch_bounds__(kTiledThreads, 1)
esb_gemm_tiled_kernel(const uint8_t* __restrict__ At, const uint8_t* __restrict__ Bt, int64_t M, int64_t N, int nkb,
                      int kbc, int nch, int stages, int n_tiles, int64_t m_tiles, float acc_scale, EpiParams ep)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    constexpr int kTileB = BN * kBK;
    constexpr int kStage = kTileA + kTileB;                      // A tile then B tile (both 1024-aligned)
    const int nbuf = kTmemCols / (nch * BN) >= 2 ? 2 : 1;       // accumulator sets (one per tile in flight)
    float* thr = reinterpret_cast<float*>(smem + stages * kStage);
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
    uint32_t tmem_cols = 32;                                     // a power of two >= the regions used
    while (tmem_cols < (uint32_t)(nbuf * nch * BN)) tmem_cols <<= 1;
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
            mbar_init(&full[s], 1);                      // the producer's arrive.expect_tx, then the copies' bytes
            mbar_init(&empty[s], 1);                     // the MMA commit that drained it
        }
        for (int a = 0; a < 2; a++) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], nch > 1 ? kWsEpiWarps : epi_warps);
        }
        mbar_init(drain, 1);
        *err = 0;
        fence_mbar_init();
    }
    ws_alloc(warp, tmem_slot, tmem_cols);
    __syncthreads();                                     // barriers initialised, TMEM allocated
    griddep_wait();                                      // the tiled operands come from the tile kernels
    if (warp < kWsEpiWarps) ws_thresholds(thr, ep, warp, lane);
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == kTiledProdWarp) {
        // ---------------------------------------------- producer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0u;
            const uint8_t* bt = Bt + (int64_t)n_tile * nkb * kTileB;   // B tiles of BN rows
            for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
                const uint8_t* at = At + (cta_in_n + ti * ctas_per_n) * nkb * (int64_t)kTileA;
                for (int kb = 0; kb < nkb; kb++) {
                    if (!wait_or_abort(&empty[s], ph ^ 1u, err)) { *err = 1; break; }
                    uint8_t* st = smem + s * kStage;
                    mbar_arrive_expect_tx(&full[s], (uint32_t)kStage);
                    bulk_copy_g2s(st, at + (int64_t)kb * kTileA, (uint32_t)kTileA, &full[s]);
                    bulk_copy_g2s(st + kTileA, bt + (int64_t)kb * kTileB, (uint32_t)kTileB, &full[s]);
                    if (++s == stages) { s = 0; ph ^= 1u; }
                }
            }
        }
    } else if (warp == kWsMmaWarp) {
        // ---------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = idesc_e4m3_f32(BN);
            const uint32_t base = smem_u32(smem);
            int s = 0;
            uint32_t ph = 0u;
            for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
                const int a = (int)(ti % nbuf);
                if (!wait_or_abort(&tempty[a], (uint32_t)((ti / nbuf) & 1) ^ 1u, err)) { *err = 1; break; }
                tc_fence_after();
                uint32_t d = tmem_base + (uint32_t)(a * nch * BN);
                uint32_t acc = 0u;
                for (int kb = 0; kb < nkb; kb++) {
                    if (kb > 0 && kb % kbc == 0) {       // next K-chunk: its own accumulator
                        d += (uint32_t)BN;
                        acc = 0u;
                    }
                    if (!wait_or_abort(&full[s], ph, err)) { *err = 1; break; }
                    tc_fence_after();
                    const uint32_t st = base + (uint32_t)(s * kStage);
                    const uint64_t ad = smem_desc_sw128(st), bd = smem_desc_sw128(st + kTileA);
                    // four K steps of 32 codes: 32 bytes along the swizzled row
                    mma_f8f6f4(d, ad, bd, idesc, acc);
                    mma_f8f6f4(d, ad + 2, bd + 2, idesc, 1u);
                    mma_f8f6f4(d, ad + 4, bd + 4, idesc, 1u);
                    mma_f8f6f4(d, ad + 6, bd + 6, idesc, 1u);
                    acc = 1u;
                    mma_commit(&empty[s]);
                    if (++s == stages) { s = 0; ph ^= 1u; }
                }
                if (*err) break;
                mma_commit(&tfull[a]);
            }
            ws_drain(drain, err);
        }
    } else if (nch > 1) {
        // ---------------------------------------------- epilogue (K in chunks)
        if (warp < kWsEpiWarps)
            tiled_chunked_epilogue<BN>(ep, thr, M, N, n0, cta_in_n, ctas_per_n, my_tiles, nch, nbuf, tmem_base,
                                       acc_scale, tfull, tempty, err, warp, lane);
    } else if (warp < epi_warps) {
        // ---------------------------------------------- epilogue
        const int64_t first = cta_in_n, ctas = ctas_per_n;
        auto rows = [=](int64_t ti, int row, int64_t& m) -> bool {
            m = (first + ti * ctas) * kBM + row;
            return m < M;
        };
        ws_epilogue<LEAN4, false>(ep, thr, rows, my_tiles, n0, N, BN, split, epi_warps, tmem_base, acc_scale, tfull, tempty,
                           err, warp, lane);
    }

    __syncthreads();
    if (*err && tid == 0) record_status(ep.status, ESB_ERR_TIMEOUT);
    if (warp == kWsMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, tmem_cols);
    }
}

// ------------------------------------------------------------- host side

static int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// K-chunking of a shape: K-blocks per chunk (each chunk's partial sums stay
// below 2^24), chunk count and N-tile width; false when the kernel cannot
// hold the chunks (more than four, or a total past the int32 range).
static bool tiled_plan(int64_t K, int ba, int ka, int bb, int kb, int* kbc, int* nch, int* BN)
{
    const int64_t nkb = cdiv(K, kBK);
    const double img = (double)fmt_max_image(ba, ka) * fmt_max_image(bb, kb);
    if ((double)K * img >= 2147483648.0) return false;
    int64_t c = nkb;
    if ((double)K * img >= 16777216.0) {
        c = (int64_t)((16777215.0 / img) / kBK);                  // whole K-blocks per chunk
        if (c < 1) return false;
    }
    const int64_t n = cdiv(nkb, c);
    if (n > 4) return false;
    *kbc = (int)c;
    *nch = (int)n;
    *BN = n <= 2 ? 256 : 128;
    return true;
}

size_t gemm_tiled_workspace_bytes(int64_t M, int64_t N, int64_t K)
{
    const int64_t nkb = cdiv(K, kBK);
    // B tiles of 256 rows bound the 128-row tiling of a chunked K from above
    return (size_t)(cdiv(M, kBM) * nkb * kTileA + cdiv(N, kTiledBN) * nkb * (int64_t)kTiledBN * kBK);
}

// The tiled path pays two extra launches and a pass over both operands:
// below about 2^32 multiply-adds the other kernels finish first (when they
// can: their decode is fast for 4-bit operands only).  ESB_GEMM_TILED_MIN_MACS
// in the environment (read per call) moves that threshold (0: every shape
// the kernel takes).
bool gemm_tiled_ok(int64_t M, int64_t N, int64_t K, int ba, int ka, int bb, int kb, int out_cpw)
{
    int kbc, nch, BN;
    // significand-split operands (k >= 4) take esb_gemm's kernels
    if (fmt_needs_split(ba, ka) || fmt_needs_split(bb, kb)) return false;
    if (M <= 0 || N < kTiledBN || K <= 0 || !tiled_plan(K, ba, ka, bb, kb, &kbc, &nch, &BN)) return false;
    if (kTiledBN % out_cpw != 0 || (nch > 1 && 16 % out_cpw != 0)) return false;
    if (nch > 1) return true;                                     // only this path takes that K
    double min_macs = (ba == 4 && bb == 4) ? 4294967296.0 : 0.0;
    if (const char* v = getenv("ESB_GEMM_TILED_MIN_MACS")) min_macs = atof(v);
    return (double)M * N * K >= min_macs;
}

static int tiled_static_smem(cudaError_t* err)
{
    static int v = -1;
    if (v < 0) {
        cudaFuncAttributes a0, a1, a2;
        *err = cudaFuncGetAttributes(&a0, esb_gemm_tiled_kernel<false, 256>);
        if (*err != cudaSuccess) return -1;
        *err = cudaFuncGetAttributes(&a1, esb_gemm_tiled_kernel<true, 256>);
        if (*err != cudaSuccess) return -1;
        *err = cudaFuncGetAttributes(&a2, esb_gemm_tiled_kernel<false, 128>);
        if (*err != cudaSuccess) return -1;
        size_t m = a0.sharedSizeBytes;
        if (a1.sharedSizeBytes > m) m = a1.sharedSizeBytes;
        if (a2.sharedSizeBytes > m) m = a2.sharedSizeBytes;
        v = (int)m;
    }
    return v;
}

static cudaError_t launch_tile(const RowsSrc& src, int64_t K, const OpFmt& f, int TH, int nkb, int64_t rblocks,
                               uint8_t* out, cudaStream_t st)
{
    const int64_t total = rblocks * nkb * (int64_t)TH * 8;
    int64_t grid = cdiv(total, 256);
    const int64_t cap = (int64_t)device_sm_count() * 8;
    if (grid > cap) grid = cap;
    esb_tile_kernel<<<(unsigned)grid, 256, 0, st>>>(src, K, f, TH, nkb, rblocks, out);
    return cudaGetLastError();
}

cudaError_t launch_gemm_tiled(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, int ba, int ka,
                              const uint32_t* B, int64_t ldb, int bb, int kb, const GemmOutputs& o, void* workspace,
                              cudaStream_t st)
{
    int kbc = 0, nch = 0, BN = 0;
    if (!tiled_plan(K, ba, ka, bb, kb, &kbc, &nch, &BN)) return cudaErrorInvalidValue;
    EpiParams ep = make_epi(o);
    ep.dq_pow2 = ldexpf(1.0f, -(ka + kb));
    ep.acc_lim = nch == 1 ? acc_fma_limit(K, ba, ka, bb, kb) : 0.0f;
    const OpFmt fa = make_opfmt(ba, ka), fb = make_opfmt(bb, kb);
    const int nkb = (int)cdiv(K, kBK);
    const int64_t m_tiles = cdiv(M, kBM), n_tiles = cdiv(N, BN);
    uint8_t* At = static_cast<uint8_t*>(workspace);
    uint8_t* Bt = At + m_tiles * nkb * (int64_t)kTileA;
    cudaError_t e = launch_tile(RowsSrc{A, lda, M}, K, fa, kBM, nkb, m_tiles, At, st);
    if (e != cudaSuccess) return e;
    e = launch_tile(RowsSrc{B, ldb, N}, K, fb, BN, nkb, n_tiles, Bt, st);
    if (e != cudaSuccess) return e;

    const int st_smem = tiled_static_smem(&e);
    if (st_smem < 0) return e;
    const int maxs = max_dyn_smem() - st_smem;
    const int64_t fixed = 1024 + 4 * 128 + 512;
    const int64_t stage_bytes = kTileA + (int64_t)BN * kBK;
    int stages = (int)((maxs - fixed) / stage_bytes);
    if (stages > kWsMaxStages) stages = kWsMaxStages;
    if (stages < 2) return cudaErrorInvalidConfiguration;
    const size_t smem = (size_t)(fixed + (int64_t)stages * stage_bytes);
    static bool configured = false;
    if (!configured) {
        e = cudaFuncSetAttribute(esb_gemm_tiled_kernel<false, 256>, cudaFuncAttributeMaxDynamicSharedMemorySize, maxs);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(esb_gemm_tiled_kernel<true, 256>, cudaFuncAttributeMaxDynamicSharedMemorySize, maxs);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(esb_gemm_tiled_kernel<false, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, maxs);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    int64_t per_n = device_sm_count() / n_tiles;
    if (per_n < 1) per_n = 1;
    if (per_n > m_tiles) per_n = m_tiles;
    const int64_t grid = per_n * n_tiles;
    const float acc_scale = ldexpf(1.0f, fa.csc + fb.csc);
    // the specialised epilogue: 4-bit codes as the only output with a scalar
    // scale and bias, whole N-tiles, a monotone requantisation, K in one chunk
    const bool fast = nch == 1 && BN == 256 && ep.codes_out && ep.out.b == 4 && !ep.scale && !ep.bias &&
                      !ep.residual && !ep.acc_out && !ep.y_out && ep.acc_lim > 0.0f && N % BN == 0 &&
                      (!ep.out.is_signed || ep.act != ESB_ACT_NONE);
    void (*kernel)(const uint8_t*, const uint8_t*, int64_t, int64_t, int, int, int, int, int, int64_t, float,
                   EpiParams) = BN == 128 ? esb_gemm_tiled_kernel<false, 128>
                                          : (fast ? esb_gemm_tiled_kernel<true, 256> : esb_gemm_tiled_kernel<false, 256>);
    return launch_pdl(kernel, dim3((unsigned)grid), dim3(kTiledThreads), smem, st, (const uint8_t*)At,
                      (const uint8_t*)Bt, M, N, nkb, kbc, nch, stages, (int)n_tiles, m_tiles, acc_scale, ep);
}

}  // namespace esb
