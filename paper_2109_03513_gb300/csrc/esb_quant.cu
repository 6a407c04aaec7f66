// esb_quant.cu -- HBM-bound element-wise kernels of libesb:
//   * projection of fp32 tensors onto packed ESB codes (Eq. cheap_projection
//     with the shift-and-round projection of Eq. fast_projection),
//   * dequantisation (Sec. IV-A, Eq. q),
//   * DDA calibration statistics and alpha (Sec. III-D).
#include <cstdint>
#include <cstdlib>
#include <mutex>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

// ----------------------------------------------------------- projection

// Granules of 128 values (lane l holds values 4l .. 4l + 3): the warps of
// the grid take equal contiguous runs of them, in the same order in every
// pass over x, so a warp's share differs by at most one granule from any
// other's.
__device__ __forceinline__ void warp_granules(int64_t gran, int64_t& g_lo, int64_t& g_hi)
{
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    g_lo = gran * gwarp / nwarps;
    g_hi = gran * (gwarp + 1) / nwarps;
}

// Codes of one granule (warp-collective): lane l turns its values 4l .. 4l
// + 3 into 16 bits of codes, lane pairs (l, l + 1) join their halves into
// code word 16 g + l / 2 with a shuffle.
template <bool SIGNED>
__device__ __forceinline__ void project_granule_b4(const float4 q, int64_t g, int64_t nw, const Thr7& t7, int k,
                                                   uint32_t* __restrict__ codes)
{
    const int lane = threadIdx.x & 31;
    const float xv4[4] = {q.x, q.y, q.z, q.w};
    uint32_t J = 0u, S = 0u;
#pragma unroll
    for (int i = 0; i < 4; i++) {
        J |= bucket7(SIGNED ? fabsf(xv4[i]) : xv4[i], t7) << (4 * i);
        if (SIGNED) S |= (__float_as_uint(xv4[i]) >> 31) << (4 * i + 3);
    }
    const uint32_t h = codes8_b4(J, S, k) & 0xffffu;          // four codes: low 16 bits
    const uint32_t other = __shfl_down_sync(0xffffffffu, h, 1);
    const int64_t wi = g * 16 + (lane >> 1);
    if ((lane & 1) == 0 && wi < nw) codes[wi] = h | (other << 16);
}

// One code word (8 values, 2 x float4) of a flat tensor.
template <bool SIGNED>
__device__ __forceinline__ uint32_t word_b4(const float4 qa, const float4 qb, const Thr7& t7, int k)
{
    const float v[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
    uint32_t J = 0u, S = 0u;
#pragma unroll
    for (int j = 0; j < 8; j++) {
        J |= bucket7(SIGNED ? fabsf(v[j]) : v[j], t7) << (4 * j);
        if (SIGNED) S |= (__float_as_uint(v[j]) >> 31) << (4 * j + 3);
    }
    return codes8_b4(J, S, k);
}

// Projection of a flat (row stride = cols, code rows without padding)
// tensor of n values (n % 8 == 0) to 4-bit codes.  The full granules are
// split among the warps exactly as in the statistics pass (warp_granules);
// each warp reads its first `stash_g` granules from its shared-memory stash
// (written by that pass) and the rest in batches of 8 coalesced 16-byte
// loads per lane; the last warp also takes the partial granule at the end.
template <bool SIGNED, bool STREAM>
__device__ __forceinline__ void project_flat_b4(const float* __restrict__ x, int64_t n, const Thr7& t7, int k,
                                                uint32_t* __restrict__ codes, const float4* stash = nullptr,
                                                int stash_g = 0)
{
    const int lane = threadIdx.x & 31;
    const int64_t gran = n / 128;
    int64_t g_lo, g_hi;
    warp_granules(gran, g_lo, g_hi);
    const float4* xv = reinterpret_cast<const float4*>(x) + lane;
    const int64_t nw = n >> 3;                        // code words
    int64_t g0 = g_lo;
    if (stash) {
        // stashed granules in pairs: lane l makes word l & 15 of granule
        // l >> 4 of the pair from two float4 (no shuffle, one store)
        const int ns = (int)(g_hi - g_lo < stash_g ? g_hi - g_lo : stash_g);
        const int half = lane >> 4, wl = lane & 15;
        int i = 0;
#pragma unroll 2
        for (; i + 2 <= ns; i += 2) {
            const float4* sp = stash + (i + half) * 32 + 2 * wl;
            codes[(g_lo + i + half) * 16 + wl] = word_b4<SIGNED>(sp[0], sp[1], t7, k);
        }
        for (g0 = g_lo + i; g0 < g_lo + ns; g0++)
            project_granule_b4<SIGNED>(stash[(g0 - g_lo) * 32 + lane], g0, nw, t7, k, codes);
    }
#pragma unroll 1
    for (; g0 < g_hi; g0 += 8) {
        float4 q[8];
#pragma unroll
        for (int u = 0; u < 8; u++) {
            q[u] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (g0 + u < g_hi) q[u] = STREAM ? __ldcs(xv + (g0 + u) * 32) : __ldg(xv + (g0 + u) * 32);
        }
#pragma unroll
        for (int u = 0; u < 8; u++) {
            if (g0 + u >= g_hi) break;                // warp-uniform
            project_granule_b4<SIGNED>(q[u], g0 + u, nw, t7, k, codes);
        }
    }
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    if (gwarp == nwarps - 1 && gran * 128 < n) {      // partial last granule
        const int64_t e = gran * 128 + 4 * lane;
        const float4 q = e < n ? __ldg(xv + gran * 32) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        project_granule_b4<SIGNED>(q, gran, nw, t7, k, codes);
    }
}

// Both projection kernels first build the threshold table of the current
// alpha (all warps, see build_thresholds), then project every element with
// it: no division per element.

// Fast path: one thread turns 4*cpw consecutive floats of a row into 4
// code words (one 16-byte store); cpw float4 loads in flight per thread,
// streaming cache hints since every byte is touched once.
template <int B>
__global__ void __launch_bounds__(256)
project_vec_kernel(const float* __restrict__ x, int64_t rows, int64_t cols, int64_t ldx,
                   float alpha, const float* __restrict__ alpha_dev, ProjParams p,
                   uint32_t* __restrict__ codes, int64_t ldc)
{
    constexpr int CPW = 32 / B;
    constexpr int L = 1 << (B - 1);
    // b = 3 and b >= 5: one 8-byte cell entry per value instead of b - 1
    // threshold loads (b = 4 keeps its register bucket search, which is faster
    // there)
    constexpr bool CELLS = B == 3 || B >= 5;
    constexpr int CAP = B <= 6 ? 1024 : 2048;
    __shared__ float T[L];
    __shared__ uint2 cells[CELLS ? CAP : 1];
    const int64_t upr = ldc >> 2;                 // 4-word units per row
    const int64_t total = rows * upr;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;

    // The first unit's loads are issued before the threshold table is built,
    // and every later unit's loads before the previous unit's store, so the
    // table set-up and the stores overlap memory latency.
    float v[4 * CPW];
    int64_t r = 0, w4 = 0, c0 = 0;
    bool full = false;
    auto fetch = [&](int64_t uu) {
        if (uu >= total) return;
        r = (rows == 1) ? 0 : uu / upr;
        w4 = uu - r * upr;
        c0 = w4 * (4 * CPW);
        full = c0 + 4 * CPW <= cols;
        if (full) {
            const float4* xr = reinterpret_cast<const float4*>(x + r * ldx + c0);
#pragma unroll
            for (int i = 0; i < CPW; i++) {
                const float4 t = __ldcs(xr + i);
                v[4 * i + 0] = t.x; v[4 * i + 1] = t.y; v[4 * i + 2] = t.z; v[4 * i + 3] = t.w;
            }
        }
    };
    int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const bool flat = (ldx == cols) && (cols % 8 == 0) && (ldc * 8 == cols);
    if (!(B == 4 && flat)) fetch(u);

    const float a = alpha_dev ? __ldg(alpha_dev) : alpha;
    build_thresholds(T, p, a, threadIdx.x >> 5, threadIdx.x & 31, 0, blockDim.x >> 5);
    __syncthreads();
    Thr7 t7;
    if (B == 4) {
#pragma unroll
        for (int i = 0; i < 7; i++) t7.t[i] = T[i];
    }
    int h0 = 0, hmax = 0;
    const bool by_cells = CELLS && build_cells<B, CAP>(cells, h0, hmax, T, p);
    const int sh = cell_shift(p.k);
    const uint32_t amask = p.is_signed ? 0x7fffffffu : 0xffffffffu;

    if (B == 4 && flat) {                                 // flat codes: coalesced warp tiles
        if (p.is_signed) project_flat_b4<true, true>(x, rows * cols, t7, p.k, codes);
        else project_flat_b4<false, true>(x, rows * cols, t7, p.k, codes);
        return;
    }

    // the loop once per per-value projection (the choice is block-uniform)
    auto run = [&](auto proj) {
        for (; u < total; u += stride) {
            uint32_t out[4];
            const int64_t rr = r, ww4 = w4, cc0 = c0;
            if (full) {
                if (B == 4) {
                    // buckets of |x| (x for the unsigned set: negatives land in bucket 0)
#pragma unroll
                    for (int w = 0; w < 4; w++) {
                        uint32_t J = 0u, S = 0u;
#pragma unroll
                        for (int j = 0; j < 8; j++) {
                            const float xv = v[w * 8 + j];
                            const uint32_t uxv = __float_as_uint(xv);
                            J |= bucket7(p.is_signed ? fabsf(xv) : xv, t7) << (4 * j);
                            S |= ((uxv >> 31) & (uint32_t)p.is_signed) << (4 * j + 3);
                        }
                        out[w] = codes8_b4(J, S, p.k);
                    }
                } else {
#pragma unroll
                    for (int w = 0; w < 4; w++) {
                        uint32_t word = 0;
#pragma unroll
                        for (int j = 0; j < CPW; j++) word |= proj(v[w * CPW + j]) << (B * j);
                        out[w] = word;
                    }
                }
            } else {
                const float* xr = x + rr * ldx + cc0;
#pragma unroll
                for (int w = 0; w < 4; w++) {
                    uint32_t word = 0;
#pragma unroll
                    for (int j = 0; j < CPW; j++) {
                        const int64_t c = cc0 + w * CPW + j;
                        const uint32_t code = (c < cols) ? proj(__ldcs(xr + w * CPW + j)) : p.zero_code;
                        word |= code << (B * j);
                    }
                    out[w] = word;
                }
            }
            fetch(u + stride);
            __stcs(reinterpret_cast<uint4*>(codes + rr * ldc + (ww4 << 2)), make_uint4(out[0], out[1], out[2], out[3]));
        }
    };
    if (by_cells)
        run([&](float xv) -> uint32_t { return project_by_cells<B>(xv, cells, h0, hmax, sh, amask); });
    else
        run([&](float xv) -> uint32_t {
            return B == 4 ? project_by_thr7(xv, t7, p) : project_by_table_t<B>(xv, T, p);
        });
}

// General path: any alignment and strides; one thread per code word.
template <int B>
__global__ void __launch_bounds__(256)
project_any_kernel(const float* __restrict__ x, int64_t rows, int64_t cols, int64_t ldx,
                   float alpha, const float* __restrict__ alpha_dev, ProjParams p,
                   uint32_t* __restrict__ codes, int64_t ldc)
{
    constexpr int CPW = 32 / B;
    constexpr int L = 1 << (B - 1);
    __shared__ float T[L];
    const float a = alpha_dev ? __ldg(alpha_dev) : alpha;
    build_thresholds(T, p, a, threadIdx.x >> 5, threadIdx.x & 31, 0, blockDim.x >> 5);
    __syncthreads();
    const int64_t total = rows * ldc;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += stride) {
        const int64_t r = u / ldc;
        const int64_t w = u - r * ldc;
        uint32_t word = 0;
#pragma unroll
        for (int j = 0; j < CPW; j++) {
            const int64_t c = w * CPW + j;
            const uint32_t code = (c < cols) ? project_by_table_t<B>(x[r * ldx + c], T, p) : p.zero_code;
            word |= code << (B * j);
        }
        codes[u] = word;  // row-major: r * ldc + w == u
    }
}

template <int B>
static cudaError_t launch_project_b(const float* x, int64_t rows, int64_t cols, int64_t ldx, float alpha,
                                    const float* alpha_dev, const ProjParams& p, uint32_t* codes,
                                    int64_t ldc, bool vec, int sms, cudaStream_t st)
{
    const int threads = 256;
    if (vec) {
        const int64_t units = rows * (ldc >> 2);
        int64_t blocks = (units + threads - 1) / threads;
        // one resident wave: every warp's share is then loaded at once
        static int per_sm = 0;
        if (!per_sm && (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, project_vec_kernel<B>, threads, 0) !=
                            cudaSuccess || per_sm < 1))
            per_sm = 2;
        const int64_t cap = (int64_t)sms * per_sm;
        if (blocks > cap) blocks = cap;
        if (blocks < 1) blocks = 1;
        project_vec_kernel<B><<<(unsigned)blocks, threads, 0, st>>>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc);
    } else {
        const int64_t units = rows * ldc;
        int64_t blocks = (units + threads - 1) / threads;
        const int64_t cap = (int64_t)sms * 8;
        if (blocks > cap) blocks = cap;
        if (blocks < 1) blocks = 1;
        project_any_kernel<B><<<(unsigned)blocks, threads, 0, st>>>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc);
    }
    return cudaGetLastError();
}

cudaError_t launch_project(const float* x, int64_t rows, int64_t cols, int64_t ldx, float alpha,
                           const float* alpha_dev, int b, int k, int is_signed, int rounding,
                           uint32_t* codes, int64_t ldc, cudaStream_t st)
{
    const ProjParams p = make_proj_params(b, k, is_signed, rounding);
    const bool vec = ((reinterpret_cast<uintptr_t>(x) & 15u) == 0) && ((reinterpret_cast<uintptr_t>(codes) & 15u) == 0)
                     && (ldx % 4 == 0) && (ldc % 4 == 0);
    const int sms = device_sm_count();
    switch (b) {
    case 2: return launch_project_b<2>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc, vec, sms, st);
    case 3: return launch_project_b<3>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc, vec, sms, st);
    case 4: return launch_project_b<4>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc, vec, sms, st);
    case 5: return launch_project_b<5>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc, vec, sms, st);
    case 6: return launch_project_b<6>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc, vec, sms, st);
    case 7: return launch_project_b<7>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc, vec, sms, st);
    default: return launch_project_b<8>(x, rows, cols, ldx, alpha, alpha_dev, p, codes, ldc, vec, sms, st);
    }
}

// ------------------------------------------------------------ dequant

__global__ void __launch_bounds__(256)
dequant_kernel(const uint32_t* __restrict__ codes, int64_t rows, int64_t cols, int64_t ldc, float alpha,
               const float* __restrict__ alpha_dev, int b, int k, float* __restrict__ y, int64_t ldy)
{
    const float a = alpha_dev ? __ldg(alpha_dev) : alpha;
    const int cpw = 32 / b;
    const uint32_t mask = (1u << b) - 1u;
    const int64_t total = rows * cols;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        const int64_t r = i / cols;
        const int64_t c = i - r * cols;
        const uint32_t code = (codes[r * ldc + c / cpw] >> (b * (int)(c % cpw))) & mask;
        y[r * ldy + c] = __fmul_rn(a, code_value(code, b, k));
    }
}

cudaError_t launch_dequant(const uint32_t* codes, int64_t rows, int64_t cols, int64_t ldc, float alpha,
                           const float* alpha_dev, int b, int k, float* y, int64_t ldy, cudaStream_t st)
{
    const int threads = 256;
    int64_t blocks = (rows * cols + threads - 1) / threads;
    const int64_t cap = (int64_t)device_sm_count() * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    dequant_kernel<<<(unsigned)blocks, threads, 0, st>>>(codes, rows, cols, ldc, alpha, alpha_dev, b, k, y, ldy);
    return cudaGetLastError();
}

// ------------------------------------------------------- DDA calibration

// Pass 1.  The data is cut into chunks of 32 values.  For each chunk the
// thread computes, from registers, the fp32 chunk mean a_c and
// M2_c = sum (x - a_c)^2; the law of total variance then gives the
// statistics from the sums of a_c, a_c^2 and M2_c with no cancellation
// inside a chunk.  Those sums are carried as unevaluated pairs of fp32
// numbers (hi + lo, error-free transformations: ~48 significant bits), so
// the reduction runs on the fp32 pipes -- GB300 has very little fp64
// throughput -- and fp64 is used only for the final few operations.
// Per-block partials go to the workspace in a fixed layout; the finalize
// kernel adds them in a fixed order, so results do not depend on
// scheduling.
constexpr int kCalThreads = 256;
constexpr int kCalChunk = 32;
constexpr int kCalMaxBlocks = 1023;   // + one 32-byte ticket record = 32 KiB of workspace
constexpr int kCalChunksPerThread = 1;
constexpr int kCalStashMax = 13;      // granules per warp kept in shared memory (4 x 8 x 13 x 512 B = 208 KiB per SM)

// (hi, lo) += x, Knuth's TwoSum with the rounding error kept in lo.
__device__ __forceinline__ void df_add(float& hi, float& lo, float x)
{
    const float s = hi + x;
    const float bp = s - hi;
    const float e = (hi - (s - bp)) + (x - bp);
    hi = s;
    lo += e;
}

// (hi, lo) += (h2, l2)
__device__ __forceinline__ void df_add2(float& hi, float& lo, float h2, float l2)
{
    df_add(hi, lo, h2);
    lo += l2;
}

// (hi, lo) += a * a, exactly split by an fma.
__device__ __forceinline__ void df_add_sq(float& hi, float& lo, float a)
{
    const float p = a * a;
    const float pe = fmaf(a, a, -p);
    df_add(hi, lo, p);
    lo += pe;
}

// Statistics of a set of values split into groups c of n_c values with
// mean a_c and within-group sum of squared deviations M2_c (law of total
// variance): n = sum n_c, s1 = sum n_c a_c, s2 = sum n_c a_c^2,
// s3 = sum M2_c, each sum an fp32 (hi, lo) pair.  One record per block in
// the workspace (32 bytes).
struct __align__(16) CalAcc {
    unsigned long long n;
    float s1h, s1l, s2h, s2l, s3h, s3l;
};
typedef CalAcc CalPartial;

__device__ __forceinline__ void cal_add(CalAcc& A, const CalAcc& B)
{
    A.n += B.n;
    df_add2(A.s1h, A.s1l, B.s1h, B.s1l);
    df_add2(A.s2h, A.s2l, B.s2h, B.s2l);
    df_add2(A.s3h, A.s3l, B.s3h, B.s3l);
}

__device__ __forceinline__ void cal_shfl(CalAcc& A, int o)
{
    CalAcc B;
    B.n = __shfl_xor_sync(0xffffffffu, A.n, o);
    B.s1h = __shfl_xor_sync(0xffffffffu, A.s1h, o); B.s1l = __shfl_xor_sync(0xffffffffu, A.s1l, o);
    B.s2h = __shfl_xor_sync(0xffffffffu, A.s2h, o); B.s2l = __shfl_xor_sync(0xffffffffu, A.s2l, o);
    B.s3h = __shfl_xor_sync(0xffffffffu, A.s3h, o); B.s3l = __shfl_xor_sync(0xffffffffu, A.s3l, o);
    cal_add(A, B);
}

// Sum over the block's threads (every thread passes its share; thread 0
// gets the total).
__device__ __forceinline__ CalAcc cal_block_reduce(CalAcc A)
{
    __shared__ CalAcc sh[kCalThreads / 32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cal_shfl(A, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) sh[warp] = A;
    __syncthreads();
    if (warp == 0) {
        // the warp totals, added pairwise by lanes 0-7 (index order fixed)
        constexpr int kW = kCalThreads / 32;
        static_assert((kW & (kW - 1)) == 0 && kW <= 32, "warp count");
        A = sh[lane < kW ? lane : 0];
#pragma unroll
        for (int o = 1; o < kW; o <<= 1) {
            CalAcc B;
            B.n = __shfl_down_sync(0xffffffffu, A.n, o);
            B.s1h = __shfl_down_sync(0xffffffffu, A.s1h, o); B.s1l = __shfl_down_sync(0xffffffffu, A.s1l, o);
            B.s2h = __shfl_down_sync(0xffffffffu, A.s2h, o); B.s2l = __shfl_down_sync(0xffffffffu, A.s2l, o);
            B.s3h = __shfl_down_sync(0xffffffffu, A.s3h, o); B.s3l = __shfl_down_sync(0xffffffffu, A.s3l, o);
            cal_add(A, B);
        }
    }
    return A;
}

// Sum of the nblocks block records in index order (fp32 pair arithmetic
// across the block: this part runs double precision at a small fraction of
// the fp32 rate); thread 0 gets the total.  Every block that calls it on
// the same records gets the same bits.
__device__ __forceinline__ CalAcc cal_reduce_records(const CalPartial* part, int nblocks)
{
    CalAcc t{0ull, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
    // nblocks <= kCalMaxBlocks < 4 * kCalThreads: at most 4 records a thread,
    // all loaded (two 16-byte loads each, from L2: other blocks wrote them)
    // before any is added
    static_assert(kCalMaxBlocks <= 4 * kCalThreads, "records per thread");
    uint4 w[4][2];
#pragma unroll
    for (int u = 0; u < 4; u++) {
        const int i = threadIdx.x + u * kCalThreads;
        const uint4* q = reinterpret_cast<const uint4*>(part + (i < nblocks ? i : 0));
        w[u][0] = __ldcg(q);
        w[u][1] = __ldcg(q + 1);
    }
#pragma unroll
    for (int u = 0; u < 4; u++) {
        if (threadIdx.x + u * kCalThreads < nblocks) {
            CalAcc r;
            r.n = (unsigned long long)w[u][0].x | ((unsigned long long)w[u][0].y << 32);
            r.s1h = __uint_as_float(w[u][0].z); r.s1l = __uint_as_float(w[u][0].w);
            r.s2h = __uint_as_float(w[u][1].x); r.s2l = __uint_as_float(w[u][1].y);
            r.s3h = __uint_as_float(w[u][1].z); r.s3l = __uint_as_float(w[u][1].w);
            cal_add(t, r);
        }
    }
    return cal_block_reduce(t);
}

// alpha = fl32(alpha* (spread + 1e-7)) from the totals (Sec. III-D); the
// spread is the standard deviation for the symmetric set and the RMS for
// the non-negative one.  fp32 pair arithmetic only (double precision runs
// at a small fraction of the fp32 rate on this part): the mean is kept as a
// pair, so s2 - s1 * mean loses nothing to the rounding of the mean even
// when |mean| >> spread; the final quotient and square root are single
// fp32 operations (relative error ~1e-7).  stats (may be null) gets
// {mean, spread, n}.
__device__ __forceinline__ float cal_alpha(const CalAcc& t, double alpha_star, int is_signed, double* stats)
{
    const float nh = (float)t.n;                                   // n as a pair (exact below 2^48)
    const float nl = (float)(t.n - (unsigned long long)nh);
    float vh, vl;                                                  // the centred (or raw) second moment sum
    // mean = s1 / n to pair precision: quotient, then the remainder's
    // quotient (products with one rounded reciprocal: ~1 ulp)
    const float rn = 1.0f / nh;
    const float mh = t.s1h * rn;
    const float ml = (fmaf(-mh, nh, t.s1h) - mh * nl + t.s1l) * rn;
    if (is_signed) {
        // s1 * mean as a pair (fma gives the product's rounding error exactly)
        const float ph = t.s1h * mh;
        const float pl = fmaf(t.s1h, mh, -ph) + t.s1h * ml + t.s1l * mh;
        // m2 = s3 + (s2 - s1 * mean)
        float dh = t.s2h, dl = t.s2l;
        df_add2(dh, dl, -ph, -pl);
        vh = t.s3h; vl = t.s3l;
        df_add2(vh, vl, dh, dl);
    } else {
        vh = t.s3h; vl = t.s3l;
        df_add2(vh, vl, t.s2h, t.s2l);
    }
    float v = vh + vl;
    if (!(v > 0.0f)) v = 0.0f;
    const float spread = sqrtf(v * rn);
    if (stats) { stats[0] = (double)mh + (double)ml; stats[1] = (double)spread; stats[2] = (double)t.n; }
    return (float)alpha_star * (spread + 1e-7f);
}

// The last block of a pass: totals and alpha.
__device__ void calibrate_finalize_block(const CalPartial* part, int nblocks, double alpha_star, int is_signed,
                                         float* alpha_out, double* stats_out)
{
    const CalAcc t = cal_reduce_records(part, nblocks);
    if (threadIdx.x == 0) *alpha_out = cal_alpha(t, alpha_star, is_signed, stats_out);
}

// Adds one group of CNT values to the accumulators: CNT = 32 keeps its mean
// in the (sa, sq) sums whose weight 32 is applied once at the end; any
// other count is weighted exactly here.
template <int CNT>
__device__ __forceinline__ void cal_group(const float (&v)[CNT], float& sa_h, float& sa_l, float& sq_h, float& sq_l,
                                          CalAcc& A, unsigned long long& full_groups)
{
    float s = 0.0f;
#pragma unroll
    for (int i = 0; i < CNT; i++) s += v[i];
    const float a = s * (1.0f / CNT);                 // CNT is a power of two: exact scaling of the sum
    float m2 = 0.0f;
#pragma unroll
    for (int i = 0; i < CNT; i++) { const float d = v[i] - a; m2 = fmaf(d, d, m2); }
    if (CNT == kCalChunk) {
        df_add(sa_h, sa_l, a);
        df_add_sq(sq_h, sq_l, a);
        full_groups += 1ull;
    } else {
        // n_c * a and n_c * a^2 as exact pairs: split the products with fmas
        const float w = (float)CNT;
        const float p1 = w * a, e1 = fmaf(w, a, -p1);
        df_add(A.s1h, A.s1l, p1); A.s1l += e1;
        const float q = a * a, qe = fmaf(a, a, -q);          // a^2 = q + qe exactly
        const float p2 = w * q, e2 = fmaf(w, q, -p2);         // w q = p2 + e2 exactly
        df_add(A.s2h, A.s2l, p2); A.s2l += e2 + w * qe;
        A.n += (unsigned long long)CNT;
    }
    df_add(A.s3h, A.s3l, m2);
}

// One value as its own group (n_c = 1, M2_c = 0).
__device__ __forceinline__ void cal_single(float a, CalAcc& A)
{
    df_add(A.s1h, A.s1l, a);
    df_add_sq(A.s2h, A.s2l, a);
    A.n += 1ull;
}

// Statistics of this block's share of x, reduced over the block; thread 0
// returns the block's record.  With a stash (this warp's region of shared
// memory) the warp also keeps its first stash_g granules there.  Each warp reads its granules in batches of
// 8 (eight coalesced 16-byte loads per lane in flight); a lane's 32 values
// of a full batch form one group, a shorter batch gives groups of 4 (any
// partition into groups serves the law of total variance).  The n % 128
// values past the last granule (all of x when it is not 16-byte aligned)
// are taken by warp 0 of block 0 one by one.
// `stream_loads` selects evict-first loads (data read once) or default loads
// (data kept in the caches for a second pass).
__device__ __forceinline__ CalAcc cal_block_partial(const float* __restrict__ x, int64_t n, int vec, bool stream_loads,
                                                    float4* stash = nullptr, int stash_g = 0)
{
    const int lane = threadIdx.x & 31;
    const int64_t gran = vec ? n / 128 : 0;
    int64_t g_lo, g_hi;
    warp_granules(gran, g_lo, g_hi);
    CalAcc A{0ull, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
    float sa_h = 0.0f, sa_l = 0.0f;   // sum of a over full groups (weight 32 applied at the end)
    float sq_h = 0.0f, sq_l = 0.0f;   // sum of a^2 over full groups
    unsigned long long full_groups = 0ull;
    const float4* xv = reinterpret_cast<const float4*>(x) + lane;
#pragma unroll 1
    for (int64_t g0 = g_lo; g0 < g_hi; g0 += 8) {
        const int cnt = (int)((g_hi - g0) < 8 ? (g_hi - g0) : 8);
        float4 q[8];
#pragma unroll
        for (int u = 0; u < 8; u++) {
            q[u] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (u < cnt) q[u] = stream_loads ? __ldcs(xv + (g0 + u) * 32) : __ldg(xv + (g0 + u) * 32);
        }
        if (stash) {                                  // keep the warp's first stash_g granules on chip
#pragma unroll
            for (int u = 0; u < 8; u++)
                if (u < cnt && g0 + u - g_lo < stash_g) stash[(g0 + u - g_lo) * 32 + lane] = q[u];
        }
        if (cnt == 8) {
            float v[kCalChunk];
#pragma unroll
            for (int u = 0; u < 8; u++) { v[4 * u] = q[u].x; v[4 * u + 1] = q[u].y; v[4 * u + 2] = q[u].z; v[4 * u + 3] = q[u].w; }
            cal_group<kCalChunk>(v, sa_h, sa_l, sq_h, sq_l, A, full_groups);
        } else {
#pragma unroll
            for (int u = 0; u < 8; u++) {
                if (u < cnt) {
                    const float v[4] = {q[u].x, q[u].y, q[u].z, q[u].w};
                    cal_group<4>(v, sa_h, sa_l, sq_h, sq_l, A, full_groups);
                }
            }
        }
    }
    const int64_t rem0 = gran * 128;
    if (blockIdx.x == 0 && threadIdx.x < 32) {
        for (int64_t i = rem0 + lane; i < n; i += 32) cal_single(x[i], A);
    }
    // full groups carry weight 32: scaling a pair by a power of two is exact
    A.n += full_groups * (unsigned long long)kCalChunk;
    df_add2(A.s1h, A.s1l, sa_h * kCalChunk, sa_l * kCalChunk);
    df_add2(A.s2h, A.s2l, sq_h * kCalChunk, sq_l * kCalChunk);
    return cal_block_reduce(A);
}

// The statistics pass of the fused kernel on a flat tensor: each warp's
// first min(granules, stash_g) granules -- a contiguous byte range, laid out
// in the stash exactly as in memory -- arrive by one bulk copy per warp
// (every byte in flight at once, no registers held), the rest by loads as
// in cal_block_partial; the statistics of the stashed granules are then
// read from shared memory.  A copy that does not complete within the wait
// limit sets *copy_timeout (after a second bounded wait for the copy).
__device__ __forceinline__ CalAcc cal_block_partial_bulk(const float* __restrict__ x, int64_t n, float4* stash,
                                                         int stash_g, int* copy_timeout)
{
    __shared__ uint64_t wbar[kCalThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t gran = n / 128;
    int64_t g_lo, g_hi;
    warp_granules(gran, g_lo, g_hi);
    const int ns = (int)((g_hi - g_lo) < stash_g ? (g_hi - g_lo) : stash_g);
    if (lane == 0 && ns > 0) {
        mbar_init(&wbar[warp], 1);
        fence_mbar_init();
        mbar_arrive_expect_tx(&wbar[warp], (uint32_t)ns * 512u);
        bulk_copy_g2s(stash, x + g_lo * 128, (uint32_t)ns * 512u, &wbar[warp]);
    }
    __syncwarp();
    CalAcc A{0ull, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
    float sa_h = 0.0f, sa_l = 0.0f, sq_h = 0.0f, sq_l = 0.0f;
    unsigned long long full_groups = 0ull;
    auto batch = [&](const float4 (&q)[8], int cnt) {
        if (cnt == 8) {
            float v[kCalChunk];
#pragma unroll
            for (int u = 0; u < 8; u++) { v[4 * u] = q[u].x; v[4 * u + 1] = q[u].y; v[4 * u + 2] = q[u].z; v[4 * u + 3] = q[u].w; }
            cal_group<kCalChunk>(v, sa_h, sa_l, sq_h, sq_l, A, full_groups);
        } else {
#pragma unroll
            for (int u = 0; u < 8; u++) {
                if (u < cnt) {
                    const float v[4] = {q[u].x, q[u].y, q[u].z, q[u].w};
                    cal_group<4>(v, sa_h, sa_l, sq_h, sq_l, A, full_groups);
                }
            }
        }
    };
    // granules past the stash: loads, while the copy is in flight
    const float4* xv = reinterpret_cast<const float4*>(x) + lane;
#pragma unroll 1
    for (int64_t g0 = g_lo + ns; g0 < g_hi; g0 += 8) {
        const int cnt = (int)((g_hi - g0) < 8 ? (g_hi - g0) : 8);
        float4 q[8];
#pragma unroll
        for (int u = 0; u < 8; u++) q[u] = (u < cnt) ? __ldcs(xv + (g0 + u) * 32) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        batch(q, cnt);
    }
    if (ns > 0) {
        if (!mbar_wait_bounded(&wbar[warp], 0u, 2000000000ull)) {
            if (lane == 0) *copy_timeout = 1;
            (void)mbar_wait_bounded(&wbar[warp], 0u, 1000000000ull);
        }
#pragma unroll 1
        for (int g0 = 0; g0 < ns; g0 += 8) {
            const int cnt = (ns - g0) < 8 ? (ns - g0) : 8;
            float4 q[8];
#pragma unroll
            for (int u = 0; u < 8; u++) q[u] = (u < cnt) ? stash[(g0 + u) * 32 + lane] : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            batch(q, cnt);
        }
    }
    const int64_t rem0 = gran * 128;
    if (blockIdx.x == 0 && threadIdx.x < 32) {
        for (int64_t i = rem0 + lane; i < n; i += 32) cal_single(x[i], A);
    }
    A.n += full_groups * (unsigned long long)kCalChunk;
    df_add2(A.s1h, A.s1l, sa_h * kCalChunk, sa_l * kCalChunk);
    df_add2(A.s2h, A.s2l, sq_h * kCalChunk, sq_l * kCalChunk);
    return cal_block_reduce(A);
}

// Workspace head record: the ticket counter, the release flag of the fused
// kernel's grid barrier, and the alpha it publishes.
// All three words are zero when a launch starts and zero again when it
// ends: the last block to leave resets them (no memset between calls).
struct CalSync {
    unsigned int ticket;          // blocks that have published their record
    unsigned int depart;          // fused kernel: blocks past the release
    unsigned long long release;   // fused kernel: (1 << 32) | bits(alpha) once alpha is known
    unsigned int pad[4];
};
static_assert(sizeof(CalSync) == sizeof(CalPartial), "head record is one partial record wide");

// Publishes the block's record and takes a ticket (thread 0); true for the
// last block.  The ticket's read-modify-write has release and acquire
// semantics at GPU scope: it releases this block's record, and the last
// block's thread 0 acquires every earlier record through it; that block's
// other threads are ordered after it by the CTA barrier that follows, and
// read the records from L2 (cal_reduce_records).
__device__ __forceinline__ bool cal_arrive(CalPartial* part, const CalAcc& mine, CalSync* sync)
{
    part[blockIdx.x] = mine;
    unsigned int old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(&sync->ticket) : "memory");
    return old == gridDim.x - 1;
}

// Leaving the fused kernel's grid barrier, at the end of the block's work
// (every block read the release word long before): the last block out
// returns the sync words to zero.
__device__ __forceinline__ void cal_depart(CalSync* sync)
{
    if (threadIdx.x == 0 && atomicAdd(&sync->depart, 1u) == gridDim.x - 1) {
        sync->ticket = 0u;
        sync->release = 0ull;
        sync->depart = 0u;
    }
}

// One launch: every block writes its partial record; the block that takes
// the last ticket adds all records in index order, finalises alpha and
// returns the ticket to zero, so the workspace needs zeroing only once,
// before its first use (never between calls).
__global__ void __launch_bounds__(kCalThreads, 4)
calibrate_pass1_kernel(const float* __restrict__ x, int64_t n, int vec, CalPartial* __restrict__ part,
                       CalSync* __restrict__ sync, double alpha_star, int is_signed,
                       float* __restrict__ alpha_out, double* __restrict__ stats_out)
{
    const CalPartial mine = cal_block_partial(x, n, vec, true);
    __shared__ bool is_last;
    if (threadIdx.x == 0) is_last = cal_arrive(part, mine, sync);
    __syncthreads();
    if (is_last) {
        calibrate_finalize_block(part, gridDim.x, alpha_star, is_signed, alpha_out, stats_out);
        if (threadIdx.x == 0) sync->ticket = 0u;      // every block has counted itself: ready for the next call
    }
}

// ------------------------------------------ empirical DDA histogram

// Histogram of |t| for the DDA of the data's own density: t = (x - mean) /
// sigma (signed formats) or x / rms (unsigned), bins of width t_max / nbins
// over [0, t_max), values past t_max in the last bin, NaN skipped.  The bin
// of a value is fixed by these fp32 operations, each rounded to nearest:
// scale = nbins / (t_max * spread), u = |x - mean| * scale, bin = floor(u).
// Each block counts into shared memory and adds its counts to the device
// array (integer additions: the result does not depend on their order).
__global__ void __launch_bounds__(256)
dda_histogram_kernel(const float* __restrict__ x, int64_t n, int is_signed, const double* __restrict__ stats,
                     int nbins, float t_max, unsigned long long* __restrict__ counts)
{
    extern __shared__ unsigned int hist[];
    for (int i = threadIdx.x; i < nbins; i += blockDim.x) hist[i] = 0u;
    griddep_wait();                                   // stats may come from the previous launch
    __syncthreads();
    const float m = is_signed ? (float)__ldg(stats) : 0.0f;
    const float sp = (float)__ldg(stats + 1);
    const float nb = (float)nbins;
    const float scale = __fdiv_rn(nb, __fmul_rn(t_max, sp));
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const float v = __ldcs(x + i);
        if (v != v) continue;
        const float u = __fmul_rn(fabsf(__fsub_rn(v, m)), scale);
        const int bin = (u < nb) ? (int)u : ((u >= nb) ? nbins - 1 : 0);   // NaN (0 * inf): bin 0
        atomicAdd(&hist[bin], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nbins; i += blockDim.x)
        if (hist[i]) atomicAdd(counts + i, (unsigned long long)hist[i]);
}

cudaError_t launch_dda_histogram(const float* x, int64_t n, int is_signed, const double* stats, int nbins,
                                 float t_max, unsigned long long* counts, cudaStream_t st)
{
    cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(unsigned long long) * (size_t)nbins, st);
    if (e != cudaSuccess) return e;
    int64_t blocks = (n + 255) / 256;
    const int64_t cap = (int64_t)device_sm_count() * 4;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    dda_histogram_kernel<<<(unsigned)blocks, 256, sizeof(unsigned int) * (size_t)nbins, st>>>(
        x, n, is_signed, stats, nbins, t_max, counts);
    return cudaGetLastError();
}

// ------------------------------------- DDA-calibrated projection, fused

// Calibration and projection of the same tensor in one launch of one
// resident wave (all blocks co-resident).  Phase 1 reduces the statistics with loads that
// leave x in L2; the last block to arrive finalises alpha, publishes it and
// raises the release flag, which every other block waits for (bounded).
// Phase 2 projects x, now read from L2, with that alpha.
template <int B>
__global__ void __launch_bounds__(kCalThreads, 4)
calibrate_project_kernel(const float* __restrict__ x, int64_t rows, int64_t cols, CalPartial* __restrict__ part,
                         CalSync* __restrict__ sync, double alpha_star, ProjParams p, float* __restrict__ alpha_out,
                         double* __restrict__ stats_out, uint32_t* __restrict__ codes, int64_t ldc,
                         int* __restrict__ status, int stash_g, unsigned long long wait_ns)
{
    // stash: stash_g granules (512 bytes each) per warp of dynamic shared memory
    extern __shared__ float4 stash_all[];
    float4* stash = stash_g > 0 ? stash_all + (size_t)(threadIdx.x >> 5) * stash_g * 32 : nullptr;
    griddep_wait();                                   // x and the workspace may be in use by the previous launch
    constexpr int CPW = 32 / B;
    constexpr int L = 1 << (B - 1);
    const int64_t n = rows * cols;
    const bool flat = B == 4 && cols % 8 == 0 && ldc * 8 == cols;
    __shared__ int copy_timeout, timed_out;
    __shared__ float s_alpha;
    __shared__ float T[L];
    if (threadIdx.x == 0) { copy_timeout = 0; timed_out = 0; }
    __syncthreads();
    const CalPartial mine = (flat && stash) ? cal_block_partial_bulk(x, n, stash, stash_g, &copy_timeout)
                                            : cal_block_partial(x, n, 1, false, nullptr, 0);
    // Grid barrier: every block publishes its record; the block that takes
    // the last ticket sums the records and publishes alpha in the release
    // word (one 64-bit store: flag and value together), which the others
    // wait for (bounded).
    __shared__ bool is_last;
    if (threadIdx.x == 0) is_last = cal_arrive(part, mine, sync);
    __syncthreads();
    if (is_last) {
        const CalAcc tot = cal_reduce_records(part, gridDim.x);
        if (threadIdx.x == 0) {
            double st[3];
            const float al = cal_alpha(tot, alpha_star, p.is_signed, stats_out ? st : nullptr);
            // alpha travels in the release word itself: nothing else has to
            // be visible to the other blocks first
            atomicExch(&sync->release, (1ull << 32) | (unsigned long long)__float_as_uint(al));
            s_alpha = al;
            *alpha_out = al;
            if (stats_out) { stats_out[0] = st[0]; stats_out[1] = st[1]; stats_out[2] = st[2]; }
        }
    } else if (threadIdx.x == 0) {
        const volatile unsigned long long* rel = &sync->release;
        const uint64_t t0 = globaltimer_ns();
        unsigned long long w = *rel;
        while ((w >> 32) == 0ull) {
            // every poll is an L2 round trip, so reading the clock each time costs nothing extra
            if (globaltimer_ns() - t0 > wait_ns) { timed_out = 1; break; }
            __nanosleep(32);
            w = *rel;
        }
        s_alpha = __uint_as_float((unsigned int)(w & 0xffffffffull));
    }
    __syncthreads();
    if (timed_out || copy_timeout) {
        if (threadIdx.x == 0) record_status(status, ESB_ERR_TIMEOUT);
        if (!timed_out) cal_depart(sync);
        return;
    }
    const float a = s_alpha;
    // every block is resident and past the barrier: a
    // dependent grid may take the SMs as these blocks finish
    griddep_launch_dependents();
    build_thresholds(T, p, a, threadIdx.x >> 5, threadIdx.x & 31, 0, blockDim.x >> 5);
    __syncthreads();
    Thr7 t7;
    if (B == 4) {
#pragma unroll
        for (int i = 0; i < 7; i++) t7.t[i] = T[i];
        if (flat) {                                     // flat codes: the statistics pass's granules
            if (p.is_signed) project_flat_b4<true, true>(x, n, t7, p.k, codes, stash, stash_g);
            else project_flat_b4<false, true>(x, n, t7, p.k, codes, stash, stash_g);
            cal_depart(sync);
            return;
        }
    }
    const int64_t upr = ldc >> 2;
    const int64_t total = rows * upr;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += stride) {
        const int64_t r = (rows == 1) ? 0 : u / upr;
        const int64_t w4 = u - r * upr;
        const int64_t c0 = w4 * (4 * CPW);
        const float* xr = x + r * cols + c0;
        uint32_t out[4];
        if (c0 + 4 * CPW <= cols) {
            float v[4 * CPW];
#pragma unroll
            for (int i = 0; i < CPW; i++) {
                const float4 t = __ldcs(reinterpret_cast<const float4*>(xr) + i);
                v[4 * i + 0] = t.x; v[4 * i + 1] = t.y; v[4 * i + 2] = t.z; v[4 * i + 3] = t.w;
            }
            if (B == 4) {
#pragma unroll
                for (int w = 0; w < 4; w++) {
                    uint32_t J = 0u, S = 0u;
#pragma unroll
                    for (int j = 0; j < 8; j++) {
                        const float xv = v[w * 8 + j];
                        J |= bucket7(p.is_signed ? fabsf(xv) : xv, t7) << (4 * j);
                        S |= ((__float_as_uint(xv) >> 31) & (uint32_t)p.is_signed) << (4 * j + 3);
                    }
                    out[w] = codes8_b4(J, S, p.k);
                }
            } else {
#pragma unroll
                for (int w = 0; w < 4; w++) {
                    uint32_t word = 0;
#pragma unroll
                    for (int j = 0; j < CPW; j++) word |= project_by_table_t<B>(v[w * CPW + j], T, p) << (B * j);
                    out[w] = word;
                }
            }
        } else {
#pragma unroll
            for (int w = 0; w < 4; w++) {
                uint32_t word = 0;
#pragma unroll
                for (int j = 0; j < CPW; j++) {
                    const int64_t c = c0 + w * CPW + j;
                    const uint32_t code = (c < cols) ? project_by_table_t<B>(__ldcs(xr + w * CPW + j), T, p) : p.zero_code;
                    word |= code << (B * j);
                }
                out[w] = word;
            }
        }
        __stcs(reinterpret_cast<uint4*>(codes + r * ldc + (w4 << 2)), make_uint4(out[0], out[1], out[2], out[3]));
    }
    cal_depart(sync);
}

// These kernels use almost no shared memory: ask for the largest L1 (the
// fused kernel's second pass re-reads x, which then stays on chip).
template <class F>
static void prefer_l1(F* kernel)
{
    (void)cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 0);
}

// Grid: one chunk per thread up to one resident wave (4 blocks of 256
// threads per SM at this kernel's register use), at most kCalMaxBlocks.
int calibrate_blocks(int64_t n)
{
    const int64_t per_block = (int64_t)kCalThreads * kCalChunk * kCalChunksPerThread;
    int64_t g = (n + per_block - 1) / per_block;
    const int64_t wave = (int64_t)device_sm_count() * 4;
    if (g > wave) g = wave;
    if (g > kCalMaxBlocks) g = kCalMaxBlocks;
    if (g < 1) g = 1;
    return (int)g;
}

// Workspace: [ticket record (32 B)][one CalPartial per block].
size_t calibrate_workspace_bytes(int64_t n)
{
    return sizeof(CalPartial) + (size_t)calibrate_blocks(n) * sizeof(CalPartial);
}

cudaError_t launch_calibrate(const float* x, int64_t n, int is_signed, double alpha_star, void* workspace,
                             float* alpha_out, double* stats_out, cudaStream_t st)
{
    const int g = calibrate_blocks(n);
    const int vec = ((reinterpret_cast<uintptr_t>(x) & 15u) == 0) ? 1 : 0;
    CalSync* sync = static_cast<CalSync*>(workspace);
    CalPartial* part = static_cast<CalPartial*>(workspace) + 1;
    static bool l1_set = false;
    if (!l1_set) { prefer_l1(calibrate_pass1_kernel); l1_set = true; }
    calibrate_pass1_kernel<<<g, kCalThreads, 0, st>>>(x, n, vec, part, sync, alpha_star, is_signed, alpha_out,
                                                        stats_out);
    return cudaGetLastError();
}

template <int B>
static cudaError_t launch_calibrate_project_b(const float* x, int64_t rows, int64_t cols, const ProjParams& p,
                                              double alpha_star, void* workspace, float* alpha_out, double* stats_out,
                                              uint32_t* codes, int64_t ldc, cudaStream_t st, bool* launched)
{
    *launched = false;
    const int64_t n = rows * cols;
    const int sms = device_sm_count();
    int64_t g = calibrate_blocks(n);                  // up to 4 blocks per SM
    // Stash (flat 4-bit codes): every warp keeps its granules in shared
    // memory between the two passes, up to kCalStashMax granules (4 blocks
    // of 8 warps x kCalStashMax x 512 bytes fit one SM); any rest is re-read.
    const bool flat = B == 4 && cols % 8 == 0 && ldc * 8 == cols;
    int stash_g = 0;
    if (flat) {
        const int64_t nwarps = g * (kCalThreads / 32);
        const int64_t gs = (n / 128 + nwarps - 1) / nwarps;
        stash_g = (int)(gs < kCalStashMax ? gs : kCalStashMax);
    }
    const size_t smem = (size_t)stash_g * 512 * (kCalThreads / 32);
    static bool configured = false;
    if (!configured) {
        cudaError_t e0 = cudaFuncSetAttribute(calibrate_project_kernel<B>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              kCalStashMax * 512 * (kCalThreads / 32));
        if (e0 != cudaSuccess) return e0;
        (void)cudaFuncSetAttribute(calibrate_project_kernel<B>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        configured = true;
    }
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, calibrate_project_kernel<B>, kCalThreads, smem);
    if (e != cudaSuccess) return e;
    const int64_t co_resident = (int64_t)per_sm * sms;
    if (co_resident < 1) return cudaSuccess;
    if (g > co_resident) g = co_resident;             // a partial stash still works: the rest is re-read
    CalSync* sync = static_cast<CalSync*>(workspace);
    CalPartial* part = static_cast<CalPartial*>(workspace) + 1;
    int* status = device_status_ptr();
    // Limit of the grid barrier's wait: 2 s.  ESB_BARRIER_WAIT_NS in the
    // environment (read at every launch) can only shorten it; tests use that
    // to make the wait run out.  The wait sits after every bulk copy of the
    // block has landed, so a block that gives up leaves nothing in flight.
    unsigned long long wait_ns = 2000000000ull;
    if (const char* v = getenv("ESB_BARRIER_WAIT_NS")) {
        const unsigned long long w = strtoull(v, nullptr, 10);
        if (w > 0 && w < wait_ns) wait_ns = w;
    }
    void* args[] = {(void*)&x, (void*)&rows, (void*)&cols, (void*)&part, (void*)&sync, (void*)&alpha_star,
                    (void*)&p, (void*)&alpha_out, (void*)&stats_out, (void*)&codes, (void*)&ldc, (void*)&status,
                    (void*)&stash_g, (void*)&wait_ns};
    // The grid is one resident wave (sized by the occupancy query above), so
    // every block becomes resident once the previous kernel of the stream
    // has left the SMs; the grid barrier's wait is bounded and reports
    // ESB_ERR_TIMEOUT should another tenant's work keep SMs occupied.  The
    // launch is programmatic (it may overlap the previous kernel's end; the
    // kernel's griddep_wait orders its reads and writes after it) rather
    // than cooperative: a cooperative launch waits for the whole device to
    // drain first.  ESB_FUSED_COOPERATIVE=1 selects the cooperative launch.
    static const int coop = [] {
        const char* v = getenv("ESB_FUSED_COOPERATIVE");
        return (v && v[0] == '1') ? 1 : 0;
    }();
    if (coop) {
        e = cudaLaunchCooperativeKernel((const void*)calibrate_project_kernel<B>, dim3((unsigned)g), dim3(kCalThreads),
                                        args, smem, st);
    } else {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)g);
        cfg.blockDim = dim3(kCalThreads);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelExC(&cfg, (const void*)calibrate_project_kernel<B>, args);
    }
    *launched = true;
    return e;
}

cudaError_t launch_calibrate_project(const float* x, int64_t rows, int64_t cols, int b, int k, int is_signed,
                                     int rounding, double alpha_star, void* workspace, float* alpha_out,
                                     double* stats_out, uint32_t* codes, int64_t ldc, cudaStream_t st)
{
    const bool vec = ((reinterpret_cast<uintptr_t>(x) & 15u) == 0) && ((reinterpret_cast<uintptr_t>(codes) & 15u) == 0)
                     && (cols % 4 == 0) && (ldc % 4 == 0);
    bool launched = false;
    cudaError_t e = cudaSuccess;
    if (vec) {
        const ProjParams p = make_proj_params(b, k, is_signed, rounding);
        switch (b) {
        case 2: e = launch_calibrate_project_b<2>(x, rows, cols, p, alpha_star, workspace, alpha_out, stats_out, codes, ldc, st, &launched); break;
        case 3: e = launch_calibrate_project_b<3>(x, rows, cols, p, alpha_star, workspace, alpha_out, stats_out, codes, ldc, st, &launched); break;
        case 4: e = launch_calibrate_project_b<4>(x, rows, cols, p, alpha_star, workspace, alpha_out, stats_out, codes, ldc, st, &launched); break;
        case 5: e = launch_calibrate_project_b<5>(x, rows, cols, p, alpha_star, workspace, alpha_out, stats_out, codes, ldc, st, &launched); break;
        case 6: e = launch_calibrate_project_b<6>(x, rows, cols, p, alpha_star, workspace, alpha_out, stats_out, codes, ldc, st, &launched); break;
        case 7: e = launch_calibrate_project_b<7>(x, rows, cols, p, alpha_star, workspace, alpha_out, stats_out, codes, ldc, st, &launched); break;
        default: e = launch_calibrate_project_b<8>(x, rows, cols, p, alpha_star, workspace, alpha_out, stats_out, codes, ldc, st, &launched); break;
        }
        if (e != cudaSuccess || launched) return e;
    }
    // General layouts: the two-launch form.
    e = launch_calibrate(x, rows * cols, is_signed, alpha_star, workspace, alpha_out, stats_out, st);
    if (e != cudaSuccess) return e;
    return launch_project(x, rows, cols, cols, 0.0f, alpha_out, b, k, is_signed, rounding, codes, ldc, st);
}

// ------------------------------------------- calibration without workspace

// Scratch of esb_calibrate_dda_noalloc: room for the ticket record and the
// partial record of every block the reduction can launch
// ((kCalMaxBlocks + 1) x 32 bytes = 32 KiB).  It is
// a file-scope device array, so it exists on every GPU that loads the
// library until the process exits, and every call of the variant shares it.
static_assert(sizeof(CalPartial) == 32, "partial record layout");
static __device__ __align__(256) unsigned char g_cal_noalloc_scratch[(kCalMaxBlocks + 1) * 32];

size_t calibrate_noalloc_capacity() { return sizeof(g_cal_noalloc_scratch); }

// The host-side name of the array is only a stand-in, never a device
// address: the address is looked up with the device current and cached per
// device and context (symbol_address).  The lookup allocates nothing.
static cudaError_t lookup_noalloc_scratch(void** p)
{
    return cudaGetSymbolAddress(p, g_cal_noalloc_scratch);
}

static cudaError_t noalloc_scratch_address(void** out)
{
    static SymbolCache cache;
    return symbol_address(lookup_noalloc_scratch, cache, out);
}

cudaError_t launch_calibrate_noalloc(const float* x, int64_t n, int is_signed, double alpha_star, float* alpha_out,
                                     double* stats_out, cudaStream_t st)
{
    if (calibrate_workspace_bytes(n) > sizeof(g_cal_noalloc_scratch)) return cudaErrorInvalidValue;
    void* ws = nullptr;
    cudaError_t e = noalloc_scratch_address(&ws);
    if (e != cudaSuccess) return e;
    // The array starts zero-filled and every call leaves its head record
    // zero again; every partial record is written before it is read.
    return launch_calibrate(x, n, is_signed, alpha_star, ws, alpha_out, stats_out, st);
}

}  // namespace esb
