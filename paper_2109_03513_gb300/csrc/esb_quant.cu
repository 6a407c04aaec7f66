// esb_quant.cu -- HBM-bound element-wise kernels of libesb:
//   * projection of fp32 tensors onto packed ESB codes (Eq. cheap_projection
//     with the shift-and-round projection of Eq. fast_projection),
//   * dequantisation (Sec. IV-A, Eq. q),
//   * DDA calibration statistics and alpha (Sec. III-D).
#include <cstdint>
#include <mutex>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

// ----------------------------------------------------------- projection

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
    __shared__ float T[L];
    const float a = alpha_dev ? __ldg(alpha_dev) : alpha;
    build_thresholds(T, p, a, threadIdx.x >> 5, threadIdx.x & 31, 0, blockDim.x >> 5);
    __syncthreads();
    Thr7 t7;
    if (B == 4) {
#pragma unroll
        for (int i = 0; i < 7; i++) t7.t[i] = T[i];
    }
    auto proj = [&](float v) -> uint32_t { return B == 4 ? project_by_thr7(v, t7, p) : project_by_table(v, T, p); };
    const int64_t upr = ldc >> 2;                 // 4-word units per row
    const int64_t total = rows * upr;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += stride) {
        const int64_t r = (rows == 1) ? 0 : u / upr;
        const int64_t w4 = u - r * upr;
        const int64_t c0 = w4 * (4 * CPW);
        const float* xr = x + r * ldx + c0;
        uint32_t out[4];
        if (c0 + 4 * CPW <= cols) {
            float v[4 * CPW];
#pragma unroll
            for (int i = 0; i < CPW; i++) {
                const float4 t = __ldcs(reinterpret_cast<const float4*>(xr) + i);
                v[4 * i + 0] = t.x; v[4 * i + 1] = t.y; v[4 * i + 2] = t.z; v[4 * i + 3] = t.w;
            }
            if (B == 4) {
                // buckets of |x| (x for the unsigned set: negatives land in bucket 0)
#pragma unroll
                for (int w = 0; w < 4; w++) {
                    uint32_t J = 0u, S = 0u;
#pragma unroll
                    for (int j = 0; j < 8; j++) {
                        const float xv = v[w * 8 + j];
                        const uint32_t u = __float_as_uint(xv);
                        J |= bucket7(p.is_signed ? fabsf(xv) : xv, t7) << (4 * j);
                        S |= ((u >> 31) & (uint32_t)p.is_signed) << (4 * j + 3);
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
#pragma unroll
            for (int w = 0; w < 4; w++) {
                uint32_t word = 0;
#pragma unroll
                for (int j = 0; j < CPW; j++) {
                    const int64_t c = c0 + w * CPW + j;
                    const uint32_t code = (c < cols) ? proj(__ldcs(xr + w * CPW + j)) : p.zero_code;
                    word |= code << (B * j);
                }
                out[w] = word;
            }
        }
        __stcs(reinterpret_cast<uint4*>(codes + r * ldc + (w4 << 2)), make_uint4(out[0], out[1], out[2], out[3]));
    }
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
            const uint32_t code = (c < cols) ? project_by_table(x[r * ldx + c], T, p) : p.zero_code;
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
        const int64_t cap = (int64_t)sms * 8;
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
constexpr int kCalMaxBlocks = 1024;
constexpr int kCalChunksPerThread = 1;

struct CalPartial {
    double n, s1, s2, s3;   // sum n_c, sum n_c a_c, sum n_c a_c^2, sum M2_c
};

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

struct CalAcc {
    unsigned long long n;
    float s1h, s1l, s2h, s2l, s3h, s3l;
};

__device__ __forceinline__ void cal_shfl(CalAcc& A, int o)
{
    const unsigned long long n = __shfl_xor_sync(0xffffffffu, A.n, o);
    const float a1 = __shfl_xor_sync(0xffffffffu, A.s1h, o), b1 = __shfl_xor_sync(0xffffffffu, A.s1l, o);
    const float a2 = __shfl_xor_sync(0xffffffffu, A.s2h, o), b2 = __shfl_xor_sync(0xffffffffu, A.s2l, o);
    const float a3 = __shfl_xor_sync(0xffffffffu, A.s3h, o), b3 = __shfl_xor_sync(0xffffffffu, A.s3l, o);
    A.n += n;
    df_add2(A.s1h, A.s1l, a1, b1);
    df_add2(A.s2h, A.s2l, a2, b2);
    df_add2(A.s3h, A.s3l, a3, b3);
}

__global__ void __launch_bounds__(kCalThreads)
calibrate_pass1_kernel(const float* __restrict__ x, int64_t n, int vec, CalPartial* __restrict__ part)
{
    const int64_t nfull = n / kCalChunk;
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t nthreads = (int64_t)gridDim.x * blockDim.x;
    CalAcc A{0ull, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
    float sa_h = 0.0f, sa_l = 0.0f;   // sum of a over full chunks (weight 32 applied at the end)
    float sq_h = 0.0f, sq_l = 0.0f;   // sum of a^2 over full chunks
    unsigned long long cnt = 0ull;
#pragma unroll 2
    for (int64_t c = tid; c < nfull; c += nthreads) {
        float v[kCalChunk];
        const float* xc = x + c * kCalChunk;
        if (vec) {
#pragma unroll
            for (int i = 0; i < kCalChunk / 4; i++) {
                const float4 t = __ldcs(reinterpret_cast<const float4*>(xc) + i);
                v[4 * i] = t.x; v[4 * i + 1] = t.y; v[4 * i + 2] = t.z; v[4 * i + 3] = t.w;
            }
        } else {
#pragma unroll
            for (int i = 0; i < kCalChunk; i++) v[i] = __ldcs(xc + i);
        }
        float s = 0.0f;
#pragma unroll
        for (int i = 0; i < kCalChunk; i++) s += v[i];
        const float a = s * (1.0f / kCalChunk);
        float m2 = 0.0f;
#pragma unroll
        for (int i = 0; i < kCalChunk; i++) { const float d = v[i] - a; m2 = fmaf(d, d, m2); }
        df_add(sa_h, sa_l, a);
        df_add_sq(sq_h, sq_l, a);
        df_add(A.s3h, A.s3l, m2);
        cnt += 1ull;
    }
    // full chunks carry weight 32: scaling a pair by a power of two is exact
    A.n = cnt * (unsigned long long)kCalChunk;
    A.s1h = sa_h * kCalChunk; A.s1l = sa_l * kCalChunk;
    A.s2h = sq_h * kCalChunk; A.s2l = sq_l * kCalChunk;
    // The ragged tail (< 32 values) is one weighted chunk, owned by thread 0.
    const int64_t tail0 = nfull * kCalChunk;
    if (tid == 0 && tail0 < n) {
        const int nt = (int)(n - tail0);
        float s = 0.0f;
        for (int i = 0; i < nt; i++) s += x[tail0 + i];
        const float a = s / (float)nt;
        float m2 = 0.0f;
        for (int i = 0; i < nt; i++) { const float d = x[tail0 + i] - a; m2 = fmaf(d, d, m2); }
        // n_t * a and n_t * a^2 as exact pairs: split the products with fmas
        const float w = (float)nt;
        const float p1 = w * a, e1 = fmaf(w, a, -p1);
        df_add(A.s1h, A.s1l, p1); A.s1l += e1;
        const float q = a * a, qe = fmaf(a, a, -q);          // a^2 = q + qe exactly
        const float p2 = w * q, e2 = fmaf(w, q, -p2);         // w q = p2 + e2 exactly
        df_add(A.s2h, A.s2l, p2); A.s2l += e2 + w * qe;
        df_add(A.s3h, A.s3l, m2);
        A.n += (unsigned long long)nt;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cal_shfl(A, o);
    __shared__ CalAcc sh[kCalThreads / 32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) sh[warp] = A;
    __syncthreads();
    if (threadIdx.x == 0) {
        CalAcc t = sh[0];
        for (int w = 1; w < kCalThreads / 32; w++) {
            t.n += sh[w].n;
            df_add2(t.s1h, t.s1l, sh[w].s1h, sh[w].s1l);
            df_add2(t.s2h, t.s2l, sh[w].s2h, sh[w].s2l);
            df_add2(t.s3h, t.s3l, sh[w].s3h, sh[w].s3l);
        }
        part[blockIdx.x] = CalPartial{(double)t.n, (double)t.s1h + (double)t.s1l, (double)t.s2h + (double)t.s2l,
                                      (double)t.s3h + (double)t.s3l};
    }
}

// Pass 2 (one block): fixed-order sum of the block partials, then
// mean = s1/n, M2 = s3 + (s2 - s1^2/n), sigma = sqrt(M2/n) (signed formats)
// or rms = sqrt((s3 + s2)/n) (unsigned formats), alpha = fl32(alpha* (spread + 1e-7)).
__global__ void __launch_bounds__(kCalThreads)
calibrate_finalize_kernel(const CalPartial* __restrict__ part, int nblocks, double alpha_star, int is_signed,
                          float* __restrict__ alpha_out, double* __restrict__ stats_out)
{
    __shared__ CalPartial sh[kCalThreads];
    CalPartial t{0.0, 0.0, 0.0, 0.0};
    for (int i = threadIdx.x; i < nblocks; i += kCalThreads) {
        t.n += part[i].n; t.s1 += part[i].s1; t.s2 += part[i].s2; t.s3 += part[i].s3;
    }
    sh[threadIdx.x] = t;
    __syncthreads();
    for (int h = kCalThreads / 2; h > 0; h >>= 1) {
        if (threadIdx.x < h) {
            sh[threadIdx.x].n += sh[threadIdx.x + h].n;
            sh[threadIdx.x].s1 += sh[threadIdx.x + h].s1;
            sh[threadIdx.x].s2 += sh[threadIdx.x + h].s2;
            sh[threadIdx.x].s3 += sh[threadIdx.x + h].s3;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        const CalPartial r = sh[0];
        const double mean = r.s1 / r.n;
        double spread;
        if (is_signed) {
            double m2 = r.s3 + (r.s2 - r.s1 * mean);
            if (m2 < 0.0) m2 = 0.0;
            spread = sqrt(m2 / r.n);
        } else {
            spread = sqrt((r.s3 + r.s2) / r.n);
        }
        *alpha_out = (float)(alpha_star * (spread + 1e-7));
        if (stats_out) { stats_out[0] = mean; stats_out[1] = spread; stats_out[2] = r.n; }
    }
}

int calibrate_blocks(int64_t n)
{
    const int64_t per_block = (int64_t)kCalThreads * kCalChunk * kCalChunksPerThread;
    int64_t g = (n + per_block - 1) / per_block;
    if (g > kCalMaxBlocks) g = kCalMaxBlocks;
    if (g < 1) g = 1;
    return (int)g;
}

size_t calibrate_workspace_bytes(int64_t n)
{
    return (size_t)calibrate_blocks(n) * sizeof(CalPartial);
}

cudaError_t launch_calibrate(const float* x, int64_t n, int is_signed, double alpha_star, void* workspace,
                             float* alpha_out, double* stats_out, cudaStream_t st)
{
    const int g = calibrate_blocks(n);
    const int vec = ((reinterpret_cast<uintptr_t>(x) & 15u) == 0) ? 1 : 0;
    CalPartial* part = static_cast<CalPartial*>(workspace);
    calibrate_pass1_kernel<<<g, kCalThreads, 0, st>>>(x, n, vec, part);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    calibrate_finalize_kernel<<<1, kCalThreads, 0, st>>>(part, g, alpha_star, is_signed, alpha_out, stats_out);
    return cudaGetLastError();
}

// ------------------------------------------- calibration without workspace

// Scratch of esb_calibrate_dda_noalloc: room for the partial record of every
// block the reduction can launch (kCalMaxBlocks x 32 bytes = 32 KiB).  It is
// a file-scope device array, so it exists on every GPU that loads the
// library until the process exits, and every call of the variant shares it.
static_assert(sizeof(CalPartial) == 32, "partial record layout");
static __device__ __align__(256) unsigned char g_cal_noalloc_scratch[kCalMaxBlocks * 32];

namespace {
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[64] = {nullptr};
}  // namespace

size_t calibrate_noalloc_capacity() { return sizeof(g_cal_noalloc_scratch); }

// The host-side name of the array is only a stand-in, never a device
// address: the address is looked up once per device (with that device
// current) and cached.
static cudaError_t noalloc_scratch_address(void** out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_cal_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

cudaError_t launch_calibrate_noalloc(const float* x, int64_t n, int is_signed, double alpha_star, float* alpha_out,
                                     double* stats_out, cudaStream_t st)
{
    if (calibrate_workspace_bytes(n) > sizeof(g_cal_noalloc_scratch)) return cudaErrorInvalidValue;
    void* ws = nullptr;
    cudaError_t e = noalloc_scratch_address(&ws);
    if (e != cudaSuccess) return e;
    // Pass 1 writes every partial record that pass 2 reads, so nothing in the
    // shared scratch has to be cleared between calls.
    return launch_calibrate(x, n, is_signed, alpha_star, ws, alpha_out, stats_out, st);
}

}  // namespace esb
