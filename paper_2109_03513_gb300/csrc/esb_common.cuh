// esb_common.cuh -- format arithmetic, the fp32-bit projection, and the
// inline-PTX wrappers (mbarrier, tcgen05) shared by the kernels of libesb.
//
// ESB format: Sec. III-B (value set) and Sec. IV-A (float format) of
// Gong et al., arXiv 2109.03513.  fmt = (b, k, signed), N = 2^(b-k-1) - 1,
// code = sign | e (b-k-1 bits) | f (k bits); value = 0.f if e == N, else
// 2^e * 1.f (units of alpha); integer image I = value * 2^k.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "esb.h"

namespace esb {

// ------------------------------------------------------------ format math

__host__ __device__ inline int fmt_N(int b, int k) { return (1 << (b - k - 1)) - 1; }
__host__ __device__ inline int fmt_ew(int b, int k) { return b - k - 1; }
__host__ __device__ inline int fmt_cpw(int b) { return 32 / b; }
__host__ __device__ inline uint32_t fmt_zero_code(int b, int k) { return (uint32_t)fmt_N(b, k) << k; }

// Largest non-negative code: e = N-1, f = 2^k - 1 (or e = N = 0 when k = b-1).
__host__ __device__ inline uint32_t fmt_max_code(int b, int k)
{
    int N = fmt_N(b, k);
    uint32_t fmax = (1u << k) - 1u;
    return N >= 1 ? (((uint32_t)(N - 1) << k) | fmax) : fmax;
}

// Largest integer image max|I| = (2^(k+1)-1) * 2^(N-1), or 2^k - 1 if N = 0.
__host__ inline double fmt_max_image(int b, int k)
{
    int N = fmt_N(b, k);
    if (N == 0) return (double)((1 << k) - 1);
    double m = (double)((1 << (k + 1)) - 1);
    for (int i = 0; i < N - 1; i++) m *= 2.0;
    return m;
}

// C in units of alpha, the clip bound of Eq. cheap_projection.
__host__ inline float fmt_C(int b, int k)
{
    double I = fmt_max_image(b, k);
    double c = I;
    for (int i = 0; i < k; i++) c *= 0.5;
    return (float)c;   // exact: at most 8 significant bits
}

// ---------------------------------------------------- device status word

// Kernels whose bounded waits give up record ESB_ERR_TIMEOUT in the
// library's device status word (address passed as a kernel argument).
__device__ __forceinline__ void record_status(int* status, int s)
{
    if (status) atomicCAS(status, 0, s);
}

// --------------------------------------------------------- projection

struct ProjParams {
    int b, k, is_signed, rounding;
    int N;
    uint32_t zero_code;
    uint32_t max_code;   // non-negative code of C
    uint32_t C_bits;     // fp32 bit pattern of C
};

__host__ inline ProjParams make_proj_params(int b, int k, int is_signed, int rounding)
{
    ProjParams p;
    p.b = b; p.k = k; p.is_signed = is_signed; p.rounding = rounding;
    p.N = fmt_N(b, k);
    p.zero_code = fmt_zero_code(b, k);
    p.max_code = fmt_max_code(b, k);
    float C = fmt_C(b, k);
    uint32_t cb;
    __builtin_memcpy(&cb, &C, 4);
    p.C_bits = cb;
    return p;
}

// Code of v = x / alpha (already divided).  Eq. fast_projection on the
// fp32 bits: the most significant 1 bit of |v| sets the binade n (values
// below 1 use the spacing 2^-k of xi_0), the k+1 leading significant bits
// are kept and the rest is rounded with one integer add and shift.  A
// carry into the next binade is the next set element (f = 0, e + 1).
__device__ __forceinline__ uint32_t project_scaled(float v, const ProjParams& p)
{
    const uint32_t u = __float_as_uint(v);
    const uint32_t sign = u >> 31;
    const uint32_t mag = u & 0x7fffffffu;
    if (mag > 0x7f800000u) return p.zero_code;                 // NaN
    if (sign && !p.is_signed) return p.zero_code;              // unsigned set: v < 0 -> 0
    uint32_t code;
    if (mag >= p.C_bits) {                                     // clip to C (incl. +-Inf)
        code = p.max_code;
    } else {
        const int bexp = (int)(mag >> 23);
        const uint32_t m24 = (mag & 0x7fffffu) | (bexp ? 0x800000u : 0u);
        const int E = bexp ? bexp - 127 : -126;                // unbiased exponent
        const int s = 23 - p.k - (E < 0 ? E : 0);              // bits to drop, >= 16
        uint32_t r;
        if (s > 24) {
            r = 0u;                                            // below half a quantum
        } else {
            const uint32_t half = 1u << (s - 1);
            const uint32_t add = p.rounding ? (half - 1u + ((m24 >> s) & 1u)) : half;
            r = (m24 + add) >> s;
        }
        if (r == 0u) return p.zero_code;                       // zero carries sign 0
        const uint32_t one = 1u << p.k;
        uint32_t e, f;
        if (E < 0) {                                           // r in [1, 2^k]
            if (r < one) { e = (uint32_t)p.N; f = r; } else { e = 0u; f = 0u; }
        } else {                                               // r in [2^k, 2^(k+1)]
            if (r >= 2u * one) { e = (uint32_t)E + 1u; f = 0u; } else { e = (uint32_t)E; f = r - one; }
        }
        code = (e << p.k) | f;
    }
    return code | (sign << (p.b - 1));
}

__device__ __forceinline__ uint32_t project_code(float x, float alpha, const ProjParams& p)
{
    return project_scaled(__fdiv_rn(x, alpha), p);
}

// ------------------------------------------- projection by thresholds

// For a fixed alpha the code of x depends only on which midpoints t_j
// (between consecutive non-negative set elements q_j < q_(j+1)) the value
// v = fl(|x| / alpha) reaches.  IEEE division is monotone in |x|, so
// "v >= t_j" is exactly "|x| >= T_j" for the smallest float T_j with that
// property ("v > t_j" when the tie at t_j goes down under half-to-even).
// The T_j are found once per kernel with the same division, after which a
// projection needs no division at all -- a different evaluation order of
// Eq. cheap_projection with identical results.
constexpr int kMaxThresholds = 127;    // 2^(b-1) - 1 for b = 8

// Element j (0-based, ascending) of the non-negative set, in units of alpha.
__device__ __forceinline__ float set_element(int j, int k)
{
    const int one = 1 << k;
    if (j < one) return ldexpf((float)j, -k);
    return ldexpf((float)(one + (j & (one - 1))), (j >> k) - 1 - k);
}

// T_j computed by one full warp.  Start from x0 = fl(t * alpha), which is
// within a few ulps of T_j; 32 consecutive candidates around it are tested
// at once.  If they do not bracket T_j (over/underflow ranges), fall back to
// a bisection over all non-negative fp32 bit patterns.
__device__ inline float warp_threshold(float alpha, float t, bool strict, int lane)
{
    const uint32_t b0 = __float_as_uint(__fmul_rn(t, alpha));
    if (b0 >= 16u && b0 < 0x7f800000u - 16u) {
        const uint32_t cand = b0 - 16u + (uint32_t)lane;
        const float v = __fdiv_rn(__uint_as_float(cand), alpha);
        const bool ok = strict ? (v > t) : (v >= t);
        const unsigned m = __ballot_sync(0xffffffffu, ok);
        if ((m & 1u) == 0u && (m >> 31) != 0u) return __uint_as_float(b0 - 16u + (uint32_t)(__ffs(m) - 1));
    }
    uint32_t lo = 0u, hi = 0x7f800000u;        // fl(0/alpha) < t (t > 0); fl(inf/alpha) >= t
    while (hi - lo > 1u) {
        const uint32_t mid = lo + ((hi - lo) >> 1);
        const float v = __fdiv_rn(__uint_as_float(mid), alpha);
        if (strict ? (v > t) : (v >= t)) hi = mid; else lo = mid;
    }
    return __uint_as_float(hi);
}

// Fill T[0 .. L-2] (L = 2^(b-1)) using the warps [warp0, warp0 + nwarps).
// The caller synchronises before reading T.
__device__ inline void build_thresholds(float* T, const ProjParams& p, float alpha, int warp, int lane, int warp0,
                                        int nwarps)
{
    const int L = 1 << (p.b - 1);
    for (int j = warp - warp0; j < L - 1; j += nwarps) {
        const float q0 = set_element(j, p.k), q1 = set_element(j + 1, p.k);
        const float t = 0.5f * (q0 + q1);                 // exact
        bool strict = false;
        if (p.rounding) {                                 // half-even: tie goes to the even multiple
            const int r = (int)(q1 / (q1 - q0));          // spacing is a power of two: exact
            strict = (r & 1) != 0;
        }
        const float Tj = warp_threshold(alpha, t, strict, lane);
        if (lane == 0) T[j] = Tj;
    }
}

// Code of x by the thresholds (bucket = number of T_j <= |x|).
__device__ __forceinline__ uint32_t project_by_table(float x, const float* T, const ProjParams& p)
{
    const uint32_t u = __float_as_uint(x);
    const uint32_t sign = u >> 31;
    const float a = __uint_as_float(u & 0x7fffffffu);
    const int L = 1 << (p.b - 1);
    int j = 0;
#pragma unroll 1
    for (int step = L >> 1; step > 0; step >>= 1)
        if (a >= T[j + step - 1]) j += step;
    if (j == 0 || (sign && !p.is_signed)) return p.zero_code;    // zero (and NaN) carry sign 0
    const int one = 1 << p.k;
    const uint32_t mag = (j >= one) ? (uint32_t)(j - one) : (((uint32_t)p.N << p.k) | (uint32_t)j);
    return mag | (sign << (p.b - 1));
}

// The same for a compile-time width B: the b - 1 levels of the search are
// unrolled (the 2^(B-1) - 1 <= 127 thresholds are in shared memory; for
// B <= 6 they sit in distinct banks, so lanes never conflict).
template <int B>
__device__ __forceinline__ uint32_t project_by_table_t(float x, const float* T, const ProjParams& p)
{
    constexpr int L = 1 << (B - 1);
    const uint32_t u = __float_as_uint(x);
    const uint32_t sign = u >> 31;
    const float a = __uint_as_float(u & 0x7fffffffu);
    int j = 0;
#pragma unroll
    for (int step = L >> 1; step > 0; step >>= 1)
        j += (a >= T[j + step - 1]) ? step : 0;
    const int one = 1 << p.k;
    const uint32_t mag = (j >= one) ? (uint32_t)(j - one) : (((uint32_t)p.N << p.k) | (uint32_t)j);
    const bool zero = j == 0 || (sign && !p.is_signed);        // zero (and NaN) carry sign 0
    return zero ? p.zero_code : (mag | (sign << (B - 1)));
}

// ------------------------------------------------ projection by cells
//
// For b = 3 and b >= 5 the bisection above costs b - 1 dependent
// shared-memory loads per value.  Instead the non-negative fp32 bit patterns are cut into cells
// of 2^(21-k) patterns (k + 2 leading fraction bits per binade).  Within a
// binade e of v = |x| / alpha the set's spacing is 2^(e-k) (also below 1),
// so consecutive thresholds lie at least alpha * 2^(e-k) >= two cells apart
// for every normal alpha: a cell holds at most one T_j, which the table
// build checks (and the caller keeps the bisection when it does not hold:
// subnormal thresholds, thresholds that overflow, tables over capacity).
// Entry c: the first threshold above the cell's start s_c, and the codes
// below and at/above it -- the code of x is then one load and one compare.
__host__ __device__ constexpr int cell_shift(int k) { return 21 - k; }

// Code of bucket j (0 .. L-1) of the non-negative set with the sign bit set
// where a sign is allowed (signed set, j != 0); the projection ANDs it with
// the value's sign.
__device__ __forceinline__ uint32_t bucket_code(int j, const ProjParams& p)
{
    if (j == 0) return p.zero_code;
    const int one = 1 << p.k;
    const uint32_t mag = (j >= one) ? (uint32_t)(j - one) : (((uint32_t)p.N << p.k) | (uint32_t)j);
    return mag | (p.is_signed ? (1u << (p.b - 1)) : 0u);
}

// Build the cell table of the thresholds T (all threads of the block; T is
// complete and visible).  Returns, identically in every thread, whether the
// table is usable; then h0 is the first cell's index and hmax the last
// entry.  The last cell lies above T_(L-2): every number there (and +Inf,
// and every value clamped to it) takes the top code, NaN the zero code.
template <int B, int CAP>
__device__ inline bool build_cells(uint2* cells, int& h0, int& hmax, const float* T, const ProjParams& p)
{
    constexpr int L = 1 << (B - 1);
    const int sh = cell_shift(p.k);
    const uint32_t tl = __float_as_uint(T[L - 2]);
    h0 = (int)(__float_as_uint(T[0]) >> sh) - 1;
    if (h0 < 0) h0 = 0;
    const int H = (int)(tl >> sh) + 2 - h0;
    hmax = H - 1;
    if (tl >= 0x7f800000u || H > CAP) return false;             // uniform across the block
    bool bad = false;
    for (int c = threadIdx.x; c < H; c += blockDim.x) {
        const float s = __uint_as_float((uint32_t)(h0 + c) << sh);
        int g = 0;                                              // #{T_j <= s_c}
#pragma unroll
        for (int step = L >> 1; step > 0; step >>= 1)
            g += (s >= T[g + step - 1]) ? step : 0;
        float thr;
        uint32_t lo, hi;
        if (c == H - 1) {
            thr = 0.0f; lo = p.zero_code; hi = bucket_code(L - 1, p);
        } else if (g == L - 1) {
            thr = __uint_as_float(0x7f800000u); lo = hi = bucket_code(L - 1, p);
        } else {
            if (g + 1 <= L - 2 && T[g + 1] < __uint_as_float((uint32_t)(h0 + c + 1) << sh)) bad = true;
            thr = T[g]; lo = bucket_code(g, p); hi = bucket_code(g + 1, p);
        }
        cells[c] = make_uint2(__float_as_uint(thr), lo | (hi << 16));
    }
    return !__syncthreads_or(bad);
}

// Code of x by the cell table.  amask clears the sign for a signed set; for
// the unsigned set the raw pattern is used, so negative values (negative as
// int32) clamp to cell 0, below T_0: the zero code.
template <int B>
__device__ __forceinline__ uint32_t project_by_cells(float x, const uint2* cells, int h0, int hmax, int sh,
                                                     uint32_t amask)
{
    const uint32_t u = __float_as_uint(x);
    const uint32_t ab = u & amask;
    const int h = min(max(((int)ab >> sh) - h0, 0), hmax);
    const uint2 e = cells[h];
    const uint32_t c = (__uint_as_float(ab) >= __uint_as_float(e.x)) ? (e.y >> 16) : e.y;
    return c & ((u >> (32 - B)) | ((1u << (B - 1)) - 1u));
}

// The same with the table in registers for b = 4 (7 thresholds).
struct Thr7 { float t[7]; };

__device__ __forceinline__ uint32_t project_by_thr7(float x, const Thr7& T, const ProjParams& p)
{
    const uint32_t u = __float_as_uint(x);
    const uint32_t sign = u >> 31;
    const float a = __uint_as_float(u & 0x7fffffffu);
    int j = (a >= T.t[3]) ? 4 : 0;
    j += (a >= (j ? T.t[5] : T.t[1])) ? 2 : 0;
    const float t3 = (j & 4) ? ((j & 2) ? T.t[6] : T.t[4]) : ((j & 2) ? T.t[2] : T.t[0]);
    j += (a >= t3) ? 1 : 0;
    if (j == 0 || (sign && !p.is_signed)) return p.zero_code;
    const int one = 1 << p.k;
    const uint32_t mag = (j >= one) ? (uint32_t)(j - one) : (((uint32_t)p.N << p.k) | (uint32_t)j);
    return mag | (sign << 3);
}

// Bucket (0..7) of a against 7 ascending thresholds: the number of T_j <= a.
__device__ __forceinline__ uint32_t bucket7(float a, const Thr7& T)
{
    uint32_t j = (a >= T.t[3]) ? 4u : 0u;
    j |= (a >= (j ? T.t[5] : T.t[1])) ? 2u : 0u;
    const float t3 = (j & 4u) ? ((j & 2u) ? T.t[6] : T.t[4]) : ((j & 2u) ? T.t[2] : T.t[0]);
    j |= (a >= t3) ? 1u : 0u;
    return j;
}

// Eight 4-bit codes at once from their buckets J (one per nibble, 0..7) and
// sign bits S (bit 3 of each nibble).  Element j of the non-negative set has
// the code (j - 2^k) mod 2^(b-1) -- the exponent field rotated by one, as in
// the decode -- so the whole word is one add and a mask; zero (j = 0) keeps
// sign 0.
__device__ __forceinline__ uint32_t codes8_b4(uint32_t J, uint32_t S, int k)
{
    const uint32_t C1 = 0x88888888u - (0x11111111u << k);   // 8 - 2^k per nibble: no borrow across nibbles
    const uint32_t nz = (J + 0x77777777u) & 0x88888888u;      // bit 3 set where j >= 1
    return ((J + C1) & 0x77777777u) | (S & nz);
}

// Lean-path threshold on the raw accumulator.  For a scale sc > 0,
// y(a) = fma(sc, a, b) is non-decreasing in the integer accumulator a
// (|a| < 2^24, checked on the host), and so is the activation of y; an
// output code's bucket counts the thresholds T_j (all > 0) at or below
// act(y).  For ReLU and no activation, act(y) >= T  <=>  y >= T (T > 0);
// ReLU6 never reaches a T above 6.  Returns A * rs for the smallest
// integer A with y(A) >= T (raw = a * rs exactly), +inf if none, -inf if
// every accumulator qualifies.  26 bounded bisection steps on integers.
__device__ __forceinline__ float acc_raw_threshold(float sc, float b, float T, int act, float rs)
{
    if (act == ESB_ACT_RELU6 && T > 6.0f) return __int_as_float(0x7f800000);
    const int lim = 1 << 24;
    if (!(__fmaf_rn(sc, (float)lim, b) >= T)) return __int_as_float(0x7f800000);
    if (__fmaf_rn(sc, (float)-lim, b) >= T) return __int_as_float(0xff800000);
    int lo = -lim, hi = lim;                           // y(lo) < T <= y(hi)
    for (int it = 0; it < 32 && hi - lo > 1; it++) {
        const int mid = lo + ((hi - lo) >> 1);
        if (__fmaf_rn(sc, (float)mid, b) >= T) hi = mid; else lo = mid;
    }
    return (float)hi * rs;
}

// Value of a code in units of alpha (Sec. IV-A, Eq. q), exact in fp32 for b <= 8.
__device__ __forceinline__ float code_value(uint32_t c, int b, int k)
{
    const int ew = b - k - 1;
    const int N = (1 << ew) - 1;
    const uint32_t s = (c >> (b - 1)) & 1u;
    const uint32_t e = ew > 0 ? (c >> k) & ((1u << ew) - 1u) : 0u;
    const uint32_t f = c & ((1u << k) - 1u);
    const bool sub = (int)e == N;
    const float m = (float)(sub ? f : ((1u << k) + f));
    const float mag = ldexpf(m, (sub ? 0 : (int)e) - k);   // power-of-two scaling: exact
    return s ? -mag : mag;
}

// Integer image of a code as float (exact; formats with max|I| < 2^24).
__device__ __forceinline__ float code_image_f(uint32_t c, int b, int k)
{
    const int ew = b - k - 1;
    const int N = (1 << ew) - 1;
    const uint32_t s = (c >> (b - 1)) & 1u;
    const uint32_t e = ew > 0 ? (c >> k) & ((1u << ew) - 1u) : 0u;
    const uint32_t f = c & ((1u << k) - 1u);
    const uint32_t mag = ((int)e == N) ? f : (((1u << k) + f) << e);
    const float m = (float)mag;
    return s ? -m : m;
}

// ------------------------------------------------------------- PTX helpers

__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Arrive on an mbarrier and add tx bytes to the transaction count its
// current phase waits for (the bulk copies that complete on it).
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t tx)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(tx) : "memory");
}

// Bulk copy of `bytes` (a multiple of 16; both addresses 16-byte aligned)
// from global to this CTA's shared memory, completing on mbarrier `bar`.
__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}

// Programmatic dependent launch.  griddep_wait: block until the grids this
// one depends on have completed and their memory is visible (returns at
// once when the launch has no programmatic dependency); every read of data
// an earlier launch may have written, and every write an earlier launch may
// still read, comes after it.  griddep_launch_dependents: this CTA no longer
// holds back the launch of a dependent grid.
// L2 prefetch of the line holding p.  It returns nothing to the SM, so it
// may be issued before griddep_wait: the loads after the wait still read
// whatever the previous grid leaves in L2, the point of coherence.
__device__ __forceinline__ void prefetch_l2(const void* p) { asm volatile("prefetch.global.L2 [%0];" ::"l"(p)); }

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Bytes of dynamic shared memory this launch was given.
__device__ __forceinline__ uint32_t dynamic_smem_bytes()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%dynamic_smem_size;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint64_t globaltimer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// try_wait with a suspend-time hint: the thread may be parked (issuing
// nothing) until the phase completes or about hint_ns pass.
__device__ __forceinline__ bool mbar_try_wait_hint(uint32_t bar, uint32_t parity, uint32_t hint_ns)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}

// Bounded wait: gives up after `limit_ns` of wall time (checked every 256
// polls) and returns false; the caller records ESB_ERR_TIMEOUT.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns)
{
    const uint32_t a = smem_u32(bar);
    if (mbar_try_wait(a, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(a, parity)) return true;
        if ((it & 255u) == 0u && globaltimer_ns() - t0 > limit_ns) return false;
    }
}

__device__ __forceinline__ void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// TMEM allocation (one full warp executes these).
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(slot)), "r"(ncols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f8f6f4, issued by one thread.
__device__ __forceinline__ void mma_f8f6f4(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive on an mbarrier once every previously issued tcgen05 op of this
// thread has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                 ::"r"(smem_u32(bar)) : "memory");
}

// 32 lanes x 16 columns of 32-bit TMEM words into 16 registers per thread.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 32 lanes x 4 columns.
__device__ __forceinline__ void tmem_ld4(uint32_t taddr, uint32_t (&r)[4])
{
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// 32 lanes x 32 columns in one load and one wait.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor for a K-major operand in the 128-byte
// swizzled layout: rows of 128 bytes, 8-row atoms of 1024 bytes (SBO).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);        // start address
    d |= (uint64_t)1u << 16;                         // LBO (unused for swizzled K-major)
    d |= (uint64_t)(1024u >> 4) << 32;               // SBO: 8 rows x 128 B
    d |= (uint64_t)1u << 46;                         // descriptor version (sm_100 family)
    d |= (uint64_t)2u << 61;                         // swizzle: 128 B
    return d;
}

// Shared-memory matrix descriptor, K-major without swizzle: core matrices
// of 8 rows x 16 bytes (rows 16 bytes apart); sbo = byte stride between
// 8-row groups along M/N, lbo = byte stride between 16-byte column chunks
// along K.  Any 16-byte aligned start address.
__device__ __forceinline__ uint64_t smem_desc_noswz(uint32_t saddr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);        // start address
    d |= (uint64_t)((lbo & 0x3FFFFu) >> 4) << 16;    // leading (K) byte offset
    d |= (uint64_t)((sbo & 0x3FFFFu) >> 4) << 32;    // stride (M/N) byte offset
    d |= (uint64_t)1u << 46;                         // descriptor version (sm_100 family)
    return d;                                        // swizzle field 0: none
}

// Instruction descriptor: kind::f8f6f4, A = B = E4M3, D = F32, K-major
// operands, M = 128, N = n.
__host__ __device__ inline uint32_t idesc_e4m3_f32(int n)
{
    uint32_t d = 0;
    d |= 1u << 4;                       // D format: F32
    d |= 0u << 7;                       // A format: E4M3
    d |= 0u << 10;                      // B format: E4M3
    d |= (uint32_t)(n >> 3) << 17;      // N >> 3
    d |= (uint32_t)(128 >> 4) << 24;    // M >> 4
    return d;
}

}  // namespace esb
