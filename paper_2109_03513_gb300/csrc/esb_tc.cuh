// esb_tc.cuh -- device code shared by the tcgen05 contraction kernels
// (esb_gemm.cu: GEMM and im2col convolution; esb_conv_halo.cu: stride-1
// convolution from a decoded input halo): operand decode of ESB codes to
// scaled E4M3 bytes, the fused post-processing epilogue (Sec. IV-C), the
// bounded mbarrier waits, and the setup and epilogue roles of the
// persistent warp-specialised kernels.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

constexpr int kBM = 128;           // rows per tile (TMEM lanes)
constexpr int kBK = 128;           // codes (= E4M3 bytes) per K-block: one 128-byte swizzle row
constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s

// Operand format of a contraction kernel.  A code whose integer image is an
// exact E4M3 number times 2^-(k+6) (k <= 3, exponent field <= 4 bits) is
// one E4M3 byte ("whole").  Wider significands (k >= 4: up to 8
// significant bits) take the significand split: I = (-1)^s m 2^sh with
// m = 16 m_hi + m_lo becomes two E4M3 bytes, m_hi 2^(sh+4) 2^-9 ("high")
// and m_lo 2^sh 2^-9 ("low"), each exact (at most 4 significant bits), and
// the two planes are separate 16-code units of an expanded K.  When either
// operand is split the logical K of the kernels is planes x K16 (K16 = K
// rounded up to 16): unit u' of it is plane u' % planes of code unit
// u' / planes, with the roles of pmap (2 bits per plane: 0 whole, 1 high,
// 2 low), chosen so that the products of the planes add up to I_A I_B:
// one split operand [H, L] against [W, W]; both split [H, H, L, L] against
// [H, L, H, L].  Every product is a multiple of 2^-(csc_A + csc_B), and the
// sum of their magnitudes is sum |I_A| |I_B| in that unit, so the fp32 TMEM
// accumulation is exact under the same bound as without the split.
struct OpFmt {
    int b, k, ew, cpw;
    uint32_t mask;
    int planes;          // 1, 2 or 4 units of the kernel's K per 16 codes
    uint32_t pmap;       // role of plane i in bits 2i, 2i+1
    int csc;             // operand scale: decoded values are I 2^-csc
    int64_t korig;       // codes per row before the expansion (K tail)
    int spw;             // word-slot layout: kernel-K slots per packed word (0: code-linear K)
};

// Significand split needed: the image is not an E4M3 number times a power of two.
__host__ __device__ inline bool fmt_needs_split(int b, int k)
{
    const int ew = b - k - 1;
    return k > 3 || ew > 4 || (ew == 4 && k == 3);
}

__host__ inline OpFmt make_opfmt(int b, int k)
{
    OpFmt o;
    o.b = b; o.k = k; o.ew = b - k - 1; o.cpw = 32 / b; o.mask = (1u << b) - 1u;
    o.planes = 1; o.pmap = 0u; o.csc = k + 6; o.korig = 0; o.spw = 0;
    return o;
}

// Word-slot layout of the kernels' K for a pair of whole-byte operands of
// widths other than 4 with the same codes per word: packed word w of a row
// takes the spw slots [w spw, (w + 1) spw) of K (spw = cpw rounded up to a
// power of two: 16 for 3-bit, 8 for 5/6-bit, 4 for 7/8-bit, 16 for 2-bit),
// its codes the first cpw of them and the E4M3 zero the rest.  A K-block
// (128 slots) is then a whole number of words and every code has a fixed
// byte, so a row decodes word by word without a running code offset.  Both
// operands use the same slots, so the sums are those of the code-linear K.
// korig: codes per row (the contraction length; codes of the last word past
// it count as zero); words: packed words per row that enter K.  Returns the
// kernels' K, or 0 when the pair keeps the code-linear layout (4-bit,
// significand planes, different codes per word).
__host__ inline int64_t plan_slots(OpFmt& fa, OpFmt& fb, int64_t korig, int64_t words)
{
    if (fa.planes != 1 || fb.planes != 1 || fa.cpw != fb.cpw || fa.b == 4 || fb.b == 4) return 0;
    const int spw = fa.cpw > 8 ? 16 : (fa.cpw > 4 ? 8 : 4);
    fa.spw = fb.spw = spw;
    fa.korig = fb.korig = korig;
    return words * spw;
}

// The plane layout of a pair of operands (see OpFmt) for a contraction of
// K codes; returns the kernels' K (K itself when neither is split).
__host__ inline int64_t plan_planes(OpFmt& fa, OpFmt& fb, int64_t K)
{
    const bool sa = fmt_needs_split(fa.b, fa.k), sb = fmt_needs_split(fb.b, fb.k);
    fa.korig = fb.korig = K;
    if (!sa && !sb) return K;
    const int P = (sa && sb) ? 4 : 2;
    fa.planes = fb.planes = P;
    if (sa && sb) {
        fa.pmap = 1u | (1u << 2) | (2u << 4) | (2u << 6);      // H H L L
        fb.pmap = 1u | (2u << 2) | (1u << 4) | (2u << 6);      // H L H L
    } else {
        (sa ? fa : fb).pmap = 1u | (2u << 2);                  // H L
        (sa ? fb : fa).pmap = 0u;                              // W W
    }
    if (sa) fa.csc = 9;
    if (sb) fb.csc = 9;
    return (int64_t)P * ((K + 15) / 16) * 16;
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

// One code -> the E4M3 byte of one significand plane (role 1: high part,
// role 2: low part; see OpFmt), value m_part 2^(shift - 9).
__device__ __forceinline__ uint32_t code_to_e4m3_part(uint32_t c, const OpFmt& f, uint32_t role)
{
    const uint32_t s = (c >> (f.b - 1)) & 1u;
    const uint32_t fr = c & ((1u << f.k) - 1u);
    const uint32_t N = (1u << f.ew) - 1u;
    const uint32_t e = f.ew > 0 ? (c >> f.k) & N : N;
    const uint32_t m = (e == N) ? fr : ((1u << f.k) | fr);
    const int sh = (e == N) ? 0 : (int)e;
    const uint32_t part = (role == 1u) ? (m >> 4) : (m & 15u);
    const int shift = (role == 1u) ? sh + 4 : sh;
    if (part == 0u) return 0u;
    const int t = 31 - __clz(part);                                 // 0 .. 3
    const int E = shift + t - 2;                                    // biased: (shift - 9 + t) + 7
    const uint32_t mag = (E >= 1) ? (((uint32_t)E << 3) | ((part << (3 - t)) & 7u))
                                  : (part << shift);                // subnormal: part 2^shift <= 7
    return (s << 7) | mag;
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

// Plain K-major rows: logical word w of row r is base[r * ld + w].  With
// kp > 0 the rows are convolution filters whose K runs over taps of kp
// codes (the input's codes per pixel) while each tap of the row holds ldt
// words of this operand's width: code kk is channel kk % kp of tap kk / kp,
// and channels past the tap's words read as zero (mixed code widths).
struct RowsSrc {
    const uint32_t* base;
    int64_t ld;
    int64_t rows;
    // Filter rows of an im2col convolution whose K runs over taps of kp
    // codes (kp = 0: plain rows).  Tap t of a row starts at word t * ldt.
    // kwt > 0 when a tap's K codes are whole words of this operand (kp =
    // kwt codes per word x kwt): logical word w is then word w % kwt of tap
    // w / kwt, and cursors walk the rows word by word.
    int64_t kp = 0;
    int64_t ldt = 0;
    int64_t kwt = 0;
    struct Row { const uint32_t* p; };
    struct Cursor { int64_t w; int64_t word; };        // w: offset in the row; word: index within the tap
    __host__ __device__ __forceinline__ bool linear() const { return kp == 0 || kwt > 0; }
    __host__ __device__ __forceinline__ bool vec4() const { return kp == 0 || ((kwt & 3) == 0 && (ldt & 3) == 0); }
    __device__ __forceinline__ Row row(int64_t r) const { Row x; x.p = (r < rows) ? base + r * ld : nullptr; return x; }
    __device__ __forceinline__ const uint32_t* words(const Row& x, int64_t w) const { return x.p ? x.p + w : nullptr; }
    // Word holding code kk of row x (nullptr: the zero code) and its slot.
    __device__ __forceinline__ const uint32_t* code_word(const Row& x, int64_t kk, int cpw, int& slot) const
    {
        if (kp == 0) {
            const int64_t wi = kk / cpw;
            slot = (int)(kk - wi * cpw);
            return words(x, wi);
        }
        const int64_t tap = kk / kp;
        const int64_t c = kk - tap * kp;
        const int64_t wi = c / cpw;
        slot = (int)(c - wi * cpw);
        return wi < ldt ? words(x, tap * ldt + wi) : nullptr;
    }
    __device__ __forceinline__ Cursor cursor(int64_t w) const
    {
        Cursor c;
        if (kwt > 0) {
            const int64_t tap = w / kwt;
            c.word = w - tap * kwt;
            c.w = tap * ldt + c.word;
        } else {
            c.w = w;
            c.word = 0;
        }
        return c;
    }
    __device__ __forceinline__ void advance(Cursor& c, int dw) const
    {
        c.w += dw;
        if (kwt > 0) {
            c.word += dw;
            while (c.word >= kwt) {
                c.word -= kwt;
                c.w += ldt - kwt;
            }
        }
    }
    __device__ __forceinline__ const uint32_t* at(const Row& x, const Cursor& c) const { return x.p ? x.p + c.w : nullptr; }
};

// General decode of the 16-code unit [k0, k0 + 16) of the kernel's K of
// one row (any b, K tail, significand planes: see OpFmt).
template <class Src>
__device__ __noinline__ uint4 decode_unit_any(const Src& src, const typename Src::Row& row, int64_t k0, int64_t K,
                                              const OpFmt f)
{
    uint32_t o0 = 0u, o1 = 0u, o2 = 0u, o3 = 0u;
    if (f.spw) {                                      // word-slot layout: slot j of word k0 / spw + j / spw
#pragma unroll 1
        for (int j = 0; j < 16; j++) {
            const int sl = j % f.spw;
            const int64_t kk = (k0 / f.spw + j / f.spw) * f.cpw + sl;
            if (sl >= f.cpw || kk >= f.korig) continue;
            int slot = 0;
            const uint32_t* p = src.code_word(row, kk, f.cpw, slot);
            if (!p) continue;
            const uint32_t v = code_to_e4m3((__ldg(p) >> (f.b * slot)) & f.mask, f) << (8 * (j & 3));
            switch (j >> 2) {
            case 0: o0 |= v; break;
            case 1: o1 |= v; break;
            case 2: o2 |= v; break;
            default: o3 |= v; break;
            }
        }
        return make_uint4(o0, o1, o2, o3);
    }
    uint32_t role = 0u;
    if (f.planes > 1) {                               // unit k0 / 16 = plane of code unit (k0 / 16) / planes
        const int64_t u = k0 >> 4;
        const int64_t cu = u / f.planes;
        role = (f.pmap >> (2 * (int)(u - cu * f.planes))) & 3u;
        k0 = cu * 16;
        K = f.korig;
    }
#pragma unroll 1
    for (int j = 0; j < 16; j++) {
        const int64_t kk = k0 + j;
        if (kk >= K) break;
        int slot = 0;
        const uint32_t* p = src.code_word(row, kk, f.cpw, slot);
        if (!p) continue;
        const uint32_t c = (__ldg(p) >> (f.b * slot)) & f.mask;
        const uint32_t byte = role ? code_to_e4m3_part(c, f, role) : code_to_e4m3(c, f);
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

__device__ __forceinline__ uint32_t swz(int r, int g) { return (uint32_t)(r * 128 + ((g ^ (r & 7)) << 4)); }

// Byte masks of the decoded lo/hi words of one b = 4 word when only its
// first v codes (0..8) are inside K.
__device__ __forceinline__ void tail_masks(int v, uint32_t& mlo, uint32_t& mhi)
{
    const int nlo = (v + 1) >> 1, nhi = v >> 1;       // lo holds codes 0,2,4,6; hi 1,3,5,7
    mlo = nlo >= 4 ? 0xffffffffu : ((1u << (8 * nlo)) - 1u);
    mhi = nhi >= 4 ? 0xffffffffu : ((1u << (8 * nhi)) - 1u);
}

// The E4M3 byte of each of the 2^b codes of a whole-byte format (planes ==
// 1), built by threads t = 0 .. nt-1: the table of the word-walk decoder.
__device__ __forceinline__ void build_e4m3_lut(uint8_t* lut, const OpFmt& f, int t, int nt)
{
    for (int c = t; c < (1 << f.b); c += nt) lut[c] = (uint8_t)code_to_e4m3((uint32_t)c, f);
}

// CH loaded words of B-bit codes in the word-slot layout (ok: word i
// exists; lim: codes of the chunk inside K) -> their E4M3 slots, stored as
// 16-byte units from unit g0 of stage row r.
template <int B, int CH>
__device__ __forceinline__ void store_slot_words(const uint32_t (&wv)[CH], uint32_t ok, int lim, const uint8_t* lut,
                                                 uint8_t* stage, int r, int g0)
{
    constexpr int CPW = 32 / B;
    constexpr int SPW = CPW > 8 ? 16 : (CPW > 4 ? 8 : 4);
    constexpr uint32_t MASK = (1u << B) - 1u;
    uint32_t o[CH * SPW / 4];
#pragma unroll
    for (int i = 0; i < CH; i++) {
#pragma unroll
        for (int q = 0; q < SPW / 4; q++) {
            uint32_t v = 0u;
#pragma unroll
            for (int t = 0; t < 4; t++) {
                const int j = q * 4 + t;
                if (j < CPW) {
                    const uint32_t byte = lut[(wv[i] >> (B * j)) & MASK];
                    v |= ((i * CPW + j < lim) ? byte : 0u) << (8 * t);
                }
            }
            o[i * (SPW / 4) + q] = ((ok >> i) & 1u) ? v : 0u;
        }
    }
#pragma unroll
    for (int g = 0; g < CH * SPW / 16; g++)
        *reinterpret_cast<uint4*>(stage + swz(r, g0 + g)) = make_uint4(o[4 * g], o[4 * g + 1], o[4 * g + 2], o[4 * g + 3]);
}

// NW loaded words of a 4-bit K-block from code k0 (ok: word i exists)
// decoded 8 codes at a time and stored as the NW / 2 units of stage row r
// from unit g0; codes past K give the E4M3 zero.
template <int NW>
__device__ __forceinline__ void store_b4_words(const uint32_t (&wv)[NW], uint32_t ok, int64_t k0, int64_t K,
                                               const OpFmt& f, uint8_t* stage, int r, int g0)
{
#pragma unroll
    for (int g = 0; g < NW / 2; g++) {
        uint32_t o[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const int i = 2 * g + h;
            if ((ok >> i) & 1u) {
                decode_word_b4(wv[i], f.k, f.ew, o[2 * h], o[2 * h + 1]);
                const int64_t kk = k0 + i * 8;
                if (kk + 8 > K) {                     // K tail: zero the codes past K
                    uint32_t ml, mh;
                    tail_masks((int)(K - kk), ml, mh);
                    o[2 * h] &= ml;
                    o[2 * h + 1] &= mh;
                }
            }
        }
        *reinterpret_cast<uint4*>(stage + swz(r, g0 + g)) = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

// One K-block of a row in the word-slot layout (see plan_slots) for B-bit
// codes: the block's words are loaded 16 at a time (independent loads in
// flight), then each word's codes go through the E4M3 table to their fixed
// bytes.  Words past the row's K words, outside the operand or outside the
// image, and codes past korig, give the E4M3 zero.
template <int B, class Src>
__device__ __forceinline__ void walk_row_slots(const Src& src, const typename Src::Row& row, int64_t k0,
                                               const OpFmt& f, const uint8_t* lut, uint8_t* stage, int r)
{
    constexpr int CPW = 32 / B;
    constexpr int SPW = CPW > 8 ? 16 : (CPW > 4 ? 8 : 4);
    constexpr int NW = kBK / SPW;                     // words per K-block: 8, 16 or 32
    constexpr int CH = 8;                             // words per chunk (a small loop body)
    const int64_t w0 = k0 / SPW;
    typename Src::Cursor cur = src.cursor(w0);
#pragma unroll 1
    for (int c0 = 0; c0 < NW; c0 += CH) {
        const int64_t left = f.korig - (w0 + c0) * CPW;   // codes of this chunk's words inside K
        const int lim = left < 0 ? 0 : (left > CH * CPW ? CH * CPW : (int)left);
        uint32_t wv[CH];
        uint32_t ok = 0u;
#pragma unroll
        for (int i = 0; i < CH; i++) {
            const uint32_t* p = (i * CPW < lim) ? src.at(row, cur) : nullptr;
            wv[i] = p ? __ldg(p) : 0u;
            ok |= (p ? 1u : 0u) << i;
            src.advance(cur, 1);
        }
        store_slot_words<B, CH>(wv, ok, lim, lut, stage, r, c0 * SPW / 16);
    }
}

// K-block [k0, k0 + 128) of one row decoded by walking its words once (a
// code never straddles two words): eight 16-code units of E4M3 bytes stored
// to the swizzled stage row r, in the word-slot layout when f.spw is set,
// else code-linear in unit_pos order.  For linear sources with one plane;
// codes past K and words outside the operand (rows past M or N,
// out-of-image taps) give the E4M3 zero.
template <class Src>
__device__ __forceinline__ void walk_row_kblock(const Src& src, const typename Src::Row& row, int64_t k0, int64_t K,
                                                const OpFmt& f, const uint8_t* lut, uint8_t* stage, int r)
{
    if (f.spw) {
        switch (f.b) {
        case 2: walk_row_slots<2>(src, row, k0, f, lut, stage, r); return;
        case 3: walk_row_slots<3>(src, row, k0, f, lut, stage, r); return;
        case 5: walk_row_slots<5>(src, row, k0, f, lut, stage, r); return;
        case 6: walk_row_slots<6>(src, row, k0, f, lut, stage, r); return;
        case 7: walk_row_slots<7>(src, row, k0, f, lut, stage, r); return;
        default: walk_row_slots<8>(src, row, k0, f, lut, stage, r); return;
        }
    }
    if (f.b == 4) {
        // 4-bit codes: each 16-code unit is two words (consecutive logical
        // words may lie in different pixels).  The block's 16 words are
        // loaded first (independent loads in flight), then decoded 8 codes
        // at a time.
        typename Src::Cursor cur = src.cursor(k0 >> 3);
        uint32_t wv[16];
        uint32_t ok = 0u;
#pragma unroll
        for (int i = 0; i < 16; i++) {
            const uint32_t* p = (k0 + i * 8 < K) ? src.at(row, cur) : nullptr;
            wv[i] = p ? __ldg(p) : 0u;
            ok |= (p ? 1u : 0u) << i;
            src.advance(cur, 1);
        }
        store_b4_words<16>(wv, ok, k0, K, f, stage, r, 0);
        return;
    }
    const int cpw = f.cpw;
    const int64_t wi = k0 / cpw;
    int slot = (int)(k0 - wi * cpw);
    typename Src::Cursor cur = src.cursor(wi);
    const uint32_t* p = (k0 < K) ? src.at(row, cur) : nullptr;
    uint32_t w = p ? __ldg(p) : 0u;
    bool valid = p != nullptr;
#pragma unroll 1
    for (int g = 0; g < 8; g++) {
        uint32_t o[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int j = 0; j < 16; j++) {
            const int64_t kk = k0 + g * 16 + j;
            const uint32_t byte = (valid && kk < K) ? (uint32_t)lut[(w >> (f.b * slot)) & f.mask] : 0u;
            const int pos = unit_pos(j);
            o[pos >> 2] |= byte << (8 * (pos & 3));
            if (++slot == cpw) {
                slot = 0;
                src.advance(cur, 1);
                p = (kk + 1 < K) ? src.at(row, cur) : nullptr;
                valid = p != nullptr;
                w = valid ? __ldg(p) : 0u;
            }
        }
        *reinterpret_cast<uint4*>(stage + swz(r, g)) = make_uint4(o[0], o[1], o[2], o[3]);
    }
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
    int codes_vec;            // widest safe store of code words: 1, 2 or 4 (pointer and ldo alignment)
    float acc_lim;            // K max|I_A| max|I_B| + 2 when that bound is below 2^20, else 0
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
        const int nq = (int)n / rcpw;                 // 32-bit: a column index is below 2^31
        const uint32_t rc = (__ldg(ep.residual + m * ep.res_ld + nq) >> (ep.res_b * ((int)n - nq * rcpw))) &
                            ((1u << ep.res_b) - 1u);
        y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
    }
    y = apply_act(y, ep.act);
    if (ep.y_out) ep.y_out[m * N + n] = y;
    if (!ep.codes_out) return 0u;
    return cx.b4 ? project_by_thr7(y, cx.t7, ep.out) : project_by_table(y, cx.T, ep.out);
}

// Wait on an mbarrier phase with a wall-clock bound and an abort flag
// raised by another role of the CTA.  The waiting thread is parked by the
// hardware between tries (suspend hint), so a waiting warp takes no issue
// slots from the working warps of its sub-partition.
constexpr uint32_t kSuspendHintNs = 20000;
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* err)
{
    const uint32_t a = smem_u32(bar);
    if (mbar_try_wait(a, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        if (mbar_try_wait_hint(a, parity, kSuspendHintNs)) return true;
        if (*err) return false;
        if (globaltimer_ns() - t0 > kWaitLimitNs) return false;
    }
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Arrive without release semantics: for the epilogue's "accumulator buffer
// free" signal, which orders only its TMEM reads (complete once
// tcgen05.wait::ld returns, fenced by tcgen05.fence::before_thread_sync)
// against the next MMA.  A release arrive would first wait for the warp's
// earlier global stores of output codes to be performed, once per tile.
__device__ __forceinline__ void mbar_arrive_tmem_free(uint64_t* bar)
{
    asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// ----------------------------------------- resident-B persistent kernel

constexpr int kWsEpiWarps = 8;                 // warps 0-7: epilogue (lanes 32*(w&3).., column half w>>2)
constexpr int kWsMmaWarp = 8;                  // warp 8: TMEM allocation and MMA issue
constexpr int kWsProdWarp0 = 9;                // warps 9-15: A producers, one stage at a time each
constexpr int kWsProdWarps = 7;
constexpr int kWsThreads = (kWsProdWarp0 + kWsProdWarps) * 32;   // 512: 4 warps per SM sub-partition
constexpr int kWsMaxStages = 8;


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

// Epilogue of one 16-column chunk for outputs other than the lean 4-bit
// path (general packing), out of line; reads its own TMEM chunk.
static __device__ __noinline__ void epi_chunk_any(const EpiParams* __restrict__ sep, const EpiCtx* __restrict__ scx,
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


struct Raw8 { uint32_t r[8]; };

// One packed word of 4-bit output codes (8 columns from n_first) with
// per-channel scale/bias, residual or extra outputs; out of line so the
// caller's accumulator registers stay in registers.
static __device__ __noinline__ uint32_t epi_word_b4(const EpiParams* __restrict__ sep, const EpiCtx* __restrict__ scx,
                                                    Raw8 v, float acc_scale, float sc_fixed, int64_t m, bool mrow,
                                                    int64_t n_first, int64_t N)
{
    const EpiParams& ep = *sep;
    const EpiCtx& cx = *scx;
    uint32_t J = 0u, S = 0u;
#pragma unroll 1
    for (int j = 0; j < 8; j++) {
        const int64_t n = n_first + j;
        const float af = __uint_as_float(v.r[j]) * acc_scale;
        if (mrow && n < N) {
            if (ep.acc_out) ep.acc_out[m * N + n] = __float2int_rn(af);
            float sc = sc_fixed;
            if (ep.scale) { sc = __ldg(ep.scale + n); if (cx.dq) sc = __fmul_rn(sc, cx.dqs); }
            const float bi = ep.bias ? __ldg(ep.bias + n) : ep.bias0;
            float y = __fmaf_rn(sc, af, bi);
            if (ep.residual) {
                const int rcpw = 32 / ep.res_b;
                const int nq = (int)n / rcpw;                 // 32-bit: a column index is below 2^31
        const uint32_t rc = (__ldg(ep.residual + m * ep.res_ld + nq) >> (ep.res_b * ((int)n - nq * rcpw))) &
                                    ((1u << ep.res_b) - 1u);
                y = __fmaf_rn(ep.res_scale, code_image_f(rc, ep.res_b, ep.res_k), y);
            }
            y = apply_act(y, ep.act);
            if (ep.y_out) ep.y_out[m * N + n] = y;
            const uint32_t u = __float_as_uint(y);
            J |= bucket7(ep.out.is_signed ? fabsf(y) : y, cx.t7) << (4 * j);
            S |= ((u >> 31) & (uint32_t)ep.out.is_signed) << (4 * j + 3);
        }
    }
    return codes8_b4(J, S, ep.out.k);
}

// ------------------------------------ roles of the warp-specialised kernels

// TMEM for the two accumulator buffers, allocated by the MMA warp before the
// CTA's first barrier (the caller then runs __syncthreads, and ws_setup reads
// the base address after it).
__device__ __forceinline__ void ws_alloc(int warp, uint32_t* tmem_slot, uint32_t tmem_cols)
{
    if (warp == kWsMmaWarp) {
        tmem_alloc(tmem_slot, tmem_cols);
        tc_fence_before();
    }
}

// Decode of the CTA's N-tile of B (rows n0 .. n0 + BN, every K-block) once
// into sB in the SW128 K-major layout, by threads t = 0 .. nthreads - 1 of
// the calling warps.  B4: B is known to be 4-bit.  The caller fences
// (fence_proxy_async_smem) and synchronises before the MMA reads sB.
template <bool B4>
__device__ __forceinline__ void ws_decode_b(const RowsSrc& srcB, int64_t n0, int64_t K, const OpFmt& fb, int BN,
                                            int nkb, uint8_t* sB, int t, int nthreads, const uint8_t* lutb = nullptr)
{
    if (B4 || (fb.b == 4 && fb.planes == 1 && srcB.linear() && srcB.vec4())) {
        // one row chunk per thread and pass (compact: this code runs cold,
        // once per CTA, on the path to the first MMA)
        const uint32_t zw = fmt_zero_code(4, fb.k) * 0x11111111u;
        const int rows_total = nkb * BN;
#pragma unroll 1
        for (int pr = t; pr < rows_total; pr += nthreads) {
            const int kb = pr / BN, r = pr - kb * BN;
            const RowsSrc::Row row = srcB.row(n0 + r);
            const int64_t kw0 = (int64_t)kb * 16;
            RowsSrc::Cursor cur[4];
#pragma unroll
            for (int pc = 0; pc < 4; pc++) cur[pc] = srcB.cursor(kw0 + 4 * pc);
            uint4 v[4];
            load_row_b4(srcB, row, cur, kw0, K, zw, v);
            store_row_b4(sB + kb * BN * kBK, r, v, kw0, K, fb);
        }
    } else if (lutb && fb.planes == 1 && srcB.linear()) {
        // other widths: one word walk per (K-block, row)
#pragma unroll 1
        for (int pr = t; pr < nkb * BN; pr += nthreads) {
            const int kb = pr / BN, r = pr - kb * BN;
            walk_row_kblock(srcB, srcB.row(n0 + r), (int64_t)kb * kBK, K, fb, lutb, sB + kb * BN * kBK, r);
        }
    } else {
        for (int u = t; u < nkb * BN * 8; u += nthreads) {
            const int kb = u / (BN * 8);
            const int rem = u - kb * BN * 8;
            const int r = rem >> 3, g = rem & 7;
            *reinterpret_cast<uint4*>(sB + kb * BN * kBK + swz(r, g)) =
                decode_unit_any(srcB, srcB.row(n0 + r), (int64_t)kb * kBK + g * 16, K, fb);
        }
    }
}

// Requantisation thresholds of the output format, built by warps 0-7 (the
// epilogue warps), which then meet on named barrier 3.
__device__ __forceinline__ void ws_thresholds(float* thr, const EpiParams& ep, int warp, int lane)
{
    if (ep.codes_out) {
        const float alpha_out = ep.alpha_out_dev ? __ldg(ep.alpha_out_dev) : ep.alpha_out;
        build_thresholds(thr, ep.out, alpha_out, warp, lane, 0, kWsEpiWarps);
    }
    asm volatile("bar.sync 3, %0;" ::"n"(kWsEpiWarps * 32) : "memory");
}

// Setup role (warps 0 .. kWsProdWarp0 - 1, while the producers already load
// A): all setup warps decode B (ws_decode_b); the MMA warp waits for that on
// named barrier 1 and leaves, while warps 0-7 build the thresholds
// (ws_thresholds: the MMA does not wait for them).  B4: B is known to be
// 4-bit.  Returns the TMEM base address (allocated by ws_alloc before the
// CTA barrier).
template <bool B4>
__device__ __forceinline__ uint32_t ws_setup(const RowsSrc& srcB, int64_t n0, int64_t K, const OpFmt& fb, int BN,
                                             int nkb, uint8_t* sB, float* thr, const EpiParams& ep,
                                             uint32_t* tmem_slot, int tid, const uint8_t* lutb = nullptr)
{
    constexpr int kSetupThreads = kWsProdWarp0 * 32;
    const int warp = tid >> 5, lane = tid & 31;
    griddep_wait();                                   // B and the alphas may come from the previous launch
    ws_decode_b<B4>(srcB, n0, K, fb, BN, nkb, sB, tid, kSetupThreads, lutb);
    fence_proxy_async_smem();
    if (warp == kWsMmaWarp) {
        asm volatile("bar.sync 1, %0;" ::"n"(kSetupThreads) : "memory");
    } else {
        asm volatile("bar.arrive 1, %0;" ::"n"(kSetupThreads) : "memory");
        ws_thresholds(thr, ep, warp, lane);
    }
    tc_fence_after();
    return *tmem_slot;
}

// Epilogue role (warps 0 .. epi_warps - 1): drains the accumulator tiles of
// this CTA in order, tile ti from TMEM buffer ti & 1 (columns (ti & 1) * BN
// ..), and frees the buffer on tempty once its columns are in registers.
// Warp w reads TMEM lanes 32 (w & 3) .. +31 (= tile rows); with split, warps
// 0-3 take the columns [0, BN/2) and warps 4-7 [BN/2, BN).  rows(ti, row, m)
// gives the output row m of a tile row and whether it exists.  LEAN4: the
// host has established 4-bit codes as the only output with a scalar scale
// and bias (every column chunk inside N, each warp's columns a multiple of
// 32); the instance then holds just the
// FMA-pipe requantisation and, for device values that rule it out, the
// out-of-line per-word path.  GEN: the output is not 4-bit codes; the
// instance holds the general-width code path and the out-of-line path for
// fp32/int32 outputs, and none of the 4-bit code (each instance keeps a
// small hot loop).
template <bool LEAN4, bool GEN, class RowMap>
__device__ __forceinline__ void ws_epilogue(const EpiParams& ep, const float* thr, const RowMap& rows,
                                            int64_t my_tiles, int64_t n0, int64_t N, int BN, bool split,
                                            int epi_warps, uint32_t tmem_base, float acc_scale, uint64_t* tfull,
                                            uint64_t* tempty, volatile int* err, int warp, int lane)
{
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;              // TMEM lane = tile row
    __shared__ EpiParams sh_ep;                       // copies for the out-of-line general path
    __shared__ EpiCtx sh_cx;
    const int half_cols = BN / 2;
    const int c_lo = split ? (warp >> 2) * half_cols : 0;
    const int c_hi = split ? c_lo + half_cols : BN;
    const EpiCtx cx = make_epi_ctx(ep, thr);
    const bool swar = ep.codes_out && ep.out.b == 4;
    const float sc_fixed = ep.scale ? 0.0f : (cx.dq ? __fmul_rn(ep.scale0, cx.dqs) : ep.scale0);
    const float sc_lean = sc_fixed * acc_scale;
    const bool out_signed = ep.out.is_signed != 0;
    // the lean path needs every column of the chunk inside N and a finite folded scale
    const bool lean_ok = swar && !ep.scale && !ep.bias && !ep.residual && !ep.acc_out && !ep.y_out &&
                         isfinite(sc_lean) && (sc_lean != 0.0f || sc_fixed == 0.0f);
    // With a positive scalar scale the requantised bucket is a monotone step
    // function of the exact integer accumulator, so the 7 thresholds on y
    // become 7 thresholds on the raw TMEM value (acc_raw_threshold, one lane
    // each); a signed output without activation keeps the general lean path.
    const bool raw_ok = lean_ok && sc_fixed > 0.0f && (!out_signed || ep.act != ESB_ACT_NONE);
    __shared__ float sh_raw[8];
    if (warp == 0) {
        if (lane == 0) { sh_ep = ep; sh_cx = cx; }
        if (raw_ok && lane < 7) sh_raw[lane] = acc_raw_threshold(sc_fixed, ep.bias0, thr[lane], ep.act, 1.0f / acc_scale);
    }
    // Output widths other than 4, codes only ("gen"): per element the
    // affine map, residual and activation, then the bucket by a bisection
    // over the 2^(b-1) - 1 thresholds; with a positive scalar scale (and an
    // unsigned output or an activation) over the same thresholds moved onto
    // the raw accumulator (gen_raw, as raw_ok above), one compare per level.
    const bool gen = GEN && !LEAN4 && ep.codes_out && ep.out.b != 4 && !ep.acc_out && !ep.y_out;
    const bool gen_raw = gen && !ep.scale && !ep.bias && !ep.residual && isfinite(sc_lean) && sc_fixed > 0.0f &&
                         (!out_signed || ep.act != ESB_ACT_NONE);
    // 4-bit codes out with a 4-bit residual and a scalar scale and bias
    // (ResNet's second conv of a block): per element y = fma(sc, acc, b),
    // then fma(res_scale, image of the residual code, y), activation and the
    // 7-threshold bucket, eight codes at a time; the residual's images come
    // from a 16-entry table.
    const bool lres = !LEAN4 && swar && !ep.scale && !ep.bias && !ep.acc_out && !ep.y_out && ep.residual &&
                      ep.res_b == 4 && isfinite(sc_lean) && (sc_lean != 0.0f || sc_fixed == 0.0f);
    __shared__ float sh_resimg[16];
    if (lres && warp == 0 && lane < 16) sh_resimg[lane] = code_image_f((uint32_t)lane, 4, ep.res_k);
    __shared__ float sh_rawT[128];                    // gen: the thresholds searched (raw or on y)
    __shared__ float sh_gres[GEN ? 256 : 1];          // gen: images of the residual's codes
    const bool gres = gen && !gen_raw && ep.residual;
    if (gres)
        for (int i = warp * 32 + lane; i < (1 << ep.res_b); i += epi_warps * 32)
            sh_gres[i] = code_image_f((uint32_t)i, ep.res_b, ep.res_k);
    if (gen) {
        const int nthr = (1 << (ep.out.b - 1)) - 1;
        for (int i = warp * 32 + lane; i < nthr; i += epi_warps * 32)
            sh_rawT[i] = gen_raw ? acc_raw_threshold(sc_fixed, ep.bias0, thr[i], ep.act, 1.0f / acc_scale) : thr[i];
    }
    asm volatile("bar.sync 2, %0;" ::"r"(epi_warps * 32) : "memory");   // exactly the epilogue warps in use
    const int cpw = ep.out_cpw;
    const float T0 = cx.t7.t[0], T1 = cx.t7.t[1], T2 = cx.t7.t[2], T3 = cx.t7.t[3], T4 = cx.t7.t[4],
                T5 = cx.t7.t[5], T6 = cx.t7.t[6];
    float R0 = 0.0f, R1 = 0.0f, R2 = 0.0f, R3 = 0.0f, R4 = 0.0f, R5 = 0.0f, R6 = 0.0f;
    if (raw_ok) {
        R0 = sh_raw[0]; R1 = sh_raw[1]; R2 = sh_raw[2]; R3 = sh_raw[3]; R4 = sh_raw[4]; R5 = sh_raw[5]; R6 = sh_raw[6];
    }
    // The same search on the FMA pipe when |acc| <= L - 2 < 2^20 (the ALU
    // pipe is the epilogue's bottleneck): with A_j = R_j / rs clamped to
    // [-L, L] and k_j = 1 - 2 A_j, sat(fma(raw, 2/rs, k_j)) = sat(2 acc -
    // 2 A_j + 1) is exactly [acc >= A_j] (an odd integer below 2^24 before
    // the clamp to [0, 1]); the next threshold is chosen by fmas with those
    // 0/1 factors, and the bucket bits are packed by fmas with powers of 16
    // (every intermediate an integer below 2^24: exact).
    const bool fma_ok = raw_ok && ep.acc_lim > 0.0f;
    float cK = 0.0f, K0 = 0.0f, K1 = 0.0f, K3 = 0.0f, D51 = 0.0f, D20 = 0.0f, D40 = 0.0f, E3 = 0.0f;
    if (fma_ok) {
        const float L = ep.acc_lim;
        auto kf = [&](float R) { return 1.0f - 2.0f * fminf(fmaxf(R * acc_scale, -L), L); };
        const float k0 = kf(R0), k1 = kf(R1), k2 = kf(R2), k3 = kf(R3), k4 = kf(R4), k5 = kf(R5), k6 = kf(R6);
        cK = 2.0f * acc_scale;
        K0 = k0; K1 = k1; K3 = k3;
        D51 = k5 - k1; D20 = k2 - k0; D40 = k4 - k0; E3 = (k6 - k4) - (k2 - k0);
    }
    // the warp holding the tile's last columns of the last N-tile writes the padding words
    const bool pad_words = ep.codes_out && (n0 + BN >= N) && ((n0 + BN) / cpw < ep.ldo) &&
                           (split ? (warp >> 2) == 1 : true);
    uint32_t zero_word = 0u;
    for (int j = 0; j < cpw; j++) zero_word |= ep.out.zero_code << (ep.out.b * j);
    for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
        const int a = (int)(ti & 1);
        if (!wait_or_abort(&tfull[a], (uint32_t)((ti >> 1) & 1), err)) { *err = 1; break; }
        tc_fence_after();
        int64_t m = 0;
        const bool mrow = rows(ti, row, m);
        const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(a * BN);
        uint32_t wsw[4] = {0u, 0u, (uint32_t)(((n0 + c_lo) / cpw) & 0xffffffff),
                           (uint32_t)(((n0 + c_lo) / cpw) >> 32)};   // general path: word, slot, column
        uint32_t gword = 0u;                          // gen path: word being packed, its next slot, its column
        int gslot = 0;
        int64_t gcol = (n0 + c_lo) / cpw;
        if (gen) {
            // columns [c_lo, c_end) are the warp's chunks holding outputs
            // inside N, 16 columns a chunk in four groups of four (a small
            // loop body with four independent threshold searches); the rest
            // of its columns are zero codes, written as whole words below
            const int64_t live = N - n0 - c_lo;
            const int c_end = live <= 0 ? c_lo : (int)((c_hi - c_lo < ((live + 15) >> 4) << 4)
                                                         ? c_hi : c_lo + (((live + 15) >> 4) << 4));
            if (c_end == c_lo) {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_tmem_free(&tempty[a]);
            }
            const int ob = ep.out.b, one = 1 << ep.out.k, nlev = ob - 1;
            const int half = 1 << (ob - 2);
            const uint32_t nk = (uint32_t)ep.out.N << ep.out.k;
            for (int c = c_lo; c < c_end; c += 16) {
                const bool last = c + 16 >= c_end;
#pragma unroll 1
                for (int g = 0; g < 4; g++) {
                    uint32_t r[4];
                    tmem_ld4(taddr + (uint32_t)(c + 4 * g), r);
                    if (last && g == 3) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive_tmem_free(&tempty[a]);
                    }
                    float v[4];
                    uint32_t sg[4];
                    // residual codes of the group's four columns: at most two words, one load each
                    const int rcpw = gres ? 32 / ep.res_b : 1;
                    uint32_t rw0 = 0u, rw1 = 0u;
                    int rsl0 = 0;
                    if (gres && mrow) {
                        const int col0 = (int)(n0 + c + 4 * g);
                        const int wq = col0 / rcpw;
                        rsl0 = col0 - wq * rcpw;
                        const uint32_t* rp = ep.residual + m * ep.res_ld + wq;
                        rw0 = __ldg(rp);
                        rw1 = (rsl0 + 3 >= rcpw && (int64_t)(wq + 1) * rcpw < N) ? __ldg(rp + 1) : rw0;
                    }
#pragma unroll
                    for (int i = 0; i < 4; i++) {
                        const int64_t n = n0 + c + 4 * g + i;
                        if (gen_raw) {
                            v[i] = __uint_as_float(r[i]);
                            sg[i] = 0u;
                        } else {
                            const int64_t nc = n < N ? n : N - 1;      // in-range index for the loads
                            float sc = sc_fixed;
                            if (ep.scale) { sc = __ldg(ep.scale + nc); if (cx.dq) sc = __fmul_rn(sc, cx.dqs); }
                            const float bi = ep.bias ? __ldg(ep.bias + nc) : ep.bias0;
                            float y = __fmaf_rn(sc, __uint_as_float(r[i]) * acc_scale, bi);
                            if (gres && mrow) {
                                const int sl = rsl0 + i;
                                const uint32_t wd = sl < rcpw ? rw0 : rw1;
                                const uint32_t rc = (wd >> (ep.res_b * (sl < rcpw ? sl : sl - rcpw))) &
                                                    ((1u << ep.res_b) - 1u);
                                y = __fmaf_rn(ep.res_scale, sh_gres[rc], y);
                            }
                            y = apply_act(y, ep.act);
                            sg[i] = (__float_as_uint(y) >> 31) & (out_signed ? 1u : 0u);
                            // an unsigned set maps negatives to zero: search -1
                            v[i] = (!out_signed && (__float_as_uint(y) >> 31)) ? -1.0f : fabsf(y);
                        }
                    }
                    int jb[4] = {0, 0, 0, 0};
#pragma unroll 1
                    for (int lv = 0; lv < nlev; lv++) {
                        const int step = half >> lv;
#pragma unroll
                        for (int i = 0; i < 4; i++) jb[i] += (v[i] >= sh_rawT[jb[i] + step - 1]) ? step : 0;
                    }
#pragma unroll
                    for (int i = 0; i < 4; i++) {
                        const uint32_t mag = (jb[i] >= one) ? (uint32_t)(jb[i] - one) : (nk | (uint32_t)jb[i]);
                        const bool zero = jb[i] == 0 || n0 + c + 4 * g + i >= N;
                        const uint32_t code = zero ? ep.out.zero_code : (mag | (sg[i] << (ob - 1)));
                        gword |= code << (ob * gslot);
                        if (++gslot == cpw) {
                            if (mrow && gcol < ep.ldo) ep.codes_out[m * ep.ldo + gcol] = gword;
                            gword = 0u;
                            gslot = 0;
                            gcol++;
                        }
                    }
                }
            }
            // the word in progress and the warp's remaining words: zero codes
            if (gslot != 0) {
                for (int j = gslot; j < cpw; j++) gword |= ep.out.zero_code << (ob * j);
                if (mrow && gcol < ep.ldo) ep.codes_out[m * ep.ldo + gcol] = gword;
                gword = 0u;
                gslot = 0;
                gcol++;
            }
            const int64_t wend = (n0 + c_hi) / cpw;
            if (mrow)
                for (; gcol < wend && gcol < ep.ldo; gcol++) ep.codes_out[m * ep.ldo + gcol] = zero_word;
        }
        for (int c = c_lo; c < (gen ? c_lo : c_hi); c += 16) {
            if (GEN || (!LEAN4 && !swar)) {
                epi_chunk_any(&sh_ep, &sh_cx, taddr + (uint32_t)c, acc_scale, m, mrow, n0 + c, N, wsw);
                if (c + 16 >= c_hi) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive_tmem_free(&tempty[a]);
                }
                continue;
            }
            if constexpr (!GEN) {
            // 4-bit output codes: 16 columns (two code words) per TMEM load
            // (compact code: measured faster than 32-column loads)
            constexpr int nc = 16;
            uint32_t r[16];
            tmem_ld16(taddr + (uint32_t)c, r);
            if (c + nc >= c_hi) {                     // every column of this warp is in registers
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_tmem_free(&tempty[a]);
            }
            // columns of the chunk inside N (codes past N are masked to the zero code)
            const int64_t ncl64 = N - (n0 + c);
            const int ncl = ncl64 < nc ? (int)ncl64 : nc;
            const bool lean = lean_ok && ncl > 0;
            uint32_t wds[2];
#pragma unroll
            for (int h = 0; h < 2; h++) {
                uint32_t J = 0u, S = 0u;
                const int live_h = ncl - 8 * h;       // nibbles of this word inside N
                const uint32_t nib = live_h >= 8 ? 0xffffffffu : (live_h <= 0 ? 0u : (1u << (4 * live_h)) - 1u);
                if (lean && fma_ok) {
                    float jh[2];
#pragma unroll
                    for (int q = 0; q < 2; q++) {
                        float jf = 0.0f;
#pragma unroll
                        for (int j = 3; j >= 0; j--) {
                            const float v = __uint_as_float(r[8 * h + 4 * q + j]);
                            const float b2 = __saturatef(__fmaf_rn(v, cK, K3));
                            const float b1 = __saturatef(__fmaf_rn(v, cK, __fmaf_rn(b2, D51, K1)));
                            const float t0 = __fmaf_rn(b1, __fmaf_rn(b2, E3, D20), __fmaf_rn(b2, D40, K0));
                            const float b0 = __saturatef(__fmaf_rn(v, cK, t0));
                            const float nb = __fmaf_rn(b2, 4.0f, __fmaf_rn(b1, 2.0f, b0));
                            jf = __fmaf_rn(jf, 16.0f, nb);       // nibbles of elements 3..0, element 0 lowest
                        }
                        jh[q] = jf + 8388608.0f;                   // integer jf < 2^16 in the low mantissa bits
                    }
                    J = (__float_as_uint(jh[0]) & 0xffffu) | (__float_as_uint(jh[1]) << 16);
                    wds[h] = codes8_b4(J & nib, 0u, ep.out.k);
                } else if (!LEAN4 && lean && raw_ok) {
                    // bucket = number of raw thresholds <= raw accumulator
#pragma unroll
                    for (int j = 0; j < 8; j++) {
                        const float v = __uint_as_float(r[8 * h + j]);
                        const bool b2 = v >= R3;
                        const bool b1 = v >= (b2 ? R5 : R1);
                        const bool b0 = v >= (b2 ? (b1 ? R6 : R4) : (b1 ? R2 : R0));
                        J |= ((b2 ? 4u : 0u) | (b1 ? 2u : 0u) | (b0 ? 1u : 0u)) << (4 * j);
                    }
                    wds[h] = codes8_b4(J & nib, 0u, ep.out.k);
                } else if (!LEAN4 && lean) {
                    // 4-bit output codes only, scalar scale/bias, no residual:
                    // y = fma(scale * 2^(kA+kB+12), raw, bias) equals
                    // fma(scale, acc, bias) exactly (power-of-two scaling),
                    // then the bucket of y among the 7 thresholds, eight
                    // codes per word at once.
#pragma unroll
                    for (int j = 0; j < 8; j++) {
                        float y = __fmaf_rn(sc_lean, __uint_as_float(r[8 * h + j]), ep.bias0);
                        y = apply_act(y, ep.act);
                        const float av = out_signed ? fabsf(y) : y;
                        const bool b2 = av >= T3;
                        const bool b1 = av >= (b2 ? T5 : T1);
                        const bool b0 = av >= (b2 ? (b1 ? T6 : T4) : (b1 ? T2 : T0));
                        J |= ((b2 ? 4u : 0u) | (b1 ? 2u : 0u) | (b0 ? 1u : 0u)) << (4 * j);
                        if (out_signed) S |= (__float_as_uint(y) >> 31) << (4 * j + 3);
                    }
                    wds[h] = codes8_b4(J & nib, S & nib, ep.out.k);
                } else if (!LEAN4 && lres && ncl > 0) {
                    const uint32_t rw = mrow ? __ldg(ep.residual + m * ep.res_ld + ((n0 + c) >> 3) + h) : 0u;
#pragma unroll
                    for (int j = 0; j < 8; j++) {
                        float y = __fmaf_rn(sc_lean, __uint_as_float(r[8 * h + j]), ep.bias0);
                        y = __fmaf_rn(ep.res_scale, sh_resimg[(rw >> (4 * j)) & 15u], y);
                        y = apply_act(y, ep.act);
                        const float av = out_signed ? fabsf(y) : y;
                        const bool b2 = av >= T3;
                        const bool b1 = av >= (b2 ? T5 : T1);
                        const bool b0 = av >= (b2 ? (b1 ? T6 : T4) : (b1 ? T2 : T0));
                        J |= ((b2 ? 4u : 0u) | (b1 ? 2u : 0u) | (b0 ? 1u : 0u)) << (4 * j);
                        if (out_signed) S |= (__float_as_uint(y) >> 31) << (4 * j + 3);
                    }
                    wds[h] = codes8_b4(J & nib, S & nib, ep.out.k);
                } else {
                    Raw8 v;
#pragma unroll
                    for (int j = 0; j < 8; j++) v.r[j] = r[8 * h + j];
                    wds[h] = epi_word_b4(&sh_ep, &sh_cx, v, acc_scale, sc_fixed, m, mrow, n0 + c + 8 * h, N);
                }
            }
            if (mrow) {
                // words w0, w0 + 1 of row m; a vector store only where the
                // address is aligned and both words are inside the row
                const int64_t w0 = (n0 + c) >> 3;
                uint32_t* dst = ep.codes_out + m * ep.ldo + w0;
                if (ep.codes_vec >= 2 && (w0 & 1) == 0 && w0 + 2 <= ep.ldo) {
                    *reinterpret_cast<uint2*>(dst) = make_uint2(wds[0], wds[1]);
                } else {
                    for (int q = 0; q < 2; q++)
                        if (w0 + q < ep.ldo) dst[q] = wds[q];
                }
            }
            }
        }
        // the last N-tile also fills the row's words past its columns (the
        // output row stride may hold more codes than the tiles cover) with
        // the zero code
        if (pad_words && mrow) {
            for (int64_t wq = (n0 + BN) / cpw; wq < ep.ldo; wq++) ep.codes_out[m * ep.ldo + wq] = zero_word;
        }
    }
}

// Bounded wait of the MMA thread for its own last commit before TMEM is
// freed (also on the abort path).
__device__ __forceinline__ void ws_drain(uint64_t* drain, volatile int* err)
{
    mma_commit(drain);
    volatile int no_abort = 0;
    if (!wait_or_abort(drain, 0u, &no_abort)) *err = 1;
}

// ------------------------------------------------------------- host side

// Launch with programmatic stream serialisation: the grid may start while
// the previous kernel of the stream finishes; the kernel's griddep_wait
// orders its dependent reads and writes after it.
template <class... KArgs, class... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

int pick_bn(int64_t N, int out_cpw);          // N-tile width (esb_gemm.cu)
int max_dyn_smem();                           // opt-in shared memory per block
EpiParams make_epi(const GemmOutputs& o);     // epilogue parameters of a call
float acc_fma_limit(int64_t K, int ba, int ka, int bb, int kb);   // FMA-pipe requantisation bound (esb_gemm.cu)

// Stride-1 convolution from a decoded input halo (esb_conv_halo.cu).  Returns
// false, launching nothing, when the shape does not suit it (stride != 1,
// A not 4-bit, rows wider than 128 - pad, too little of the tile used, or
// too little shared memory); otherwise launches and stores the launch
// status in *err.  BN is the preferred N-tile width; a smaller one is used
// when the resident filters would not fit.
bool conv_halo_ok(const esb_conv_desc& d, int P, int Q, int64_t ldx, int bx, int kx, int out_cpw);
bool launch_conv_halo(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, const OpFmt& fa,
                      const uint32_t* W, int64_t ldw, const OpFmt& fb, int BN, const EpiParams& ep, cudaStream_t st,
                      cudaError_t* err);

}  // namespace esb
