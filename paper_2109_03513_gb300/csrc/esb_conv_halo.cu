// esb_conv_halo.cu -- stride-1 ESB convolution from a decoded input halo
// (Sec. IV-B: the r x s x c_in x c_out convolution of the computing logic).
//
// The im2col kernel (esb_gemm.cu) decodes every input code once per filter
// tap.  Here a 128-row output tile is rows_out = 128 / Ws whole output rows
// of one image, each padded to a pitch of Ws pixel slots (Ws = the power of
// two >= w + pad).  The producers decode the rows_out + r - 1 input rows
// that tile needs ONCE into shared memory, pixel-linear: slot
// (i * Ws + j + pad) holds input pixel (row p0 - pad + i, column j), and the
// slots of columns w .. Ws - 1, of the left padding and of rows outside the
// image hold E4M3 zero bytes (the decoded zero code).  Each 16-code channel
// chunk is its own plane of slots x 16 bytes.
//
// Output pixel (p0 + pl, q) is tile row pl * Ws + q, and its tap (r, s)
// reads slot (pl * Ws + q) + r * Ws + s.  So tap (r, s) of the whole tile is
// the same buffer seen from a start address shifted by (r * Ws + s) * 16
// bytes: with A in the K-major no-swizzle layout (rows 16 bytes apart in
// 8-row core matrices, SBO = 128 bytes between them, LBO = one plane between
// 16-code chunks), every tap is one descriptor, and the MMA warp issues
// r * s * (chunks / 2) tcgen05.mma (K = 32) per tile from a single decode.
// B (the filters, K = (tap, channel)) is resident as in the GEMM kernel, and
// the epilogue is the shared one; rows with q >= Q or past the image's last
// output row are computed from zero slots and not stored.
//
// Channel blocks of 128 codes are separate stages, so a tile's halo never
// needs more than 8 planes of shared memory at once.
#include <cstdint>
#include <cuda_runtime.h>

#include "esb_tc.cuh"

namespace esb {

constexpr int kHaloDecoders = kWsProdWarps - 1;   // bulk path: warps decoding each tile together

struct HaloGeom {
    const uint32_t* X;   // n*h*w pixels of ldx words
    int ldx;             // words per pixel (multiple of 4)
    int H, W, P, Q, R, S, pad;
    int lws;             // log2(Ws)
    int rows_out;        // output rows per tile (128 / Ws)
    int tpi;             // tiles per image
    int hr;              // halo rows (rows_out + R - 1)
    int ns;              // slots per plane (128 + (R-1) * Ws + S - 1)
    int pb;              // bytes per plane (ns * 16)
    int cblocks;         // channel blocks of 16 words
    int spw;             // K slots per input word: 8 (4-bit codes, 5/6-bit word slots) or 16 (2/3-bit word slots)
    int stage_bytes;     // planes of one channel block (<= 8 planes), then raw rows
    int planes_bytes;    // the planes part of a stage
    int raw_bytes;       // raw code rows of a tile (one channel block only), or 0: register path
};

// The MMAs of one stage (channel block) with every offset a compile-time
// constant: slot pitch WS, an R x S filter, UT K steps of 32 codes per tap
// of which this block holds PAIRS, N-tile BN.  Straight-line issue, nothing
// but the tcgen05.mma between two MMAs.
template <int WS, int R, int S, int UT, int PAIRS, int BN>
__device__ __forceinline__ void halo_mma_fixed(uint32_t d, uint32_t a_st, uint32_t b_blk, uint32_t idesc,
                                               uint32_t& acc)
{
    constexpr int NS = 128 + (R - 1) * WS + S - 1;
    constexpr uint32_t PB = NS * 16;
    const uint64_t a_desc = smem_desc_noswz(a_st, PB, 128u);
    const uint64_t b_desc = smem_desc_sw128(b_blk);
#pragma unroll
    for (int t = 0; t < R * S; t++) {
#pragma unroll
        for (int j = 0; j < PAIRS; j++) {
            const uint32_t ao = (uint32_t)((((t / S) * WS + (t % S)) * 16 + 2 * j * (int)PB) >> 4);
            const int kq = t * UT + j;
            const uint32_t bo = (uint32_t)(((kq >> 2) * BN * 128 + (kq & 3) * 32) >> 4);
            mma_f8f6f4(d, a_desc + ao, b_desc + bo, idesc, acc);
            acc = 1u;
        }
    }
}

// One packed word of a 5- or 6-bit format in the word-slot layout (8 K
// slots per word, see plan_slots): code j to byte j through the E4M3 table,
// the slots past the word's codes zero.
__device__ __forceinline__ void decode_word_slot8(uint32_t w, const uint8_t* lut, int b, uint32_t& lo, uint32_t& hi)
{
    const int cpw = 32 / b;
    const uint32_t mask = (1u << b) - 1u;
    uint32_t o[2] = {0u, 0u};
#pragma unroll
    for (int j = 0; j < 8; j++)
        if (j < cpw) o[j >> 2] |= (uint32_t)lut[(w >> (b * j)) & mask] << (8 * (j & 3));
    lo = o[0];
    hi = o[1];
}

// One packed word of a 2- or 3-bit format in the word-slot layout (16 K
// slots per word): a whole 16-byte plane entry.
__device__ __forceinline__ uint4 decode_word_slot16(uint32_t w, const uint8_t* lut, int b)
{
    const int cpw = 32 / b;
    const uint32_t mask = (1u << b) - 1u;
    uint32_t o[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int j = 0; j < 16; j++)
        if (j < cpw) o[j >> 2] |= (uint32_t)lut[(w >> (b * j)) & mask] << (8 * (j & 3));
    return make_uint4(o[0], o[1], o[2], o[3]);
}

// Decode modes of the halo fill: 4-bit codes (SWAR), 5/6-bit word slots
// (8 per word), 2/3-bit word slots (16 per word).
enum { kHaloB4 = 0, kHaloSlot8 = 1, kHaloSlot16 = 2 };

// One 4-word piece (piece pc of the pixel in slot `slot`) into its planes:
// 2 planes (pc * 2 ..) for 8-slot words, 4 planes (pc * 4 ..) for 16-slot
// words; ok = false writes the E4M3 zero (outside the image).
template <int MODE>
__device__ __forceinline__ void halo_store_piece(uint8_t* st, int pb, int slot, int pc, bool ok, const uint4 v, int k,
                                                 int ew, const uint8_t* lut, int b)
{
    if (MODE == kHaloSlot16) {
        uint8_t* dst = st + (4 * pc) * pb + slot * 16;
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; i++)
            *reinterpret_cast<uint4*>(dst + i * pb) = ok ? decode_word_slot16(w[i], lut, b) : make_uint4(0u, 0u, 0u, 0u);
        return;
    }
    uint4 c0 = make_uint4(0u, 0u, 0u, 0u), c1 = c0;
    if (ok) {
        if (MODE == kHaloSlot8) {
            decode_word_slot8(v.x, lut, b, c0.x, c0.y);
            decode_word_slot8(v.y, lut, b, c0.z, c0.w);
            decode_word_slot8(v.z, lut, b, c1.x, c1.y);
            decode_word_slot8(v.w, lut, b, c1.z, c1.w);
        } else {
            decode_word_b4(v.x, k, ew, c0.x, c0.y);
            decode_word_b4(v.y, k, ew, c0.z, c0.w);
            decode_word_b4(v.z, k, ew, c1.x, c1.y);
            decode_word_b4(v.w, k, ew, c1.z, c1.w);
        }
    }
    uint8_t* dst = st + (2 * pc) * pb + slot * 16;
    *reinterpret_cast<uint4*>(dst) = c0;
    *reinterpret_cast<uint4*>(dst + pb) = c1;
}

// Producer: decode one channel block of one tile's halo into stage st.
// Lane l owns slots l, l + 32, ...; each slot takes NPC 16-byte pieces
// (4 words = two 16-code chunks each) of its pixel.  The pieces of up to
// 16 / NPC slot groups are loaded before any decode, so a fill makes at
// most a few round trips to memory.
template <int NPC, int MODE>
__device__ __forceinline__ void halo_fill_t(const HaloGeom& g, int p0, const uint32_t* xi, uint8_t* st, int lane,
                                            int k, int ew, const uint8_t* lut, int b)
{
    constexpr int GB = 16 / NPC;                                   // slot groups per batch
    const int groups = (g.ns + 31) >> 5;
    const int nb = (groups + GB - 1) / GB;
    const int per = (groups + nb - 1) / nb;                        // balanced batches
    const int wsm = (1 << g.lws) - 1;
#pragma unroll 1
    for (int g0 = 0; g0 < groups; g0 += per) {
        uint4 v[GB][NPC];
        uint32_t okm = 0u;
#pragma unroll
        for (int u = 0; u < GB; u++) {
            const int slot = (g0 + u) * 32 + lane;
            const int rel = slot - g.pad;
            const int hi = rel >> g.lws;                           // halo row (-1: left guard)
            const int j = rel & wsm;
            const int h = p0 - g.pad + hi;
            const bool ok = u < per && slot < g.ns && rel >= 0 && hi < g.hr && j < g.W && (unsigned)h < (unsigned)g.H;
            const uint4* px = reinterpret_cast<const uint4*>(xi + ((int64_t)h * g.W + j) * g.ldx);
#pragma unroll
            for (int pc = 0; pc < NPC; pc++) v[u][pc] = ok ? __ldg(px + pc) : make_uint4(0u, 0u, 0u, 0u);
            okm |= (ok ? 1u : 0u) << u;
        }
#pragma unroll
        for (int u = 0; u < GB; u++) {
            const int slot = (g0 + u) * 32 + lane;
            if (u >= per || slot >= g.ns) break;
            const bool ok = (okm >> u) & 1u;
#pragma unroll
            for (int pc = 0; pc < NPC; pc++) halo_store_piece<MODE>(st, g.pb, slot, pc, ok, v[u][pc], k, ew, lut, b);
        }
    }
}

// Bulk-copy fills (one channel block, ldx <= 16 words).  The copy issuer
// (one thread) copies the input rows of tile T that lie inside the image,
// whole (w pixels of ldx words, contiguous in NHWC), into the stage's raw
// area with one cp.async.bulk each, completing on mbarrier `raw_bar`.
__device__ __forceinline__ void halo_issue_rows(const HaloGeom& g, int64_t T, uint8_t* st, uint64_t* raw_bar)
{
    const int nimg = (int)(T / g.tpi);
    const int p0 = (int)(T - (int64_t)nimg * g.tpi) * g.rows_out;
    uint8_t* raw = st + g.planes_bytes;
    const int row_words = g.W * g.ldx;
    int valid = 0;
    for (int i = 0; i < g.hr; i++) {
        const int h = p0 - g.pad + i;
        valid += (h >= 0 && h < g.H) ? 1 : 0;
    }
    mbar_arrive_expect_tx(raw_bar, (uint32_t)(valid * row_words * 4));
    for (int i = 0; i < g.hr; i++) {
        const int h = p0 - g.pad + i;
        if (h >= 0 && h < g.H)
            bulk_copy_g2s(raw + (size_t)i * row_words * 4, g.X + ((int64_t)nimg * g.H + h) * row_words,
                          (uint32_t)(row_words * 4), raw_bar);
    }
}

// The decoders' share of one bulk-filled tile: slots first, first + stride,
// ... (zeros for padding slots and rows outside the image).
template <int NPC, int MODE>
__device__ __forceinline__ void halo_decode_t(const HaloGeom& g, int64_t T, uint8_t* st, int first, int stride, int k,
                                              int ew, const uint8_t* lut, int b)
{
    const int nimg = (int)(T / g.tpi);
    const int p0 = (int)(T - (int64_t)nimg * g.tpi) * g.rows_out;
    const uint8_t* raw = st + g.planes_bytes;
    const int wsm = (1 << g.lws) - 1;
#pragma unroll 1                                      // compact: it shares the SM's instruction cache
    for (int slot = first; slot < g.ns; slot += stride) {
        const int rel = slot - g.pad;
        const int hi = rel >> g.lws;
        const int j = rel & wsm;
        const int h = p0 - g.pad + hi;
        const bool ok = rel >= 0 && hi < g.hr && j < g.W && (unsigned)h < (unsigned)g.H;
        const uint4* src = reinterpret_cast<const uint4*>(raw + ((size_t)hi * g.W + j) * g.ldx * 4);
#pragma unroll 1                                      // one piece at a time: a small loop body
        for (int pc = 0; pc < NPC; pc++)
            halo_store_piece<MODE>(st, g.pb, slot, pc, ok, ok ? src[pc] : make_uint4(0u, 0u, 0u, 0u), k, ew, lut, b);
    }
}

// lut: the E4M3 table of a 5/6-bit word-slot input (nullptr: 4-bit codes).
__device__ __noinline__ void halo_decode(const HaloGeom g, int64_t T, uint8_t* st, int first, int stride, int k, int ew,
                                         const uint8_t* lut, int b)
{
    if (lut && g.spw == 16) {
        switch (g.ldx >> 2) {
        case 1: halo_decode_t<1, kHaloSlot16>(g, T, st, first, stride, k, ew, lut, b); break;
        case 2: halo_decode_t<2, kHaloSlot16>(g, T, st, first, stride, k, ew, lut, b); break;
        case 3: halo_decode_t<3, kHaloSlot16>(g, T, st, first, stride, k, ew, lut, b); break;
        default: halo_decode_t<4, kHaloSlot16>(g, T, st, first, stride, k, ew, lut, b); break;
        }
        return;
    }
    if (lut) {
        switch (g.ldx >> 2) {
        case 1: halo_decode_t<1, kHaloSlot8>(g, T, st, first, stride, k, ew, lut, b); break;
        case 2: halo_decode_t<2, kHaloSlot8>(g, T, st, first, stride, k, ew, lut, b); break;
        case 3: halo_decode_t<3, kHaloSlot8>(g, T, st, first, stride, k, ew, lut, b); break;
        default: halo_decode_t<4, kHaloSlot8>(g, T, st, first, stride, k, ew, lut, b); break;
        }
        return;
    }
    switch (g.ldx >> 2) {
    case 1: halo_decode_t<1, kHaloB4>(g, T, st, first, stride, k, ew, lut, b); break;
    case 2: halo_decode_t<2, kHaloB4>(g, T, st, first, stride, k, ew, lut, b); break;
    case 3: halo_decode_t<3, kHaloB4>(g, T, st, first, stride, k, ew, lut, b); break;
    default: halo_decode_t<4, kHaloB4>(g, T, st, first, stride, k, ew, lut, b); break;
    }
}

// Channel block cb (words 16 cb .. of each pixel) of tile T's halo.
__device__ __noinline__ void halo_fill(const HaloGeom g, int64_t T, int cb, uint8_t* st, int lane, int k, int ew,
                                       const uint8_t* lut, int b)
{
    const int nimg = (int)(T / g.tpi);
    const int p0 = (int)(T - (int64_t)nimg * g.tpi) * g.rows_out;
    const int w0 = cb * 16;
    const int npc = min(16, g.ldx - w0) >> 2;                      // pieces per slot (1..4)
    const uint32_t* xi = g.X + (int64_t)nimg * g.H * g.W * g.ldx + w0;
    if (lut && g.spw == 16) {
        switch (npc) {
        case 1: halo_fill_t<1, kHaloSlot16>(g, p0, xi, st, lane, k, ew, lut, b); break;
        case 2: halo_fill_t<2, kHaloSlot16>(g, p0, xi, st, lane, k, ew, lut, b); break;
        case 3: halo_fill_t<3, kHaloSlot16>(g, p0, xi, st, lane, k, ew, lut, b); break;
        default: halo_fill_t<4, kHaloSlot16>(g, p0, xi, st, lane, k, ew, lut, b); break;
        }
        return;
    }
    if (lut) {
        switch (npc) {
        case 1: halo_fill_t<1, kHaloSlot8>(g, p0, xi, st, lane, k, ew, lut, b); break;
        case 2: halo_fill_t<2, kHaloSlot8>(g, p0, xi, st, lane, k, ew, lut, b); break;
        case 3: halo_fill_t<3, kHaloSlot8>(g, p0, xi, st, lane, k, ew, lut, b); break;
        default: halo_fill_t<4, kHaloSlot8>(g, p0, xi, st, lane, k, ew, lut, b); break;
        }
        return;
    }
    switch (npc) {
    case 1: halo_fill_t<1, kHaloB4>(g, p0, xi, st, lane, k, ew, lut, b); break;
    case 2: halo_fill_t<2, kHaloB4>(g, p0, xi, st, lane, k, ew, lut, b); break;
    case 3: halo_fill_t<3, kHaloB4>(g, p0, xi, st, lane, k, ew, lut, b); break;
    default: halo_fill_t<4, kHaloB4>(g, p0, xi, st, lane, k, ew, lut, b); break;
    }
}

template <bool FAST, bool GEN>
__global__ void __launch_bounds__(kWsThreads, 1)
esb_conv_halo_kernel(HaloGeom g, RowsSrc srcB, int64_t N, int64_t K, OpFmt fa, OpFmt fb, int BN, int nkb,
                     int stages, int n_tiles, int64_t m_tiles, float acc_scale, EpiParams ep)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sB = smem;                                        // nkb blocks of BN x 128 bytes (SW128)
    uint8_t* sA = sB + nkb * BN * kBK;                         // stages x stage_bytes (halo planes)
    float* thr = reinterpret_cast<float*>(sA + stages * g.stage_bytes);
    uint64_t* full = reinterpret_cast<uint64_t*>(thr + 128);
    uint64_t* empty = full + kWsMaxStages;
    uint64_t* tfull = empty + kWsMaxStages;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint64_t* rawb = drain + 1;                                // kWsMaxStages: bulk-copy fills
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(rawb + kWsMaxStages);
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
    const int half_cols = BN / 2;
    const bool split = (half_cols % 16 == 0) && (half_cols % ep.out_cpw == 0);
    const int epi_warps = split ? 8 : 4;
    const int cbs = g.cblocks;
    // E4M3 tables of 5/6-bit word-slot operands (4-bit codes decode by SWAR)
    __shared__ uint8_t lut_a[64], lut_b[64];
    const bool slot_a = fa.spw != 0;
    if (slot_a) build_e4m3_lut(lut_a, fa, tid, kWsThreads);
    if (fb.spw != 0) build_e4m3_lut(lut_b, fb, tid, kWsThreads);
    // the layout above must fit the dynamic allocation (uniform for the CTA)
    if ((uintptr_t)(reinterpret_cast<const volatile uint8_t*>(err) + 4 - smem_raw) > dynamic_smem_bytes()) {
        if (tid == 0) record_status(ep.status, ESB_ERR_INTERNAL);
        return;
    }

    {
        // the CTA's rows of B into L2 while the previous grid may still be
        // finishing (weights are often no longer in L2 by the next call)
        const int64_t rows_b = (srcB.rows - n0) < (int64_t)BN ? (srcB.rows - n0) : (int64_t)BN;
        const char* b0 = reinterpret_cast<const char*>(srcB.base + n0 * srcB.ld);
        const int64_t bytes = rows_b > 0 ? rows_b * srcB.ld * 4 : 0;
        for (int64_t off = (int64_t)tid * 128; off < bytes; off += (int64_t)kWsThreads * 128) prefetch_l2(b0 + off);
    }
    if (tid == 0) {
        for (int s = 0; s < stages; s++) {
            // bulk path: the kKHaloDecoders decoder warps fill a stage together
            mbar_init(&full[s], g.raw_bytes > 0 ? kHaloDecoders : 1);
            mbar_init(&empty[s], 1);
            mbar_init(&rawb[s], 1);                   // the issuer's arrive.expect_tx, then the copies' bytes
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
    griddep_wait();                                   // X, B and the alphas may come from the previous launch
    griddep_launch_dependents();                      // every CTA is resident: the next grid may queue behind it

    // Setup.  Every warp but the bulk issuer (which starts the first tiles'
    // row copies at once) decodes its share of B, one row chunk per thread
    // where it can, so that B is ready after about one load round trip; the
    // MMA warp waits for all of it on named barrier 1, the others only
    // arrive.  The epilogue warps then build the requantisation thresholds
    // (named barrier 3) while the first tile is filled and multiplied.
    const bool bulk = FAST || g.raw_bytes > 0;
    if (!(bulk && warp == kWsProdWarp0)) {
        const int nbdec = bulk ? kWsThreads - 32 : kWsThreads;
        const int t = (bulk && warp > kWsProdWarp0) ? tid - 32 : tid;
        ws_decode_b<FAST>(srcB, n0, K, fb, BN, nkb, sB, t, nbdec, fb.spw ? lut_b : nullptr);
        fence_proxy_async_smem();
        if (warp == kWsMmaWarp) asm volatile("bar.sync 1, %0;" ::"r"(nbdec) : "memory");
        else asm volatile("bar.arrive 1, %0;" ::"r"(nbdec) : "memory");
    }
    if (warp < kWsEpiWarps) ws_thresholds(thr, ep, warp, lane);
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp >= kWsProdWarp0) {
        // ---------------------------------------------- halo producers
        const int p = warp - kWsProdWarp0;
        if (bulk) {
            // Bulk path, tiles in order: producer warp 0 issues the row copies
            // of every tile as soon as its stage is free (up to `stages` tiles
            // ahead); the other kHaloDecoders warps decode each tile together,
            // so the first tile is ready after one copy and a short decode.
            int s = 0;
            uint32_t ph = 0u;
            if (p == 0) {
                if (lane == 0) {
                    for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
                        if (!wait_or_abort(&empty[s], ph ^ 1u, err)) { *err = 1; break; }
                        halo_issue_rows(g, cta_in_n + ti * ctas_per_n, sA + s * g.stage_bytes, &rawb[s]);
                        if (++s == stages) { s = 0; ph ^= 1u; }
                    }
                }
            } else {
                const int d = p - 1;                  // decoder index 0 .. kHaloDecoders - 1
                for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
                    if (!wait_or_abort(&rawb[s], ph, err)) { *err = 1; break; }
                    halo_decode(g, cta_in_n + ti * ctas_per_n, sA + s * g.stage_bytes, d * 32 + lane,
                                kHaloDecoders * 32, fa.k, fa.ew, slot_a ? lut_a : nullptr, fa.b);
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&full[s]);
                    if (++s == stages) { s = 0; ph ^= 1u; }
                }
            }
        } else {
        // Register path (several channel blocks): warp p fills iterations p,
        // p + nprod, ... of this CTA's (tile, channel block) sequence; at most
        // `stages` producers are active (an mbarrier's parity tells apart
        // only adjacent phases).
        const int nprod = stages < kWsProdWarps ? stages : kWsProdWarps;
        const int64_t total_it = (p < nprod) ? my_tiles * cbs : 0;
        // stage s and its phase ph follow it incrementally (no division in
        // the loop): it advances by nprod <= stages, so s wraps at most once
        int s = p;
        uint32_t ph = 0u;
        for (int64_t it = p; it < total_it && !*err; it += nprod) {
            const int64_t ti = (cbs == 1) ? it : it / cbs;
            const int cb = (int)(it - ti * cbs);
            if (!wait_or_abort(&empty[s], ph ^ 1u, err)) { *err = 1; break; }
            halo_fill(g, cta_in_n + ti * ctas_per_n, cb, sA + s * g.stage_bytes, lane, fa.k, fa.ew,
                      slot_a ? lut_a : nullptr, fa.b);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&full[s]);
            s += nprod;
            if (s >= stages) { s -= stages; ph ^= 1u; }
        }
        }
    } else if (warp == kWsMmaWarp) {
        // ---------------------------------------------- MMA issue
        // Common geometries issue straight-line MMAs with constant offsets
        // (halo_mma_fixed); others compute the offsets in the loop.
        // Descriptors never come from shared memory: the tensor core's own
        // operand reads keep it close to saturated.
        if (lane == 0) {
            const uint32_t idesc = idesc_e4m3_f32(BN);
            const uint32_t b_base = smem_u32(sB), a_base = smem_u32(sA);
            const int ws = 1 << g.lws;
            const int units_tap = (g.ldx * g.spw) >> 5;        // 32-slot K steps per tap
            const bool r3 = g.R == 3 && g.S == 3;
            int s = 0;                                         // stage and phase of the next K-block
            uint32_t ph = 0u;
            for (int64_t ti = 0; ti < my_tiles && !*err; ti++) {
                const int a = (int)(ti & 1);
                if (!wait_or_abort(&tempty[a], (uint32_t)((ti >> 1) & 1) ^ 1u, err)) { *err = 1; break; }
                tc_fence_after();
                const uint32_t d = tmem_base + (uint32_t)(a * BN);
                uint32_t acc = 0u;
                for (int cb = 0; cb < cbs; cb++) {
                    if (!wait_or_abort(&full[s], ph, err)) { *err = 1; break; }
                    tc_fence_after();
                    const uint32_t a_st = a_base + (uint32_t)(s * g.stage_bytes);
                    const uint32_t b_blk = b_base + (uint32_t)(cb * BN * kBK);   // block cb: 4 K steps on
                    const int pairs = (min(16, g.ldx - cb * 16) * g.spw) >> 5;   // K steps (plane pairs) of the block
                    if (r3 && ws == 64 && units_tap == 2 && BN == 64) {           // 56 x 56 x 64
                        halo_mma_fixed<64, 3, 3, 2, 2, 64>(d, a_st, b_blk, idesc, acc);
                    } else if (r3 && ws == 32 && units_tap == 4 && BN == 128) {   // 28 x 28 x 128
                        halo_mma_fixed<32, 3, 3, 4, 4, 128>(d, a_st, b_blk, idesc, acc);
                    } else if (r3 && ws == 16 && units_tap == 8 && pairs == 4 && BN == 64) {   // 14 x 14 x 256
                        halo_mma_fixed<16, 3, 3, 8, 4, 64>(d, a_st, b_blk, idesc, acc);
                    } else {
                        for (int r = 0; r < g.R; r++) {
                            for (int sx = 0; sx < g.S; sx++) {
                                const uint32_t at = a_st + (uint32_t)((r * ws + sx) * 16);
                                const int kq0 = (r * g.S + sx) * units_tap + cb * (g.spw >> 1);
                                for (int j = 0; j < pairs; j++) {
                                    const int kq = kq0 + j;
                                    const uint32_t bb = b_base + (uint32_t)((kq >> 2) * BN * kBK + (kq & 3) * 32);
                                    mma_f8f6f4(d, smem_desc_noswz(at + (uint32_t)(2 * j * g.pb), (uint32_t)g.pb, 128u),
                                               smem_desc_sw128(bb), idesc, acc);
                                    acc = 1u;
                                }
                            }
                        }
                    }
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
        const int ctas = (int)ctas_per_n, first = (int)cta_in_n;   // tile counts fit in 32 bits (host check)
        const int tpi = g.tpi, rows_out = g.rows_out, lws = g.lws, P = g.P, Q = g.Q;
        auto rows = [=](int64_t ti, int row, int64_t& m) -> bool {
            const int T = first + (int)ti * ctas;
            const int nimg = T / tpi;
            const int p = (T - nimg * tpi) * rows_out + (row >> lws);
            const int q = row & ((1 << lws) - 1);
            m = ((int64_t)nimg * P + p) * Q + q;
            return q < Q && p < P;
        };
        ws_epilogue<FAST, GEN>(ep, thr, rows, my_tiles, n0, N, BN, split, epi_warps, tmem_base, acc_scale, tfull, tempty, err,
                    warp, lane);
    }

    __syncthreads();
    if (*err && tid == 0) record_status(ep.status, ESB_ERR_TIMEOUT);
    if (warp == kWsMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, tmem_cols);
    }
}

// Minimum share of the computed tile rows that are real output pixels for
// the halo path to be taken (56 x 56: 87.5 %; 7 x 7: 38 %, im2col instead).
constexpr double kHaloMinUse = 0.7;

struct HaloPlan {
    HaloGeom g;
    int BN, nkb, stages;
    int64_t K, smem;
};

// Static shared memory of the kernel (the larger of its two instances).
static int halo_static_smem(cudaError_t* err)
{
    static int v = -1;
    if (v < 0) {
        cudaFuncAttributes a0, a1, a2;
        *err = cudaFuncGetAttributes(&a0, esb_conv_halo_kernel<false, false>);
        if (*err != cudaSuccess) return -1;
        *err = cudaFuncGetAttributes(&a1, esb_conv_halo_kernel<true, false>);
        if (*err != cudaSuccess) return -1;
        *err = cudaFuncGetAttributes(&a2, esb_conv_halo_kernel<false, true>);
        if (*err != cudaSuccess) return -1;
        size_t m = a0.sharedSizeBytes > a1.sharedSizeBytes ? a0.sharedSizeBytes : a1.sharedSizeBytes;
        if (a2.sharedSizeBytes > m) m = a2.sharedSizeBytes;
        v = (int)m;
    }
    return v;
}

// Geometry, N-tile width and shared-memory budget of the halo path, or
// false when the shape does not suit it.  BN starts at bn0 and shrinks
// (keeping whole output words) until the resident B and two halo stages fit.
static bool halo_plan(const esb_conv_desc& d, int P, int Q, int64_t ldx, const OpFmt& fa, int bn0, int out_cpw,
                      HaloPlan* hp, cudaError_t* err)
{
    *err = cudaSuccess;
    // 4-bit codes, or 5/6-bit codes in the word-slot layout (8 K slots per
    // word, the same K per pixel word as 4-bit codes)
    const bool slot8 = fa.spw == 8 && (fa.b == 5 || fa.b == 6);
    const bool slot16 = fa.spw == 16 && (fa.b == 2 || fa.b == 3);
    if (d.stride != 1 || !(fa.b == 4 || slot8 || slot16) || fa.planes != 1 || ldx % 4 != 0 || ldx > (1 << 20) ||
        d.pad > d.r - 1 || d.pad > d.s - 1)
        return false;
    int lws = 0;
    while ((1 << lws) < d.w + d.pad) lws++;
    const int ws = 1 << lws;
    if (ws > kBM || Q > ws) return false;
    HaloGeom& g = hp->g;
    g.X = nullptr; g.ldx = (int)ldx; g.H = d.h; g.W = d.w; g.P = P; g.Q = Q; g.R = d.r; g.S = d.s; g.pad = d.pad;
    g.lws = lws;
    g.rows_out = kBM / ws;
    g.tpi = (P + g.rows_out - 1) / g.rows_out;
    if ((double)P * Q / ((double)g.tpi * kBM) < kHaloMinUse) return false;
    g.hr = g.rows_out + d.r - 1;
    g.ns = kBM + (d.r - 1) * ws + d.s - 1;
    g.pb = g.ns * 16;
    g.cblocks = (int)((ldx + 15) / 16);
    g.spw = slot16 ? 16 : 8;
    const int planes = (int)((ldx >= 16 ? 16 : ldx) * g.spw / 16);      // planes of one channel block
    g.planes_bytes = ((planes * g.pb + 127) / 128) * 128;
    // one channel block: the fill bulk-copies whole input rows to a raw area of the stage
    g.raw_bytes = (g.cblocks == 1) ? ((g.hr * d.w * (int)ldx * 4 + 127) / 128) * 128 : 0;
    g.stage_bytes = g.planes_bytes + g.raw_bytes;
    if ((int64_t)d.n * g.tpi >= (1ll << 30)) return false;
    const int st_smem = halo_static_smem(err);
    if (st_smem < 0) return false;
    const int maxs = max_dyn_smem() - st_smem;
    hp->K = (int64_t)d.r * d.s * ldx * g.spw;
    hp->nkb = (int)((hp->K + kBK - 1) / kBK);
    static const int cands[] = {256, 240, 224, 208, 192, 176, 160, 144, 128, 112, 96, 80, 64, 48, 32, 16};
    for (int i = -1; i < (int)(sizeof(cands) / sizeof(cands[0])); i++) {
        const int bn = i < 0 ? bn0 : cands[i];
        if (bn <= 0 || (i >= 0 && bn >= bn0) || bn % out_cpw != 0) continue;
        const int64_t fixed = 1024 + (int64_t)hp->nkb * bn * kBK + 4 * 128 + 512;
        int64_t stg = (maxs - fixed) / g.stage_bytes;
        if (stg > kWsMaxStages) stg = kWsMaxStages;
        if (stg < 2) continue;
        hp->BN = bn;
        hp->stages = (int)stg;
        hp->smem = fixed + stg * (int64_t)g.stage_bytes;
        return true;
    }
    return false;
}

bool conv_halo_ok(const esb_conv_desc& d, int P, int Q, int64_t ldx, int bx, int kx, int out_cpw)
{
    HaloPlan hp;
    cudaError_t e;
    OpFmt fa = make_opfmt(bx, kx);
    if (bx == 5 || bx == 6) fa.spw = 8;               // as plan_slots for same-width input and filters
    if (bx == 2 || bx == 3) fa.spw = 16;
    return halo_plan(d, P, Q, ldx, fa, pick_bn(d.cout, out_cpw), out_cpw, &hp, &e);
}

bool launch_conv_halo(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, const OpFmt& fa,
                      const uint32_t* W, int64_t ldw, const OpFmt& fb, int BN, const EpiParams& ep, cudaStream_t st,
                      cudaError_t* err)
{
    HaloPlan hp;
    if (!halo_plan(d, P, Q, ldx, fa, BN, ep.out_cpw, &hp, err)) return *err != cudaSuccess;
    if (hp.smem <= 0 || hp.smem > max_dyn_smem() - halo_static_smem(err)) {
        *err = cudaErrorInvalidConfiguration;
        return true;
    }
    hp.g.X = X;
    static bool configured = false;
    if (!configured) {
        *err = cudaFuncSetAttribute(esb_conv_halo_kernel<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    max_dyn_smem() - halo_static_smem(err));
        if (*err != cudaSuccess) return true;
        *err = cudaFuncSetAttribute(esb_conv_halo_kernel<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    max_dyn_smem() - halo_static_smem(err));
        if (*err != cudaSuccess) return true;
        *err = cudaFuncSetAttribute(esb_conv_halo_kernel<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    max_dyn_smem() - halo_static_smem(err));
        if (*err != cudaSuccess) return true;
        configured = true;
    }
    const int64_t N = d.cout;
    const int n_tiles = (int)((N + hp.BN - 1) / hp.BN);
    const int64_t m_tiles = (int64_t)d.n * hp.g.tpi;
    int64_t per_n = device_sm_count() / n_tiles;
    if (per_n < 1) per_n = 1;
    if (per_n > m_tiles) per_n = m_tiles;
    const int64_t grid = per_n * n_tiles;
    RowsSrc b{W, (int64_t)d.r * d.s * ldw, N};
    const float acc_scale = ldexpf(1.0f, fa.csc + fb.csc);
    // The specialised instance: 4-bit B, bulk-copied input rows and 4-bit
    // codes as the only output, with a scalar scale and bias, in whole N-tiles
    // and with a monotone requantisation (unsigned codes or an activation).
    const int half = hp.BN / 2;
    const bool split = (half % 16 == 0) && (half % ep.out_cpw == 0);
    const bool fast = fb.b == 4 && hp.g.raw_bytes > 0 && ep.codes_out && ep.out.b == 4 && !ep.scale && !ep.bias &&
                      !ep.residual && !ep.acc_out && !ep.y_out && ep.acc_lim > 0.0f && N % hp.BN == 0 &&
                      (!ep.out.is_signed || ep.act != ESB_ACT_NONE) && (split ? half : hp.BN) % 32 == 0;
    const bool gen = !(ep.codes_out && ep.out.b == 4);       // the general-width epilogue instance
    *err = launch_pdl(fast ? esb_conv_halo_kernel<true, false>
                           : (gen ? esb_conv_halo_kernel<false, true> : esb_conv_halo_kernel<false, false>),
                      dim3((unsigned)grid), dim3(kWsThreads), (size_t)hp.smem, st, hp.g, b, N,
                      hp.K, fa, fb, hp.BN, hp.nkb, hp.stages, n_tiles, m_tiles, acc_scale, ep);
    return true;
}

}  // namespace esb
