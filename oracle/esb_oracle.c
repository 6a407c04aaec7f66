/*
 * esb_oracle.c -- plain, slow, obviously-correct CPU reference of Elastic
 * Significant Bit (ESB) quantization (Gong et al., "Elastic Significant Bit
 * Quantization and Acceleration for Deep Neural Networks", arXiv 2109.03513).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call this file:
 * only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg load it.
 * It shares no code, header, table or constant generator with the CUDA
 * library; the two are written independently from the paper.
 *
 * Every function follows one passage of the paper (cited per function) and
 * uses no blocking, fusion or reordering beyond it.  Floating point is fp64
 * except where the method itself fixes fp32 (the x/alpha division of
 * Eq. cheap_projection and the fp32 epilogue, whose op order is pinned).
 * Build: gcc -O2 -std=c11 -ffp-contract=off -fno-fast-math -shared -fPIC.
 *
 * Conventions shared with the test-suite (not with the CUDA code):
 *   fmt = (b, k, is_signed); N = 2^(b-k-1) - 1 (Sec. III-B).
 *   Values are handled "in units of alpha": q = element of the set
 *   U_{i=0..N} xi_i * Omega_i, and the integer image is I = q * 2^k.
 *   Code bit layout (Sec. IV-A, ESB float format): sign | e (b-k-1 bits) |
 *   f (k bits), MSB to LSB; e = N marks the "0.f" values; zero has sign 0.
 *   Packing: floor(32/b) codes per 32-bit word, code j of a row in bits
 *   [b*(j%cpw), b*(j%cpw)+b) of word j/cpw; unused slots hold the zero code,
 *   unused high bits are 0.
 */
#define _GNU_SOURCE
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_MAX_SET 4096

/* N = 2^(b-k-1) - 1: the number of shifted fraction sets beyond Omega_0
 * (Sec. III-B, Eq. epot_quantization_expression). */
int oracle_N(int b, int k) { return (1 << (b - k - 1)) - 1; }

int oracle_format_ok(int b, int k) { return b >= 2 && b <= 8 && k >= 0 && k <= b - 1; }

/* Non-negative part of the set, in units of alpha, ascending.
 * Sec. III-B: Omega_0 = {0..2^k-1}, Omega_i = {2^k..2^(k+1)-1} (i>0),
 * xi_0 = 2^-k, xi_i = 2^(i-k-1) (i>0).  Returns the element count 2^(b-1). */
int oracle_set_nonneg(int b, int k, double *out)
{
    int N = oracle_N(b, k);
    int n = 0;
    for (int f = 0; f < (1 << k); f++)            /* xi_0 * Omega_0 */
        out[n++] = ldexp((double)f, -k);
    for (int i = 1; i <= N; i++)                   /* xi_i * Omega_i */
        for (int f = 0; f < (1 << k); f++)
            out[n++] = ldexp((double)((1 << k) + f), i - k - 1);
    return n;
}

/* Full signed set (2^b - 1 elements, one zero), ascending. */
int oracle_set_full(int b, int k, double *out)
{
    double pos[ORACLE_MAX_SET];
    int n = oracle_set_nonneg(b, k, pos);
    int m = 0;
    for (int j = n - 1; j >= 1; j--) out[m++] = -pos[j];
    for (int j = 0; j < n; j++) out[m++] = pos[j];
    return m;
}

/* C = max(xi_N * Omega_N) (Sec. III-C, below Eq. thresholing_func). */
double oracle_C(int b, int k)
{
    double s[ORACLE_MAX_SET];
    int n = oracle_set_nonneg(b, k, s);
    return s[n - 1];
}

/* Eq. thresholing_func: the look-up projection P(a) of a magnitude a in
 * [0, C] onto the non-negative set.  Element q_j owns the half-open
 * interval [ (q_{j-1}+q_j)/2, (q_j+q_{j+1})/2 ); the first interval starts
 * at 0, the last one ends at C inclusive.  A value on a midpoint therefore
 * goes to the larger element ("half away from zero" on the magnitude).
 * rounding = 1 replaces that tie rule by "the element whose multiple of the
 * local spacing is even" (optional rounding; not the paper's default).
 * Midpoints of dyadic set elements are exact in fp64, and a is an fp32
 * value, so every comparison below is exact. */
static double lookup_projection(double a, const double *s, int n, int rounding)
{
    for (int j = n - 1; j >= 1; j--) {
        double lo = 0.5 * (s[j - 1] + s[j]);
        if (a > lo) return s[j];
        if (a == lo) {
            if (rounding == 0) return s[j];
            double spacing = s[j] - s[j - 1];
            double r = s[j] / spacing;          /* integer-valued */
            return (fmod(r, 2.0) == 0.0) ? s[j] : s[j - 1];
        }
    }
    return s[0];
}

/* Eq. cheap_projection: v = fl32(x / alpha) (one IEEE single division),
 * clip to [-C, C], project the magnitude with Eq. thresholing_func, restore
 * the sign.  Returns the projected value in units of alpha (q; the
 * quantized weight is alpha * q).  Unsigned formats use the non-negative
 * half of the set, so negative inputs go to 0.  NaN goes to 0. */
double oracle_project_value(float x, float alpha, int b, int k, int is_signed, int rounding)
{
    double s[ORACLE_MAX_SET];
    int n = oracle_set_nonneg(b, k, s);
    float v = x / alpha;
    if (isnan(v)) return 0.0;
    int neg = v < 0.0f;
    double a = fabs((double)v);
    if (neg && !is_signed) return 0.0;
    double C = s[n - 1];
    if (a > C) a = C;
    double q = lookup_projection(a, s, n, rounding);
    return neg ? -q : q;
}

/* Eq. fast_projection, written independently as a second formulation of
 * the same projection: keep k+1 significant bits of |v| starting at its
 * most significant 1 bit n, round the rest.  The paper's n = max{i: v>=2^i}
 * is read as max(floor(log2|v|), 0) so that values below 1 use the spacing
 * of xi_0 (the reading that makes Eq. fast_projection equal
 * Eq. thresholing_func).  Used only to cross-check the look-up form. */
double oracle_project_value_shift(float x, float alpha, int b, int k, int is_signed, int rounding)
{
    float v = x / alpha;
    if (isnan(v)) return 0.0;
    int neg = v < 0.0f;
    if (neg && !is_signed) return 0.0;
    double a = fabs((double)v);
    double C = oracle_C(b, k);
    if (a > C) a = C;
    int n = 0;
    if (a >= 1.0) {
        int ex;
        frexp(a, &ex);            /* a = m * 2^ex, m in [0.5,1) */
        n = ex - 1;
    }
    double quantum = ldexp(1.0, n - k);
    double r = a / quantum;       /* exact: power-of-two scaling */
    double fl = floor(r);
    double R;
    if (r - fl > 0.5) R = fl + 1.0;
    else if (r - fl < 0.5) R = fl;
    else R = (rounding == 0) ? fl + 1.0 : ((fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0);
    double q = R * quantum;
    return neg ? -q : q;
}

/* Array form of oracle_project_value_shift (values in units of alpha). */
void oracle_project_values_shift(const float *x, int64_t n, float alpha, int b, int k,
                                 int is_signed, int rounding, double *q)
{
    for (int64_t i = 0; i < n; i++)
        q[i] = oracle_project_value_shift(x[i], alpha, b, k, is_signed, rounding);
}

/* Array form of oracle_project_value (values in units of alpha). */
void oracle_project_values(const float *x, int64_t n, float alpha, int b, int k,
                           int is_signed, int rounding, double *q)
{
    for (int64_t i = 0; i < n; i++)
        q[i] = oracle_project_value(x[i], alpha, b, k, is_signed, rounding);
}

/* Sec. IV-A, ESB float format: the code of a set element q (units of
 * alpha): q = 0.f for e = N, q = 2^e * 1.f otherwise.  Found by searching
 * every (e, f) pair.  Returns 0xFFFFFFFF if q is not in the set. */
uint32_t oracle_encode(double q, int b, int k, int is_signed)
{
    int N = oracle_N(b, k);
    uint32_t sign = (q < 0.0) ? 1u : 0u;
    double m = fabs(q);
    if (m == 0.0) sign = 0;                 /* zero always carries sign 0 */
    if (sign && !is_signed) return 0xFFFFFFFFu;
    int ew = b - k - 1;
    for (int e = 0; e <= N; e++) {
        for (int f = 0; f < (1 << k); f++) {
            double val = (e == N) ? ldexp((double)f, -k)
                                  : ldexp(1.0 + ldexp((double)f, -k), e);
            if (val == m)
                return (sign << (b - 1)) | ((uint32_t)e << k) | (uint32_t)f;
        }
    }
    (void)ew;
    return 0xFFFFFFFFu;
}

/* Sec. IV-A, Eq. q: value (units of alpha) of a b-bit code. */
double oracle_decode(uint32_t code, int b, int k)
{
    int N = oracle_N(b, k);
    uint32_t sign = (code >> (b - 1)) & 1u;
    uint32_t e = (b - k - 1 > 0) ? (code >> k) & ((1u << (b - k - 1)) - 1u) : 0u;
    uint32_t f = code & ((1u << k) - 1u);
    double mag = ((int)e == N) ? ldexp((double)f, -k)
                               : ldexp(1.0 + ldexp((double)f, -k), (int)e);
    return sign ? -mag : mag;
}

uint32_t oracle_zero_code(int b, int k) { return oracle_encode(0.0, b, k, 1); }

/* Projection of an fp32 array to codes (one code per uint32, unpacked). */
void oracle_project_codes(const float *x, int64_t n, float alpha, int b, int k,
                          int is_signed, int rounding, uint32_t *codes)
{
    for (int64_t i = 0; i < n; i++)
        codes[i] = oracle_encode(oracle_project_value(x[i], alpha, b, k, is_signed, rounding),
                                 b, k, is_signed);
}

/* Packing of a rows x cols code matrix into rows of ld_words 32-bit words. */
void oracle_pack(const uint32_t *codes, int64_t rows, int64_t cols, int b, int k,
                 int64_t ld_words, uint32_t *out)
{
    int cpw = 32 / b;
    uint32_t zero = oracle_zero_code(b, k);
    for (int64_t r = 0; r < rows; r++)
        for (int64_t w = 0; w < ld_words; w++) {
            uint32_t word = 0;
            for (int j = 0; j < cpw; j++) {
                int64_t c = w * cpw + j;
                uint32_t code = (c < cols) ? codes[r * cols + c] : zero;
                word |= code << (b * j);
            }
            out[r * ld_words + w] = word;
        }
}

void oracle_unpack(const uint32_t *words, int64_t rows, int64_t cols, int b,
                   int64_t ld_words, uint32_t *codes)
{
    int cpw = 32 / b;
    uint32_t mask = (1u << b) - 1u;
    for (int64_t r = 0; r < rows; r++)
        for (int64_t c = 0; c < cols; c++)
            codes[r * cols + c] = (words[r * ld_words + c / cpw] >> (b * (c % cpw))) & mask;
}

/* ---------------------------------------------------------------------- */
/* Distribution difference aligner (Sec. III-D).                           */

static double std_phi(double t) { return exp(-0.5 * t * t) / 2.5066282746310002; }
static double std_Q(double t) { return 0.5 * erfc(t / sqrt(2.0)); }   /* 1 - Phi(t) */

/* Integral of (t-q)^2 phi(t) over [lo, hi] (hi may be +inf), from the
 * antiderivative (1+q^2) Phi(t) + (2q - t) phi(t), written with the upper
 * tail Q = 1 - Phi for accuracy at large t. */
static double cell_error(double lo, double hi, double q)
{
    double up = isinf(hi) ? 0.0 : (2.0 * q - hi) * std_phi(hi);
    double Qhi = isinf(hi) ? 0.0 : std_Q(hi);
    return (1.0 + q * q) * (std_Q(lo) - Qhi) + up - (2.0 * q - lo) * std_phi(lo);
}

/* Eq. objective_function_expansion: D(alpha, b, k) over the non-negative
 * half with p(t) = N(0, 1) (Sec. III-D, "Resolving extremum"); the cell of
 * each element alpha*q_j is bounded by the midpoints to its neighbours, the
 * first cell starts at 0 and the last runs to infinity. */
double oracle_D(double alpha, int b, int k)
{
    double s[ORACLE_MAX_SET];
    int n = oracle_set_nonneg(b, k, s);
    double D = 0.0;
    for (int j = 0; j < n; j++) {
        double q = alpha * s[j];
        double lo = (j == 0) ? 0.0 : alpha * 0.5 * (s[j - 1] + s[j]);
        double hi = (j == n - 1) ? INFINITY : alpha * 0.5 * (s[j] + s[j + 1]);
        D += cell_error(lo, hi, q);
    }
    return D;
}

/* dD/dalpha.  Differentiating Eq. objective_function_expansion, the terms
 * from the moving cell boundaries cancel (a boundary is the midpoint of its
 * two elements, equally far from both), leaving
 *   D'(alpha) = -2 sum_j q_j int_{cell j} (t - alpha q_j) phi(t) dt,
 * with int t phi = phi(lo) - phi(hi) and int phi = Q(lo) - Q(hi). */
double oracle_dD(double alpha, int b, int k)
{
    double s[ORACLE_MAX_SET];
    int n = oracle_set_nonneg(b, k, s);
    double g = 0.0;
    for (int j = 0; j < n; j++) {
        double lo = (j == 0) ? 0.0 : alpha * 0.5 * (s[j - 1] + s[j]);
        double m1, m0;
        if (j == n - 1) { m1 = std_phi(lo); m0 = std_Q(lo); }
        else {
            double hi = alpha * 0.5 * (s[j] + s[j + 1]);
            m1 = std_phi(lo) - std_phi(hi);
            m0 = std_Q(lo) - std_Q(hi);
        }
        g += -2.0 * s[j] * (m1 - alpha * s[j] * m0);
    }
    return g;
}

/* Eq. optimal_alpha_seeking: alpha* = argmin D.  D is not convex for large
 * N; the reading used here is "the first local minimum from small alpha"
 * (Sec. III-D resolves the extremum of the differentiable D; Fig. 7 plots
 * D and its first and second derivatives).  The minimum is bracketed on a
 * 20000-point log grid over [1e-4, 4], then located as the zero of D' by
 * bisection to full fp64 precision.  Returns alpha*, and D(alpha*) via D_out. */
double oracle_alpha_star(int b, int k, double *D_out)
{
    const int G = 20000;
    const double lo = 1e-4, hi = 4.0;
    double *a = (double *)malloc(sizeof(double) * G);
    double *d = (double *)malloc(sizeof(double) * G);
    for (int i = 0; i < G; i++) {
        a[i] = lo * pow(hi / lo, (double)i / (double)(G - 1));
        d[i] = oracle_D(a[i], b, k);
    }
    int im = G - 1;
    for (int i = 1; i < G - 1; i++)
        if (d[i] <= d[i - 1] && d[i] < d[i + 1]) { im = i; break; }
    double x0 = a[im > 0 ? im - 1 : 0], x1 = a[im < G - 1 ? im + 1 : G - 1];
    free(a);
    free(d);
    /* D' < 0 at x0 and > 0 at x1 around an interior minimum. */
    for (int it = 0; it < 200; it++) {
        double xm = 0.5 * (x0 + x1);
        if (xm <= x0 || xm >= x1) break;
        if (oracle_dD(xm, b, k) < 0.0) x0 = xm; else x1 = xm;
    }
    double as = 0.5 * (x0 + x1);
    if (D_out) *D_out = oracle_D(as, b, k);
    return as;
}

/* Sec. III-D, Normalization: mu = (1/d) sum x, sigma = sqrt((1/d) sum (x-mu)^2),
 * two passes in fp64.  Signed formats: alpha = fl32(alpha* (sigma + 1e-7)).
 * Unsigned formats (post-ReLU data, the non-negative half of the set):
 * alpha = fl32(alpha* (rms + 1e-7)) with rms = sqrt((1/d) sum x^2), the scale
 * of the underlying normal of a half-normal.  stats = {mu, sigma|rms, d}.
 * alpha_star is oracle_alpha_star(b, k) of the format, solved once by the caller. */
float oracle_calibrate_with(const float *x, int64_t d, double alpha_star, int is_signed, double *stats)
{
    double s = 0.0;
    for (int64_t i = 0; i < d; i++) s += (double)x[i];
    double mu = s / (double)d;
    double ss = 0.0;
    for (int64_t i = 0; i < d; i++) {
        double c = is_signed ? ((double)x[i] - mu) : (double)x[i];
        ss += c * c;
    }
    double spread = sqrt(ss / (double)d);
    if (stats) { stats[0] = mu; stats[1] = spread; stats[2] = (double)d; }
    return (float)(alpha_star * (spread + 1e-7));
}

/* ---------------------------------------------------------------------- */
/* Contraction and the post-processing of Sec. IV-B/IV-C.                  */

/* Integer image I = q * 2^k of a code (exact; fits int64 for the formats
 * the contraction accepts). */
static int64_t image_of(uint32_t code, int b, int k)
{
    return (int64_t)ldexp(oracle_decode(code, b, k), k);
}

/* Table of image_of over all 2^b codes (built once per call). */
static void image_table(int b, int k, int64_t *t)
{
    for (uint32_t c = 0; c < (1u << b); c++) t[c] = image_of(c, b, k);
}

/* C[m][n] = sum_k I(A[m][k]) * I(B[n][k]) in int64 (Sec. III-B: the product
 * of two set elements is the product of their fraction values and shifts;
 * Sec. IV-B: a convolution is a multiply-accumulate over c_in * K * K).
 * A: M x K codes packed in rows of lda words, B: N x K packed in rows of
 * ldb words (both K-major). */
void oracle_gemm_i64(const uint32_t *A, int64_t lda, int ba, int ka,
                     const uint32_t *B, int64_t ldb, int bb, int kb,
                     int64_t M, int64_t N, int64_t K, int64_t *C)
{
    int cpa = 32 / ba, cpb = 32 / bb;
    uint32_t ma = (1u << ba) - 1u, mb = (1u << bb) - 1u;
    int64_t ta[256], tb[256];
    image_table(ba, ka, ta);
    image_table(bb, kb, tb);
    for (int64_t m = 0; m < M; m++)
        for (int64_t n = 0; n < N; n++) {
            int64_t acc = 0;
            for (int64_t kk = 0; kk < K; kk++) {
                uint32_t ca = (A[m * lda + kk / cpa] >> (ba * (kk % cpa))) & ma;
                uint32_t cb = (B[n * ldb + kk / cpb] >> (bb * (kk % cpb))) & mb;
                acc += ta[ca] * tb[cb];
            }
            C[m * N + n] = acc;
        }
}

/* One entry C[m][n] (for sampled checks of large problems). */
int64_t oracle_gemm_entry(const uint32_t *A, int64_t lda, int ba, int ka,
                          const uint32_t *B, int64_t ldb, int bb, int kb,
                          int64_t K, int64_t m, int64_t n)
{
    int cpa = 32 / ba, cpb = 32 / bb;
    uint32_t ma = (1u << ba) - 1u, mb = (1u << bb) - 1u;
    int64_t ta[256], tb[256];
    image_table(ba, ka, ta);
    image_table(bb, kb, tb);
    int64_t acc = 0;
    for (int64_t kk = 0; kk < K; kk++) {
        uint32_t ca = (A[m * lda + kk / cpa] >> (ba * (kk % cpa))) & ma;
        uint32_t cb = (B[n * ldb + kk / cpb] >> (bb * (kk % cpb))) & mb;
        acc += ta[ca] * tb[cb];
    }
    return acc;
}

/* Post-processing of one accumulator (Sec. IV-C "BN and DN" and "ESB
 * quantization" steps, with this library's pinned fp32 op order):
 *   y = fmaf(scale, (float)acc, bias)
 *   y = fmaf(res_scale, (float)I_res, y)          (if has_res)
 *   y = max(y, 0) / min(max(y, 0), 6)             (act 1 / act 2)
 *   code = projection of y with alpha_out         (Eq. cheap_projection)
 * Returns y; writes the output code. */
float oracle_epilogue_one(int64_t acc, float scale, float bias, int has_res, int64_t I_res,
                          float res_scale, int act, float alpha_out, int bo, int ko,
                          int so, int rounding, uint32_t *code_out)
{
    float y = fmaf(scale, (float)acc, bias);
    if (has_res) y = fmaf(res_scale, (float)I_res, y);
    if (act == 1) y = (y > 0.0f) ? y : 0.0f;
    else if (act == 2) { y = (y > 0.0f) ? y : 0.0f; y = (y < 6.0f) ? y : 6.0f; }
    if (code_out)
        *code_out = oracle_encode(oracle_project_value(y, alpha_out, bo, ko, so, rounding), bo, ko, so);
    return y;
}

/* oracle_epilogue_one over an M x N accumulator; scale/bias per column n;
 * res_images (nullable) is M x N; y (nullable) M x N; codes M x N unpacked. */
void oracle_epilogue_array(const int64_t *acc, int64_t M, int64_t N, const float *scale, const float *bias,
                           const int64_t *res_images, float res_scale, int act, float alpha_out,
                           int bo, int ko, int so, int rounding, float *y, uint32_t *codes)
{
    for (int64_t m = 0; m < M; m++)
        for (int64_t n = 0; n < N; n++) {
            int64_t i = m * N + n;
            uint32_t c = 0;
            float v = oracle_epilogue_one(acc[i], scale[n], bias[n], res_images != 0,
                                          res_images ? res_images[i] : 0, res_scale, act, alpha_out,
                                          bo, ko, so, rounding, &c);
            if (y) y[i] = v;
            if (codes) codes[i] = c;
        }
}

/* Sec. IV-B computing logic of a convolution layer, NHWC: X codes are rows
 * of C codes per pixel (ldx words), W codes are rows of C codes per
 * (cout, r, s) (ldw words).  acc[n][p][q][co] = sum_{r,s,c} I(X)*I(W) with
 * zero padding outside the image, for the output rows p in [p0, p1) only:
 * acc holds (p1 - p0) rows per image (the bounded samples of the CPU
 * baseline).  oracle_conv2d_i64 below is the whole output, p in [0, P). */
void oracle_conv2d_rows_i64(const uint32_t *X, int64_t ldx, int bx, int kx,
                            const uint32_t *W, int64_t ldw, int bw, int kw,
                            int Nb, int H, int Wd, int C, int Cout, int R, int S,
                            int stride, int pad, int P, int Q, int p0, int p1, int64_t *acc)
{
    int cpx = 32 / bx, cpw_ = 32 / bw;
    uint32_t mx = (1u << bx) - 1u, mw = (1u << bw) - 1u;
    int64_t tx[256], tw[256];
    image_table(bx, kx, tx);
    image_table(bw, kw, tw);
    int rows = p1 - p0;
    (void)P;
    for (int n = 0; n < Nb; n++)
        for (int p = p0; p < p1; p++)
            for (int q = 0; q < Q; q++)
                for (int co = 0; co < Cout; co++) {
                    int64_t s = 0;
                    for (int r = 0; r < R; r++)
                        for (int t = 0; t < S; t++) {
                            int h = p * stride - pad + r, w = q * stride - pad + t;
                            if (h < 0 || h >= H || w < 0 || w >= Wd) continue;
                            const uint32_t *xr = X + (((int64_t)n * H + h) * Wd + w) * ldx;
                            const uint32_t *wr = W + (((int64_t)co * R + r) * S + t) * ldw;
                            for (int c = 0; c < C; c++) {
                                uint32_t cx = (xr[c / cpx] >> (bx * (c % cpx))) & mx;
                                uint32_t cw = (wr[c / cpw_] >> (bw * (c % cpw_))) & mw;
                                s += tx[cx] * tw[cw];
                            }
                        }
                    acc[(((int64_t)n * rows + (p - p0)) * Q + q) * Cout + co] = s;
                }
}

void oracle_conv2d_i64(const uint32_t *X, int64_t ldx, int bx, int kx,
                       const uint32_t *W, int64_t ldw, int bw, int kw,
                       int Nb, int H, int Wd, int C, int Cout, int R, int S,
                       int stride, int pad, int P, int Q, int64_t *acc)
{
    oracle_conv2d_rows_i64(X, ldx, bx, kx, W, ldw, bw, kw, Nb, H, Wd, C, Cout, R, S,
                           stride, pad, P, Q, 0, P, acc);
}

/* Depthwise convolution (one filter per channel; MobileNetV2's 3x3 layers):
 * W codes are rows of C codes per tap (r, s), ldw words. */
void oracle_dwconv_i64(const uint32_t *X, int64_t ldx, int bx, int kx,
                       const uint32_t *W, int64_t ldw, int bw, int kw,
                       int Nb, int H, int Wd, int C, int R, int S,
                       int stride, int pad, int P, int Q, int64_t *acc)
{
    int cpx = 32 / bx, cpw_ = 32 / bw;
    uint32_t mx = (1u << bx) - 1u, mw = (1u << bw) - 1u;
    int64_t tx[256], tw[256];
    image_table(bx, kx, tx);
    image_table(bw, kw, tw);
    for (int n = 0; n < Nb; n++)
        for (int p = 0; p < P; p++)
            for (int q = 0; q < Q; q++)
                for (int c = 0; c < C; c++) {
                    int64_t s = 0;
                    for (int r = 0; r < R; r++)
                        for (int t = 0; t < S; t++) {
                            int h = p * stride - pad + r, w = q * stride - pad + t;
                            if (h < 0 || h >= H || w < 0 || w >= Wd) continue;
                            const uint32_t *xr = X + (((int64_t)n * H + h) * Wd + w) * ldx;
                            const uint32_t *wr = W + ((int64_t)r * S + t) * ldw;
                            uint32_t cx = (xr[c / cpx] >> (bx * (c % cpx))) & mx;
                            uint32_t cw = (wr[c / cpw_] >> (bw * (c % cpw_))) & mw;
                            s += tx[cx] * tw[cw];
                        }
                    acc[(((int64_t)n * P + p) * Q + q) * C + c] = s;
                }
}

/* Sec. IV-B max pooling with the intersection window: window p x p (here
 * win), stride s, windows that run past the border are cut to the part
 * inside the image ("the intersection window").  Works on codes through
 * their values (the projection is monotone, so pooling codes equals
 * pooling the quantized values).  Output P = ceil((H + 2 pad - win)/s) + 1
 * rows is supplied by the caller. */
void oracle_maxpool_codes(const uint32_t *X, int64_t ldx, int b, int k,
                          int Nb, int H, int Wd, int C, int win, int stride, int pad,
                          int P, int Q, int64_t ldy, uint32_t *Y)
{
    int cpw = 32 / b;
    uint32_t mask = (1u << b) - 1u;
    uint32_t zero = oracle_zero_code(b, k);
    for (int n = 0; n < Nb; n++)
        for (int p = 0; p < P; p++)
            for (int q = 0; q < Q; q++) {
                uint32_t *yr = Y + (((int64_t)n * P + p) * Q + q) * ldy;
                for (int64_t w = 0; w < ldy; w++) {
                    uint32_t word = 0;
                    for (int j = 0; j < cpw; j++) {
                        int c = (int)(w * cpw + j);
                        uint32_t best_code = zero;
                        if (c < C) {
                            double best = -INFINITY;
                            for (int r = 0; r < win; r++)
                                for (int t = 0; t < win; t++) {
                                    int h = p * stride - pad + r, ww = q * stride - pad + t;
                                    if (h < 0 || h >= H || ww < 0 || ww >= Wd) continue;
                                    const uint32_t *xr = X + (((int64_t)n * H + h) * Wd + ww) * ldx;
                                    uint32_t cx = (xr[c / cpw] >> (b * (c % cpw))) & mask;
                                    double v = oracle_decode(cx, b, k);
                                    if (v > best) { best = v; best_code = cx; }
                                }
                            if (best == 0.0) best_code = zero;
                        }
                        word |= best_code << (b * j);
                    }
                    yr[w] = word;
                }
            }
}

/* Global average pooling of codes: sum of integer images over H x W per
 * (n, c) in int64. */
void oracle_avgpool_sum_i64(const uint32_t *X, int64_t ldx, int b, int k,
                            int Nb, int HW, int C, int64_t *sums)
{
    int cpw = 32 / b;
    uint32_t mask = (1u << b) - 1u;
    for (int n = 0; n < Nb; n++)
        for (int c = 0; c < C; c++) {
            int64_t s = 0;
            for (int i = 0; i < HW; i++) {
                const uint32_t *xr = X + ((int64_t)n * HW + i) * ldx;
                s += image_of((xr[c / cpw] >> (b * (c % cpw))) & mask, b, k);
            }
            sums[(int64_t)n * C + c] = s;
        }
}

/* ---------------------------------------------------------------------- */
/* DDA for data densities other than N(0,1) (the paper assumes N(0,1) in    */
/* Sec. III-D "Resolving extremum").  D(alpha) is Eq.                      */
/* objective_function_expansion with another p(t), written out as the      */
/* integral of (t - alpha q)^2 p(t) over the cell of each element q of the */
/* non-negative set; alpha* is its first local minimum from small alpha.   */

/* Composite Simpson rule of (t - q)^2 * p(t) over [lo, hi] with m (even)
 * subintervals; p(t) = (lam / 2) exp(-lam t), the Laplace density with
 * unit variance (lam = sqrt 2). */
static double laplace_cell(double lo, double hi, double q, int m)
{
    const double lam = sqrt(2.0);
    double h = (hi - lo) / m, s = 0.0;
    for (int i = 0; i <= m; i++) {
        double t = lo + i * h;
        double f = (t - q) * (t - q) * 0.5 * lam * exp(-lam * t);
        s += (i == 0 || i == m) ? f : ((i & 1) ? 4.0 * f : 2.0 * f);
    }
    return s * h / 3.0;
}

/* D(alpha) for Laplace data: the last cell runs to lo + 60 / lam (the tail
 * beyond holds e^-60 of the mass); m subintervals per cell. */
static double laplace_D_m(double alpha, int b, int k, int m)
{
    double s[ORACLE_MAX_SET];
    int n = oracle_set_nonneg(b, k, s);
    double D = 0.0;
    for (int j = 0; j < n; j++) {
        double lo = (j == 0) ? 0.0 : alpha * 0.5 * (s[j - 1] + s[j]);
        double hi = (j == n - 1) ? lo + 60.0 / sqrt(2.0) : alpha * 0.5 * (s[j] + s[j + 1]);
        D += laplace_cell(lo, hi, alpha * s[j], m);
    }
    return D;
}

double oracle_D_laplace(double alpha, int b, int k) { return laplace_D_m(alpha, b, k, 4000); }

/* First local minimum of f on a geometric grid of G points over [1e-4, 4]
 * (coarse evaluation fc), refined by golden-section search on f between
 * the grid neighbours of that point. */
static double first_minimum_golden(double (*fc)(double, const void *), double (*f)(double, const void *),
                                   const void *ctx, double *f_out)
{
    const int G = 4000;
    const double lo = 1e-4, hi = 4.0;
    double prev2 = fc(lo, ctx), a1 = lo * pow(hi / lo, 1.0 / (G - 1)), prev = fc(a1, ctx);
    double x0 = lo, x1 = hi;
    for (int i = 2; i < G; i++) {
        double ai = lo * pow(hi / lo, (double)i / (double)(G - 1));
        double cur = fc(ai, ctx);
        if (prev < prev2 && prev <= cur) {
            x0 = lo * pow(hi / lo, (double)(i - 2) / (double)(G - 1));
            x1 = ai;
            break;
        }
        prev2 = prev;
        prev = cur;
    }
    const double g = 0.5 * (sqrt(5.0) - 1.0);
    double c = x1 - g * (x1 - x0), d = x0 + g * (x1 - x0);
    double fc_ = f(c, ctx), fd = f(d, ctx);
    for (int it = 0; it < 300 && x1 - x0 > 1e-14 * x1; it++) {
        if (fc_ < fd) { x1 = d; d = c; fd = fc_; c = x1 - g * (x1 - x0); fc_ = f(c, ctx); }
        else { x0 = c; c = d; fc_ = fd; d = x0 + g * (x1 - x0); fd = f(d, ctx); }
    }
    double as = 0.5 * (x0 + x1);
    if (f_out) *f_out = f(as, ctx);
    return as;
}

typedef struct { int b, k; } bk_ctx;

static double laplace_coarse(double a, const void *c)
{
    const bk_ctx *p = (const bk_ctx *)c;
    return laplace_D_m(a, p->b, p->k, 200);
}

static double laplace_fine(double a, const void *c)
{
    const bk_ctx *p = (const bk_ctx *)c;
    return oracle_D_laplace(a, p->b, p->k);
}

/* alpha* for Laplace data with unit variance; D(alpha*) via D_out. */
double oracle_alpha_star_laplace(int b, int k, double *D_out)
{
    bk_ctx c = {b, k};
    return first_minimum_golden(laplace_coarse, laplace_fine, &c, D_out);
}

/* Histogram of the normalised magnitudes of x (the empirical density of
 * the data): t = (x - mean) / spread for signed formats, x / spread for
 * unsigned ones; bin = floor(u) with u = |x - mean| * (nbins / (t_max *
 * spread)), each step an fp32 operation rounded to nearest; u >= nbins goes
 * to the last bin; NaN values are skipped. */
void oracle_histogram_abs(const float *x, int64_t n, int is_signed, double mean, double spread, int nbins,
                          float t_max, uint64_t *counts)
{
    volatile float m = is_signed ? (float)mean : 0.0f;
    volatile float sp = (float)spread;
    volatile float nb = (float)nbins;
    volatile float den = t_max * sp;
    volatile float scale = nb / den;
    for (int i = 0; i < nbins; i++) counts[i] = 0;
    for (int64_t i = 0; i < n; i++) {
        if (isnan(x[i])) continue;
        volatile float d = x[i] - m;
        volatile float u = fabsf(d) * scale;
        int bin;
        if (u < nb) bin = (int)floorf(u);
        else if (u >= nb) bin = nbins - 1;
        else bin = 0;
        counts[bin]++;
    }
}

typedef struct { const uint64_t *counts; int nbins; double t_max; int b, k; } hist_ctx;

/* D(alpha) for the empirical density: bin i of width w = t_max / nbins
 * holds counts[i] / (2 n) of the mass, spread evenly over it (the
 * non-negative half holds 1/2, as for the symmetric densities).  Each bin
 * is cut at the cell boundaries alpha (s_j + s_{j+1}) / 2 inside it; on each
 * piece the integrand (t - alpha q)^2 is a quadratic, which Simpson's rule
 * with one interval integrates exactly.  q of a piece: the projection of
 * its midpoint (Eq. thresholing_func). */
double oracle_D_hist(double alpha, const uint64_t *counts, int nbins, double t_max, int b, int k)
{
    double s[ORACLE_MAX_SET];
    int ns = oracle_set_nonneg(b, k, s);
    double total = 0.0;
    for (int i = 0; i < nbins; i++) total += (double)counts[i];
    double w = t_max / nbins, D = 0.0;
    int j = 0;                                  /* next boundary index (boundary between s[j], s[j+1]) */
    for (int i = 0; i < nbins; i++) {
        double e0 = i * w, e1 = (i + 1) * w;
        double p = (double)counts[i] / (2.0 * total * w);
        while (j < ns - 1 && alpha * 0.5 * (s[j] + s[j + 1]) <= e0) j++;
        double u = e0;
        for (;;) {
            int jj = j;
            double v = e1;
            while (jj < ns - 1 && alpha * 0.5 * (s[jj] + s[jj + 1]) < e1) {
                double bd = alpha * 0.5 * (s[jj] + s[jj + 1]);
                if (bd > u) { v = bd; break; }
                jj++;
            }
            if (p > 0.0) {
                double tm = 0.5 * (u + v);
                double q = alpha * lookup_projection(tm / alpha, s, ns, 0);
                double fu = (u - q) * (u - q), fm = (tm - q) * (tm - q), fv = (v - q) * (v - q);
                D += p * (v - u) / 6.0 * (fu + 4.0 * fm + fv);
            }
            if (v >= e1) break;
            u = v;
        }
    }
    return D;
}

static double hist_f(double a, const void *c)
{
    const hist_ctx *h = (const hist_ctx *)c;
    return oracle_D_hist(a, h->counts, h->nbins, h->t_max, h->b, h->k);
}

/* alpha* of the empirical density (first local minimum of oracle_D_hist). */
double oracle_alpha_star_hist(const uint64_t *counts, int nbins, double t_max, int b, int k, double *D_out)
{
    hist_ctx c = {counts, nbins, t_max, b, k};
    return first_minimum_golden(hist_f, hist_f, &c, D_out);
}

/* ---------------------------------------------------------------------- */
/* Quantisation-aware training (Algorithm 1; Sec. III-D "Normalization").  */

/* Forward of one tensor: DN, x_hat = fl32(fl32(x - fl32(mu)) / fl32(sigma +
 * 1e-7)), then the projection of x_hat with scale alpha (alpha* of the
 * format, in fp32): codes (unpacked) and the fake-quantised values
 * fl32(alpha * q). */
void oracle_dn_project(const float *x, int64_t n, double mu, double sigma, float alpha, int b, int k, int is_signed,
                       int rounding, uint32_t *codes, float *xq)
{
    volatile float m = (float)mu;
    volatile float s = (float)(sigma + 1e-7);
    for (int64_t i = 0; i < n; i++) {
        volatile float c = x[i] - m;
        volatile float xh = c / s;
        double q = oracle_project_value(xh, alpha, b, k, is_signed, rounding);
        codes[i] = oracle_encode(q, b, k, is_signed);
        if (xq) xq[i] = alpha * (float)q;
    }
}

/* Backward: the straight-through estimator passes the gradient of the
 * fake-quantised values to x_hat unchanged; DN's derivative, with c = x -
 * mu, s = sigma + 1e-7 and both mu and sigma functions of all of x:
 *   d x_hat_i / d x_j = (delta_ij - 1/d) / s - c_i c_j / (d sigma s^2),
 * so grad_x_j = sum_i g_i d x_hat_i / d x_j (fp64, rounded to fp32 at the
 * end; the second term is 0 when sigma = 0). */
void oracle_dn_backward(const float *g, const float *x, int64_t n, double mu, double sigma, float *gx)
{
    double s = sigma + 1e-7, sg = 0.0, sgc = 0.0, d = (double)n;
    for (int64_t i = 0; i < n; i++) {
        sg += (double)g[i];
        sgc += (double)g[i] * ((double)x[i] - mu);
    }
    for (int64_t j = 0; j < n; j++) {
        double cj = (double)x[j] - mu;
        double t = ((double)g[j] - sg / d) / s;
        if (sigma > 0.0) t -= cj * sgc / (d * sigma * s * s);
        gx[j] = (float)t;
    }
}

/* Exponential moving average of (mu, sigma): r <- (1 - gamma) r + gamma b. */
void oracle_ema(const double *batch, double *running, double gamma)
{
    for (int i = 0; i < 2; i++) {
        volatile double a = (1.0 - gamma) * running[i];
        volatile double c = gamma * batch[i];
        running[i] = a + c;
    }
}
