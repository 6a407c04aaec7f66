/*
 * esb.h -- C ABI of libesb.so: Elastic Significant Bit (ESB) quantization
 * and ESB-coded contraction on one Blackwell-Ultra GPU (sm_103a).
 *
 * Method: Gong et al., "Elastic Significant Bit Quantization and
 * Acceleration for Deep Neural Networks" (arXiv 2109.03513).
 *
 * Conventions for every entry point
 * ---------------------------------
 * - Pointers marked [device] are CUDA device pointers owned by the caller;
 *   [host] pointers are ordinary host memory owned by the caller.  The
 *   library never keeps a pointer after a call returns and allocates no
 *   device memory; scratch memory is passed in by the caller (workspace).
 * - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *   stream).  All device work is enqueued asynchronously on that stream;
 *   nothing synchronises unless stated.
 * - Arguments are validated on the host before any launch.  A non-zero
 *   esb_status means nothing was enqueued.  ESB_ERR_CUDA means a launch
 *   failed (cudaGetLastError is left set for the caller to inspect).
 * - Kernels that wait on the tensor-core pipeline bound every wait; when a
 *   wait gives up the kernel records ESB_ERR_TIMEOUT in a device status word
 *   (read with esb_get_status) and returns without hanging.
 *
 * ESB format (Sec. III-B set, Sec. IV-A float format)
 * ---------------------------------------------------
 * fmt = {b, k, is_signed}, 2 <= b <= 8, 0 <= k <= b-1, N = 2^(b-k-1) - 1.
 * A b-bit code is  sign (1 bit) | e (b-k-1 bits) | f (k bits), MSB..LSB.
 * Its value in units of alpha is 0.f (= f * 2^-k) when e == N and
 * 2^e * 1.f otherwise; its integer image is I = value * 2^k.  Zero is
 * always encoded with sign 0 (e = N, f = 0), so the all-zero bit pattern
 * is NOT zero.  Unsigned formats (is_signed = 0) use the non-negative half
 * of the set with the same codes (sign bit always 0).
 *
 * Packed code matrices: floor(32/b) codes per little-endian 32-bit word,
 * code j of a row in bits [b*(j % cpw), b*(j % cpw) + b) of word j / cpw;
 * slots past the last column hold the zero code; unused high bits are 0.
 * Each row starts at a word boundary; `ld*` arguments give the row stride
 * in 32-bit words.
 */
#ifndef ESB_H_
#define ESB_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum esb_status {
    ESB_OK = 0,
    ESB_ERR_INVALID_ARG = 1,  /* null pointer, negative size, bad enum, ld too small, alpha <= 0 ... */
    ESB_ERR_UNSUPPORTED = 2,  /* (b,k) outside the range the entry point implements */
    ESB_ERR_RANGE = 3,        /* an exactness bound (int32 / fp32 accumulation) would be exceeded */
    ESB_ERR_ALIGN = 4,        /* a pointer or stride violates the stated alignment */
    ESB_ERR_CUDA = 5,         /* a CUDA runtime call or launch failed */
    ESB_ERR_TIMEOUT = 6,      /* (device status only) a bounded pipeline wait gave up */
    ESB_ERR_INTERNAL = 7      /* (device status only) a kernel found its shared-memory
                                 allocation smaller than its layout and did no work */
} esb_status;

typedef struct esb_format {
    int32_t b;          /* total bits, 2..8 */
    int32_t k;          /* fraction bits (k+1 significant bits), 0..b-1 */
    int32_t is_signed;  /* 1: symmetric set; 0: non-negative half */
} esb_format;

/* Tie rule of the projection.  Sec. III-C gives half-open look-up
 * intervals, so a value on a midpoint goes to the element of larger
 * magnitude (ESB_ROUND_HALF_AWAY, the default).  ESB_ROUND_HALF_EVEN picks
 * the neighbour whose multiple of the local spacing is even. */
enum { ESB_ROUND_HALF_AWAY = 0, ESB_ROUND_HALF_EVEN = 1 };

/* Activation of the fused epilogue (Sec. IV-B "MP&ReLU"; ReLU6 for
 * MobileNetV2-shaped networks). */
enum { ESB_ACT_NONE = 0, ESB_ACT_RELU = 1, ESB_ACT_RELU6 = 2 };

/* Post-processing fused into the contraction (Sec. IV-C: "BN and DN"
 * affine, activation, ESB quantization of the next layer's input).
 * For accumulator acc[m][n] (exact int32) the epilogue computes, in fp32
 * with this exact op order:
 *   s = scale[n] (or scale0)
 *   s = s * (fl32(alpha_a * alpha_b) * 2^-(kA+kB))     if alpha_a_dev and alpha_b_dev
 *   y = fmaf(s, (float)acc, bias[n])
 *   y = fmaf(res_scale, (float)I_res[m][n], y)         if residual != NULL
 *   y = max(y, 0) (RELU) or min(max(y, 0), 6) (RELU6)
 *   code = projection of y with alpha_out, fmt_out, rounding_out
 *          (same as esb_project)
 * The BN/DN fold of Sec. IV-C becomes scale[n]/bias[n] (esb_fold_bn_dn). */
typedef struct esb_epilogue {
    const float* scale;        /* [device] N floats, or NULL -> scale0 for every n */
    const float* alpha_a_dev;  /* [device] 1 float (scale of A / X), or NULL; with alpha_b_dev */
    const float* alpha_b_dev;  /* [device] 1 float (scale of B / W), or NULL: the "Scale" stage */
    const float* bias;         /* [device] N floats, or NULL -> bias0 for every n */
    float scale0;
    float bias0;
    int32_t act;               /* ESB_ACT_* */
    const uint32_t* residual;  /* [device] packed codes, M rows of res_ld words, or NULL */
    int64_t res_ld;            /* row stride of residual in words */
    esb_format res_fmt;        /* format of the residual codes */
    float res_scale;           /* multiplies the residual integer image */
    float alpha_out;           /* requantisation scale (> 0), used if alpha_out_dev == NULL */
    const float* alpha_out_dev;/* [device] 1 float, read by the kernel; overrides alpha_out */
    esb_format fmt_out;        /* format of the output codes */
    int32_t rounding_out;      /* ESB_ROUND_* */
} esb_epilogue;

/* Convolution geometry, NHWC activations, weights [cout][r][s][c]. */
typedef struct esb_conv_desc {
    int32_t n, h, w, c;        /* input batch, height, width, channels */
    int32_t cout;              /* output channels (must equal c when groups == c) */
    int32_t r, s;              /* filter height, width */
    int32_t stride, pad;       /* same stride / zero padding in both dimensions */
    int32_t groups;            /* 1 (dense) or c (depthwise) */
} esb_conv_desc;

/* ---------------------------------------------------------------- info */

/* Library version: major*10000 + minor*100 + patch. */
int32_t esb_version(void);

/* Human-readable name of an esb_status value (static string). */
const char* esb_status_string(int32_t status);

/* ESB_OK if 2 <= b <= 8, 0 <= k <= b-1 and is_signed is 0 or 1. */
esb_status esb_format_check(esb_format f);

/* floor(32 / b) codes per 32-bit word; 0 for b outside 2..8. */
int32_t esb_codes_per_word(int32_t b);

/* Smallest row stride (words) for `cols` codes that keeps rows 16-byte
 * aligned: ceil(cols / cpw) rounded up to a multiple of 4. */
int64_t esb_row_words(int64_t cols, int32_t b);

/* The code of zero (sign 0, e = N, f = 0); 0xFFFFFFFF for a bad format. */
uint32_t esb_zero_code(esb_format f);

/* alpha*(b,k) of Eq. optimal_alpha_seeking: the scale minimising the
 * distribution difference D(alpha,b,k) of Eq. objective_function_expansion
 * for N(0,1) data (Sec. III-D "Resolving extremum"; Table 1 prints it).
 * Where D has several local minima (large N) the first one from small
 * alpha is returned.  `dda` (nullable) receives the squared error over both
 * halves, 2*D(alpha*), the quantity Table 1 prints as DDA.  Host only;
 * cached per (b,k); thread-safe. */
esb_status esb_alpha_star(int32_t b, int32_t k, double* alpha_star, double* dda);

/* ----------------------------------------------------------- calibrate */

/* Bytes of device workspace esb_calibrate_dda needs for n values on the
 * current device (the reduction grid follows its SM count). */
size_t esb_calibrate_dda_workspace_bytes(int64_t n);

/* DDA calibration of Sec. III-D ("Normalization" and "Resolving extremum"):
 * statistics of x, then alpha = fl32(alpha*(b,k) * (spread + 1e-7)), where
 * spread is the standard deviation sigma (signed formats: data normalised
 * to zero mean and unit variance as in Sec. III-D) or the root mean square
 * (unsigned formats: post-ReLU data, the scale of the underlying normal).
 *   x          [device] n floats (16-byte aligned for the vector path; any
 *              alignment accepted)
 *   n          > 0
 *   workspace  [device] >= esb_calibrate_dda_workspace_bytes(n) bytes,
 *              16-byte aligned, zero-filled before its first use (e.g.
 *              cudaMemset once); every call that completes leaves its first
 *              32 bytes zero again (the block records after them are
 *              scratch), so it needs no clearing between calls.  After a
 *              device status of ESB_ERR_TIMEOUT zero it again.
 *   alpha_out  [device] 1 float written by the kernel (no host sync)
 *   stats_out  [device] 3 doubles {mean, sigma or rms, n}, or NULL
 * One kernel launch; the reduction order is fixed, so results are
 * bit-reproducible on a device.
 * Errors: INVALID_ARG, UNSUPPORTED (bad format), ALIGN (workspace), CUDA. */
esb_status esb_calibrate_dda(const float* x, int64_t n, esb_format f,
                             void* workspace, size_t workspace_bytes,
                             float* alpha_out, double* stats_out, void* stream);

/* Statistics and alpha of a tensor that is split into `count` parts, from
 * the parts' statistics (Sec. III-D "Normalization": the mean and standard
 * deviation of the whole tensor, then alpha = fl32(alpha*(b,k) * (spread +
 * 1e-7)) as esb_calibrate_dda computes it).  The parts' statistics combine
 * by the law of total variance, in fp64:
 *   n = sum n_i,  mean = sum n_i mean_i / n,
 *   signed:   n sigma^2 = sum n_i (sigma_i^2 + (mean_i - mean)^2)
 *   unsigned: n rms^2   = sum n_i rms_i^2
 * (the mean first, so the second sum has no cancellation).  This is the
 * one exchange of a data-parallel calibration: every rank gathers all
 * ranks' stats and calls this, so every rank gets the same alpha.  Host
 * only, no device work.
 *   stats      [host] count x 3 doubles {mean, spread, n}, as stats_out of
 *              esb_calibrate_dda writes them; parts with n == 0 are skipped
 *   stats_out  [host] 3 doubles {mean, spread, n} of the whole, or NULL
 *   alpha_out  [host] 1 float, or NULL
 * Errors: INVALID_ARG (NULL stats, count <= 0, a non-finite entry, a
 * negative n or spread, total n == 0), UNSUPPORTED (bad format). */
esb_status esb_dda_combine(const double* stats, int64_t count, esb_format f, double* stats_out, float* alpha_out);

/* Size of the fixed scratch array behind esb_calibrate_dda_noalloc. */
#define ESB_CALIBRATE_NOALLOC_SCRATCH_BYTES 32768

/* esb_calibrate_dda without a workspace argument (the paper has no
 * counterpart; this is a deployment convenience).  Some callers cannot
 * allocate device memory: a plug-in that only receives input and output
 * pointers from its host application and has no allocator to call, a
 * framework whose caching allocator already holds the device's memory (a
 * direct cudaMalloc can then fail, or fragment memory it manages), or a
 * serving loop that must not allocate after start-up.  This entry point
 * computes the same alpha and statistics as esb_calibrate_dda but keeps its
 * scratch (one 32-byte record per reduction block, at most
 * ESB_CALIBRATE_NOALLOC_SCRATCH_BYTES) in a fixed array inside the library;
 * every GPU that loads the library holds that array until the process
 * exits.  It calls no cudaMalloc, cudaFree or other allocating routine.
 *   x          [device] n floats; n > 0
 *   alpha_out  [device] 1 float; stats_out [device] 3 doubles or NULL
 * The first call on a device looks up the array's device address (with
 * that device current) and caches it for that device's context (a new
 * context, e.g. after cudaDeviceReset, looks it up again); make that first
 * call before any stream capture.  All calls share the one array (zero-filled when the
 * library loads; each call leaves its head record zero and overwrites every
 * block record it later reads): calls whose kernels overlap on the GPU (on
 * different streams without ordering) race on it and must be serialised.
 * Errors: INVALID_ARG, UNSUPPORTED, RANGE (scratch need above the array's
 * size; the reduction uses at most 1023 blocks plus one ticket record, so
 * no n exceeds it), CUDA. */
esb_status esb_calibrate_dda_noalloc(const float* x, int64_t n, esb_format f,
                                     float* alpha_out, double* stats_out, void* stream);

/* ------------------------------------------ DDA for other data densities */

/* Sec. III-D derives alpha* for N(0,1) data ("Resolving extremum": the
 * paper assumes p(t) is the standard normal).  These entry points run the
 * same objective, Eq. objective_function_expansion, and the same rule (the
 * first local minimum of D from small alpha on [1e-4, 4], alpha =
 * fl32(alpha* (spread + 1e-7))) for other densities of the normalised data
 * t: a Laplace density with unit variance (heavy tails), or the data's own
 * density, taken from a histogram of |t|. */
enum { ESB_DIST_GAUSSIAN = 0, ESB_DIST_LAPLACE = 1 };

/* Most bins of an empirical DDA histogram (one 32-bit shared-memory counter
 * per bin and block). */
#define ESB_DDA_MAX_BINS 12288

/* alpha*(b,k) and 2 D(alpha*) for density `dist` (ESB_DIST_*); GAUSSIAN is
 * esb_alpha_star.  Host only; cached per (b,k); thread-safe.
 * Errors: UNSUPPORTED (format), INVALID_ARG (dist, NULL alpha_star). */
esb_status esb_alpha_star_dist(int32_t b, int32_t k, int32_t dist, double* alpha_star, double* dda);

/* esb_calibrate_dda with the alpha* of density `dist` (same statistics,
 * same arguments and workspace rules). */
esb_status esb_calibrate_dda_dist(const float* x, int64_t n, esb_format f, int32_t dist,
                                  void* workspace, size_t workspace_bytes,
                                  float* alpha_out, double* stats_out, void* stream);

/* Histogram of the normalised magnitudes |t| of x: t = (x - mean) / sigma
 * for signed formats, x / rms for unsigned ones, with {mean, spread} read
 * from `stats` (as esb_calibrate_dda's stats_out writes them).  Bin i
 * counts the values with floor(u) == i, u = |x - mean| * (nbins / (t_max *
 * spread)) in fp32 (each operation rounded to nearest); values past t_max
 * go to the last bin, NaN is skipped.
 *   x       [device] n floats
 *   stats   [device] 3 doubles
 *   counts  [device] nbins uint64, overwritten (zero-filled by the call)
 *   nbins   2 .. ESB_DDA_MAX_BINS;  t_max > 0 (in units of the spread)
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
esb_status esb_dda_histogram(const float* x, int64_t n, esb_format f, const double* stats,
                             int32_t nbins, float t_max, unsigned long long* counts, void* stream);

/* alpha* of the empirical density: the density of |t| is the histogram's,
 * even within each bin of width t_max / nbins (half the mass on the
 * non-negative half, as for the symmetric densities), and D is Eq.
 * objective_function_expansion with it.  Host only.
 *   counts [host] nbins uint64 (at least one non-zero)
 * Errors: UNSUPPORTED (format), INVALID_ARG. */
esb_status esb_alpha_star_hist(const unsigned long long* counts, int32_t nbins, float t_max,
                               int32_t b, int32_t k, double* alpha_star, double* dda);

/* DDA calibration with the data's own density: the statistics pass of
 * esb_calibrate_dda, esb_dda_histogram of x, then esb_alpha_star_hist on
 * the host and alpha = fl32(alpha* (spread + 1e-7)) written to alpha_out.
 * Synchronises `stream` (the histogram comes back to the host).
 *   workspace as esb_calibrate_dda; counts [device] nbins uint64 (scratch);
 *   stats_out [device] 3 doubles (required); alpha_star_out [host] or NULL.
 * Errors: INVALID_ARG, UNSUPPORTED, ALIGN (workspace), CUDA. */
esb_status esb_calibrate_dda_empirical(const float* x, int64_t n, esb_format f,
                                       void* workspace, size_t workspace_bytes,
                                       int32_t nbins, float t_max, unsigned long long* counts,
                                       float* alpha_out, double* stats_out, double* alpha_star_out,
                                       void* stream);

/* ------------------------------------------------------------- project */

/* Cheap projection operator of Eq. cheap_projection with the
 * shift-and-round projection of Eq. fast_projection: for each element,
 * v = x / alpha (IEEE fp32 division, round to nearest), clip to [-C, C]
 * (C = largest set element), keep k+1 significant bits of |v| (the
 * spacing of values below 1 is 2^-k), round by `rounding`, restore the
 * sign, emit the b-bit code.  NaN -> zero code; +-Inf -> +-C; negative
 * values -> zero code for unsigned formats.
 *   x        [device] rows x cols floats, row stride ldx (>= cols) floats
 *   alpha    > 0 and finite; used when alpha_dev == NULL
 *   alpha_dev[device] 1 float (e.g. written by esb_calibrate_dda), or NULL
 *   codes    [device] rows x ldc words, ldc >= ceil(cols / cpw); every word
 *            of every row is written (slots past cols hold the zero code)
 * Fast path when x, codes are 16-byte aligned and ldx, ldc are multiples
 * of 4; otherwise a slower general path.  The two ranges must not overlap.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
esb_status esb_project(const float* x, int64_t rows, int64_t cols, int64_t ldx,
                       float alpha, const float* alpha_dev, esb_format f, int32_t rounding,
                       uint32_t* codes, int64_t ldc, void* stream);

/* DDA-calibrated projection of one tensor: the statistics and alpha of
 * esb_calibrate_dda (Sec. III-D), then esb_project of the same tensor with
 * that alpha (Eq. cheap_projection), in one launch of one resident wave
 * with a grid barrier between the passes: each warp keeps its share of the
 * tensor on chip (shared memory) between them, so x is read from memory
 * once.  The barrier needs every block resident; its wait is bounded, and
 * should another tenant's work keep SMs occupied for seconds the call
 * reports ESB_ERR_TIMEOUT through esb_get_status; the workspace must then
 * be zero-filled again before the next call.  (ESB_FUSED_COOPERATIVE=1
 * in the environment selects a cooperative launch, which waits for the
 * whole device instead.  ESB_BARRIER_WAIT_NS, read at every call, can only
 * shorten the wait's 2 s limit: a test aid that makes the wait run out.)
 *   x          [device] rows x cols floats, contiguous (row stride cols)
 *   workspace  [device] >= esb_calibrate_dda_workspace_bytes(rows * cols),
 *              16-byte aligned, zero-filled before its first use, as for
 *              esb_calibrate_dda (the two may share one workspace when
 *              their calls are ordered)
 *   alpha_out  [device] 1 float written with the alpha used
 *   stats_out  [device] 3 doubles {mean, sigma or rms, n}, or NULL
 *   codes      [device] rows x ldc words, as esb_project
 * 16-byte-aligned x and codes with cols and ldc multiples of 4 take the
 * fused path; other layouts run the two steps as separate launches.
 * Errors: INVALID_ARG, UNSUPPORTED, ALIGN (workspace), CUDA. */
esb_status esb_project_dda(const float* x, int64_t rows, int64_t cols, esb_format f, int32_t rounding,
                           void* workspace, size_t workspace_bytes, float* alpha_out, double* stats_out,
                           uint32_t* codes, int64_t ldc, void* stream);

/* Dequantisation (test aid and fp32 export): y = fl32(alpha * q), q the
 * value of each code in units of alpha (Sec. IV-A, Eq. q).
 *   codes [device] rows x ldc words; y [device] rows x ldy floats. */
esb_status esb_dequant(const uint32_t* codes, int64_t rows, int64_t cols, int64_t ldc,
                       float alpha, const float* alpha_dev, esb_format f,
                       float* y, int64_t ldy, void* stream);

/* ----------------------------------------- quantisation-aware training */

/* Forward of one tensor in Algorithm 1 (DNN training with ESB): data
 * normalisation (Sec. III-D "Normalization"), x_hat = (x - mu) / (sigma +
 * 1e-7), then ESB projection of x_hat with the DDA scale alpha*(b,k) of
 * N(0,1) data (Eq. optimal_alpha_seeking; the normalised data need no
 * other scale).  In fp32, each operation rounded to nearest:
 * x_hat = fl32(fl32(x - fl32(mu)) / fl32(sigma + 1e-7)), code = projection
 * of x_hat as esb_project with alpha = fl32(alpha*), xq = fl32(alpha * q),
 * q the code's value (the fake-quantised value the forward multiplies).
 *   x      [device] rows x cols floats (row stride cols)
 *   stats  [device] doubles {mu, sigma}: the batch's (stats_out of
 *          esb_calibrate_dda with a signed format) in training, the moving
 *          averages of esb_ema_update at test time
 *   codes  [device] rows x ldc words; xq [device] rows x cols floats or NULL
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
esb_status esb_dn_project(const float* x, int64_t rows, int64_t cols, const double* stats, esb_format f,
                          int32_t rounding, uint32_t* codes, int64_t ldc, float* xq, void* stream);

/* Backward of esb_dn_project (Algorithm 1, backward loop): the gradient
 * with respect to the fake-quantised values passes the projection unchanged
 * (straight-through: Algorithm 1 multiplies no derivative of ESB), then
 * through DN with the batch's mean and sigma, which depend on every
 * element: with c = x - mu, s = sigma + 1e-7 and d = n,
 *   grad_x[j] = (grad[j] - mean(grad)) / s - c[j] sum_i(grad[i] c[i]) / (d sigma s^2)
 * (the second term is 0 when sigma = 0).  Sums in fp64 in a fixed order;
 * grad_x rounded to fp32.
 *   grad, x [device] n floats; stats [device] {mu, sigma} of the forward
 *   workspace [device] >= esb_dn_backward_workspace_bytes(n), 16-byte aligned
 *   grad_x [device] n floats
 * Errors: INVALID_ARG, ALIGN, CUDA. */
size_t esb_dn_backward_workspace_bytes(int64_t n);
esb_status esb_dn_backward(const float* grad, const float* x, int64_t n, const double* stats, void* workspace,
                           size_t workspace_bytes, float* grad_x, void* stream);

/* Exponential moving average of activation statistics (Sec. III-D,
 * "Normalization", training phase):
 *   mu <- (1 - gamma) mu + gamma mu_i,  sigma <- (1 - gamma) sigma + gamma sigma_i,
 * in fp64, each product and sum rounded separately.
 *   batch_stats [device] {mu_i, sigma_i, ...}; running_stats [device] {mu, sigma}
 *   gamma in [0, 1] (the paper's momentum coefficient)
 * Errors: INVALID_ARG, CUDA. */
esb_status esb_ema_update(const double* batch_stats, double* running_stats, double gamma, void* stream);

/* ---------------------------------------------------------------- gemm */

/* ESB-coded GEMM (Sec. III-B products of set elements; Sec. IV-B/IV-C
 * computing logic): acc[m][n] = sum_k I(A[m][k]) * I(B[n][k]) exactly, then
 * the fused epilogue (esb_epilogue) on each element.
 *   A  [device] M rows of lda words (K codes each, K-major), 16-byte aligned rows
 *   B  [device] N rows of ldb words (K codes each, K-major), 16-byte aligned rows
 *   ep [host] epilogue parameters; may be NULL when codes_out == NULL and
 *      y_out == NULL
 *   acc_out   [device] M x N int32 (row stride N), or NULL
 *   y_out     [device] M x N floats (row stride N), or NULL
 *   codes_out [device] M rows of ldo words (N codes in fmt_out), or NULL
 * The contraction runs on the tcgen05 tensor cores (kind::f8f6f4, E4M3
 * operands).  A format with k <= 3 and b-k-1 <= 4 decodes to one exact
 * E4M3 byte per code; a format with k >= 4 (5 to 8 significant bits, e.g.
 * (6,4), (7,5), (8,6)) takes the significand split: each code becomes two
 * exact E4M3 bytes (high and low 4-bit parts of its significand), and the
 * contraction runs over 2 (one operand split) or 4 (both) planes of K.
 * Formats with an exponent field of 5 or more bits ((6,0), (7,0), (7,1),
 * (8,0)..(8,3)) are UNSUPPORTED.  Either way the sum must satisfy
 * K * max|I_A| * max|I_B| < 2^24 (else ESB_ERR_RANGE).
 * Errors: INVALID_ARG, UNSUPPORTED, RANGE, ALIGN, CUDA. */
esb_status esb_gemm(int64_t M, int64_t N, int64_t K,
                    const uint32_t* A, int64_t lda, esb_format fa,
                    const uint32_t* B, int64_t ldb, esb_format fb,
                    const esb_epilogue* ep,
                    int32_t* acc_out, float* y_out, uint32_t* codes_out, int64_t ldo,
                    void* stream);

/* The same contraction and epilogue as esb_gemm for large operands, with
 * caller-provided scratch: each operand is first decoded once into a tiled
 * image of E4M3 bytes in the workspace (tiles of 128 rows of A or 256 rows
 * of B by 128 codes, each one contiguous block in the MMA operand layout),
 * then a persistent tcgen05 kernel streams whole tiles into shared memory
 * by bulk copies.  Arguments, outputs and errors are those of esb_gemm; the
 * exactness bound is wider: with K max|I_A| max|I_B| >= 2^24 the kernel
 * splits K into up to four chunks that each stay below 2^24 (each chunk
 * exact in fp32) and adds them as integers (the int32 accumulator, and
 * float(acc) rounded to nearest for the epilogue), so the call takes
 * K max|I_A| max|I_B| < 2^31 when the chunks fit (four) and the output
 * codes hold a divisor of 16 per word; RANGE otherwise.  Significand-split
 * formats (k >= 4) always run esb_gemm's kernels, with its 2^24 bound.  Plus
 *   workspace  [device] >= esb_gemm_tiled_workspace_bytes(M, N, K) bytes,
 *              16-byte aligned, contents undefined before and after (the
 *              call overwrites it)
 * Shapes the tiled kernel does not take (N < 256, 256 not a multiple of the
 * output's codes per word, or fewer than 2^32 multiply-adds, where the
 * other kernels finish first) run esb_gemm's kernels; the workspace is then
 * unused.  Errors: as esb_gemm, and ALIGN (workspace) or INVALID_ARG
 * (workspace too small). */
size_t esb_gemm_tiled_workspace_bytes(int64_t M, int64_t N, int64_t K);
esb_status esb_gemm_tiled(int64_t M, int64_t N, int64_t K,
                          const uint32_t* A, int64_t lda, esb_format fa,
                          const uint32_t* B, int64_t ldb, esb_format fb,
                          const esb_epilogue* ep,
                          int32_t* acc_out, float* y_out, uint32_t* codes_out, int64_t ldo,
                          void* workspace, size_t workspace_bytes, void* stream);

/* The "Scale" stage of Sec. IV-C on the host: the fp32 factor that turns
 * the integer accumulator of codes in formats fa and fb into the product of
 * their values, fl32(alpha_a * alpha_b) * 2^-(ka+kb) -- the value the
 * epilogue computes on the device from alpha_a_dev and alpha_b_dev.
 * Errors: INVALID_ARG (alpha not finite and > 0, NULL out), UNSUPPORTED. */
esb_status esb_dequant_scale(float alpha_a, esb_format fa, float alpha_b, esb_format fb, float* scale_out);

/* The "BN and DN" fold of Sec. IV-C: batch normalisation (per channel
 * mean, standard deviation, gamma, beta) and the next layer's data
 * normalisation (mean dn_mean, standard deviation dn_std) applied to the
 * dequantised product become one affine map of the integer accumulator,
 *   DN(BN(Scale(acc))) = scale[n] * acc + bias[n],
 *   scale[n] = alpha_a 2^-ka alpha_w 2^-kw gamma_n / (std_n dn_std)
 *   bias[n]  = (std_n beta_n - mean_n gamma_n - std_n dn_mean) / (dn_std std_n),
 * computed in fp64.  The paper also folds the division by the next
 * layer's alpha into it; here that division stays in the requantisation
 * (esb_epilogue.alpha_out), so scale/bias (cast to fp32) are the
 * epilogue's scale and bias arrays.  Host only.
 *   bn_*       [host] n doubles each; bn_std > 0
 *   scale_out, bias_out [host] n doubles each
 * Errors: INVALID_ARG (NULL pointer, n < 0, non-positive or non-finite
 * alpha / std), UNSUPPORTED (bad format). */
esb_status esb_fold_bn_dn(float alpha_a, esb_format fa, float alpha_w, esb_format fw,
                          const double* bn_mean, const double* bn_std, const double* bn_gamma,
                          const double* bn_beta, int64_t n, double dn_mean, double dn_std,
                          double* scale_out, double* bias_out);

/* ---------------------------------------------------------------- conv */

/* ESB-coded convolution, NHWC (Sec. IV-B: a K x K x c_in x c_out
 * convolution over an h x w x c_in feature map), as an implicit GEMM with
 * M = n*P*Q output pixels, N = cout, K = r*s*c, followed by the fused
 * epilogue.  P = (h + 2 pad - r)/stride + 1, Q likewise.
 *   X [device] n*h*w pixel rows of ldx words (c codes each), ldx % 4 == 0
 *   W [device] cout*r*s rows of ldw words (c codes each, in fw, which may
 *     differ from fx in width and k), ldw % 4 == 0
 *   outputs as esb_gemm with M = n*P*Q rows (pixel-major NHWC).
 * The formats follow esb_gemm (one E4M3 byte per code, or the significand
 * split for k >= 4), with K = r*s*c real terms in the 2^24 bound.
 * groups == c selects the depthwise path (one r x s filter per channel, W
 * holds r*s rows of ldw words with c codes each, cout == c), which runs on
 * CUDA cores (no dense contraction): exact int32 sums of r*s products, the
 * same epilogue; there fmt_out.b must equal fx.b and
 * r*s*max|I_X|*max|I_W| < 2^31.
 * Errors: INVALID_ARG, UNSUPPORTED, RANGE, ALIGN, CUDA. */
esb_status esb_conv2d_nhwc(const esb_conv_desc* d,
                           const uint32_t* X, int64_t ldx, esb_format fx,
                           const uint32_t* W, int64_t ldw, esb_format fw,
                           const esb_epilogue* ep,
                           int32_t* acc_out, float* y_out, uint32_t* codes_out, int64_t ldo,
                           void* stream);

/* Kernels behind esb_conv2d_nhwc. */
enum {
    ESB_CONV_KERNEL_HALO = 1,      /* stride 1, 4-bit X: input rows decoded once,
                                      each filter tap a shifted view (tcgen05) */
    ESB_CONV_KERNEL_IM2COL = 2,    /* implicit im2col, filters resident in shared memory */
    ESB_CONV_KERNEL_STREAMED = 3,  /* implicit im2col, filters streamed per K-block */
    ESB_CONV_KERNEL_DEPTHWISE = 4  /* groups == c, CUDA cores */
};

/* Which of the kernels above esb_conv2d_nhwc launches for geometry d, X
 * row stride ldx and formats fx, fw, when its packed output codes have
 * out_b bits (0: no code output).  The filter stride is taken to be ldx
 * when fw.b == fx.b and esb_row_words(c, fw.b) otherwise; the halo kernel
 * needs 4-bit codes of the same layout on both sides.  The choice depends only on these and on
 * the device's shared memory (queried on the current device); results are
 * identical whichever kernel runs.  Setting ESB_CONV_IM2COL=1 in the
 * environment before the first call disables the halo kernel.
 *   kernel [host] receives one ESB_CONV_KERNEL_* value
 * Errors: INVALID_ARG (bad geometry, or the call would be rejected),
 * CUDA (no device). */
esb_status esb_conv2d_kernel(const esb_conv_desc* d, int64_t ldx, esb_format fx, esb_format fw, int32_t out_b,
                             int32_t* kernel);

/* ------------------------------------------------- int64 contraction */

/* The ESB contraction on the CUDA cores with exact int64 accumulators, for
 * formats and sizes outside the tensor-core path (power-of-two-like sets
 * such as (5,0), (6,1), (6,0), whose images reach 2^30, or sums past
 * 2^24).  Eq. esb_multiplication: each product of two set elements is the
 * product of their significands shifted by the sum of their exponents;
 * every multiply-accumulate here is one small integer product, one 64-bit
 * shift and one 64-bit add.
 *   A, lda, fa, B, ldb, fb, ep, y_out, codes_out, ldo: as esb_gemm (any
 *       formats; no alignment requirement)
 *   acc_out [device] M x N int64 (row stride N), or NULL
 * The epilogue takes float(acc) rounded to nearest.  Requires
 * K * max|I_A| * max|I_B| < 2^62 (else ESB_ERR_RANGE).
 * Errors: INVALID_ARG, UNSUPPORTED, RANGE, CUDA. */
esb_status esb_gemm_i64(int64_t M, int64_t N, int64_t K,
                        const uint32_t* A, int64_t lda, esb_format fa,
                        const uint32_t* B, int64_t ldb, esb_format fb,
                        const esb_epilogue* ep,
                        int64_t* acc_out, float* y_out, uint32_t* codes_out, int64_t ldo,
                        void* stream);

/* esb_conv2d_nhwc (groups == 1) on the int64 path of esb_gemm_i64: any
 * formats, input and filter codes of different widths, ldx and ldw any
 * strides that hold c codes; acc_out [device] n*P*Q x cout int64 or NULL.
 * Requires r*s*c * max|I_X| * max|I_W| < 2^62.
 * Errors: INVALID_ARG, UNSUPPORTED, RANGE, CUDA. */
esb_status esb_conv2d_nhwc_i64(const esb_conv_desc* d,
                               const uint32_t* X, int64_t ldx, esb_format fx,
                               const uint32_t* W, int64_t ldw, esb_format fw,
                               const esb_epilogue* ep,
                               int64_t* acc_out, float* y_out, uint32_t* codes_out, int64_t ldo,
                               void* stream);

/* -------------------------------------------------------------- pooling */

/* Max pooling of ESB codes, NHWC (Sec. IV-B "MP" stage with the
 * intersection window: a window that runs past the border is cut to the
 * part inside the image).  The projection is monotone, so the maximum of
 * the codes' values is the value of the projected maximum; each output
 * slot holds the input code of largest value (the zero code for zero).
 *   X [device] n*h*w pixel rows of ldx words (c codes each, format f)
 *   Y [device] n*P*Q rows of ldy words, P = (h + 2 pad - win)/stride + 1
 *     (for 3x3/2 pad 1 this is ceil(h/2), the paper's output size)
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
esb_status esb_maxpool_nhwc(const uint32_t* X, int64_t ldx, esb_format f,
                            int32_t n, int32_t h, int32_t w, int32_t c,
                            int32_t win, int32_t stride, int32_t pad,
                            uint32_t* Y, int64_t ldy, void* stream);

/* Global average pooling of ESB codes (the pooling before ResNet18's and
 * MobileNetV2's classifier): s[i][ch] = sum over the hw pixels of the
 * integer images (exact int32), y = fl32(scale * (float)s) (scale carries
 * alpha * 2^-k / hw), then y is projected with alpha_out / fmt_out as in
 * esb_project.  fmt_out.b must equal f.b.
 *   X [device] n*hw pixel rows of ldx words; y_out [device] n x c floats
 *   or NULL; codes_out [device] n rows of ldo words or NULL.
 * Errors: INVALID_ARG, UNSUPPORTED, RANGE, CUDA. */
esb_status esb_avgpool_nhwc(const uint32_t* X, int64_t ldx, esb_format f,
                            int32_t n, int32_t hw, int32_t c, float scale,
                            float alpha_out, esb_format fmt_out, int32_t rounding,
                            float* y_out, uint32_t* codes_out, int64_t ldo, void* stream);

/* ----------------------------------------------------- peak measurement */

/* Microbenchmarks of the tensor-pipe rates the contraction's roofline is
 * measured against (no paper counterpart): one launch of `iters` rounds of
 * back-to-back MMAs on every SM, operands zero.  Time it with CUDA events on
 * `stream`; *ops receives its operation count (2 per multiply-add).
 *   ESB_PEAK_TCGEN05_F8F6F4: tcgen05.mma kind::f8f6f4, E4M3 x E4M3 -> fp32
 *     TMEM, M = 128, N = 256, K = 32, one issuing thread per SM (4 per round)
 *   ESB_PEAK_MMA_SYNC_S8: mma.sync m16n8k32 s8 x s8 -> s32, 8 per round per
 *     warp, 4 blocks of 8 warps per SM
 * Errors: INVALID_ARG, CUDA. */
enum { ESB_PEAK_TCGEN05_F8F6F4 = 0, ESB_PEAK_MMA_SYNC_S8 = 1 };
esb_status esb_peak_launch(int32_t kind, int64_t iters, int64_t* ops, void* stream);

/* ------------------------------------------------------------- status */

/* Synchronises `stream`, then returns and clears the device status word
 * (ESB_OK or ESB_ERR_TIMEOUT) in *device_status.  Returns ESB_ERR_CUDA if
 * the synchronisation fails. */
esb_status esb_get_status(void* stream, int32_t* device_status);

#ifdef __cplusplus
}
#endif

#endif /* ESB_H_ */
