// esb_api.cu -- the extern "C" entry points of libesb.so: host-side argument
// validation, path selection and launches.  Declarations and contracts are
// in include/esb.h.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <vector>

#include <cuda.h>
#include <cuda_runtime.h>

#include "esb.h"
#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

__device__ int g_esb_device_status = 0;

// Id of the current context (unique for the life of the process).  The two
// driver calls are fetched through the runtime, so the library needs no
// link-time dependency on the driver library.
static bool current_context_id(unsigned long long* id)
{
    using GetCurrent = CUresult (*)(CUcontext*);
    using GetId = CUresult (*)(CUcontext, unsigned long long*);
    static GetCurrent get_current = nullptr;
    static GetId get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrent>(f);
        f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<GetId>(f);
    });
    if (!get_current || !get_id) return false;
    CUcontext ctx = nullptr;
    return get_current(&ctx) == CUDA_SUCCESS && ctx && get_id(ctx, id) == CUDA_SUCCESS;
}

cudaError_t symbol_address(cudaError_t (*lookup)(void**), SymbolCache& cache, void** out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= SymbolCache::kDevices) return cudaErrorInvalidDevice;
    // The context's id is unique for the life of the process, so a context
    // created after a cudaDeviceReset (which reloads the module, moving its
    // arrays) never matches an entry of the one before.
    unsigned long long id = 0;
    const bool have_id = current_context_id(&id);
    std::lock_guard<std::mutex> lk(cache.mu);
    if (!have_id || !cache.ptr[dev] || cache.ctx_id[dev] != id) {
        void* p = nullptr;
        e = lookup(&p);
        if (e != cudaSuccess) return e;
        // the lookup makes the device's primary context current if none was
        if (!have_id && !current_context_id(&id)) {
            *out = p;  // no id to key on: use the address without caching it
            return cudaSuccess;
        }
        cache.ptr[dev] = p;
        cache.ctx_id[dev] = id;
    }
    *out = cache.ptr[dev];
    return cudaSuccess;
}

static cudaError_t lookup_device_status(void** p) { return cudaGetSymbolAddress(p, g_esb_device_status); }

int* device_status_ptr()
{
    static SymbolCache cache;
    void* p = nullptr;
    if (symbol_address(lookup_device_status, cache, &p) != cudaSuccess) return nullptr;
    return static_cast<int*>(p);
}

int device_sm_count()
{
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 132;
    if (cache[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 132;
        cache[dev] = n;
    }
    return cache[dev];
}

}  // namespace esb

using namespace esb;

namespace {

bool fmt_ok(const esb_format& f)
{
    return f.b >= 2 && f.b <= 8 && f.k >= 0 && f.k <= f.b - 1 && (f.is_signed == 0 || f.is_signed == 1);
}

// The tensor-core operand routes: one scaled E4M3 byte per code needs
// k <= 3 and an exponent field of at most 4 bits, and must avoid the E4M3
// NaN pattern (exponent 15 with mantissa 111, i.e. b-k-1 = 4 and k = 3);
// wider significands (k >= 4, at most 8 significant bits, shifts up to 6
// for b <= 8) take the significand split into two exact E4M3 planes.
// Other formats (exponent fields of 5+ bits) have images far past the
// int32 bound and are not contracted.
bool fmt_tc_ok(const esb_format& f)
{
    const int ew = f.b - f.k - 1;
    return (f.k <= 3 && ew <= 4 && !(ew == 4 && f.k == 3)) || f.k >= 4;
}

int64_t words_for(int64_t cols, int b) { return (cols + (32 / b) - 1) / (32 / b); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

std::mutex g_astar_mu;
double g_astar[9][9];
double g_dda[9][9];
bool g_astar_have[9][9];

double g_astar_lap[9][9];
double g_dda_lap[9][9];
bool g_astar_lap_have[9][9];

esb_status alpha_star_laplace_cached(int b, int k, double* a, double* d)
{
    std::lock_guard<std::mutex> lk(g_astar_mu);
    if (!g_astar_lap_have[b][k]) {
        g_astar_lap[b][k] = alpha_star_solve_laplace(b, k, &g_dda_lap[b][k]);
        g_astar_lap_have[b][k] = true;
    }
    if (a) *a = g_astar_lap[b][k];
    if (d) *d = g_dda_lap[b][k];
    return ESB_OK;
}

esb_status alpha_star_cached(int b, int k, double* a, double* d)
{
    std::lock_guard<std::mutex> lk(g_astar_mu);
    if (!g_astar_have[b][k]) {
        g_astar[b][k] = alpha_star_solve(b, k, &g_dda[b][k]);
        g_astar_have[b][k] = true;
    }
    if (a) *a = g_astar[b][k];
    if (d) *d = g_dda[b][k];
    return ESB_OK;
}

esb_status check_epilogue(const esb_epilogue* ep, int64_t M, int64_t N, bool want_codes)
{
    if (!ep) return want_codes ? ESB_ERR_INVALID_ARG : ESB_OK;
    if (ep->act < ESB_ACT_NONE || ep->act > ESB_ACT_RELU6) return ESB_ERR_INVALID_ARG;
    if (ep->residual) {
        if (!fmt_ok(ep->res_fmt)) return ESB_ERR_UNSUPPORTED;
        if (ep->res_ld < words_for(N, ep->res_fmt.b)) return ESB_ERR_INVALID_ARG;
        if (esb::fmt_max_image(ep->res_fmt.b, ep->res_fmt.k) >= 16777216.0) return ESB_ERR_RANGE;
    }
    if (want_codes) {
        if (!fmt_ok(ep->fmt_out)) return ESB_ERR_UNSUPPORTED;
        if (ep->rounding_out != ESB_ROUND_HALF_AWAY && ep->rounding_out != ESB_ROUND_HALF_EVEN) return ESB_ERR_INVALID_ARG;
        if (!ep->alpha_out_dev && !(std::isfinite(ep->alpha_out) && ep->alpha_out > 0.0f)) return ESB_ERR_INVALID_ARG;
    }
    (void)M;
    return ESB_OK;
}

}  // namespace

extern "C" {

int32_t esb_version(void) { return 100; }

const char* esb_status_string(int32_t s)
{
    switch (s) {
    case ESB_OK: return "ok";
    case ESB_ERR_INVALID_ARG: return "invalid argument";
    case ESB_ERR_UNSUPPORTED: return "unsupported format or configuration";
    case ESB_ERR_RANGE: return "exactness bound exceeded";
    case ESB_ERR_ALIGN: return "misaligned pointer or stride";
    case ESB_ERR_CUDA: return "CUDA error";
    case ESB_ERR_TIMEOUT: return "device pipeline wait timed out";
    case ESB_ERR_INTERNAL: return "kernel launch configuration inconsistent (no work done)";
    default: return "unknown status";
    }
}

esb_status esb_format_check(esb_format f) { return fmt_ok(f) ? ESB_OK : ESB_ERR_UNSUPPORTED; }

int32_t esb_codes_per_word(int32_t b) { return (b >= 2 && b <= 8) ? 32 / b : 0; }

int64_t esb_row_words(int64_t cols, int32_t b)
{
    if (b < 2 || b > 8 || cols < 0) return 0;
    return (words_for(cols, b) + 3) & ~int64_t(3);
}

uint32_t esb_zero_code(esb_format f) { return fmt_ok(f) ? fmt_zero_code(f.b, f.k) : 0xFFFFFFFFu; }

esb_status esb_alpha_star(int32_t b, int32_t k, double* alpha_star, double* dda)
{
    if (b < 2 || b > 8 || k < 0 || k > b - 1) return ESB_ERR_UNSUPPORTED;
    if (!alpha_star) return ESB_ERR_INVALID_ARG;
    return alpha_star_cached(b, k, alpha_star, dda);
}

size_t esb_calibrate_dda_workspace_bytes(int64_t n) { return n > 0 ? calibrate_workspace_bytes(n) : 0; }

esb_status esb_calibrate_dda(const float* x, int64_t n, esb_format f, void* workspace, size_t workspace_bytes,
                             float* alpha_out, double* stats_out, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (!x || n <= 0 || !workspace || !alpha_out) return ESB_ERR_INVALID_ARG;
    if (workspace_bytes < calibrate_workspace_bytes(n)) return ESB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(workspace) & 15u) != 0) return ESB_ERR_ALIGN;
    double as = 0.0;
    alpha_star_cached(f.b, f.k, &as, nullptr);
    cudaError_t e = launch_calibrate(x, n, f.is_signed, as, workspace, alpha_out, stats_out,
                                     static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_calibrate_dda_noalloc(const float* x, int64_t n, esb_format f, float* alpha_out, double* stats_out,
                                     void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (!x || n <= 0 || !alpha_out) return ESB_ERR_INVALID_ARG;
    if (calibrate_workspace_bytes(n) > calibrate_noalloc_capacity()) return ESB_ERR_RANGE;
    double as = 0.0;
    alpha_star_cached(f.b, f.k, &as, nullptr);
    cudaError_t e = launch_calibrate_noalloc(x, n, f.is_signed, as, alpha_out, stats_out,
                                             static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_alpha_star_dist(int32_t b, int32_t k, int32_t dist, double* alpha_star, double* dda)
{
    if (b < 2 || b > 8 || k < 0 || k > b - 1) return ESB_ERR_UNSUPPORTED;
    if (!alpha_star) return ESB_ERR_INVALID_ARG;
    if (dist == ESB_DIST_GAUSSIAN) return alpha_star_cached(b, k, alpha_star, dda);
    if (dist == ESB_DIST_LAPLACE) return alpha_star_laplace_cached(b, k, alpha_star, dda);
    return ESB_ERR_INVALID_ARG;
}

esb_status esb_calibrate_dda_dist(const float* x, int64_t n, esb_format f, int32_t dist, void* workspace,
                                  size_t workspace_bytes, float* alpha_out, double* stats_out, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (dist != ESB_DIST_GAUSSIAN && dist != ESB_DIST_LAPLACE) return ESB_ERR_INVALID_ARG;
    if (!x || n <= 0 || !workspace || !alpha_out) return ESB_ERR_INVALID_ARG;
    if (workspace_bytes < calibrate_workspace_bytes(n)) return ESB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(workspace) & 15u) != 0) return ESB_ERR_ALIGN;
    double as = 0.0;
    esb_alpha_star_dist(f.b, f.k, dist, &as, nullptr);
    const cudaError_t e = launch_calibrate(x, n, f.is_signed, as, workspace, alpha_out, stats_out,
                                           static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_dda_histogram(const float* x, int64_t n, esb_format f, const double* stats, int32_t nbins, float t_max,
                             unsigned long long* counts, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (n < 0 || nbins < 2 || nbins > ESB_DDA_MAX_BINS || !(std::isfinite(t_max) && t_max > 0.0f))
        return ESB_ERR_INVALID_ARG;
    if (!stats || !counts || (n > 0 && !x)) return ESB_ERR_INVALID_ARG;
    const cudaError_t e = launch_dda_histogram(x, n, f.is_signed, stats, nbins, t_max, counts,
                                               static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_alpha_star_hist(const unsigned long long* counts, int32_t nbins, float t_max, int32_t b, int32_t k,
                               double* alpha_star, double* dda)
{
    if (b < 2 || b > 8 || k < 0 || k > b - 1) return ESB_ERR_UNSUPPORTED;
    if (!counts || !alpha_star || nbins < 2 || nbins > ESB_DDA_MAX_BINS || !(std::isfinite(t_max) && t_max > 0.0f))
        return ESB_ERR_INVALID_ARG;
    unsigned long long total = 0;
    for (int i = 0; i < nbins; i++) total += counts[i];
    if (total == 0) return ESB_ERR_INVALID_ARG;
    *alpha_star = alpha_star_solve_hist(counts, nbins, (double)t_max, b, k, dda);
    return ESB_OK;
}

esb_status esb_calibrate_dda_empirical(const float* x, int64_t n, esb_format f, void* workspace,
                                       size_t workspace_bytes, int32_t nbins, float t_max,
                                       unsigned long long* counts, float* alpha_out, double* stats_out,
                                       double* alpha_star_out, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (!x || n <= 0 || !workspace || !alpha_out || !stats_out || !counts) return ESB_ERR_INVALID_ARG;
    if (nbins < 2 || nbins > ESB_DDA_MAX_BINS || !(std::isfinite(t_max) && t_max > 0.0f)) return ESB_ERR_INVALID_ARG;
    if (workspace_bytes < calibrate_workspace_bytes(n)) return ESB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(workspace) & 15u) != 0) return ESB_ERR_ALIGN;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    double as = 0.0;
    alpha_star_cached(f.b, f.k, &as, nullptr);
    // 1. statistics (and the Gaussian alpha, overwritten below)
    cudaError_t e = launch_calibrate(x, n, f.is_signed, as, workspace, alpha_out, stats_out, st);
    if (e != cudaSuccess) return ESB_ERR_CUDA;
    // 2. histogram of the normalised magnitudes
    e = launch_dda_histogram(x, n, f.is_signed, stats_out, nbins, t_max, counts, st);
    if (e != cudaSuccess) return ESB_ERR_CUDA;
    // 3. alpha* of the histogram on the host
    std::vector<unsigned long long> h((size_t)nbins);
    double stats[3] = {0.0, 0.0, 0.0};
    if (cudaMemcpyAsync(h.data(), counts, sizeof(unsigned long long) * (size_t)nbins, cudaMemcpyDeviceToHost, st) !=
            cudaSuccess ||
        cudaMemcpyAsync(stats, stats_out, sizeof(stats), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return ESB_ERR_CUDA;
    const double ash = alpha_star_solve_hist(h.data(), nbins, (double)t_max, f.b, f.k, nullptr);
    if (alpha_star_out) *alpha_star_out = ash;
    const float alpha = static_cast<float>(ash * (stats[1] + 1e-7));
    if (cudaMemcpyAsync(alpha_out, &alpha, sizeof(float), cudaMemcpyHostToDevice, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return ESB_ERR_CUDA;
    return ESB_OK;
}

esb_status esb_dn_project(const float* x, int64_t rows, int64_t cols, const double* stats, esb_format f,
                          int32_t rounding, uint32_t* codes, int64_t ldc, float* xq, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (rows < 0 || cols < 0 || ldc < words_for(cols, f.b)) return ESB_ERR_INVALID_ARG;
    if (rounding != ESB_ROUND_HALF_AWAY && rounding != ESB_ROUND_HALF_EVEN) return ESB_ERR_INVALID_ARG;
    if (rows == 0 || ldc == 0) return ESB_OK;
    if (!stats || !codes || (cols > 0 && !x)) return ESB_ERR_INVALID_ARG;
    double as = 0.0;
    alpha_star_cached(f.b, f.k, &as, nullptr);
    const cudaError_t e = launch_dn_project(x, rows, cols, stats, f.b, f.k, f.is_signed, rounding, (float)as, codes,
                                            ldc, xq, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

size_t esb_dn_backward_workspace_bytes(int64_t n) { return n > 0 ? dn_grad_workspace_bytes(n) : 0; }

esb_status esb_dn_backward(const float* grad, const float* x, int64_t n, const double* stats, void* workspace,
                           size_t workspace_bytes, float* grad_x, void* stream)
{
    if (n < 0) return ESB_ERR_INVALID_ARG;
    if (n == 0) return ESB_OK;
    if (!grad || !x || !stats || !workspace || !grad_x) return ESB_ERR_INVALID_ARG;
    if (workspace_bytes < dn_grad_workspace_bytes(n)) return ESB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(workspace) & 15u) != 0) return ESB_ERR_ALIGN;
    const cudaError_t e = launch_dn_grad(grad, x, n, stats, workspace, grad_x, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_ema_update(const double* batch_stats, double* running_stats, double gamma, void* stream)
{
    if (!batch_stats || !running_stats || !(gamma >= 0.0 && gamma <= 1.0)) return ESB_ERR_INVALID_ARG;
    const cudaError_t e = launch_ema(batch_stats, running_stats, gamma, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_dda_combine(const double* stats, int64_t count, esb_format f, double* stats_out, float* alpha_out)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (!stats || count <= 0) return ESB_ERR_INVALID_ARG;
    double n = 0.0, s1 = 0.0;
    for (int64_t i = 0; i < count; i++) {
        const double m = stats[3 * i], sp = stats[3 * i + 1], ni = stats[3 * i + 2];
        if (!std::isfinite(m) || !std::isfinite(sp) || !std::isfinite(ni) || ni < 0.0 || sp < 0.0)
            return ESB_ERR_INVALID_ARG;
        n += ni;
        s1 += ni * m;
    }
    if (!(n > 0.0)) return ESB_ERR_INVALID_ARG;
    const double mean = s1 / n;
    double m2 = 0.0;
    for (int64_t i = 0; i < count; i++) {
        const double m = stats[3 * i], sp = stats[3 * i + 1], ni = stats[3 * i + 2];
        if (ni == 0.0) continue;
        m2 += f.is_signed ? ni * (sp * sp + (m - mean) * (m - mean)) : ni * sp * sp;
    }
    const double spread = std::sqrt(m2 / n);
    if (stats_out) {
        stats_out[0] = mean;
        stats_out[1] = spread;
        stats_out[2] = n;
    }
    if (alpha_out) {
        double as = 0.0;
        alpha_star_cached(f.b, f.k, &as, nullptr);
        *alpha_out = static_cast<float>(as * (spread + 1e-7));
    }
    return ESB_OK;
}

esb_status esb_dequant_scale(float alpha_a, esb_format fa, float alpha_b, esb_format fb, float* scale_out)
{
    if (!fmt_ok(fa) || !fmt_ok(fb)) return ESB_ERR_UNSUPPORTED;
    if (!scale_out || !(std::isfinite(alpha_a) && alpha_a > 0.0f) || !(std::isfinite(alpha_b) && alpha_b > 0.0f))
        return ESB_ERR_INVALID_ARG;
    const float ab = alpha_a * alpha_b;  // one fp32 rounding, as on the device
    *scale_out = ab * std::ldexp(1.0f, -(fa.k + fb.k));
    return ESB_OK;
}

esb_status esb_fold_bn_dn(float alpha_a, esb_format fa, float alpha_w, esb_format fw, const double* bn_mean,
                          const double* bn_std, const double* bn_gamma, const double* bn_beta, int64_t n,
                          double dn_mean, double dn_std, double* scale_out, double* bias_out)
{
    if (!fmt_ok(fa) || !fmt_ok(fw)) return ESB_ERR_UNSUPPORTED;
    if (n < 0 || !(std::isfinite(alpha_a) && alpha_a > 0.0f) || !(std::isfinite(alpha_w) && alpha_w > 0.0f) ||
        !(std::isfinite(dn_std) && dn_std > 0.0) || !std::isfinite(dn_mean))
        return ESB_ERR_INVALID_ARG;
    if (n == 0) return ESB_OK;
    if (!bn_mean || !bn_std || !bn_gamma || !bn_beta || !scale_out || !bias_out) return ESB_ERR_INVALID_ARG;
    const double s = std::ldexp((double)alpha_a, -fa.k) * std::ldexp((double)alpha_w, -fw.k);
    for (int64_t i = 0; i < n; i++)
        if (!(std::isfinite(bn_std[i]) && bn_std[i] > 0.0)) return ESB_ERR_INVALID_ARG;
    for (int64_t i = 0; i < n; i++) {
        scale_out[i] = s * bn_gamma[i] / (bn_std[i] * dn_std);
        bias_out[i] = (bn_std[i] * bn_beta[i] - bn_mean[i] * bn_gamma[i] - bn_std[i] * dn_mean) / (dn_std * bn_std[i]);
    }
    return ESB_OK;
}

esb_status esb_project(const float* x, int64_t rows, int64_t cols, int64_t ldx, float alpha, const float* alpha_dev,
                       esb_format f, int32_t rounding, uint32_t* codes, int64_t ldc, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (rows < 0 || cols < 0 || ldx < cols || ldc < words_for(cols, f.b)) return ESB_ERR_INVALID_ARG;
    if (rounding != ESB_ROUND_HALF_AWAY && rounding != ESB_ROUND_HALF_EVEN) return ESB_ERR_INVALID_ARG;
    if (!alpha_dev && !(std::isfinite(alpha) && alpha > 0.0f)) return ESB_ERR_INVALID_ARG;
    if (rows == 0 || ldc == 0) return ESB_OK;
    if (!codes || (cols > 0 && !x)) return ESB_ERR_INVALID_ARG;
    cudaError_t e = launch_project(x, rows, cols, ldx, alpha, alpha_dev, f.b, f.k, f.is_signed, rounding, codes, ldc,
                                   static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_project_dda(const float* x, int64_t rows, int64_t cols, esb_format f, int32_t rounding,
                           void* workspace, size_t workspace_bytes, float* alpha_out, double* stats_out,
                           uint32_t* codes, int64_t ldc, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (rows <= 0 || cols <= 0 || ldc < words_for(cols, f.b)) return ESB_ERR_INVALID_ARG;
    if (rounding != ESB_ROUND_HALF_AWAY && rounding != ESB_ROUND_HALF_EVEN) return ESB_ERR_INVALID_ARG;
    if (!x || !workspace || !alpha_out || !codes) return ESB_ERR_INVALID_ARG;
    if (workspace_bytes < calibrate_workspace_bytes(rows * cols)) return ESB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(workspace) & 15u) != 0) return ESB_ERR_ALIGN;
    double as = 0.0;
    alpha_star_cached(f.b, f.k, &as, nullptr);
    cudaError_t e = launch_calibrate_project(x, rows, cols, f.b, f.k, f.is_signed, rounding, as, workspace, alpha_out,
                                             stats_out, codes, ldc, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_dequant(const uint32_t* codes, int64_t rows, int64_t cols, int64_t ldc, float alpha,
                       const float* alpha_dev, esb_format f, float* y, int64_t ldy, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (rows < 0 || cols < 0 || ldc < words_for(cols, f.b) || ldy < cols) return ESB_ERR_INVALID_ARG;
    if (!alpha_dev && !(std::isfinite(alpha) && alpha > 0.0f)) return ESB_ERR_INVALID_ARG;
    if (rows == 0 || cols == 0) return ESB_OK;
    if (!codes || !y) return ESB_ERR_INVALID_ARG;
    cudaError_t e = launch_dequant(codes, rows, cols, ldc, alpha, alpha_dev, f.b, f.k, y, ldy,
                                   static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

// Validation shared by esb_gemm and esb_gemm_tiled: ESB_OK with *run set
// when there is work to launch.  acc_bound: the exactness bound on
// K max|I_A| max|I_B| of the path (2^24 for one fp32 accumulation, 2^31
// for the chunked one of the tiled path, which checks the rest itself).
static esb_status gemm_check(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, esb_format fa,
                             const uint32_t* B, int64_t ldb, esb_format fb, const esb_epilogue* ep,
                             int32_t* acc_out, float* y_out, uint32_t* codes_out, int64_t ldo, bool* run,
                             double acc_bound = 16777216.0)
{
    *run = false;
    if (!fmt_ok(fa) || !fmt_ok(fb)) return ESB_ERR_UNSUPPORTED;
    if (M < 0 || N < 0 || K < 0) return ESB_ERR_INVALID_ARG;
    if (lda < words_for(K, fa.b) || ldb < words_for(K, fb.b)) return ESB_ERR_INVALID_ARG;
    if (!fmt_tc_ok(fa) || !fmt_tc_ok(fb)) return ESB_ERR_UNSUPPORTED;
    const bool want_codes = codes_out != nullptr;
    esb_status s = check_epilogue(ep, M, N, want_codes || y_out != nullptr);
    if (s != ESB_OK) return s;
    if (want_codes && ldo < words_for(N, ep->fmt_out.b)) return ESB_ERR_INVALID_ARG;
    if ((double)K * fmt_max_image(fa.b, fa.k) * fmt_max_image(fb.b, fb.k) >= acc_bound) return ESB_ERR_RANGE;
    if (M > (int64_t)65535 * 128 * 256 || N > (int64_t)65535 * 16) return ESB_ERR_UNSUPPORTED;
    if (M == 0 || N == 0) return ESB_OK;
    if (!A || !B) return ESB_ERR_INVALID_ARG;
    if (!acc_out && !y_out && !codes_out) return ESB_OK;
    if (!aligned16(A) || !aligned16(B) || (lda & 3) || (ldb & 3)) return ESB_ERR_ALIGN;
    if (!gemm_pick_ok(N, want_codes ? ep->fmt_out.b : 4)) return ESB_ERR_UNSUPPORTED;
    *run = true;
    return ESB_OK;
}

esb_status esb_gemm(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, esb_format fa,
                    const uint32_t* B, int64_t ldb, esb_format fb, const esb_epilogue* ep, int32_t* acc_out,
                    float* y_out, uint32_t* codes_out, int64_t ldo, void* stream)
{
    bool run = false;
    const esb_status s = gemm_check(M, N, K, A, lda, fa, B, ldb, fb, ep, acc_out, y_out, codes_out, ldo, &run);
    if (s != ESB_OK || !run) return s;
    GemmOutputs o{ep, acc_out, y_out, codes_out, ldo};
    cudaError_t e = launch_gemm(M, N, K, A, lda, fa.b, fa.k, B, ldb, fb.b, fb.k, o, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

size_t esb_gemm_tiled_workspace_bytes(int64_t M, int64_t N, int64_t K)
{
    return (M > 0 && N > 0 && K > 0) ? gemm_tiled_workspace_bytes(M, N, K) : 0;
}

esb_status esb_gemm_tiled(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, esb_format fa,
                          const uint32_t* B, int64_t ldb, esb_format fb, const esb_epilogue* ep, int32_t* acc_out,
                          float* y_out, uint32_t* codes_out, int64_t ldo, void* workspace, size_t workspace_bytes,
                          void* stream)
{
    bool run = false;
    const esb_status s =
        gemm_check(M, N, K, A, lda, fa, B, ldb, fb, ep, acc_out, y_out, codes_out, ldo, &run, 2147483648.0);
    if (s != ESB_OK || !run) return s;
    GemmOutputs o{ep, acc_out, y_out, codes_out, ldo};
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int out_cpw = codes_out ? 32 / ep->fmt_out.b : 8;
    if (!gemm_tiled_ok(M, N, K, fa.b, fa.k, fb.b, fb.k, out_cpw)) {
        // esb_gemm's kernels: one fp32 accumulation
        if ((double)K * fmt_max_image(fa.b, fa.k) * fmt_max_image(fb.b, fb.k) >= 16777216.0) return ESB_ERR_RANGE;
        const cudaError_t e = launch_gemm(M, N, K, A, lda, fa.b, fa.k, B, ldb, fb.b, fb.k, o, st);
        return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
    }
    if (!workspace || workspace_bytes < gemm_tiled_workspace_bytes(M, N, K)) return ESB_ERR_INVALID_ARG;
    if (!aligned16(workspace)) return ESB_ERR_ALIGN;
    const cudaError_t e = launch_gemm_tiled(M, N, K, A, lda, fa.b, fa.k, B, ldb, fb.b, fb.k, o, workspace, st);
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_conv2d_nhwc(const esb_conv_desc* d, const uint32_t* X, int64_t ldx, esb_format fx, const uint32_t* W,
                           int64_t ldw, esb_format fw, const esb_epilogue* ep, int32_t* acc_out, float* y_out,
                           uint32_t* codes_out, int64_t ldo, void* stream)
{
    if (!d) return ESB_ERR_INVALID_ARG;
    if (!fmt_ok(fx) || !fmt_ok(fw)) return ESB_ERR_UNSUPPORTED;
    if (d->n < 0 || d->h <= 0 || d->w <= 0 || d->c <= 0 || d->cout <= 0 || d->r <= 0 || d->s <= 0 ||
        d->stride <= 0 || d->pad < 0)
        return ESB_ERR_INVALID_ARG;
    if (d->h + 2 * d->pad < d->r || d->w + 2 * d->pad < d->s) return ESB_ERR_INVALID_ARG;
    if (d->pad >= d->r || d->pad >= d->s) return ESB_ERR_INVALID_ARG;
    if (ldx < words_for(d->c, fx.b)) return ESB_ERR_INVALID_ARG;
    const int P = (d->h + 2 * d->pad - d->r) / d->stride + 1;
    const int Q = (d->w + 2 * d->pad - d->s) / d->stride + 1;
    const int64_t M = (int64_t)d->n * P * Q;
    const bool want_codes = codes_out != nullptr;
    if (d->groups == d->c && d->c > 1) {
        if (d->cout != d->c) return ESB_ERR_INVALID_ARG;
        if (ldw < words_for(d->c, fw.b)) return ESB_ERR_INVALID_ARG;
        esb_status s = check_epilogue(ep, M, d->c, want_codes || y_out != nullptr);
        if (s != ESB_OK) return s;
        if (want_codes && (ep->fmt_out.b != fx.b || ldo < words_for(d->c, fx.b))) return ESB_ERR_INVALID_ARG;
        if ((double)d->r * d->s * fmt_max_image(fx.b, fx.k) * fmt_max_image(fw.b, fw.k) >= 2147483648.0)
            return ESB_ERR_RANGE;
        if (M == 0 || (!acc_out && !y_out && !codes_out)) return ESB_OK;
        if (!X || !W) return ESB_ERR_INVALID_ARG;
        GemmOutputs o{ep, acc_out, y_out, codes_out, ldo};
        cudaError_t e = launch_dwconv(*d, P, Q, X, ldx, fx.b, fx.k, W, ldw, fw.b, fw.k, o,
                                      static_cast<cudaStream_t>(stream));
        return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
    }
    if (d->groups != 1) return ESB_ERR_UNSUPPORTED;
    if (ldw < words_for(d->c, fw.b)) return ESB_ERR_INVALID_ARG;
    if (!fmt_tc_ok(fx) || !fmt_tc_ok(fw)) return ESB_ERR_UNSUPPORTED;
    esb_status s = check_epilogue(ep, M, d->cout, want_codes || y_out != nullptr);
    if (s != ESB_OK) return s;
    if (want_codes && ldo < words_for(d->cout, ep->fmt_out.b)) return ESB_ERR_INVALID_ARG;
    // the exactness bound counts the r*s*c real terms: padding slots hold the
    // zero code, whose image is 0
    const int64_t K = (int64_t)d->r * d->s * d->c;
    if ((double)K * fmt_max_image(fx.b, fx.k) * fmt_max_image(fw.b, fw.k) >= 16777216.0) return ESB_ERR_RANGE;
    if (M == 0) return ESB_OK;
    if (!X || !W) return ESB_ERR_INVALID_ARG;
    if (!acc_out && !y_out && !codes_out) return ESB_OK;
    if (!aligned16(X) || !aligned16(W) || (ldx & 3) || (ldw & 3)) return ESB_ERR_ALIGN;
    if (M > (int64_t)65535 * 128 * 256) return ESB_ERR_UNSUPPORTED;
    if (!gemm_pick_ok(d->cout, want_codes ? ep->fmt_out.b : 4)) return ESB_ERR_UNSUPPORTED;
    GemmOutputs o{ep, acc_out, y_out, codes_out, ldo};
    cudaError_t e = launch_conv_tc(*d, P, Q, X, ldx, fx.b, fx.k, W, ldw, fw.b, fw.k, o, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

// Bound of the int64 path: the sum of |I_A| |I_B| over K stays below 2^62.
static bool i64_bound_ok(int64_t K, esb_format fa, esb_format fb)
{
    return (double)K * fmt_max_image(fa.b, fa.k) * fmt_max_image(fb.b, fb.k) < 4611686018427387904.0;
}

esb_status esb_gemm_i64(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, esb_format fa,
                        const uint32_t* B, int64_t ldb, esb_format fb, const esb_epilogue* ep, int64_t* acc_out,
                        float* y_out, uint32_t* codes_out, int64_t ldo, void* stream)
{
    if (!fmt_ok(fa) || !fmt_ok(fb)) return ESB_ERR_UNSUPPORTED;
    if (M < 0 || N < 0 || K < 0) return ESB_ERR_INVALID_ARG;
    if (lda < words_for(K, fa.b) || ldb < words_for(K, fb.b)) return ESB_ERR_INVALID_ARG;
    const bool want_codes = codes_out != nullptr;
    esb_status s = check_epilogue(ep, M, N, want_codes || y_out != nullptr);
    if (s != ESB_OK) return s;
    if (want_codes && ldo < words_for(N, ep->fmt_out.b)) return ESB_ERR_INVALID_ARG;
    if (!i64_bound_ok(K, fa, fb)) return ESB_ERR_RANGE;
    if (!shiftadd_grid_ok(M, N, want_codes ? ep->fmt_out.b : 4)) return ESB_ERR_UNSUPPORTED;
    if (M == 0 || N == 0 || (!acc_out && !y_out && !codes_out)) return ESB_OK;
    if (K > 0 && (!A || !B)) return ESB_ERR_INVALID_ARG;
    GemmOutputs o{ep, nullptr, y_out, codes_out, ldo};
    const cudaError_t e = launch_gemm_i64(M, N, K, A, lda, fa.b, fa.k, B, ldb, fb.b, fb.k, acc_out, o,
                                          static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_conv2d_nhwc_i64(const esb_conv_desc* d, const uint32_t* X, int64_t ldx, esb_format fx,
                               const uint32_t* W, int64_t ldw, esb_format fw, const esb_epilogue* ep,
                               int64_t* acc_out, float* y_out, uint32_t* codes_out, int64_t ldo, void* stream)
{
    if (!d) return ESB_ERR_INVALID_ARG;
    if (!fmt_ok(fx) || !fmt_ok(fw)) return ESB_ERR_UNSUPPORTED;
    if (d->n < 0 || d->h <= 0 || d->w <= 0 || d->c <= 0 || d->cout <= 0 || d->r <= 0 || d->s <= 0 ||
        d->stride <= 0 || d->pad < 0 || d->pad >= d->r || d->pad >= d->s)
        return ESB_ERR_INVALID_ARG;
    if (d->h + 2 * d->pad < d->r || d->w + 2 * d->pad < d->s) return ESB_ERR_INVALID_ARG;
    if (d->groups != 1) return ESB_ERR_UNSUPPORTED;
    if (ldx < words_for(d->c, fx.b) || ldw < words_for(d->c, fw.b)) return ESB_ERR_INVALID_ARG;
    const int P = (d->h + 2 * d->pad - d->r) / d->stride + 1;
    const int Q = (d->w + 2 * d->pad - d->s) / d->stride + 1;
    const int64_t M = (int64_t)d->n * P * Q;
    const bool want_codes = codes_out != nullptr;
    esb_status s = check_epilogue(ep, M, d->cout, want_codes || y_out != nullptr);
    if (s != ESB_OK) return s;
    if (want_codes && ldo < words_for(d->cout, ep->fmt_out.b)) return ESB_ERR_INVALID_ARG;
    if (!i64_bound_ok((int64_t)d->r * d->s * d->c, fx, fw)) return ESB_ERR_RANGE;
    if (!shiftadd_grid_ok(M, d->cout, want_codes ? ep->fmt_out.b : 4)) return ESB_ERR_UNSUPPORTED;
    if (M == 0 || (!acc_out && !y_out && !codes_out)) return ESB_OK;
    if (!X || !W) return ESB_ERR_INVALID_ARG;
    GemmOutputs o{ep, nullptr, y_out, codes_out, ldo};
    const cudaError_t e = launch_conv_i64(*d, P, Q, X, ldx, fx.b, fx.k, W, ldw, fw.b, fw.k, acc_out, o,
                                          static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_conv2d_kernel(const esb_conv_desc* d, int64_t ldx, esb_format fx, esb_format fw, int32_t out_b,
                             int32_t* kernel)
{
    if (!d || !kernel) return ESB_ERR_INVALID_ARG;
    if (!fmt_ok(fx) || !fmt_ok(fw)) return ESB_ERR_INVALID_ARG;
    if (d->n < 0 || d->h <= 0 || d->w <= 0 || d->c <= 0 || d->cout <= 0 || d->r <= 0 || d->s <= 0 ||
        d->stride <= 0 || d->pad < 0 || d->pad >= d->r || d->pad >= d->s)
        return ESB_ERR_INVALID_ARG;
    if (d->h + 2 * d->pad < d->r || d->w + 2 * d->pad < d->s) return ESB_ERR_INVALID_ARG;
    if (ldx < words_for(d->c, fx.b)) return ESB_ERR_INVALID_ARG;
    if (out_b != 0 && (out_b < 2 || out_b > 8)) return ESB_ERR_INVALID_ARG;
    if (d->groups == d->c && d->c > 1) {
        *kernel = ESB_CONV_KERNEL_DEPTHWISE;
        return ESB_OK;
    }
    if (d->groups != 1 || !fmt_tc_ok(fx) || !fmt_tc_ok(fw) || (ldx & 3)) return ESB_ERR_INVALID_ARG;
    const int P = (d->h + 2 * d->pad - d->r) / d->stride + 1;
    const int Q = (d->w + 2 * d->pad - d->s) / d->stride + 1;
    // the filter stride: ldx for the same code width, else the smallest one
    const int64_t ldw = fw.b == fx.b ? ldx : esb_row_words(d->c, fw.b);
    const int k = conv_kernel_choice(*d, P, Q, ldx, fx.b, fx.k, ldw, fw.b, fw.k, out_b ? out_b : 4);
    if (k < 0) return ESB_ERR_CUDA;
    *kernel = k;
    return ESB_OK;
}

esb_status esb_maxpool_nhwc(const uint32_t* X, int64_t ldx, esb_format f, int32_t n, int32_t h, int32_t w, int32_t c,
                            int32_t win, int32_t stride, int32_t pad, uint32_t* Y, int64_t ldy, void* stream)
{
    if (!fmt_ok(f)) return ESB_ERR_UNSUPPORTED;
    if (n < 0 || h <= 0 || w <= 0 || c <= 0 || win <= 0 || stride <= 0 || pad < 0 || pad >= win) return ESB_ERR_INVALID_ARG;
    if (h + 2 * pad < win || w + 2 * pad < win) return ESB_ERR_INVALID_ARG;
    if (ldx < words_for(c, f.b) || ldy < words_for(c, f.b)) return ESB_ERR_INVALID_ARG;
    const int P = (h + 2 * pad - win) / stride + 1, Q = (w + 2 * pad - win) / stride + 1;
    if (n == 0) return ESB_OK;
    if (!X || !Y) return ESB_ERR_INVALID_ARG;
    cudaError_t e = launch_maxpool(X, ldx, f.b, f.k, n, h, w, c, win, stride, pad, P, Q, Y, ldy,
                                   static_cast<cudaStream_t>(stream), f.is_signed);
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_avgpool_nhwc(const uint32_t* X, int64_t ldx, esb_format f, int32_t n, int32_t hw, int32_t c, float scale,
                            float alpha_out, esb_format fmt_out, int32_t rounding, float* y_out, uint32_t* codes_out,
                            int64_t ldo, void* stream)
{
    if (!fmt_ok(f) || !fmt_ok(fmt_out)) return ESB_ERR_UNSUPPORTED;
    if (n < 0 || hw <= 0 || c <= 0 || ldx < words_for(c, f.b)) return ESB_ERR_INVALID_ARG;
    if (fmt_out.b != f.b) return ESB_ERR_INVALID_ARG;
    if (codes_out && ldo < words_for(c, f.b)) return ESB_ERR_INVALID_ARG;
    if (rounding != ESB_ROUND_HALF_AWAY && rounding != ESB_ROUND_HALF_EVEN) return ESB_ERR_INVALID_ARG;
    if (!std::isfinite(scale) || !(std::isfinite(alpha_out) && alpha_out > 0.0f)) return ESB_ERR_INVALID_ARG;
    if ((double)hw * fmt_max_image(f.b, f.k) >= 2147483648.0) return ESB_ERR_RANGE;
    if (n == 0 || (!y_out && !codes_out)) return ESB_OK;
    if (!X) return ESB_ERR_INVALID_ARG;
    if ((int64_t)n > 65535) return ESB_ERR_UNSUPPORTED;
    cudaError_t e = launch_avgpool(X, ldx, f.b, f.k, n, hw, c, scale, alpha_out, fmt_out.b, fmt_out.k, fmt_out.is_signed,
                                   rounding, y_out, codes_out, ldo, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_peak_launch(int32_t kind, int64_t iters, int64_t* ops, void* stream)
{
    if ((kind != ESB_PEAK_TCGEN05_F8F6F4 && kind != ESB_PEAK_MMA_SYNC_S8) || iters <= 0 || iters > (1ll << 30) || !ops)
        return ESB_ERR_INVALID_ARG;
    const cudaError_t e = launch_peak(kind, iters, ops, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? ESB_OK : ESB_ERR_CUDA;
}

esb_status esb_get_status(void* stream, int32_t* device_status)
{
    if (!device_status) return ESB_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return ESB_ERR_CUDA;
    int v = 0;
    if (cudaMemcpyFromSymbol(&v, esb::g_esb_device_status, sizeof(int)) != cudaSuccess) return ESB_ERR_CUDA;
    const int zero = 0;
    if (cudaMemcpyToSymbol(esb::g_esb_device_status, &zero, sizeof(int)) != cudaSuccess) return ESB_ERR_CUDA;
    *device_status = v;
    return ESB_OK;
}

}  // extern "C"
