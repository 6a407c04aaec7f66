// esb_qat.cu -- kernels of the quantisation-aware training step of
// Algorithm 1 (DNN training with ESB):
//   * DN followed by ESB projection (Sec. III-D "Normalization": x_hat =
//     (x - mu) / (sigma + eps), eps = 1e-7; the normalised data meet the
//     DDA scale alpha*(b,k) directly), emitting the codes and the
//     fake-quantised values alpha* q the forward pass multiplies;
//   * the backward pass through it: the straight-through estimator (the
//     gradient w.r.t. the normalised data passes the projection unchanged,
//     Algorithm 1 multiplies no derivative of ESB) and the exact derivative
//     of DN, whose mean and sigma depend on every element:
//       dL/dx_j = (g_j - mean(g)) / s - c_j sum_i(g_i c_i) / (d sigma s^2),
//     c = x - mu, s = sigma + eps;
//   * the exponential moving average of the activation statistics
//     (Sec. III-D: mu <- (1 - gamma) mu + gamma mu_i, likewise sigma).
// The reductions run in fp64 with a fixed order (per-block partials, then
// one block), so results are reproducible.
#include <cstdint>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

namespace {

constexpr int kQatThreads = 256;

// x_hat = fl32(fl32(x - mu) / fl32(sigma + eps)), then its projection with
// scale alpha*; codes packed cpw per word (rows of ldc words, cols codes).
__global__ void __launch_bounds__(kQatThreads)
dn_project_kernel(const float* __restrict__ x, int64_t rows, int64_t cols, const double* __restrict__ stats,
                  float alpha, ProjParams p, uint32_t* __restrict__ codes, int64_t ldc, float* __restrict__ xq)
{
    __shared__ float T[128];
    griddep_wait();                                   // stats may come from the previous launch
    build_thresholds(T, p, alpha, threadIdx.x >> 5, threadIdx.x & 31, 0, kQatThreads / 32);
    __syncthreads();
    const float m = (float)__ldg(stats);
    const float s = (float)(__ldg(stats + 1) + 1e-7);
    const int cpw = 32 / p.b;
    const int64_t total = rows * ldc;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < total; u += stride) {
        const int64_t r = u / ldc, w = u - r * ldc;
        uint32_t word = 0u;
        for (int j = 0; j < cpw; j++) {
            const int64_t c = w * cpw + j;
            uint32_t code = p.zero_code;
            if (c < cols) {
                const float xh = __fdiv_rn(__fsub_rn(x[r * cols + c], m), s);
                code = project_by_table(xh, T, p);
                if (xq) xq[r * cols + c] = __fmul_rn(alpha, code_value(code, p.b, p.k));
            }
            word |= code << (p.b * j);
        }
        codes[u] = word;
    }
}

// Per-block fp64 partials of sum g and sum g (x - mu), in a fixed order.
__global__ void __launch_bounds__(kQatThreads)
dn_grad_partials_kernel(const float* __restrict__ g, const float* __restrict__ x, int64_t n,
                        const double* __restrict__ stats, double2* __restrict__ part)
{
    __shared__ double2 sh[kQatThreads];
    griddep_wait();
    const double mu = __ldg(stats);
    double s1 = 0.0, s2 = 0.0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const double gi = (double)g[i];
        s1 += gi;
        s2 = fma(gi, (double)x[i] - mu, s2);
    }
    sh[threadIdx.x] = make_double2(s1, s2);
    __syncthreads();
    for (int o = kQatThreads / 2; o > 0; o >>= 1) {
        if (threadIdx.x < o) {
            sh[threadIdx.x].x += sh[threadIdx.x + o].x;
            sh[threadIdx.x].y += sh[threadIdx.x + o].y;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) part[blockIdx.x] = sh[0];
}

// One block: the partials in index order -> part[nblocks] = totals.
__global__ void __launch_bounds__(kQatThreads) dn_grad_total_kernel(double2* __restrict__ part, int nblocks)
{
    __shared__ double2 sh[kQatThreads];
    double s1 = 0.0, s2 = 0.0;
    for (int i = threadIdx.x; i < nblocks; i += blockDim.x) { s1 += part[i].x; s2 += part[i].y; }
    sh[threadIdx.x] = make_double2(s1, s2);
    __syncthreads();
    for (int o = kQatThreads / 2; o > 0; o >>= 1) {
        if (threadIdx.x < o) {
            sh[threadIdx.x].x += sh[threadIdx.x + o].x;
            sh[threadIdx.x].y += sh[threadIdx.x + o].y;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) part[nblocks] = sh[0];
}

__global__ void __launch_bounds__(kQatThreads)
dn_grad_kernel(const float* __restrict__ g, const float* __restrict__ x, int64_t n, const double* __restrict__ stats,
               const double2* __restrict__ tot, float* __restrict__ gx)
{
    const double mu = __ldg(stats), sigma = __ldg(stats + 1);
    const double s = sigma + 1e-7;
    const double2 t = tot[0];
    const double d = (double)n;
    const double gm = t.x / d;
    const double k2 = sigma > 0.0 ? t.y / (d * sigma * s * s) : 0.0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const double c = (double)x[i] - mu;
        gx[i] = (float)(((double)g[i] - gm) / s - c * k2);
    }
}

// mu <- (1 - gamma) mu + gamma mu_i; sigma likewise (products and sums
// rounded separately, no fused multiply-add).
__global__ void ema_kernel(const double* __restrict__ batch, double* __restrict__ running, double gamma)
{
    if (threadIdx.x < 2) {
        const double a = __dmul_rn(1.0 - gamma, running[threadIdx.x]);
        const double b = __dmul_rn(gamma, batch[threadIdx.x]);
        running[threadIdx.x] = __dadd_rn(a, b);
    }
}

int qat_blocks(int64_t units)
{
    int64_t b = (units + kQatThreads - 1) / kQatThreads;
    const int64_t cap = (int64_t)device_sm_count() * 4;
    if (b > cap) b = cap;
    return (int)(b < 1 ? 1 : b);
}

}  // namespace

size_t dn_grad_workspace_bytes(int64_t n) { return sizeof(double2) * (size_t)(qat_blocks(n) + 1); }

cudaError_t launch_dn_project(const float* x, int64_t rows, int64_t cols, const double* stats, int b, int k,
                              int is_signed, int rounding, float alpha, uint32_t* codes, int64_t ldc, float* xq,
                              cudaStream_t st)
{
    const ProjParams p = make_proj_params(b, k, is_signed, rounding);
    dn_project_kernel<<<qat_blocks(rows * ldc), kQatThreads, 0, st>>>(x, rows, cols, stats, alpha, p, codes, ldc, xq);
    return cudaGetLastError();
}

cudaError_t launch_dn_grad(const float* g, const float* x, int64_t n, const double* stats, void* workspace, float* gx,
                           cudaStream_t st)
{
    const int nb = qat_blocks(n);
    double2* part = static_cast<double2*>(workspace);
    dn_grad_partials_kernel<<<nb, kQatThreads, 0, st>>>(g, x, n, stats, part);
    dn_grad_total_kernel<<<1, kQatThreads, 0, st>>>(part, nb);
    dn_grad_kernel<<<nb, kQatThreads, 0, st>>>(g, x, n, stats, part + nb, gx);
    return cudaGetLastError();
}

cudaError_t launch_ema(const double* batch, double* running, double gamma, cudaStream_t st)
{
    ema_kernel<<<1, 32, 0, st>>>(batch, running, gamma);
    return cudaGetLastError();
}

}  // namespace esb
