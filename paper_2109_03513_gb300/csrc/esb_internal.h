// esb_internal.h -- launchers and host helpers shared by the libesb sources
// (not part of the public C ABI).
#pragma once

#include <cstddef>
#include <cstdint>
#include <mutex>
#include <cuda_runtime.h>

#include "esb.h"

namespace esb {

int device_sm_count();

// Device address of a __device__ symbol of this library in the current
// context, cached per device and keyed by the context's id.  `lookup` runs
// cudaGetSymbolAddress in the symbol's own translation unit (in host code
// the symbol's name is only a stand-in for the device array).
struct SymbolCache {
    static constexpr int kDevices = 64;
    std::mutex mu;
    unsigned long long ctx_id[kDevices] = {};
    void* ptr[kDevices] = {};
};
cudaError_t symbol_address(cudaError_t (*lookup)(void**), SymbolCache& cache, void** out);

// Device address of the library status word on the current device.
int* device_status_ptr();

cudaError_t launch_project(const float* x, int64_t rows, int64_t cols, int64_t ldx, float alpha,
                           const float* alpha_dev, int b, int k, int is_signed, int rounding,
                           uint32_t* codes, int64_t ldc, cudaStream_t st);

cudaError_t launch_dequant(const uint32_t* codes, int64_t rows, int64_t cols, int64_t ldc, float alpha,
                           const float* alpha_dev, int b, int k, float* y, int64_t ldy, cudaStream_t st);

size_t calibrate_workspace_bytes(int64_t n);
cudaError_t launch_calibrate(const float* x, int64_t n, int is_signed, double alpha_star, void* workspace,
                             float* alpha_out, double* stats_out, cudaStream_t st);

cudaError_t launch_calibrate_project(const float* x, int64_t rows, int64_t cols, int b, int k, int is_signed,
                                     int rounding, double alpha_star, void* workspace, float* alpha_out,
                                     double* stats_out, uint32_t* codes, int64_t ldc, cudaStream_t st);

size_t calibrate_noalloc_capacity();
cudaError_t launch_calibrate_noalloc(const float* x, int64_t n, int is_signed, double alpha_star, float* alpha_out,
                                     double* stats_out, cudaStream_t st);

struct GemmOutputs {
    const esb_epilogue* ep;
    int32_t* acc_out;
    float* y_out;
    uint32_t* codes_out;
    int64_t ldo;
};

cudaError_t launch_gemm(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, int ba, int ka,
                        const uint32_t* B, int64_t ldb, int bb, int kb, const GemmOutputs& o, cudaStream_t st);

cudaError_t launch_conv_tc(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int bx, int kx,
                           const uint32_t* W, int64_t ldw, int bw, int kw, const GemmOutputs& o, cudaStream_t st);

bool gemm_pick_ok(int64_t N, int out_b);

// Large GEMMs (esb_gemm_tiled.cu): both operands decoded once into tiled
// E4M3 images in the caller's workspace, then a persistent tcgen05 kernel
// over whole-tile bulk copies.
size_t gemm_tiled_workspace_bytes(int64_t M, int64_t N, int64_t K);
bool gemm_tiled_ok(int64_t M, int64_t N, int64_t K, int ba, int ka, int bb, int kb, int out_cpw);
cudaError_t launch_gemm_tiled(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, int ba, int ka,
                              const uint32_t* B, int64_t ldb, int bb, int kb, const GemmOutputs& o, void* workspace,
                              cudaStream_t st);
// Kernel esb_conv2d_nhwc launches for a dense convolution (an
// esb_conv_kernel value), or -1 when the device cannot be queried.
int conv_kernel_choice(const esb_conv_desc& d, int P, int Q, int64_t ldx, int bx, int kx, int64_t ldw, int bw,
                       int kw, int out_b);

cudaError_t launch_dwconv(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int bx, int kx,
                          const uint32_t* W, int64_t ldw, int bw, int kw, const GemmOutputs& o, cudaStream_t st);
cudaError_t launch_maxpool(const uint32_t* X, int64_t ldx, int b, int k, int n, int H, int Wd, int C, int win,
                           int stride, int pad, int P, int Q, uint32_t* Y, int64_t ldy, cudaStream_t st,
                           int is_signed);
cudaError_t launch_avgpool(const uint32_t* X, int64_t ldx, int b, int k, int n, int HW, int C, float scale,
                           float alpha_out, int bo, int ko, int so, int rounding, float* y_out, uint32_t* codes_out,
                           int64_t ldo, cudaStream_t st);

// CUDA-core contraction with int64 accumulators (esb_shiftadd.cu).
bool shiftadd_grid_ok(int64_t M, int64_t N, int out_b);
cudaError_t launch_gemm_i64(int64_t M, int64_t N, int64_t K, const uint32_t* A, int64_t lda, int ba, int ka,
                            const uint32_t* B, int64_t ldb, int bb, int kb, int64_t* acc64, const GemmOutputs& o,
                            cudaStream_t st);
cudaError_t launch_conv_i64(const esb_conv_desc& d, int P, int Q, const uint32_t* X, int64_t ldx, int bx, int kx,
                            const uint32_t* W, int64_t ldw, int bw, int kw, int64_t* acc64, const GemmOutputs& o,
                            cudaStream_t st);

// Quantisation-aware training kernels (esb_qat.cu).
size_t dn_grad_workspace_bytes(int64_t n);
cudaError_t launch_dn_project(const float* x, int64_t rows, int64_t cols, const double* stats, int b, int k,
                              int is_signed, int rounding, float alpha, uint32_t* codes, int64_t ldc, float* xq,
                              cudaStream_t st);
cudaError_t launch_dn_grad(const float* g, const float* x, int64_t n, const double* stats, void* workspace, float* gx,
                           cudaStream_t st);
cudaError_t launch_ema(const double* batch, double* running, double gamma, cudaStream_t st);

// Tensor-pipe peak microbenchmarks (esb_peak.cu): kind 0 tcgen05 f8f6f4,
// kind 1 mma.sync s8; *flops receives the operations of the launch.
cudaError_t launch_peak(int kind, int64_t iters, int64_t* flops, cudaStream_t st);

// alpha*(b,k) and 2*D(alpha*) (Sec. III-D), solved on the host in fp64.
double alpha_star_solve(int b, int k, double* dda);
// The same for Laplace data with unit variance, and for the empirical
// density of a histogram of |t| (nbins bins over [0, t_max), t in spreads).
double alpha_star_solve_laplace(int b, int k, double* dda);
double alpha_star_solve_hist(const unsigned long long* counts, int nbins, double t_max, int b, int k, double* dda);
cudaError_t launch_dda_histogram(const float* x, int64_t n, int is_signed, const double* stats, int nbins,
                                 float t_max, unsigned long long* counts, cudaStream_t st);

}  // namespace esb
