// esb_peak.cu -- microbenchmark kernels that measure the tensor-pipe peaks
// the contraction's roofline divides by (the library has no paper
// counterpart for these): back-to-back tcgen05.mma kind::f8f6f4 (E4M3
// operands from shared memory, fp32 accumulators in TMEM, M = 128, N = 256,
// K = 32) and back-to-back legacy mma.sync s8 (m16n8k32, int32 accumulators
// in registers).  One CTA per SM; operands are zeros (the instruction rate
// does not depend on the values).  The host times a launch with CUDA events.
#include <cstdint>
#include <cuda_runtime.h>

#include "esb_common.cuh"
#include "esb_internal.h"

namespace esb {

namespace {

constexpr int kPeakN = 256;
constexpr uint64_t kPeakWaitNs = 2000000000ull;

__global__ void __launch_bounds__(128, 1) peak_tcgen05_kernel(int64_t iters, int* status)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sa = smem;                                // 128 rows x 128 bytes
    uint8_t* sb = smem + 128 * 128;                    // 256 rows x 128 bytes
    __shared__ uint64_t bar;
    __shared__ uint32_t tslot;
    const int tid = threadIdx.x;
    for (int i = tid; i < (128 + kPeakN) * 128 / 16; i += blockDim.x)
        reinterpret_cast<uint4*>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
    if (tid == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
    }
    if (tid < 32) {
        tmem_alloc(&tslot, 256);
        tc_fence_before();
    }
    fence_proxy_async_smem();
    __syncthreads();
    tc_fence_after();
    const uint32_t d = tslot;
    if (tid == 0) {
        const uint32_t idesc = idesc_e4m3_f32(kPeakN);
        const uint64_t ad = smem_desc_sw128(smem_u32(sa)), bd = smem_desc_sw128(smem_u32(sb));
        for (int64_t it = 0; it < iters; it++) {
#pragma unroll
            for (int j = 0; j < 4; j++) mma_f8f6f4(d, ad + 2 * j, bd + 2 * j, idesc, (it > 0 || j > 0) ? 1u : 0u);
        }
        mma_commit(&bar);
        if (!mbar_wait_bounded(&bar, 0u, kPeakWaitNs)) record_status(status, ESB_ERR_TIMEOUT);
    }
    __syncthreads();
    if (tid < 32) {
        tc_fence_after();
        tmem_dealloc(d, 256);
    }
}

// Eight independent m16n8k32 s8 accumulations per warp in flight.
__global__ void __launch_bounds__(256) peak_mma_s8_kernel(int64_t iters, int* sink)
{
    int acc[8][4];
#pragma unroll
    for (int i = 0; i < 8; i++)
#pragma unroll
        for (int j = 0; j < 4; j++) acc[i][j] = 0;
    const uint32_t a0 = threadIdx.x & 1u, a1 = 0u, a2 = 0u, a3 = 0u, b0 = 0u, b1 = 0u;
    for (int64_t it = 0; it < iters; it++) {
#pragma unroll
        for (int i = 0; i < 8; i++) {
            asm volatile(
                "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                "{%0,%1,%2,%3};"
                : "+r"(acc[i][0]), "+r"(acc[i][1]), "+r"(acc[i][2]), "+r"(acc[i][3])
                : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
        }
    }
    int s = 0;
#pragma unroll
    for (int i = 0; i < 8; i++) s += acc[i][0] + acc[i][1] + acc[i][2] + acc[i][3];
    if (sink && s == 123456789) *sink = s;            // never true: keeps the loop
}

}  // namespace

cudaError_t launch_peak(int kind, int64_t iters, int64_t* flops, cudaStream_t st)
{
    const int sms = device_sm_count();
    if (kind == 0) {
        const size_t smem = 1024 + (size_t)(128 + kPeakN) * 128;
        static bool configured = false;
        if (!configured) {
            const cudaError_t e = cudaFuncSetAttribute(peak_tcgen05_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                       (int)smem);
            if (e != cudaSuccess) return e;
            configured = true;
        }
        peak_tcgen05_kernel<<<sms, 128, smem, st>>>(iters, device_status_ptr());
        *flops = (int64_t)sms * iters * 4 * 2 * 128 * kPeakN * 32;
    } else {
        const int blocks = sms * 4;
        peak_mma_s8_kernel<<<blocks, 256, 0, st>>>(iters, device_status_ptr());
        *flops = (int64_t)blocks * 8 * iters * 8 * 2 * 16 * 8 * 32;
    }
    return cudaGetLastError();
}

}  // namespace esb
