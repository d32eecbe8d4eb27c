// Measurement aids: kernels that exercise one execution pipe of the SM at
// full rate, so that the roofline of the linear layer (Section 4.4) can be
// stated against rates measured on the device at hand rather than derived
// from nominal figures.  Neither computes anything the paper defines.
//
//   probe_fp32_kernel    paired fp32 multiply / fused multiply-add
//                        (mul.rn.f32x2, fma.rn.f32x2): the two operations the
//                        GEMM's dequant epilogue issues per output and group
//   probe_mma_f8_kernel  back-to-back tcgen05.mma kind::f8f6f4 (E4M3 x E4M3 ->
//                        fp32) of the GEMM's shape, M128 N256 K32, operands in
//                        shared memory with the GEMM's 64-byte swizzle layout
#include <cuda_runtime.h>

#include "ptx.cuh"
#include "quartz_internal.h"

namespace quartz {
namespace {

constexpr int kProbeThreads = 256;
constexpr int kProbeChains = 8;

__global__ void __launch_bounds__(kProbeThreads) probe_fp32_kernel(int64_t iters, float *sink)
{
    uint64_t x[kProbeChains];
    const float seed = 1.0f + static_cast<float>(threadIdx.x) * 1e-6f;
#pragma unroll
    for (int j = 0; j < kProbeChains; ++j) {
        const float v = seed + static_cast<float>(j) * 1e-3f;
        x[j] = (static_cast<uint64_t>(__float_as_uint(v)) << 32) | __float_as_uint(v);
    }
    const uint64_t m = (static_cast<uint64_t>(__float_as_uint(0.999f)) << 32) | __float_as_uint(0.999f);
    const uint64_t c = (static_cast<uint64_t>(__float_as_uint(1e-3f)) << 32) | __float_as_uint(1e-3f);
    for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
        for (int j = 0; j < kProbeChains; ++j)
            asm volatile("fma.rn.f32x2 %0, %0, %1, %2;" : "+l"(x[j]) : "l"(m), "l"(c));
#pragma unroll
        for (int j = 0; j < kProbeChains; ++j) asm volatile("mul.rn.f32x2 %0, %0, %1;" : "+l"(x[j]) : "l"(m));
    }
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < kProbeChains; ++j)
        s += __uint_as_float(static_cast<uint32_t>(x[j])) + __uint_as_float(static_cast<uint32_t>(x[j] >> 32));
    sink[static_cast<int64_t>(blockIdx.x) * kProbeThreads + threadIdx.x] = s;
}

// One CTA per SM: warp 0 allocates 256 TMEM columns, thread 0 issues
// 2 * iters MMAs into one accumulator from a 24 KB operand stage (128 x 64
// A bytes, 256 x 64 B bytes, the GEMM's layout), commits once and waits for
// completion with the bounded wait.  The operands hold E4M3 bytes of
// magnitude at most 240 (no NaN encodings), so the sums stay finite.
constexpr int kProbeABytes = 128 * 64;
constexpr int kProbeStageBytes = kProbeABytes + 256 * 64;
// The dynamic shared memory request (far above what the kernel uses) keeps one
// CTA per SM, so a grid of one CTA per SM loads every tensor pipe once.
constexpr int kProbeSmem = 200 * 1024;

__global__ void __launch_bounds__(128, 1) probe_mma_f8_kernel(int64_t iters, int *dev_err)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t base = smem_u32(smem);
    const uint32_t bar = base + kProbeStageBytes;
    uint32_t *holder = reinterpret_cast<uint32_t *>(smem + kProbeStageBytes + 8);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + kProbeStageBytes + 12);
    uint32_t *ops = reinterpret_cast<uint32_t *>(smem);
    for (int i = threadIdx.x; i < kProbeStageBytes / 4; i += blockDim.x) {
        uint32_t h = static_cast<uint32_t>(i) * 0x9E3779B1u + blockIdx.x * 0x85EBCA77u;
        h ^= h >> 15;
        ops[i] = h & 0x77777777u;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (threadIdx.x == 0) {
        mbar_init(bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (threadIdx.x < 32) {
        tmem_alloc(smem_u32(holder), 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *holder;
    if (threadIdx.x == 0) {
        const uint32_t idesc = idesc_e4m3_f32(128, 256);
        for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
            for (int kk = 0; kk < 2; ++kk)
                mma_f8_ss(tmem, sdesc_k_major_sw64(base + kk * 32), sdesc_k_major_sw64(base + kProbeABytes + kk * 32),
                          idesc, (i > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(bar);
        mbar_wait_bounded(bar, 0, abort_flag, dev_err, kWaitLimitNs);
    }
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x < 32) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

}  // namespace

cudaError_t launch_probe_fp32(int blocks, int64_t iters, float *sink, cudaStream_t s)
{
    probe_fp32_kernel<<<blocks, kProbeThreads, 0, s>>>(iters, sink);
    return cudaGetLastError();
}

cudaError_t launch_probe_mma_f8(int blocks, int64_t iters, int *dev_err, cudaStream_t s)
{
    cudaError_t e = cudaFuncSetAttribute(probe_mma_f8_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kProbeSmem);
    if (e != cudaSuccess) return e;
    probe_mma_f8_kernel<<<blocks, 128, kProbeSmem, s>>>(iters, dev_err);
    return cudaGetLastError();
}

}  // namespace quartz
