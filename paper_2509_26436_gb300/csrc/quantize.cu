// QuaRTZ encoder (Section 3, Eq. 1 then Eq. 2) and dequantiser for sm_103a.
//
// The encoder is HBM-bound: per element it reads 2 bytes (fp16) and writes
// half a byte of code, 1/G_s bytes of FLAG and 2/64 bytes of scale.  Each
// thread owns one 16-byte chunk (8 consecutive elements along K) and eight
// consecutive lanes own one 64-element quantization group, so a warp reads
// 512 contiguous bytes, the group reductions are 3 xor-shuffles and the
// code words of a warp form one contiguous 128-byte store.  Several chunks
// per thread are loaded before any is processed to keep enough bytes in
// flight to saturate HBM.
#include <cuda_fp16.h>

#include "quartz_internal.h"

namespace quartz {
namespace {

constexpr int kThreads = 256;
constexpr int kChunksPerThread = 4;
constexpr int kGroupQ = 64;

__device__ __forceinline__ uint4 ldg_stream(const uint4 *p)
{
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void unpack8(const uint4 &raw, float (&x)[8])
{
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&w[i]));
        x[2 * i] = f.x;
        x[2 * i + 1] = f.y;
    }
}

// Encode the 8 elements of one chunk.  All 32 lanes must call this together
// (the group and subgroup reductions are warp shuffles); `valid` only gates
// the stores.
template <int GS, int MODE>
__device__ __forceinline__ void encode_chunk(const uint4 raw, int64_t chunk, bool valid, int lane,
                                             uint32_t *__restrict__ codes,
                                             uint8_t *__restrict__ flags,
                                             __half *__restrict__ scales,
                                             int8_t *__restrict__ zeros,
                                             int32_t *__restrict__ gsum)
{
    float x[8];
    unpack8(raw, x);

    // --- Eq. 1: group statistics over the 8 lanes of the group ------------
    float s32, lo = 0.f;
    if (MODE == QUARTZ_SYMMETRIC) {
        float amax = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) amax = fmaxf(amax, fabsf(x[i]));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 2));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 4));
        s32 = __fdiv_rn(amax, 127.0f);
    } else {
        float hi = 0.f;  // the range always contains 0
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            lo = fminf(lo, x[i]);
            hi = fmaxf(hi, x[i]);
        }
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) {
            lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
            hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
        }
        s32 = __fdiv_rn(__fsub_rn(hi, lo), 255.0f);
    }
    const __half s16 = __float2half_rn(s32);
    const float s = __half2float(s16);
    const float r = (s > 0.f) ? __frcp_rn(s) : 0.f;
    int z = 0;
    if (MODE == QUARTZ_ASYMMETRIC && s > 0.f) z = __float2int_rn(__fmul_rn(-lo, r)) - 128;

    int q[8];
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const float t = fminf(fmaxf(__fmul_rn(x[i], r), -1024.0f), 1024.0f);
        q[i] = min(max(__float2int_rn(t) + z, -127), 127);
        m |= static_cast<uint32_t>(abs(q[i]));
    }

    // --- Eq. 2: OR of the magnitudes over the subgroup, FLAG --------------
    if (GS >= 16) m |= __shfl_xor_sync(0xffffffffu, m, 1);
    if (GS >= 32) m |= __shfl_xor_sync(0xffffffffu, m, 2);
    if (GS >= 64) m |= __shfl_xor_sync(0xffffffffu, m, 4);
    const int flag = max(29 - __clz(static_cast<int>(m)), 0);

    uint32_t word = 0;
    int vsum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int mag = abs(q[i]) >> flag;  // truncation toward zero
        const int c = q[i] < 0 ? -mag : mag;
        word |= (static_cast<uint32_t>(c) & 0xFu) << (4 * i);
        if (MODE == QUARTZ_ASYMMETRIC) vsum += c;
    }
    if (MODE == QUARTZ_ASYMMETRIC) {
        vsum *= (1 << flag);  // sum of decoded values v = c * 2^FLAG
        vsum += __shfl_xor_sync(0xffffffffu, vsum, 1);
        vsum += __shfl_xor_sync(0xffffffffu, vsum, 2);
        vsum += __shfl_xor_sync(0xffffffffu, vsum, 4);
    }
    if (!valid) return;

    codes[chunk] = word;
    constexpr int kChunksPerSub = GS / 8;
    if ((lane & (kChunksPerSub - 1)) == 0) flags[chunk / kChunksPerSub] = static_cast<uint8_t>(flag);
    if ((lane & 7) == 0) {
        const int64_t g = chunk >> 3;
        scales[g] = s16;
        if (MODE == QUARTZ_ASYMMETRIC) {
            zeros[g] = static_cast<int8_t>(z);
            gsum[g] = vsum;
        }
    }
}

template <int GS, int MODE>
__global__ void __launch_bounds__(kThreads) quantize_kernel(const uint4 *__restrict__ x,
                                                            int64_t n_chunks,
                                                            uint32_t *__restrict__ codes,
                                                            uint8_t *__restrict__ flags,
                                                            __half *__restrict__ scales,
                                                            int8_t *__restrict__ zeros,
                                                            int32_t *__restrict__ gsum)
{
    const int lane = threadIdx.x & 31;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * (kThreads * kChunksPerThread) + threadIdx.x;
    uint4 raw[kChunksPerThread];
#pragma unroll
    for (int j = 0; j < kChunksPerThread; ++j) {
        const int64_t c = base + j * kThreads;
        raw[j] = (c < n_chunks) ? ldg_stream(x + c) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int j = 0; j < kChunksPerThread; ++j) {
        const int64_t c = base + j * kThreads;
        encode_chunk<GS, MODE>(raw[j], c, c < n_chunks, lane, codes, flags, scales, zeros, gsum);
    }
}

// x_hat = s * (v - z), v = sgn(c) (|c| << FLAG); one thread per 8 elements.
__global__ void __launch_bounds__(kThreads) dequantize_kernel(
    const uint32_t *__restrict__ codes, const uint8_t *__restrict__ flags,
    const __half *__restrict__ scales, const int8_t *__restrict__ zeros, int group_s,
    int64_t n_chunks, uint4 *__restrict__ out)
{
    const int64_t c = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x;
    if (c >= n_chunks) return;
    const uint32_t word = codes[c];
    const int flag = flags[(c * 8) / group_s];
    const int64_t g = c >> 3;
    const float s = __half2float(scales[g]);
    const int z = zeros ? zeros[g] : 0;
    uint32_t o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int c0 = static_cast<int>(word << (28 - 8 * i)) >> 28;
        const int c1 = static_cast<int>(word << (24 - 8 * i)) >> 28;
        const float y0 = __fmul_rn(s, static_cast<float>(c0 * (1 << flag) - z));
        const float y1 = __fmul_rn(s, static_cast<float>(c1 * (1 << flag) - z));
        const __half2 h = __floats2half2_rn(y0, y1);
        o[i] = *reinterpret_cast<const uint32_t *>(&h);
    }
    out[c] = make_uint4(o[0], o[1], o[2], o[3]);
}

template <int GS, int MODE>
cudaError_t launch_q(const void *x, const quartz_encoded_t *e, cudaStream_t s)
{
    const int64_t n_chunks = e->rows * e->K / 8;
    const int64_t per_block = kThreads * kChunksPerThread;
    const int64_t blocks = (n_chunks + per_block - 1) / per_block;
    quantize_kernel<GS, MODE><<<static_cast<unsigned>(blocks), kThreads, 0, s>>>(
        static_cast<const uint4 *>(x), n_chunks, reinterpret_cast<uint32_t *>(e->codes), e->flags,
        reinterpret_cast<__half *>(e->scales), e->zeros, e->gsum);
    return cudaGetLastError();
}

template <int MODE>
cudaError_t launch_q_mode(const void *x, const quartz_encoded_t *e, cudaStream_t s)
{
    switch (e->p.group_s) {
        case 8: return launch_q<8, MODE>(x, e, s);
        case 16: return launch_q<16, MODE>(x, e, s);
        case 32: return launch_q<32, MODE>(x, e, s);
        default: return launch_q<64, MODE>(x, e, s);
    }
}

}  // namespace

cudaError_t launch_quantize(const void *x, const quartz_encoded_t *out, cudaStream_t s)
{
    static_assert(kGroupQ == 64, "one quantization group is 8 lanes x 8 elements");
    if (out->rows == 0) return cudaSuccess;
    return out->p.mode == QUARTZ_SYMMETRIC ? launch_q_mode<QUARTZ_SYMMETRIC>(x, out, s)
                                           : launch_q_mode<QUARTZ_ASYMMETRIC>(x, out, s);
}

cudaError_t launch_dequantize(const quartz_encoded_t *e, void *y, cudaStream_t s)
{
    const int64_t n_chunks = e->rows * e->K / 8;
    if (n_chunks == 0) return cudaSuccess;
    const int64_t blocks = (n_chunks + kThreads - 1) / kThreads;
    dequantize_kernel<<<static_cast<unsigned>(blocks), kThreads, 0, s>>>(
        reinterpret_cast<const uint32_t *>(e->codes), e->flags,
        reinterpret_cast<const __half *>(e->scales),
        e->p.mode == QUARTZ_ASYMMETRIC ? e->zeros : nullptr, e->p.group_s, n_chunks,
        static_cast<uint4 *>(y));
    return cudaGetLastError();
}

}  // namespace quartz
