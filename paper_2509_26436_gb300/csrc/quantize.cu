// QuaRTZ encoder (Section 3, Eq. 1 then Eq. 2) and dequantiser for sm_103a.
//
// The encoder is HBM-bound: per element it reads 2 bytes (fp16) and writes
// half a byte of code, 1/G_s bytes of FLAG and 2/64 bytes of scale.
//
// Symmetric mode (the default) keeps the per-element instruction count low
// enough for HBM to be the limit: each thread owns 16 consecutive elements
// (two 16-byte loads; four lanes form one 64-element group, so the group
// maximum takes two xor-shuffles), the scale and FLAG come from the group and
// subgroup maxima (max |q| = min(rne(max|x| * r), 127), since rounding and the
// cap are monotonic), and the codes are formed four elements per 32-bit word:
// rne(|x| r) is produced by the 1.5 * 2^23 rounding addend, which leaves the
// integer in the low byte of the float, the bytes are gathered with byte
// permutes, shifted right by FLAG in one 32-bit shift, and the sign applied
// per byte in 4-bit two's complement.
//
// Asymmetric mode, and the 16-bit-code LLM variant of Section 5, use one
// thread per 8-element chunk (eight lanes per group) with the same arithmetic
// written per element.
#include <cuda_fp16.h>

#include "lzs_e4m3.cuh"
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

// ---------------------------------------------------------------------------
// Symmetric encoder: 16 elements per thread
// ---------------------------------------------------------------------------
constexpr int kUnitsPerThread = 2;
// Adding 1.5 * 2^23 to a float of magnitude below 2^22 rounds it to an
// integer (round-to-nearest-even, the rounding of the addition) and leaves
// that integer in the low mantissa bits: for 0 <= n < 256 the low byte of the
// sum's bit pattern is n.
constexpr float kRoundAddend = 12582912.0f;

// a * b on float pairs, rounded to nearest even (PTX mul.rn.f32x2).
__device__ __forceinline__ float2 mul2_rn(float2 a, float2 b)
{
    float2 d;
    asm("{\n\t.reg .b64 a, b, d;\n\t"
        "mov.b64 a, {%2, %3};\n\t"
        "mov.b64 b, {%4, %5};\n\t"
        "mul.rn.f32x2 d, a, b;\n\t"
        "mov.b64 {%0, %1}, d;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// Per byte: m (0..7) with the sign s (0x00 or 0xFF) applied in 4-bit two's
// complement: m for s = 0, (16 - m) & 15 for s = 0xFF.
__device__ __forceinline__ uint32_t signed_nibbles(uint32_t m, uint32_t s)
{
    return ((m ^ (s & 0x0F0F0F0Fu)) + (s & 0x01010101u)) & 0x0F0F0F0Fu;
}

// Eq. 2 codes of 8 elements given as four fp16 pairs `w` (the raw words) and
// their sign-cleared copies `a`: q = rne(x r) (capped at +-127 when CAP), c =
// sgn(q) (|q| >> flag), packed as 8 nibbles, element k in bits 4k..4k+3.
template <bool CAP>
__device__ __forceinline__ uint32_t lzs_word8(const uint32_t *w, const uint32_t *a, float r, int flag)
{
    uint32_t u[4][2];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&a[i]));
        float2 t = mul2_rn(f, make_float2(r, r));
        if (CAP) {
            t.x = fminf(t.x, 127.0f);
            t.y = fminf(t.y, 127.0f);
        }
        // Two scalar additions: a paired multiply followed by a paired add
        // was observed to be fused into one multiply-add (parity tests
        // failed on exact ties of x r), which rounds the unrounded product.
        const float2 m = make_float2(__fadd_rn(t.x, kRoundAddend), __fadd_rn(t.y, kRoundAddend));
        u[i][0] = __float_as_uint(m.x);
        u[i][1] = __float_as_uint(m.y);
    }
    // byte k of ev / od: |q| of element 2k / 2k + 1
    const uint32_t ev = prmt(prmt(u[0][0], u[1][0], 0x0040u), prmt(u[2][0], u[3][0], 0x0040u), 0x5410u);
    const uint32_t od = prmt(prmt(u[0][1], u[1][1], 0x0040u), prmt(u[2][1], u[3][1], 0x0040u), 0x5410u);
    // byte k of sev / sod: 0xFF when element 2k / 2k + 1 is negative (a
    // selector nibble 8 + b replicates the sign bit of byte b)
    const uint32_t sev = prmt(prmt(w[0], w[1], 0x00D9u), prmt(w[2], w[3], 0x00D9u), 0x5410u);
    const uint32_t sod = prmt(prmt(w[0], w[1], 0x00FBu), prmt(w[2], w[3], 0x00FBu), 0x5410u);
    const uint32_t keep = 0x01010101u * (0xFFu >> flag);
    const uint32_t cev = signed_nibbles((ev >> flag) & keep, sev);
    const uint32_t cod = signed_nibbles((od >> flag) & keep, sod);
    return cev | (cod << 4);
}

__device__ __forceinline__ int lzs_flag_of(float amax_sub, float r)
{
    const int qmax = min(__float2int_rn(__fmul_rn(amax_sub, r)), 127);
    return max(29 - __clz(qmax), 0);
}

// 16-element units per LZS subgroup (G_s >= 16).
template <int GS>
__host__ __device__ constexpr int kUnitsPerSub()
{
    return GS >= 16 ? GS / 16 : 1;
}

// Eq. 1 + Eq. 2 on the 16 elements of one unit (lo, hi: eight fp16 pairs):
// the group scale and, per 8-element half, the FLAG and the eight codes.  All
// 32 lanes must call it together (group and subgroup maxima are shuffles).
struct UnitCodes {
    uint32_t c0, c1;   // codes of elements 0-7 and 8-15 (element k in bits 4k..4k+3)
    int flag0, flag1;  // their FLAGs (equal unless G_s = 8)
    int flag_next;     // G_s >= 16: FLAG of the next subgroup (packed FLAG storage)
    __half s16;        // the group's fp16 scale
};

template <int GS>
__device__ __forceinline__ UnitCodes encode_unit_sym(const uint4 lo, const uint4 hi)
{
    const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
    uint32_t a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i] = w[i] & 0x7FFF7FFFu;
    // --- maxima of |x|: each 8-element half, the unit, the group ----------
    __half2 m0 = __hmax2(__hmax2(*reinterpret_cast<const __half2 *>(&a[0]), *reinterpret_cast<const __half2 *>(&a[1])),
                         __hmax2(*reinterpret_cast<const __half2 *>(&a[2]), *reinterpret_cast<const __half2 *>(&a[3])));
    __half2 m1 = __hmax2(__hmax2(*reinterpret_cast<const __half2 *>(&a[4]), *reinterpret_cast<const __half2 *>(&a[5])),
                         __hmax2(*reinterpret_cast<const __half2 *>(&a[6]), *reinterpret_cast<const __half2 *>(&a[7])));
    const float2 f0 = __half22float2(m0), f1 = __half22float2(m1);
    const float sub0 = fmaxf(f0.x, f0.y), sub1 = fmaxf(f1.x, f1.y);
    const float unit_max = fmaxf(sub0, sub1);
    const float pair_max = fmaxf(unit_max, __shfl_xor_sync(0xffffffffu, unit_max, 1));
    const float amax = fmaxf(pair_max, __shfl_xor_sync(0xffffffffu, pair_max, 2));

    // --- Eq. 1: scale and reciprocal (as the per-element path) ------------
    UnitCodes u;
    u.s16 = __float2half_rn(__fdiv_rn(amax, 127.0f));
    const float s = __half2float(u.s16);
    const float r = (s > 0.f) ? __frcp_rn(s) : 0.f;

    // --- Eq. 2: FLAG of each subgroup from its maximum --------------------
    if (GS == 8) {
        u.flag0 = lzs_flag_of(sub0, r);
        u.flag1 = lzs_flag_of(sub1, r);
    } else {
        const float m = GS == 16 ? unit_max : GS == 32 ? pair_max : amax;
        u.flag0 = u.flag1 = lzs_flag_of(m, r);
    }
    if (__float2int_rn(__fmul_rn(amax, r)) > 127) {  // only when the fp16 scale rounded far down
        u.c0 = lzs_word8<true>(w, a, r, u.flag0);
        u.c1 = lzs_word8<true>(w + 4, a + 4, r, u.flag1);
    } else {
        u.c0 = lzs_word8<false>(w, a, r, u.flag0);
        u.c1 = lzs_word8<false>(w + 4, a + 4, r, u.flag1);
    }
    u.flag_next = 0;
    if (GS >= 16) u.flag_next = __shfl_down_sync(0xffffffffu, u.flag0, kUnitsPerSub<GS>());
    return u;
}

// The same encoding with a scale fixed beforehand (one per row, or a static
// calibrated one): FLAGs from the subgroup maxima (shuffles over 2 or 4
// lanes for G_s = 32, 64; all 32 lanes call it together) and codes capped at
// +-127 when an element of this thread exceeds the scale's range.
template <int GS>
__device__ __forceinline__ UnitCodes encode_unit_sym_scaled(const uint4 lo, const uint4 hi, __half s16, float r)
{
    const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
    uint32_t a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i] = w[i] & 0x7FFF7FFFu;
    __half2 m0 = __hmax2(__hmax2(*reinterpret_cast<const __half2 *>(&a[0]), *reinterpret_cast<const __half2 *>(&a[1])),
                         __hmax2(*reinterpret_cast<const __half2 *>(&a[2]), *reinterpret_cast<const __half2 *>(&a[3])));
    __half2 m1 = __hmax2(__hmax2(*reinterpret_cast<const __half2 *>(&a[4]), *reinterpret_cast<const __half2 *>(&a[5])),
                         __hmax2(*reinterpret_cast<const __half2 *>(&a[6]), *reinterpret_cast<const __half2 *>(&a[7])));
    const float2 f0 = __half22float2(m0), f1 = __half22float2(m1);
    const float sub0 = fmaxf(f0.x, f0.y), sub1 = fmaxf(f1.x, f1.y);
    const float unit_max = fmaxf(sub0, sub1);
    UnitCodes u;
    u.s16 = s16;
    if (GS == 8) {
        u.flag0 = lzs_flag_of(sub0, r);
        u.flag1 = lzs_flag_of(sub1, r);
    } else {
        float m = unit_max;
        if (GS >= 32) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 1));
        if (GS >= 64) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 2));
        u.flag0 = u.flag1 = lzs_flag_of(m, r);
    }
    if (__float2int_rn(fminf(__fmul_rn(unit_max, r), 1024.0f)) > 127) {
        u.c0 = lzs_word8<true>(w, a, r, u.flag0);
        u.c1 = lzs_word8<true>(w + 4, a + 4, r, u.flag1);
    } else {
        u.c0 = lzs_word8<false>(w, a, r, u.flag0);
        u.c1 = lzs_word8<false>(w + 4, a + 4, r, u.flag1);
    }
    u.flag_next = 0;
    if (GS >= 16) u.flag_next = __shfl_down_sync(0xffffffffu, u.flag0, kUnitsPerSub<GS>());
    return u;
}

// The LLM variant of Section 5 on one unit (symmetric): Eq. 1 with 32767
// levels (16-bit codes), then Eq. 2 straight to 4 bits with FLAG =
// max(29 - clz(m), 0) in 0..12, m the OR of the subgroup's |q|.  The OR has
// the bit length of the subgroup's largest |q|, and |q| = rne(min(|x| r,
// 32767)) grows with |x|, so the FLAG comes from the subgroup's largest
// |x| (one conversion per subgroup, as in the 8-bit encoder) and each code
// is bits F .. F+2 of |q|, taken from the 1.5 * 2^23 rounding sum, with the
// sign of x applied in 4-bit two's complement.  q comes from the binary32
// operations of the definition (x r with r = RN(1/s), round half to even,
// the 32767 cap), so codes, FLAGs and scales are exactly Eq. 1 + Eq. 2's
// (compared bit for bit in the GPU tests).  All 32 lanes call it together
// (4 lanes per group).
__device__ __forceinline__ int lzs_flag_wide(float amax_sub, float r)
{
    const int qmax = min(__float2int_rn(__fmul_rn(amax_sub, r)), 32767);
    return max(29 - __clz(qmax), 0);
}

// Codes of 8 elements (four fp16 pairs `w`, sign-cleared copies `a`) for
// 16-bit stage-1 codes: c = sgn(x) (min(rne(|x| r), 32767) >> flag), element
// k in bits 4k..4k+3.  Branch-free cap: the fp16 scale can round down (by up
// to half of it for the smallest subnormal scales), so rne(|x| r) reaches
// up to 49151 for the elements nearest the group maximum.  Such an element
// lies in a subgroup with FLAG 12 (its capped maximum is 32767), where its
// shifted magnitude is 8..11 against the capped value's 7, while every
// shifted magnitude in a subgroup with a lower FLAG is at most 7; so each
// packed magnitude byte b <= 15 becomes (b & 7) | 7 * (bit 3 of b).  (A
// branch on the cap, as the 8-bit encoder has, diverges here: with 32767
// levels the fp16 rounding of the scale takes it in about half the groups.)
__device__ __forceinline__ uint32_t lzs_word8_wide(const uint32_t *w, const uint32_t *a, float r, int flag)
{
    uint32_t u[4][2];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&a[i]));
        const float2 t = mul2_rn(f, make_float2(r, r));
        // scalar additions (see lzs_word8); the low 22 bits of the sum are
        // rne(|x| r), and its value >> flag (at most 11) lands in the low byte
        u[i][0] = __float_as_uint(__fadd_rn(t.x, kRoundAddend)) >> flag;
        u[i][1] = __float_as_uint(__fadd_rn(t.y, kRoundAddend)) >> flag;
    }
    const uint32_t ev = prmt(prmt(u[0][0], u[1][0], 0x0040u), prmt(u[2][0], u[3][0], 0x0040u), 0x5410u);
    const uint32_t od = prmt(prmt(u[0][1], u[1][1], 0x0040u), prmt(u[2][1], u[3][1], 0x0040u), 0x5410u);
    const uint32_t sev = prmt(prmt(w[0], w[1], 0x00D9u), prmt(w[2], w[3], 0x00D9u), 0x5410u);
    const uint32_t sod = prmt(prmt(w[0], w[1], 0x00FBu), prmt(w[2], w[3], 0x00FBu), 0x5410u);
    const uint32_t mev = (ev & 0x07070707u) | (((ev >> 3) & 0x01010101u) * 7u);  // bytes 8..15 -> 7
    const uint32_t mod = (od & 0x07070707u) | (((od >> 3) & 0x01010101u) * 7u);
    const uint32_t cev = signed_nibbles(mev, sev);
    const uint32_t cod = signed_nibbles(mod, sod);
    return cev | (cod << 4);
}

template <int GS>
__device__ __forceinline__ UnitCodes encode_unit_wide(const uint4 lo, const uint4 hi)
{
    const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
    uint32_t a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i] = w[i] & 0x7FFF7FFFu;
    __half2 m0 = __hmax2(__hmax2(*reinterpret_cast<const __half2 *>(&a[0]), *reinterpret_cast<const __half2 *>(&a[1])),
                         __hmax2(*reinterpret_cast<const __half2 *>(&a[2]), *reinterpret_cast<const __half2 *>(&a[3])));
    __half2 m1 = __hmax2(__hmax2(*reinterpret_cast<const __half2 *>(&a[4]), *reinterpret_cast<const __half2 *>(&a[5])),
                         __hmax2(*reinterpret_cast<const __half2 *>(&a[6]), *reinterpret_cast<const __half2 *>(&a[7])));
    const float2 f0 = __half22float2(m0), f1 = __half22float2(m1);
    const float sub0 = fmaxf(f0.x, f0.y), sub1 = fmaxf(f1.x, f1.y);
    const float unit_max = fmaxf(sub0, sub1);
    const float pair_max = fmaxf(unit_max, __shfl_xor_sync(0xffffffffu, unit_max, 1));
    const float amax = fmaxf(pair_max, __shfl_xor_sync(0xffffffffu, pair_max, 2));

    UnitCodes u;
    u.s16 = __float2half_rn(__fdiv_rn(amax, 32767.0f));
    const float s = __half2float(u.s16);
    const float r = (s > 0.f) ? __frcp_rn(s) : 0.f;
    if (GS == 8) {
        u.flag0 = lzs_flag_wide(sub0, r);
        u.flag1 = lzs_flag_wide(sub1, r);
    } else {
        const float m = GS == 16 ? unit_max : GS == 32 ? pair_max : amax;
        u.flag0 = u.flag1 = lzs_flag_wide(m, r);
    }
    u.c0 = lzs_word8_wide(w, a, r, u.flag0);
    u.c1 = lzs_word8_wide(w + 4, a + 4, r, u.flag1);
    u.flag_next = 0;
    if (GS >= 16) u.flag_next = __shfl_down_sync(0xffffffffu, u.flag0, kUnitsPerSub<GS>());
    return u;
}

// Store one unit's FLAGs: one byte per subgroup, or (packed) two per byte,
// subgroup 2j in the low nibble of byte j; a packed byte is written by the
// lane holding its first subgroup.
template <int GS>
__device__ __forceinline__ void store_unit_flags(const UnitCodes &u, int64_t unit, int lane,
                                                 uint8_t *__restrict__ flags, bool packed)
{
    constexpr int ups = kUnitsPerSub<GS>();
    if (GS == 8) {
        if (packed)
            flags[unit] = static_cast<uint8_t>(u.flag0 | (u.flag1 << 4));
        else
            reinterpret_cast<uint16_t *>(flags)[unit] = static_cast<uint16_t>(u.flag0 | (u.flag1 << 8));
    } else if (packed) {
        if ((lane & (2 * ups - 1)) == 0) flags[unit / (2 * ups)] = static_cast<uint8_t>(u.flag0 | (u.flag_next << 4));
    } else if ((lane & (ups - 1)) == 0) {
        flags[unit / ups] = static_cast<uint8_t>(u.flag0);
    }
}

// Store one unit's encoding: codes, FLAGs, and the scale once per group.
template <int GS>
__device__ __forceinline__ void store_unit_sym(const UnitCodes &u, int64_t unit, int lane,
                                               uint2 *__restrict__ codes, uint8_t *__restrict__ flags,
                                               __half *__restrict__ scales, bool packed)
{
    codes[unit] = make_uint2(u.c0, u.c1);
    store_unit_flags<GS>(u, unit, lane, flags, packed);
    if ((lane & 3) == 0) scales[unit >> 2] = u.s16;
}

template <int GS, bool WIDE>
__global__ void __launch_bounds__(kThreads) quantize_sym_kernel(const uint4 *__restrict__ x, int64_t n_units,
                                                                uint2 *__restrict__ codes,
                                                                uint8_t *__restrict__ flags,
                                                                __half *__restrict__ scales, int packed)
{
    griddep_wait();
    const int lane = threadIdx.x & 31;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * (kThreads * kUnitsPerThread) + threadIdx.x;
    uint4 raw[kUnitsPerThread][2];
#pragma unroll
    for (int j = 0; j < kUnitsPerThread; ++j) {
        const int64_t u = base + j * kThreads;
        const bool in = u < n_units;
        raw[j][0] = in ? ldg_stream(x + 2 * u) : make_uint4(0, 0, 0, 0);
        raw[j][1] = in ? ldg_stream(x + 2 * u + 1) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int j = 0; j < kUnitsPerThread; ++j) {
        const int64_t u = base + j * kThreads;
        const UnitCodes c = WIDE ? encode_unit_wide<GS>(raw[j][0], raw[j][1]) : encode_unit_sym<GS>(raw[j][0], raw[j][1]);
        if (u < n_units) store_unit_sym<GS>(c, u, lane, codes, flags, scales, packed != 0);
    }
}

// One block per row, for scales that are not per 64-group: either the row's
// own scale (group_q = K, per-token / per-channel: a first pass over the row
// finds max |x|), or a static calibrated scale `static_s16` given by the
// caller (any group_q; every group's stored scale is that value).  A second
// pass encodes the row with it.
template <int GS>
__global__ void __launch_bounds__(kThreads) quantize_row_sym_kernel(const uint4 *__restrict__ x, int64_t K,
                                                                    int group_q, int use_static,
                                                                    unsigned short static_s16,
                                                                    uint2 *__restrict__ codes,
                                                                    uint8_t *__restrict__ flags,
                                                                    __half *__restrict__ scales, int packed)
{
    griddep_wait();
    __shared__ float warp_max[kThreads / 32];
    const int lane = threadIdx.x & 31;
    const int64_t row = blockIdx.x;
    const int64_t U = K / 16;                       // units per row (a multiple of 4)
    const int64_t rounds = (U + kThreads - 1) / kThreads;
    const uint4 *xr = x + row * U * 2;
    __half s16;
    if (use_static) {
        s16 = __ushort_as_half(static_s16);
    } else {
        float m = 0.f;
        for (int64_t it = 0; it < rounds; ++it) {
            const int64_t j = it * kThreads + threadIdx.x;
            if (j >= U) break;
            const uint4 lo = ldg_stream(xr + 2 * j), hi = ldg_stream(xr + 2 * j + 1);
            const uint32_t w[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
            __half2 h = __habs2(*reinterpret_cast<const __half2 *>(&w[0]));
#pragma unroll
            for (int i = 1; i < 8; ++i) h = __hmax2(h, __habs2(*reinterpret_cast<const __half2 *>(&w[i])));
            const float2 f = __half22float2(h);
            m = fmaxf(m, fmaxf(f.x, f.y));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (lane == 0) warp_max[threadIdx.x >> 5] = m;
        __syncthreads();
        m = 0.f;
#pragma unroll
        for (int i = 0; i < kThreads / 32; ++i) m = fmaxf(m, warp_max[i]);
        s16 = __float2half_rn(__fdiv_rn(m, 127.0f));
    }
    const float s = __half2float(s16);
    const float r = (s > 0.f) ? __frcp_rn(s) : 0.f;
    for (int64_t it = 0; it < rounds; ++it) {   // the same trip count in every lane (shuffles)
        const int64_t j = it * kThreads + threadIdx.x;
        const bool in = j < U;
        const uint4 lo = in ? ldg_stream(xr + 2 * j) : make_uint4(0, 0, 0, 0);
        const uint4 hi = in ? ldg_stream(xr + 2 * j + 1) : make_uint4(0, 0, 0, 0);
        const UnitCodes c = encode_unit_sym_scaled<GS>(lo, hi, s16, r);
        if (!in) continue;
        const int64_t u = row * U + j;
        codes[u] = make_uint2(c.c0, c.c1);
        store_unit_flags<GS>(c, u, lane, flags, packed != 0);
        if ((j * 16) % group_q == 0) scales[(u * 16) / group_q] = s16;
    }
}

// Fused activation path of the linear layer: the same encoding, decoded at
// once to the GEMM's E4M3 operand (16 bytes per unit, row-major) and its
// scale side values (fp32, [G][m_pad], rows at perm32(r)); units of the
// padding rows [M, m_pad) write zero scales.  When `codes` is not NULL the
// encoded tensor is stored as well.
template <int GS, bool WIDE>
__global__ void __launch_bounds__(kThreads) encode_operand_kernel(
    const uint4 *__restrict__ x, int64_t n_units, int64_t n_units_pad, int64_t units_per_row, int64_t m_pad,
    uint4 *__restrict__ a_op, float *__restrict__ a_side, uint2 *__restrict__ codes,
    uint8_t *__restrict__ flags, __half *__restrict__ scales, int packed)
{
    griddep_wait();
    const int lane = threadIdx.x & 31;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * (kThreads * kUnitsPerThread) + threadIdx.x;
    uint4 raw[kUnitsPerThread][2];
#pragma unroll
    for (int j = 0; j < kUnitsPerThread; ++j) {
        const int64_t u = base + j * kThreads;
        const bool in = u < n_units;
        raw[j][0] = in ? ldg_stream(x + 2 * u) : make_uint4(0, 0, 0, 0);
        raw[j][1] = in ? ldg_stream(x + 2 * u + 1) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int j = 0; j < kUnitsPerThread; ++j) {
        const int64_t u = base + j * kThreads;
        const UnitCodes c = WIDE ? encode_unit_wide<GS>(raw[j][0], raw[j][1]) : encode_unit_sym<GS>(raw[j][0], raw[j][1]);
        if (u >= n_units_pad) continue;
        const int64_t row = u / units_per_row;
        if ((lane & 3) == 0) {
            const int64_t g = (u - row * units_per_row) >> 2;
            a_side[g * m_pad + perm32(row)] = u < n_units ? __half2float(c.s16) : 0.f;
        }
        if (u >= n_units) continue;
        uint4 o;
        if (WIDE) {
            e5m2_from_codes8(c.c0, c.flag0, o.x, o.y);
            e5m2_from_codes8(c.c1, c.flag1, o.z, o.w);
        } else {
            e4m3_from_codes8(c.c0, c.flag0, o.x, o.y);
            e4m3_from_codes8(c.c1, c.flag1, o.z, o.w);
        }
        a_op[u] = o;
        if (codes) store_unit_sym<GS>(c, u, lane, codes, flags, scales, packed != 0);
    }
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
// the stores.  (16-bit codes, symmetric: encode_unit_wide.)
template <int GS, int MODE>
__device__ __forceinline__ void encode_chunk(const uint4 raw, int64_t chunk, bool valid, int lane,
                                             uint32_t *__restrict__ codes,
                                             uint8_t *__restrict__ flags,
                                             __half *__restrict__ scales,
                                             int8_t *__restrict__ zeros,
                                             int32_t *__restrict__ gsum, bool packed)
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
        constexpr float kT = 1024.0f;  // beyond the cap, below int overflow
        constexpr int kQ = 127;
        const float t = fminf(fmaxf(__fmul_rn(x[i], r), -kT), kT);
        q[i] = min(max(__float2int_rn(t) + z, -kQ), kQ);
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
    constexpr int kChunksPerSub = GS / 8;
    const int flag_next = __shfl_down_sync(0xffffffffu, flag, kChunksPerSub);  // next subgroup's
    if (!valid) return;

    codes[chunk] = word;
    if (packed) {
        if ((lane & (2 * kChunksPerSub - 1)) == 0)
            flags[chunk / (2 * kChunksPerSub)] = static_cast<uint8_t>(flag | (flag_next << 4));
    } else if ((lane & (kChunksPerSub - 1)) == 0) {
        flags[chunk / kChunksPerSub] = static_cast<uint8_t>(flag);
    }
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
                                                            int32_t *__restrict__ gsum, int packed)
{
    griddep_wait();
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
        encode_chunk<GS, MODE>(raw[j], c, c < n_chunks, lane, codes, flags, scales, zeros, gsum,
                                     packed != 0);
    }
}

// Cache append (attention decode step): x [BH, T, d] fp16 is encoded into
// rows bh * L_max + t0 + j of an encoded cache, symmetric 8-bit codes.  The
// chunk encoder is the one above; only the output chunk index is remapped
// (d % 128 == 0 keeps every 64-group and every FLAG byte inside one row).
template <int GS>
__global__ void __launch_bounds__(kThreads) kv_append_kernel(const uint4 *__restrict__ x, int64_t n_chunks,
                                                             int64_t chunks_per_row, int64_t T, int64_t L_max,
                                                             int64_t t0, uint32_t *__restrict__ codes,
                                                             uint8_t *__restrict__ flags,
                                                             __half *__restrict__ scales, int packed)
{
    griddep_wait();
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
        const int64_t r = c / chunks_per_row;
        const int64_t dst_row = (r / T) * L_max + t0 + (r % T);
        const int64_t dst = dst_row * chunks_per_row + (c - r * chunks_per_row);
        encode_chunk<GS, QUARTZ_SYMMETRIC>(raw[j], dst, c < n_chunks, lane, codes, flags, scales,
                                                  nullptr, nullptr, packed != 0);
    }
}

// x_hat = s * (v - z), v = sgn(c) (|c| << FLAG); one thread per 8 elements.
// Dequantiser: x_hat = s * (v - z), v = c << FLAG, in binary32, rounded once to
// fp16.  Each thread takes kDeqChunksPerThread chunks of 8 elements (one
// 32-bit code word in, one 16-byte fp16 vector out) spaced a block apart, so
// that every load and store instruction of a warp is contiguous; all loads
// are issued before any arithmetic, which keeps several of them in flight
// per thread.  Subgroup and group indices are shifts (G_s and a 64-wide
// group are powers of two); one scale per row (group_q = K, any K % 64 == 0)
// divides by K.
constexpr int kDeqChunksPerThread = 4;

template <int GS>
__global__ void __launch_bounds__(kThreads) dequantize_kernel(
    const uint32_t *__restrict__ codes, const uint8_t *__restrict__ flags,
    const __half *__restrict__ scales, const int8_t *__restrict__ zeros, int64_t group_q,
    int packed, int64_t n_chunks, uint4 *__restrict__ out)
{
    griddep_wait();
    constexpr int kSubShift = GS == 8 ? 3 : GS == 16 ? 4 : GS == 32 ? 5 : 6;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * (kThreads * kDeqChunksPerThread) + threadIdx.x;
    uint32_t word[kDeqChunksPerThread];
    int flag[kDeqChunksPerThread], z[kDeqChunksPerThread];
    float sc[kDeqChunksPerThread];
#pragma unroll
    for (int j = 0; j < kDeqChunksPerThread; ++j) {
        const int64_t c = base + j * kThreads;
        word[j] = 0u;
        flag[j] = z[j] = 0;
        sc[j] = 0.f;
        if (c < n_chunks) {
            word[j] = __ldcs(codes + c);
            flag[j] = load_flag(flags, (c * 8) >> kSubShift, packed != 0);
            const int64_t g = group_q == 64 ? (c >> 3) : (c * 8) / group_q;
            sc[j] = __half2float(scales[g]);
            if (zeros) z[j] = zeros[g];
        }
    }
#pragma unroll
    for (int j = 0; j < kDeqChunksPerThread; ++j) {
        const int64_t c = base + j * kThreads;
        if (c >= n_chunks) continue;
        uint32_t o[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int c0 = static_cast<int>(word[j] << (28 - 8 * i)) >> 28;
            const int c1 = static_cast<int>(word[j] << (24 - 8 * i)) >> 28;
            const float y0 = __fmul_rn(sc[j], static_cast<float>(c0 * (1 << flag[j]) - z[j]));
            const float y1 = __fmul_rn(sc[j], static_cast<float>(c1 * (1 << flag[j]) - z[j]));
            const __half2 h = __floats2half2_rn(y0, y1);
            o[i] = *reinterpret_cast<const uint32_t *>(&h);
        }
        __stcs(out + c, make_uint4(o[0], o[1], o[2], o[3]));
    }
}

template <int GS, int MODE, bool WIDE = false>
cudaError_t launch_q(const void *x, const quartz_encoded_t *e, cudaStream_t s)
{
    if constexpr (MODE == QUARTZ_SYMMETRIC) {
        const int64_t n_units = e->rows * e->K / 16;
        const int64_t per_block = kThreads * kUnitsPerThread;
        const int64_t blocks = (n_units + per_block - 1) / per_block;
        launch_pdl(quantize_sym_kernel<GS, WIDE>, dim3(static_cast<unsigned>(blocks)), dim3(kThreads), 0, s, 
            static_cast<const uint4 *>(x), n_units, reinterpret_cast<uint2 *>(e->codes), e->flags,
            reinterpret_cast<__half *>(e->scales), e->p.flag_bits == 4);
        return cudaGetLastError();
    } else {
        const int64_t n_chunks = e->rows * e->K / 8;
        const int64_t per_block = kThreads * kChunksPerThread;
        const int64_t blocks = (n_chunks + per_block - 1) / per_block;
        launch_pdl(quantize_kernel<GS, MODE>, dim3(static_cast<unsigned>(blocks)), dim3(kThreads), 0, s, 
            static_cast<const uint4 *>(x), n_chunks, reinterpret_cast<uint32_t *>(e->codes), e->flags,
            reinterpret_cast<__half *>(e->scales), e->zeros, e->gsum, e->p.flag_bits == 4);
        return cudaGetLastError();
    }
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

cudaError_t launch_q_wide(const void *x, const quartz_encoded_t *e, cudaStream_t s)
{
    switch (e->p.group_s) {
        case 8: return launch_q<8, QUARTZ_SYMMETRIC, true>(x, e, s);
        case 16: return launch_q<16, QUARTZ_SYMMETRIC, true>(x, e, s);
        case 32: return launch_q<32, QUARTZ_SYMMETRIC, true>(x, e, s);
        default: return launch_q<64, QUARTZ_SYMMETRIC, true>(x, e, s);
    }
}

template <int GS>
cudaError_t launch_row(const void *x, const quartz_encoded_t *e, int use_static, unsigned short s16,
                       cudaStream_t s)
{
    launch_pdl(quantize_row_sym_kernel<GS>, dim3(static_cast<unsigned>(e->rows)), dim3(kThreads), 0, s, 
        static_cast<const uint4 *>(x), e->K, e->p.group_q, use_static, s16, reinterpret_cast<uint2 *>(e->codes),
        e->flags, reinterpret_cast<__half *>(e->scales), e->p.flag_bits == 4);
    return cudaGetLastError();
}

cudaError_t launch_quantize_row(const void *x, const quartz_encoded_t *e, int use_static, unsigned short s16,
                                cudaStream_t s)
{
    switch (e->p.group_s) {
        case 8: return launch_row<8>(x, e, use_static, s16, s);
        case 16: return launch_row<16>(x, e, use_static, s16, s);
        case 32: return launch_row<32>(x, e, use_static, s16, s);
        default: return launch_row<64>(x, e, use_static, s16, s);
    }
}

}  // namespace

cudaError_t launch_kv_append(const void *x, int64_t BH, int64_t T, const quartz_encoded_t *cache, int64_t L_max,
                             int64_t t0, cudaStream_t s)
{
    const int64_t cpr = cache->K / 8;
    const int64_t n_chunks = BH * T * cpr;
    if (n_chunks == 0) return cudaSuccess;
    const int64_t per_block = kThreads * kChunksPerThread;
    const unsigned blocks = static_cast<unsigned>((n_chunks + per_block - 1) / per_block);
    const uint4 *xv = static_cast<const uint4 *>(x);
    uint32_t *codes = reinterpret_cast<uint32_t *>(cache->codes);
    __half *scales = reinterpret_cast<__half *>(cache->scales);
    const int packed = cache->p.flag_bits == 4;
    switch (cache->p.group_s) {
        case 8: launch_pdl(kv_append_kernel<8>, dim3(blocks), dim3(kThreads), 0, s, xv, n_chunks, cpr, T, L_max, t0, codes, cache->flags, scales, packed); break;
        case 16: launch_pdl(kv_append_kernel<16>, dim3(blocks), dim3(kThreads), 0, s, xv, n_chunks, cpr, T, L_max, t0, codes, cache->flags, scales, packed); break;
        case 32: launch_pdl(kv_append_kernel<32>, dim3(blocks), dim3(kThreads), 0, s, xv, n_chunks, cpr, T, L_max, t0, codes, cache->flags, scales, packed); break;
        default: launch_pdl(kv_append_kernel<64>, dim3(blocks), dim3(kThreads), 0, s, xv, n_chunks, cpr, T, L_max, t0, codes, cache->flags, scales, packed); break;
    }
    return cudaGetLastError();
}

cudaError_t launch_quantize_static(const void *x, const quartz_encoded_t *out, uint16_t s16, cudaStream_t s)
{
    if (out->rows == 0) return cudaSuccess;
    return launch_quantize_row(x, out, 1, s16, s);
}

cudaError_t launch_quantize(const void *x, const quartz_encoded_t *out, cudaStream_t s)
{
    static_assert(kGroupQ == 64, "one quantization group is 8 lanes x 8 elements");
    if (out->rows == 0) return cudaSuccess;
    if (out->p.code_bits == 16) return launch_q_wide(x, out, s);   // Section 5 LLM variant
    if (out->p.group_q != kGroupQ) return launch_quantize_row(x, out, 0, 0, s);  // group_q == K
    return out->p.mode == QUARTZ_SYMMETRIC ? launch_q_mode<QUARTZ_SYMMETRIC>(x, out, s)
                                           : launch_q_mode<QUARTZ_ASYMMETRIC>(x, out, s);
}

cudaError_t launch_encode_operand(const void *x, int64_t M, int64_t K, const quartz_params_t *p,
                                  const LinearWorkspace &ws, const quartz_encoded_t *enc, cudaStream_t s)
{
    const int64_t upr = K / 16;
    const int64_t n_units = M * upr;
    const int64_t n_units_pad = ws.m_pad * upr;
    const int64_t per_block = kThreads * kUnitsPerThread;
    const unsigned blocks = static_cast<unsigned>((n_units_pad + per_block - 1) / per_block);
    const uint4 *xv = static_cast<const uint4 *>(x);
    uint4 *op = static_cast<uint4 *>(ws.a_op);
    uint2 *codes = enc ? reinterpret_cast<uint2 *>(enc->codes) : nullptr;
    uint8_t *flags = enc ? enc->flags : nullptr;
    __half *scales = enc ? reinterpret_cast<__half *>(enc->scales) : nullptr;
    const int packed = enc && enc->p.flag_bits == 4;
    if (p->code_bits == 16) {  // Section 5 LLM variant: E5M2 operand
        switch (p->group_s) {
            case 8: launch_pdl(encode_operand_kernel<8, true>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
            case 16: launch_pdl(encode_operand_kernel<16, true>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
            case 32: launch_pdl(encode_operand_kernel<32, true>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
            default: launch_pdl(encode_operand_kernel<64, true>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
        }
        return cudaGetLastError();
    }
    switch (p->group_s) {
        case 8: launch_pdl(encode_operand_kernel<8, false>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
        case 16: launch_pdl(encode_operand_kernel<16, false>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
        case 32: launch_pdl(encode_operand_kernel<32, false>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
        default: launch_pdl(encode_operand_kernel<64, false>, dim3(blocks), dim3(kThreads), 0, s, xv, n_units, n_units_pad, upr, ws.m_pad, op, ws.a_side, codes, flags, scales, packed); break;
    }
    return cudaGetLastError();
}

cudaError_t launch_dequantize(const quartz_encoded_t *e, void *y, cudaStream_t s)
{
    const int64_t n_chunks = e->rows * e->K / 8;
    if (n_chunks == 0) return cudaSuccess;
    const int64_t per_block = kThreads * kDeqChunksPerThread;
    const unsigned blocks = static_cast<unsigned>((n_chunks + per_block - 1) / per_block);
    const uint32_t *codes = reinterpret_cast<const uint32_t *>(e->codes);
    const __half *scales = reinterpret_cast<const __half *>(e->scales);
    const int8_t *zeros = e->p.mode == QUARTZ_ASYMMETRIC ? e->zeros : nullptr;
    const int packed = e->p.flag_bits == 4;
    uint4 *out = static_cast<uint4 *>(y);
    switch (e->p.group_s) {
        case 8: launch_pdl(dequantize_kernel<8>, dim3(blocks), dim3(kThreads), 0, s, codes, e->flags, scales, zeros, e->p.group_q, packed, n_chunks, out); break;
        case 16: launch_pdl(dequantize_kernel<16>, dim3(blocks), dim3(kThreads), 0, s, codes, e->flags, scales, zeros, e->p.group_q, packed, n_chunks, out); break;
        case 32: launch_pdl(dequantize_kernel<32>, dim3(blocks), dim3(kThreads), 0, s, codes, e->flags, scales, zeros, e->p.group_q, packed, n_chunks, out); break;
        default: launch_pdl(dequantize_kernel<64>, dim3(blocks), dim3(kThreads), 0, s, codes, e->flags, scales, zeros, e->p.group_q, packed, n_chunks, out); break;
    }
    return cudaGetLastError();
}

}  // namespace quartz
