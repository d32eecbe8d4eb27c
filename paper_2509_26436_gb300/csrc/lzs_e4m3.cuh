// Device helpers shared by the encoder and the operand preparation: decode
// of 4-bit LZS codes (Eq. 2) to FP8 E4M3 (or, for 16-bit stage-1 codes,
// E5M2) tensor-core operands.
#pragma once
#include <cstdint>

namespace quartz {

// Byte permute (PTX prmt, default mode: a selector nibble b < 8 copies byte b
// of {hi:lo}, b + 8 replicates that byte's sign bit).
__device__ __forceinline__ uint32_t prmt_b32(uint32_t lo, uint32_t hi, uint32_t sel)
{
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(lo), "r"(hi), "r"(sel));
    return d;
}

// Four table lookups at once: byte k of x (0..15) selects byte x_k of the
// 16-byte table {t0, t1, t2, t3}.
__device__ __forceinline__ uint32_t lut16(uint32_t x, uint32_t t0, uint32_t t1, uint32_t t2, uint32_t t3)
{
    const uint32_t y = x & 0x07070707u;
    const uint32_t sel = prmt_b32(y | (y >> 4), 0u, 0x0020u);  // nibble k = low 3 bits of byte k
    const uint32_t lo = prmt_b32(t0, t1, sel);
    const uint32_t hi = prmt_b32(t2, t3, sel);
    const uint32_t use_hi = prmt_b32(x << 4, 0u, 0xBA98u);      // 0xFF where bit 3 of byte k is set
    return (hi & use_hi) | (lo & ~use_hi);
}

// Decode eight 4-bit codes (one 32-bit word, code k in bits 4k..4k+3) of one
// subgroup with FLAG `flag` to E4M3 bytes of v = c * 2^flag, written to the
// eight bytes of {lo, hi} in code order.  The E4M3 byte of a nonzero c is
// sign | (7 + e + flag) << 3 | m for |c| = (1 + m/8) 2^e, so the table for
// FLAG f is the FLAG-0 table with 8 f added to every nonzero entry (no carry
// leaves a byte: the largest entry, 7 * 2^4 = 112, is 0x6E / 0xEE).
__device__ __forceinline__ void e4m3_from_codes8(uint32_t word, int flag, uint32_t &lo, uint32_t &hi)
{
    const uint32_t add = (static_cast<uint32_t>(flag) << 3) * 0x01010101u;
    // entries for codes 0..15 (two's complement -8..7; -8 never occurs)
    const uint32_t t0 = 0x44403800u + (add & 0xFFFFFF00u);  //  0,  1,  2,  3
    const uint32_t t1 = 0x4E4C4A48u + add;                  //  4,  5,  6,  7
    const uint32_t t2 = 0xCACCCE00u + (add & 0xFFFFFF00u);  // -8, -7, -6, -5
    const uint32_t t3 = 0xB8C0C4C8u + add;                  // -4, -3, -2, -1
    const uint32_t ev = lut16(word & 0x0F0F0F0Fu, t0, t1, t2, t3);         // codes 0, 2, 4, 6
    const uint32_t od = lut16((word >> 4) & 0x0F0F0F0Fu, t0, t1, t2, t3);  // codes 1, 3, 5, 7
    lo = prmt_b32(ev, od, 0x5140u);
    hi = prmt_b32(ev, od, 0x7362u);
}

// The same for codes with FLAGs up to 12 (16-bit stage-1 codes, Section 5
// LLM variant), to E5M2 bytes: |v| reaches 7 * 2^12 = 28672, beyond E4M3's
// range but exact in E5M2, whose 2-bit mantissa holds every |c| <= 7
// (1, 1.5 or 1.75 times a power of two) and whose exponent reaches 2^15.
// The byte of a nonzero c is sign | (15 + e + flag) << 2 | m, so FLAG f adds
// 4 f to every nonzero entry (largest 0x47 + 48 = 0x77: no carry leaves a
// byte).
__device__ __forceinline__ void e5m2_from_codes8(uint32_t word, int flag, uint32_t &lo, uint32_t &hi)
{
    const uint32_t add = (static_cast<uint32_t>(flag) << 2) * 0x01010101u;
    const uint32_t t0 = 0x42403C00u + (add & 0xFFFFFF00u);  //  0,  1,  2,  3
    const uint32_t t1 = 0x47464544u + add;                  //  4,  5,  6,  7
    const uint32_t t2 = 0xC5C6C700u + (add & 0xFFFFFF00u);  // -8, -7, -6, -5
    const uint32_t t3 = 0xBCC0C2C4u + add;                  // -4, -3, -2, -1
    const uint32_t ev = lut16(word & 0x0F0F0F0Fu, t0, t1, t2, t3);
    const uint32_t od = lut16((word >> 4) & 0x0F0F0F0Fu, t0, t1, t2, t3);
    lo = prmt_b32(ev, od, 0x5140u);
    hi = prmt_b32(ev, od, 0x7362u);
}

// FLAG of subgroup k (global index over the flattened [rows, K/G_s] array):
// one byte per FLAG, or packed two per byte (subgroup 2j in the low nibble).
__device__ __forceinline__ int load_flag(const uint8_t *flags, int64_t k, bool packed)
{
    return packed ? (flags[k >> 1] >> ((k & 1) * 4)) & 0xF : flags[k];
}

}  // namespace quartz
