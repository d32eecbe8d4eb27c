/*
 * QuaRTZ CPU oracle -- TEST INFRASTRUCTURE, NOT PART OF THE PRODUCT PATH.
 *
 * A plain, slow, single-threaded C restatement of what the W4A4 QuaRTZ
 * linear layer computes (arXiv 2509.26436):
 *   stage 1  per-group 8-bit min-max quantization        (Section 3, Eq. 1)
 *   stage 2  Leading Zero Suppression to 4-bit + FLAG    (Section 3, Eq. 2)
 *   LLM variant  16-bit codes straight to 4 bits, FLAG 0..12   (Section 5)
 *   GEMM     s4 x s4 -> integer partial sums per 64-wide group, then the
 *            16-bit-scale / zero-point dequantisation    (Section 4.4;
 *            Appendix C: groups of 64 along K with 16-bit scales)
 *
 * Only the test suite, the package smoke check and the benchmark's
 * CPU-baseline / reference leg load this library.  It shares no source,
 * header, table or helper with the CUDA library; the two only see the same
 * seeded fp16 inputs.
 *
 * Floating point: built with -O2 -ffp-contract=off so that every float
 * expression below is exactly one IEEE-754 binary32 round-to-nearest-even
 * operation (no fused multiply-add).  The paper fixes the storage
 * precisions (fp16 inputs, 16-bit scales, int8 / 4-bit codes, 32-bit
 * integer accumulation); the quantizer's intermediate arithmetic is binary32
 * (the precision the integer codes are decided in on both sides), and the
 * final dequantised product is accumulated in binary64.
 *
 * Readings of the paper used here (where it is silent or inconsistent):
 *   R1  Eq. 1 prints s = (xmax-xmin)/255 with a clamp to [-127,127] and
 *       z = round(-xmin/s), which do not fit together.  Default mode is the
 *       symmetric midtread quantizer of Appendix A: s = max|x|/127, z = 0.
 *       The asymmetric mode keeps Eq. 1's 255 levels and its zero point,
 *       widens [xmin, xmax] to contain 0, and stores z - 128 as int8.
 *   R2  round() is round-half-to-even.
 *   R3  x/s is evaluated as x * r with r = RN(1/s), both in binary32.
 *   R4  the 16-bit scale is IEEE binary16, rounded to nearest even, and the
 *       rounded scale is the one used to quantize.
 *   R5  a group whose scale rounds to 0 gets all-zero codes and z = 0.
 *   R6  the 4-bit code is two's complement in [-7, 7]; two codes per byte,
 *       element with even index in the low nibble.
 *   R7  the LZS shift truncates toward zero (Appendix A).
 *   R8  FLAG is stored unpacked, one byte per subgroup (Section 4.4).
 *   R9  groups and subgroups run along K, the reduction axis.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_ERR_ARG -1
#define ORACLE_ERR_CODE128 -2

/* ---------------------------------------------------------------------------
 * IEEE-754 binary16 <-> binary32, written from the format's definition:
 * 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits; exponent field 0
 * encodes zero / subnormals (fraction * 2^-24), 31 encodes inf / NaN.
 * ------------------------------------------------------------------------- */
float oracle_half_to_float(uint16_t h)
{
    int sign = (h >> 15) & 1;
    int e = (h >> 10) & 31;
    int f = h & 1023;
    float v;
    if (e == 0)
        v = ldexpf((float)f, -24);
    else if (e == 31)
        v = f ? NAN : INFINITY;
    else
        v = ldexpf((float)(1024 + f), e - 25);
    return sign ? -v : v;
}

uint16_t oracle_float_to_half_rn(float x)
{
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    float a = fabsf(x);
    if (isnan(x))
        return 0x7E00;
    if (a >= 65520.0f) /* halfway between 65504 and 2^16 rounds (to even) up */
        return sign | 0x7C00;
    if (a < ldexpf(1.0f, -14)) {
        /* subnormal range: quantum 2^-24; scaling by 2^24 is exact */
        float n = rintf(ldexpf(a, 24)); /* round half to even */
        return sign | (uint16_t)n;      /* n == 1024 encodes 2^-14 exactly */
    }
    int ex;
    frexpf(a, &ex);           /* a = fr * 2^ex, fr in [0.5, 1) */
    int E = ex - 1;           /* a in [2^E, 2^(E+1)) */
    float n = rintf(ldexpf(a, 10 - E)); /* significand * 2^10, in [1024, 2048] */
    if (n == 2048.0f) {
        n = 1024.0f;
        E += 1;
    }
    if (E + 15 >= 31)
        return sign | 0x7C00;
    return sign | (uint16_t)(((E + 15) << 10) | ((int)n - 1024));
}

/* round half to even, binary32 -> int (R2); |t| is bounded by the caller */
static int rne_int(float t) { return (int)rintf(t); }

static int clamp_int(int v, int lo, int hi) { return v < lo ? lo : (v > hi ? hi : v); }

static float clamp_float(float v, float lo, float hi) { return v < lo ? lo : (v > hi ? hi : v); }

/* ---------------------------------------------------------------------------
 * Stage 1: per-group 8-bit min-max quantization (Section 3, Eq. 1), groups of
 * `group_q` consecutive elements along K (Appendix C uses 64).
 *   mode 0 (symmetric, R1):  s = fp16(max|x| / 127), z = 0
 *   mode 1 (asymmetric, R1): xmin = min(min x, 0), xmax = max(max x, 0),
 *                            s = fp16((xmax - xmin) / 255),
 *                            z = round(-xmin / s) - 128   (stored offset)
 *   x_hat = clamp(round(x / s) + z, -127, 127)
 * Outputs: q [rows*K] int8, scales [rows*K/group_q] fp16 bits,
 *          zeros [rows*K/group_q] int8 (may be NULL in mode 0).
 * ------------------------------------------------------------------------- */
int oracle_quantize(const uint16_t *x, int64_t rows, int64_t K, int group_q, int mode,
                    int8_t *q, uint16_t *scales, int8_t *zeros)
{
    if (rows < 0 || K <= 0 || group_q <= 0 || K % group_q != 0 || (mode != 0 && mode != 1))
        return ORACLE_ERR_ARG;
    int64_t G = K / group_q;
    for (int64_t row = 0; row < rows; ++row) {
        for (int64_t g = 0; g < G; ++g) {
            const uint16_t *xg = x + row * K + g * group_q;
            int8_t *qg = q + row * K + g * group_q;
            float x_min = oracle_half_to_float(xg[0]);
            float x_max = x_min;
            for (int k = 1; k < group_q; ++k) {
                float v = oracle_half_to_float(xg[k]);
                if (v < x_min) x_min = v;
                if (v > x_max) x_max = v;
            }
            float s_f32;
            if (mode == 0) {
                float amax = fabsf(x_min) > fabsf(x_max) ? fabsf(x_min) : fabsf(x_max);
                s_f32 = amax / 127.0f;
            } else {
                if (x_min > 0.0f) x_min = 0.0f;
                if (x_max < 0.0f) x_max = 0.0f;
                float range = x_max - x_min;
                s_f32 = range / 255.0f;
            }
            uint16_t s16 = oracle_float_to_half_rn(s_f32);
            float s = oracle_half_to_float(s16);
            int z = 0;
            if (s == 0.0f) {
                /* R5: degenerate group */
                for (int k = 0; k < group_q; ++k) qg[k] = 0;
            } else {
                float r = 1.0f / s; /* R3 */
                if (mode == 1) {
                    float t = (-x_min) * r;
                    z = rne_int(t) - 128;
                }
                for (int k = 0; k < group_q; ++k) {
                    float t = oracle_half_to_float(xg[k]) * r;
                    t = clamp_float(t, -1024.0f, 1024.0f);
                    qg[k] = (int8_t)clamp_int(rne_int(t) + z, -127, 127);
                }
            }
            scales[row * G + g] = s16;
            if (zeros) zeros[row * G + g] = (int8_t)z;
        }
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------------
 * Static per-tensor quantization (Appendix C: the latent-diffusion setting
 * quantizes activations statically per tensor).  The scale s (fp16 bits) is
 * calibrated beforehand and given; every element is quantized with it as in
 * Eq. 1 (symmetric, z = 0): x_hat = clamp(round(x / s), -127, 127), x / s
 * evaluated as x * r with r = RN(1/s) (R3); s = 0 gives all-zero codes (R5).
 * Values beyond 127 s saturate.  Output q [n].
 * ------------------------------------------------------------------------- */
int oracle_quantize_static(const uint16_t *x, int64_t n, uint16_t s16, int8_t *q)
{
    float s = oracle_half_to_float(s16);
    if (n < 0 || !(s >= 0.0f) || s > 65504.0f) return ORACLE_ERR_ARG;
    if (s == 0.0f) {
        for (int64_t i = 0; i < n; ++i) q[i] = 0;
        return ORACLE_OK;
    }
    float r = 1.0f / s;
    for (int64_t i = 0; i < n; ++i) {
        float t = oracle_half_to_float(x[i]) * r;
        t = clamp_float(t, -1024.0f, 1024.0f);
        q[i] = (int8_t)clamp_int(rne_int(t), -127, 127);
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------------
 * Stage 2: Leading Zero Suppression (Section 3, Eq. 2).
 * Each int8 code is viewed as sign + 7-bit magnitude; per subgroup of G_s
 * codes the magnitudes are OR-ed into m, FLAG = max(29 - clz(m), 0), and
 * every magnitude is shifted right by FLAG (truncation toward zero, R7).
 * ------------------------------------------------------------------------- */

/* number of consecutive zero bits from the top of a 32-bit word (0..32) */
int oracle_clz32(uint32_t v)
{
    int n = 0;
    for (int b = 31; b >= 0; --b) {
        if ((v >> b) & 1u) break;
        ++n;
    }
    return n;
}

/* FLAG of one subgroup of `gs` int8 codes; ORACLE_ERR_CODE128 for code -128,
 * which Eq. 1 never produces and whose magnitude would need FLAG 5. */
int oracle_lzs_flag(const int8_t *q, int gs)
{
    uint32_t m = 0;
    for (int i = 0; i < gs; ++i) {
        if (q[i] == -128) return ORACLE_ERR_CODE128;
        uint32_t mag = (uint32_t)(q[i] < 0 ? -q[i] : q[i]);
        m |= mag;
    }
    int flag = 29 - oracle_clz32(m);
    return flag > 0 ? flag : 0;
}

/* codes q [n] -> flags [n/gs] and 4-bit values c [n] in [-7, 7] */
int oracle_lzs_encode(const int8_t *q, int64_t n, int gs, uint8_t *flags, int8_t *c)
{
    if (gs <= 0 || n % gs != 0) return ORACLE_ERR_ARG;
    for (int64_t b = 0; b < n / gs; ++b) {
        int flag = oracle_lzs_flag(q + b * gs, gs);
        if (flag < 0) return flag;
        flags[b] = (uint8_t)flag;
        for (int i = 0; i < gs; ++i) {
            int v = q[b * gs + i];
            int sgn = v < 0 ? -1 : 1;
            int mag = v < 0 ? -v : v;
            c[b * gs + i] = (int8_t)(sgn * (mag >> flag));
        }
    }
    return ORACLE_OK;
}

/* 4-bit values c [n] + flags -> decoded integers v = sgn * (|c| << FLAG):
 * every value of a subgroup was shifted by the same FLAG, so shifting back by
 * FLAG restores its magnitude (minus the truncated low bits). */
int oracle_lzs_decode(const int8_t *c, const uint8_t *flags, int64_t n, int gs, int16_t *v)
{
    if (gs <= 0 || n % gs != 0) return ORACLE_ERR_ARG;
    for (int64_t i = 0; i < n; ++i) {
        int ci = c[i];
        int sgn = ci < 0 ? -1 : 1;
        int mag = ci < 0 ? -ci : ci;
        v[i] = (int16_t)(sgn * (mag << flags[i / gs]));
    }
    return ORACLE_OK;
}

/* R6: two signed 4-bit codes per byte, even index in the low nibble */
void oracle_pack_nibbles(const int8_t *c, int64_t n, uint8_t *packed)
{
    for (int64_t i = 0; i < n; i += 2) {
        uint8_t lo = (uint8_t)(c[i] & 0xF);
        uint8_t hi = (uint8_t)((i + 1 < n ? c[i + 1] : 0) & 0xF);
        packed[i / 2] = (uint8_t)(lo | (hi << 4));
    }
}

void oracle_unpack_nibbles(const uint8_t *packed, int64_t n, int8_t *c)
{
    for (int64_t i = 0; i < n; ++i) {
        int nib = (packed[i / 2] >> ((i & 1) * 4)) & 0xF;
        c[i] = (int8_t)(nib >= 8 ? nib - 16 : nib);
    }
}

/* ---------------------------------------------------------------------------
 * Full encoder: fp16 [rows, K] -> packed codes [rows, K/2], flags
 * [rows, K/gs], scales [rows, K/gq] (fp16 bits), zeros [rows, K/gq] and
 * gsum [rows, K/gq] = sum of the decoded values of each quantization group
 * (needed by the zero-point correction; zeros/gsum may be NULL in mode 0).
 * ------------------------------------------------------------------------- */
int oracle_encode(const uint16_t *x, int64_t rows, int64_t K, int gq, int gs, int mode,
                  uint8_t *codes, uint8_t *flags, uint16_t *scales, int8_t *zeros,
                  int32_t *gsum)
{
    if (gs <= 0 || gq % gs != 0 || K % gq != 0 || K % 2 != 0) return ORACLE_ERR_ARG;
    int8_t q[65536];
    int8_t c[65536];
    int16_t v[65536];
    if (K > 65536) return ORACLE_ERR_ARG;
    int64_t G = K / gq;
    for (int64_t row = 0; row < rows; ++row) {
        int rc = oracle_quantize(x + row * K, 1, K, gq, mode, q, scales + row * G,
                                 zeros ? zeros + row * G : 0);
        if (rc) return rc;
        rc = oracle_lzs_encode(q, K, gs, flags + row * (K / gs), c);
        if (rc) return rc;
        oracle_pack_nibbles(c, K, codes + row * (K / 2));
        if (gsum) {
            oracle_lzs_decode(c, flags + row * (K / gs), K, gs, v);
            for (int64_t g = 0; g < G; ++g) {
                int32_t s = 0;
                for (int k = 0; k < gq; ++k) s += v[g * gq + k];
                gsum[row * G + g] = s;
            }
        }
    }
    return ORACLE_OK;
}

/* Encoder with a static scale: Eq. 1 with the given scale (above), then
 * Eq. 2 as oracle_encode; scales [rows, K/gq] all receive s16 (symmetric). */
int oracle_encode_static(const uint16_t *x, int64_t rows, int64_t K, uint16_t s16, int gq, int gs,
                         uint8_t *codes, uint8_t *flags, uint16_t *scales)
{
    if (gs <= 0 || gq % gs != 0 || K % gq != 0 || K % 2 != 0) return ORACLE_ERR_ARG;
    int8_t q[65536];
    int8_t c[65536];
    if (K > 65536) return ORACLE_ERR_ARG;
    int64_t G = K / gq;
    for (int64_t row = 0; row < rows; ++row) {
        int rc = oracle_quantize_static(x + row * K, K, s16, q);
        if (rc) return rc;
        rc = oracle_lzs_encode(q, K, gs, flags + row * (K / gs), c);
        if (rc) return rc;
        oracle_pack_nibbles(c, K, codes + row * (K / 2));
        for (int64_t g = 0; g < G; ++g) scales[row * G + g] = s16;
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------------
 * LLM variant (Section 5: activations quantized to 16-bit integers and
 * then LZS-coded to 4 bits, subgroups of G_s = 8).  Stage 1 quantizes
 * each group to 16-bit integers, symmetric: s = fp16(max|x| / 32767),
 * q = clamp(round(x * r), -32767, 32767) with r = RN(1/s) (R3); a zero scale
 * gives all-zero codes (R5).  Stage 2 is Eq. 2 unchanged on the wider codes:
 * FLAG = max(29 - clz(m), 0) now ranges over 0..12, and the 4-bit code keeps
 * the three bits below the leading one: c = sgn(q) (|q| >> FLAG).
 * ------------------------------------------------------------------------- */
int oracle_quantize16(const uint16_t *x, int64_t rows, int64_t K, int group_q, int16_t *q,
                      uint16_t *scales)
{
    if (rows < 0 || K <= 0 || group_q <= 0 || K % group_q != 0) return ORACLE_ERR_ARG;
    int64_t G = K / group_q;
    for (int64_t row = 0; row < rows; ++row) {
        for (int64_t g = 0; g < G; ++g) {
            const uint16_t *xg = x + row * K + g * group_q;
            int16_t *qg = q + row * K + g * group_q;
            float amax = 0.0f;
            for (int k = 0; k < group_q; ++k) {
                float v = fabsf(oracle_half_to_float(xg[k]));
                if (v > amax) amax = v;
            }
            uint16_t s16 = oracle_float_to_half_rn(amax / 32767.0f);
            float s = oracle_half_to_float(s16);
            if (s == 0.0f) {
                for (int k = 0; k < group_q; ++k) qg[k] = 0;
            } else {
                float r = 1.0f / s;
                for (int k = 0; k < group_q; ++k) {
                    float t = clamp_float(oracle_half_to_float(xg[k]) * r, -65536.0f, 65536.0f);
                    qg[k] = (int16_t)clamp_int(rne_int(t), -32767, 32767);
                }
            }
            scales[row * G + g] = s16;
        }
    }
    return ORACLE_OK;
}

/* Eq. 2 on 16-bit codes q [n]: flags [n/gs] (0..12), 4-bit values c [n] */
int oracle_lzs_encode16(const int16_t *q, int64_t n, int gs, uint8_t *flags, int8_t *c)
{
    if (gs <= 0 || n % gs != 0) return ORACLE_ERR_ARG;
    for (int64_t b = 0; b < n / gs; ++b) {
        uint32_t m = 0;
        for (int i = 0; i < gs; ++i) {
            int v = q[b * gs + i];
            if (v == -32768) return ORACLE_ERR_CODE128;
            m |= (uint32_t)(v < 0 ? -v : v);
        }
        int flag = 29 - oracle_clz32(m);
        if (flag < 0) flag = 0;
        flags[b] = (uint8_t)flag;
        for (int i = 0; i < gs; ++i) {
            int v = q[b * gs + i];
            int mag = v < 0 ? -v : v;
            c[b * gs + i] = (int8_t)((v < 0 ? -1 : 1) * (mag >> flag));
        }
    }
    return ORACLE_OK;
}

/* Full LLM-variant encoder: codes [rows, K/2], flags [rows, K/gs], scales [rows, K/gq] */
int oracle_encode16(const uint16_t *x, int64_t rows, int64_t K, int gq, int gs, uint8_t *codes,
                    uint8_t *flags, uint16_t *scales)
{
    if (gs <= 0 || gq % gs != 0 || K % gq != 0 || K % 2 != 0 || K > 65536) return ORACLE_ERR_ARG;
    int16_t q[65536];
    int8_t c[65536];
    int64_t G = K / gq;
    for (int64_t row = 0; row < rows; ++row) {
        int rc = oracle_quantize16(x + row * K, 1, K, gq, q, scales + row * G);
        if (rc) return rc;
        rc = oracle_lzs_encode16(q, K, gs, flags + row * (K / gs), c);
        if (rc) return rc;
        oracle_pack_nibbles(c, K, codes + row * (K / 2));
    }
    return ORACLE_OK;
}

/* decode packed codes + flags of `rows` rows back to integers v [rows, K] */
int oracle_decode_codes(const uint8_t *codes, const uint8_t *flags, int64_t rows, int64_t K,
                        int gs, int16_t *v)
{
    int8_t c[65536];
    if (K > 65536 || gs <= 0 || K % gs != 0) return ORACLE_ERR_ARG;
    for (int64_t row = 0; row < rows; ++row) {
        oracle_unpack_nibbles(codes + row * (K / 2), K, c);
        int rc = oracle_lzs_decode(c, flags + row * (K / gs), K, gs, v + row * K);
        if (rc) return rc;
    }
    return ORACLE_OK;
}

/* dequantised values x_hat = s * (v - z) of one encoded tensor, binary64 */
int oracle_dequantize(const uint8_t *codes, const uint8_t *flags, const uint16_t *scales,
                      const int8_t *zeros, int64_t rows, int64_t K, int gq, int gs, double *out)
{
    int16_t v[65536];
    if (K > 65536 || gq <= 0 || K % gq != 0) return ORACLE_ERR_ARG;
    int64_t G = K / gq;
    for (int64_t row = 0; row < rows; ++row) {
        int rc = oracle_decode_codes(codes + row * (K / 2), flags + row * (K / gs), 1, K, gs, v);
        if (rc) return rc;
        for (int64_t k = 0; k < K; ++k) {
            int64_t g = k / gq;
            double s = (double)oracle_half_to_float(scales[row * G + g]);
            int z = zeros ? zeros[row * G + g] : 0;
            out[row * K + k] = s * (double)(v[k] - z);
        }
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------------
 * GEMM (Section 4.4): the integer MMA over decoded LZS values, one partial
 * sum per quantization group g of 64 along K:
 *     P_g[m, n] = sum_{k in g} v_a[m, k] * v_w[n, k]          (int64)
 * for the selected activation rows `rows_sel` (NULL = all M rows).
 * Output P [G][n_sel][N].
 * ------------------------------------------------------------------------- */
int oracle_group_partials(const int16_t *va, const int16_t *vw, int64_t M, int64_t N, int64_t K,
                          int gq, const int64_t *rows_sel, int64_t n_sel, int64_t *P)
{
    if (gq <= 0 || K % gq != 0) return ORACLE_ERR_ARG;
    int64_t G = K / gq;
    int64_t nr = rows_sel ? n_sel : M;
    for (int64_t i = 0; i < nr; ++i) {
        int64_t m = rows_sel ? rows_sel[i] : i;
        if (m < 0 || m >= M) return ORACLE_ERR_ARG;
        for (int64_t n = 0; n < N; ++n) {
            for (int64_t g = 0; g < G; ++g) {
                int64_t acc = 0;
                for (int64_t k = g * gq; k < (g + 1) * gq; ++k)
                    acc += (int64_t)va[m * K + k] * (int64_t)vw[n * K + k];
                P[(g * nr + i) * N + n] = acc;
            }
        }
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------------
 * W4A4 linear (Section 4.4 with Appendix C's 16-bit group scales):
 *     y[m, n] = sum_g s_a[m,g] * s_w[n,g] * D_g[m, n]  (+ bias[n])
 *     D_g[m, n] = sum_{k in g} (v_a[m,k] - z_a[m,g]) * (v_w[n,k] - z_w[n,g])
 * i.e. the exact product of the two dequantised operands x_hat = s (v - z),
 * evaluated with integer group sums and binary64 scaling.
 * Encoded operands are passed as (codes, flags, scales, zeros); zeros may be
 * NULL (symmetric).  bias is fp16 bits or NULL.  y [n_sel, N] binary64 for
 * the selected rows (rows_sel NULL = all M rows).  When `yabs` is not NULL it
 * receives sum_g |s_a s_w D_g| + |bias[n]|, the magnitude a rounding error
 * bound of any evaluation order scales with.
 * ------------------------------------------------------------------------- */
int oracle_linear(const uint8_t *a_codes, const uint8_t *a_flags, const uint16_t *a_scales,
                  const int8_t *a_zeros, const uint8_t *w_codes, const uint8_t *w_flags,
                  const uint16_t *w_scales, const int8_t *w_zeros, int64_t M, int64_t N,
                  int64_t K, int gq, int gs, const uint16_t *bias, const int64_t *rows_sel,
                  int64_t n_sel, int16_t *w_scratch /* [N*K] */, double *y, double *yabs)
{
    int16_t va[65536];
    if (K > 65536 || gq <= 0 || K % gq != 0 || gs <= 0 || gq % gs != 0) return ORACLE_ERR_ARG;
    int64_t G = K / gq;
    int rc = oracle_decode_codes(w_codes, w_flags, N, K, gs, w_scratch);
    if (rc) return rc;
    int64_t nr = rows_sel ? n_sel : M;
    for (int64_t i = 0; i < nr; ++i) {
        int64_t m = rows_sel ? rows_sel[i] : i;
        if (m < 0 || m >= M) return ORACLE_ERR_ARG;
        rc = oracle_decode_codes(a_codes + m * (K / 2), a_flags + m * (K / gs), 1, K, gs, va);
        if (rc) return rc;
        for (int64_t n = 0; n < N; ++n) {
            const int16_t *vw = w_scratch + n * K;
            double acc = 0.0, mag = 0.0;
            for (int64_t g = 0; g < G; ++g) {
                int za = a_zeros ? a_zeros[m * G + g] : 0;
                int zw = w_zeros ? w_zeros[n * G + g] : 0;
                int64_t d = 0;
                for (int64_t k = g * gq; k < (g + 1) * gq; ++k)
                    d += (int64_t)(va[k] - za) * (int64_t)(vw[k] - zw);
                double sa = (double)oracle_half_to_float(a_scales[m * G + g]);
                double sw = (double)oracle_half_to_float(w_scales[n * G + g]);
                acc += sa * sw * (double)d;
                mag += fabs(sa * sw * (double)d);
            }
            if (bias) {
                acc += (double)oracle_half_to_float(bias[n]);
                mag += fabs((double)oracle_half_to_float(bias[n]));
            }
            y[i * N + n] = acc;
            if (yabs) yabs[i * N + n] = mag;
        }
    }
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------------
 * QuaRTZ attention, one decode step (Appendix D, Table 6: QuaRTZ kernels for
 * attention with heads x 128 dimensions and LZS groups of 8 / 16 / 32).  The
 * paper gives no formula; the reading used here: the query and the
 * key / value caches are encoded with Eq. 1 + Eq. 2 per token, groups of
 * `gq` along the head dimension d, and for each of the BH (batch x head)
 * rows
 *     score_t = scale * sum_g s_q[g] s_k[t,g] sum_{k in g} v_q[k] v_k[t,k]
 *     p_t     = exp(score_t - max_t score) / sum_t exp(score_t - max_t score)
 *     o[k]    = sum_t p_t * s_v[t,g(k)] * v_v[t,k]
 * over the first L tokens of the head, the integer group sums in int64 and
 * everything else in binary64.  The caches hold the tokens of head bh in
 * rows bh * L_max .. bh * L_max + L - 1.  Output o [BH, d]; when `oabs` is
 * not NULL it receives sum_t p_t |s_v v_v[t,k]|, the magnitude a rounding
 * error bound of o scales with.  Symmetric encodings (no zero points).
 * ------------------------------------------------------------------------- */
int oracle_attention_decode(const uint8_t *q_codes, const uint8_t *q_flags, const uint16_t *q_scales,
                            const uint8_t *k_codes, const uint8_t *k_flags, const uint16_t *k_scales,
                            const uint8_t *v_codes, const uint8_t *v_flags, const uint16_t *v_scales,
                            int64_t BH, int64_t L_max, int64_t L, int64_t d, int gq, int gs,
                            double scale, double *o, double *oabs)
{
    static double score[65536];
    int16_t vq[4096], vk[4096];
    if (d <= 0 || d > 4096 || gq <= 0 || d % gq != 0 || gs <= 0 || gq % gs != 0 || L <= 0 ||
        L > L_max || L > 65536 || BH < 0)
        return ORACLE_ERR_ARG;
    int64_t G = d / gq;
    for (int64_t bh = 0; bh < BH; ++bh) {
        int rc = oracle_decode_codes(q_codes + bh * (d / 2), q_flags + bh * (d / gs), 1, d, gs, vq);
        if (rc) return rc;
        double smax = -INFINITY;
        for (int64_t t = 0; t < L; ++t) {
            int64_t row = bh * L_max + t;
            rc = oracle_decode_codes(k_codes + row * (d / 2), k_flags + row * (d / gs), 1, d, gs, vk);
            if (rc) return rc;
            double acc = 0.0;
            for (int64_t g = 0; g < G; ++g) {
                int64_t P = 0;
                for (int64_t k = g * gq; k < (g + 1) * gq; ++k) P += (int64_t)vq[k] * (int64_t)vk[k];
                acc += (double)oracle_half_to_float(q_scales[bh * G + g]) *
                       (double)oracle_half_to_float(k_scales[row * G + g]) * (double)P;
            }
            score[t] = scale * acc;
            if (score[t] > smax) smax = score[t];
        }
        double denom = 0.0;
        for (int64_t t = 0; t < L; ++t) {
            score[t] = exp(score[t] - smax);
            denom += score[t];
        }
        for (int64_t k = 0; k < d; ++k) {
            o[bh * d + k] = 0.0;
            if (oabs) oabs[bh * d + k] = 0.0;
        }
        for (int64_t t = 0; t < L; ++t) {
            int64_t row = bh * L_max + t;
            double p = score[t] / denom;
            rc = oracle_decode_codes(v_codes + row * (d / 2), v_flags + row * (d / gs), 1, d, gs, vk);
            if (rc) return rc;
            for (int64_t k = 0; k < d; ++k) {
                double vhat = (double)oracle_half_to_float(v_scales[row * G + k / gq]) * (double)vk[k];
                o[bh * d + k] += p * vhat;
                if (oabs) oabs[bh * d + k] += p * fabs(vhat);
            }
        }
    }
    return ORACLE_OK;
}
