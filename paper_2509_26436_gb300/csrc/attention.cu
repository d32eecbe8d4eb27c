// QuaRTZ attention, one decode step (Appendix D, Table 6: attention with
// heads x 128 dimensions on LZS-coded operands, groups of 8 / 16 / 32), for
// sm_103a.
//
// One query per (batch x head) row attends over the first L tokens of that
// head's key / value cache.  Query, keys and values are QuaRTZ-encoded per
// token (Eq. 1 + Eq. 2, 64-wide groups along the head dimension):
//     score_t = scale * sum_g s_q[g] s_k[t,g] P_g[t],
//     P_g[t]  = sum_{k in g} v_q[k] v_k[t,k]            (exact integers)
//     o       = sum_t softmax(score)_t * s_v[t,g] v_v[t,.]
// The step is HBM-bound: per token and head it reads 2 x (64 code bytes +
// 128/G_s FLAG bytes + 4 scale bytes) and does about 2 operations per cached
// element, so the kernel streams the caches once, split over enough CTAs to
// keep every SM's memory pipe busy (split-L with a combine pass):
//
//   attn_decode_kernel<G_s>: CTA (split, bh), 128 threads, tokens in tiles
//     of 128.  Keys: one token per thread; the integer group sums are dp4a
//     products of the query's decoded values (int8, |v| <= 112, computed
//     once per CTA) with the key codes placed in the high nibble of each
//     byte (16 c), shifted per subgroup by the key's FLAG — the paper's
//     accumulator-shift schedule (Section 4.4) on the key side, exact.
//     Softmax: running maximum and sum per CTA in the log2 domain; each key
//     thread then writes p_t s_v 2^FLAG for its token's value subgroups
//     (the FLAG added to the scale's exponent field).  Values: 4 threads per
//     token row (one 16-byte chunk of 32 codes each) x 32 token slots; each
//     code becomes a float exactly through the 2^23 magic number, and
//     o += p_t s_v 2^FLAG c with paired f32x2 subtract and fused
//     multiply-add (two instructions per two codes).  The code tiles of
//     both caches (8 KB each per 128 tokens) stream through a 2-stage
//     shared-memory ring filled by cp.async (chunks XOR-swizzled against
//     bank conflicts) one tile ahead (more stages measured slower: fewer
//     CTAs fit an SM); FLAGs and scales of the next tile are prefetched
//     into registers.  Output per CTA: unnormalised o, running
//     max, running sum.
//   attn_combine_kernel: one CTA per bh merges the splits.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <atomic>

#include "lzs_e4m3.cuh"
#include "quartz_internal.h"

namespace quartz {
namespace {

constexpr int kD = 128;              // head dimension
constexpr int kWords = kD / 8;       // 32-bit code words per token row
constexpr int kTile = 128;           // tokens per tile = threads per CTA
constexpr int kAttnThreads = 128;
constexpr int kPfStride = kTile + 2;           // s_pf row stride: conflict-free reads and writes
constexpr int kPartStride = kD + 4;  // o[128], m, l (+ pad) per split
constexpr int kMaxSplits = 64;
constexpr float kLog2e = 1.4426950408889634f;

struct AttnArgs {
    const uint32_t *q_codes;
    const uint8_t *q_flags;
    const __half *q_scales;
    const uint32_t *k_codes;
    const uint8_t *k_flags;
    const __half *k_scales;
    const uint32_t *v_codes;
    const uint8_t *v_flags;
    const __half *v_scales;
    int q_packed, k_packed, v_packed;
    int64_t L_max;
    int L, n_split, chunk;
    float scale_log2;  // softmax scale * log2(e)
    float *part;       // [BH][n_split][kPartStride]
};

// The FLAG bytes (or nibbles) of one token row: S = 128 / G_s subgroups,
// stored at subgroup index row * S + j (one byte each, or two per byte).
template <int GS>
__device__ __forceinline__ void load_row_flags(const uint8_t *flags, int64_t row, bool packed, uint32_t (&f)[4])
{
    constexpr int S = kD / GS;
    f[0] = f[1] = f[2] = f[3] = 0u;
    const int bytes = packed ? S / 2 : S;
    const uint8_t *p = flags + row * bytes;
    if (bytes == 16) {
        const uint4 v = *reinterpret_cast<const uint4 *>(p);
        f[0] = v.x, f[1] = v.y, f[2] = v.z, f[3] = v.w;
    } else if (bytes == 8) {
        const uint2 v = *reinterpret_cast<const uint2 *>(p);
        f[0] = v.x, f[1] = v.y;
    } else if (bytes == 4) {
        f[0] = *reinterpret_cast<const uint32_t *>(p);
    } else if (bytes == 2) {
        f[0] = *reinterpret_cast<const uint16_t *>(p);
    } else {
        f[0] = *p;
    }
}

__device__ __forceinline__ int row_flag(const uint32_t (&f)[4], int j, bool packed)
{
    return packed ? static_cast<int>((f[j >> 3] >> (4 * (j & 7))) & 0xFu)
                  : static_cast<int>((f[j >> 2] >> (8 * (j & 3))) & 0xFFu);
}

__device__ __forceinline__ float2 load_scales2(const __half *scales, int64_t row)
{
    const uint32_t w = *reinterpret_cast<const uint32_t *>(scales + 2 * row);
    return __half22float2(*reinterpret_cast<const __half2 *>(&w));
}

// The float 2^23 + (c + 8) for the biased code byte selected by `sel` (byte
// b of `biased_bytes` into byte 0, 0x4B above it: 0x4B0000xx = 2^23 + xx).
__device__ __forceinline__ float magic_float(uint32_t biased_bytes, uint32_t sel)
{
    return __int_as_float(prmt_b32(biased_bytes, 0x4B000000u, sel));
}

__device__ __forceinline__ uint4 lds_u4(uint32_t addr)
{
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

// s v 2^F for a float s that is 0 or normal: the exponent field grows by F
// (exact; for s = 0 the result is a tiny normal, only ever multiplied by 0).
__device__ __forceinline__ float scale_pow2(float s, int F)
{
    return __int_as_float(__float_as_int(s) + (F << 23));
}

// (acc0, acc1) += p * (c0, c1), where c = f - (2^23 + 8) for the magic floats
// f: one paired subtraction and one paired fused multiply-add.
__device__ __forceinline__ void fma_codes2(float &acc0, float &acc1, float p, float f0, float f1)
{
    asm("{\n\t.reg .b64 f, m, c, pp, acc;\n\t"
        "mov.b64 f, {%2, %3};\n\t"
        "mov.b64 m, {%5, %5};\n\t"
        "add.rn.f32x2 c, f, m;\n\t"
        "mov.b64 pp, {%4, %4};\n\t"
        "mov.b64 acc, {%0, %1};\n\t"
        "fma.rn.f32x2 acc, pp, c, acc;\n\t"
        "mov.b64 {%0, %1}, acc;\n\t}"
        : "+f"(acc0), "+f"(acc1)
        : "f"(f0), "f"(f1), "f"(p), "f"(-8388616.0f));
}

// Asynchronous 16-byte global -> shared copies (cp.async, completion tracked
// per thread in commit groups; the wait is the hardware's own).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Shared-memory offset of 16-byte chunk c (0..3) of token row r in a code
// tile: rows of 64 bytes, chunks XOR-swizzled by (r / 2) % 4 so that eight
// consecutive rows reading the same chunk hit eight different bank groups.
__device__ __forceinline__ uint32_t tile_off(int r, int c) { return r * 64 + ((c ^ ((r >> 1) & 3)) << 4); }

// The FLAGs and scales of one token row of the key and value caches.
struct RowSide {
    uint32_t kf[4], vf[4];
    float2 sk, sv;
};

template <int GS>
__device__ __forceinline__ void load_side(const AttnArgs &a, int64_t row, bool valid, RowSide &r)
{
    if (valid) {
        load_row_flags<GS>(a.k_flags, row, a.k_packed != 0, r.kf);
        load_row_flags<GS>(a.v_flags, row, a.v_packed != 0, r.vf);
        r.sk = load_scales2(a.k_scales, row);
        r.sv = load_scales2(a.v_scales, row);
    } else {
        r.kf[0] = r.kf[1] = r.kf[2] = r.kf[3] = 0u;
        r.vf[0] = r.vf[1] = r.vf[2] = r.vf[3] = 0u;
        r.sk = r.sv = make_float2(0.f, 0.f);
    }
}

constexpr int kStages = 2;                     // code tiles in flight per CTA
constexpr int kTileBytes = kTile * kD / 2;     // 8 KB of codes per tile and cache
constexpr int kAttnDynSmem = kStages * 2 * kTileBytes;
// Value phase layout: each thread takes kValDims dimensions (one piece of
// a token row's codes) of tile_tokens / slots tokens.  16 dimensions (an
// 8-byte piece, 16 accumulators) at G_s = 8 and 16: fewer registers, which
// lets G_s = 16 run 6 CTAs per SM (2-3% faster at G_s = 8 and 16); 32 (a
// 16-byte chunk) at G_s = 32 and 64, 1% faster there.
template <int GS>
constexpr int val_dims() { return GS <= 16 ? 16 : 32; }
static_assert(kAttnThreads * (16 + 1) * 4 <= kAttnDynSmem && kAttnThreads * (32 + 1) * 4 <= kAttnDynSmem,
              "slot reduction fits the code ring");

// Resident CTAs per SM the register allocation is bounded for: more warps
// cover the memory latency.  5 (at most 102 registers, no spills) measured
// 8-10% faster than the unbounded 120-register build.  At G_s = 16 and 32
// the shared memory of 6 CTAs fits and the kernel compiles to at most 80
// registers without spills (G_s = 16 with the 16-dimension value layout):
// 3-4% faster; at G_s = 8 shared memory allows only 5.
template <int GS>
constexpr int attn_min_ctas() { return GS == 16 || GS == 32 ? 6 : 5; }

template <int GS>
__global__ void __launch_bounds__(kAttnThreads, attn_min_ctas<GS>()) attn_decode_kernel(const __grid_constant__ AttnArgs a)
{
    griddep_wait();
    constexpr int S = kD / GS;            // subgroups per row
    constexpr int kWordsPerSub = GS / 8;  // code words per subgroup
    extern __shared__ __align__(128) uint8_t s_ring[];  // [kStages][K, V][kTileBytes]
    __shared__ float s_pf[S][kPfStride];  // p_t s_v 2^FLAG per value subgroup and token
    __shared__ __align__(16) uint32_t s_q[2 * kWords];  // the query's decoded values (even, odd codes)
    __shared__ float s_wmax[kAttnThreads / 32];
    __shared__ float s_wsum[kAttnThreads / 32];

    const int tid = threadIdx.x;
    const int split = blockIdx.x;
    const int64_t bh = blockIdx.y;
    const int t_begin = split * a.chunk;
    const int t_end = min(t_begin + a.chunk, a.L);
    const int n_tiles = (t_end - t_begin + kTile - 1) / kTile;
    const uint32_t ring = static_cast<uint32_t>(__cvta_generic_to_shared(s_ring));
    const uint8_t *kbytes = reinterpret_cast<const uint8_t *>(a.k_codes);
    const uint8_t *vbytes = reinterpret_cast<const uint8_t *>(a.v_codes);

    // Copies of tile `it` (both caches) into stage it % kStages; every thread
    // commits one group per call, empty past the last tile.
    auto issue = [&](int it) {
        if (it < n_tiles) {
            const int tile = t_begin + it * kTile;
            const uint32_t kdst = ring + (it % kStages) * 2 * kTileBytes;
            const uint32_t vdst = kdst + kTileBytes;
#pragma unroll
            for (int k = 0; k < kTileBytes / 16 / kAttnThreads; ++k) {
                const int ci = tid + k * kAttnThreads;
                const int r = ci >> 2, c = ci & 3;
                if (tile + r < t_end) {
                    const int64_t src = (bh * a.L_max + tile + r) * (kD / 2) + c * 16;
                    cp_async16(kdst + tile_off(r, c), kbytes + src);
                    cp_async16(vdst + tile_off(r, c), vbytes + src);
                }
            }
        }
        cp_async_commit();
    };
#pragma unroll
    for (int it = 0; it < kStages - 1; ++it) issue(it);

    // ---- the query's decoded values, as int8 (even codes, odd codes) -------
    // decoded once per CTA by the first 16 threads (one code word each)
    if (tid < kWords) {
        uint32_t f[4];
        load_row_flags<GS>(a.q_flags, bh, a.q_packed != 0, f);
        const uint32_t word = a.q_codes[bh * kWords + tid];
        const int F = row_flag(f, tid / kWordsPerSub, a.q_packed != 0);
        uint32_t e = 0u, o = 0u;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int c0 = static_cast<int>(word << (28 - 8 * b)) >> 28;  // code 2b
            const int c1 = static_cast<int>(word << (24 - 8 * b)) >> 28;  // code 2b + 1
            e |= (static_cast<uint32_t>(c0 * (1 << F)) & 0xFFu) << (8 * b);
            o |= (static_cast<uint32_t>(c1 * (1 << F)) & 0xFFu) << (8 * b);
        }
        s_q[tid] = e;
        s_q[kWords + tid] = o;
    }
    const float2 sq = load_scales2(a.q_scales, bh);
    RowSide cur;
    load_side<GS>(a, bh * a.L_max + t_begin + tid, t_begin + tid < t_end, cur);
    __syncthreads();
    const uint32_t sq_addr = static_cast<uint32_t>(__cvta_generic_to_shared(s_q));

    constexpr int kValDims = val_dims<GS>();          // value phase: dimensions per thread
    constexpr int kPieces = kD / kValDims;             // code pieces per token row
    constexpr int kSlots = kAttnThreads / kPieces;     // token slots
    constexpr int kWordsPerPiece = kValDims / 8;       // 32-bit code words per piece
    const int vc = tid % kPieces;   // value phase: code piece (dims kValDims vc ..)
    const int slot = tid / kPieces; // value phase: token slot
    float acc[kValDims];
#pragma unroll
    for (int k = 0; k < kValDims; ++k) acc[k] = 0.f;
    float m_run = -INFINITY;  // running maximum (log2 domain)
    float l_thr = 0.f;        // this thread's share of the running sum

    for (int it = 0; it < n_tiles; ++it) {
        const int tile = t_begin + it * kTile;
        issue(it + kStages - 1);     // into the stage tile it - 1 used
        cp_async_wait<kStages - 1>();  // this thread's copies of tile `it` have landed
        __syncthreads();     // ... and everyone else's
        const uint32_t kst = ring + (it % kStages) * 2 * kTileBytes;
        const uint32_t vst = kst + kTileBytes;
        // FLAGs and scales of the next tile, while this one is processed
        RowSide nxt;
        load_side<GS>(a, bh * a.L_max + tile + kTile + tid, tile + kTile + tid < t_end, nxt);

        // ---- keys: one token per thread -----------------------------------
        const bool valid = tile + tid < t_end;
        float s2 = -INFINITY;
        if (valid) {
            uint32_t kw[kWords], qe[kWords], qo[kWords];  // the query words: broadcast shared loads
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const uint4 v = lds_u4(kst + tile_off(tid, c));
                kw[4 * c] = v.x, kw[4 * c + 1] = v.y, kw[4 * c + 2] = v.z, kw[4 * c + 3] = v.w;
                const uint4 e = lds_u4(sq_addr + 16 * c);
                qe[4 * c] = e.x, qe[4 * c + 1] = e.y, qe[4 * c + 2] = e.z, qe[4 * c + 3] = e.w;
                const uint4 o = lds_u4(sq_addr + 4 * kWords + 16 * c);
                qo[4 * c] = o.x, qo[4 * c + 1] = o.y, qo[4 * c + 2] = o.z, qo[4 * c + 3] = o.w;
            }
            int P[2] = {0, 0};
#pragma unroll
            for (int j = 0; j < S; ++j) {
                int dot = 0;  // 16 x the code dot product of subgroup j
#pragma unroll
                for (int w = j * kWordsPerSub; w < (j + 1) * kWordsPerSub; ++w) {
                    dot = __dp4a(static_cast<int>(qe[w]), static_cast<int>((kw[w] << 4) & 0xF0F0F0F0u), dot);
                    dot = __dp4a(static_cast<int>(qo[w]), static_cast<int>(kw[w] & 0xF0F0F0F0u), dot);
                }
                P[(j * GS) / 64] += (dot >> 4) * (1 << row_flag(cur.kf, j, a.k_packed != 0));
            }
            const float sc = __fmul_rn(__fmul_rn(sq.x, cur.sk.x), static_cast<float>(P[0])) +
                             __fmul_rn(__fmul_rn(sq.y, cur.sk.y), static_cast<float>(P[1]));
            s2 = sc * a.scale_log2;
        }

        // ---- softmax: tile maximum, rescale, weights ----------------------
        float wm = s2;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
        if ((tid & 31) == 0) s_wmax[tid >> 5] = wm;
        __syncthreads();
        float tmax = s_wmax[0];
#pragma unroll
        for (int w = 1; w < kAttnThreads / 32; ++w) tmax = fmaxf(tmax, s_wmax[w]);
        const float m_new = fmaxf(m_run, tmax);
        const float alpha = exp2f(m_run - m_new);  // 0 on the first tile
        const float p = valid ? exp2f(s2 - m_new) : 0.f;
        l_thr = l_thr * alpha + p;
#pragma unroll
        for (int j = 0; j < S; ++j)  // p_t s_v 2^FLAG of every value subgroup (0 past the end)
            s_pf[j][tid] = p * scale_pow2((j * GS) / 64 ? cur.sv.y : cur.sv.x, row_flag(cur.vf, j, a.v_packed != 0));
        if (m_new != m_run) {  // CTA-uniform: rescale only when the maximum grew
#pragma unroll
            for (int k = 0; k < kValDims; ++k) acc[k] *= alpha;
        }
        m_run = m_new;
        __syncthreads();

        // ---- values: o += p_t s_v 2^FLAG c_t -------------------------------
#pragma unroll
        for (int i = 0; i < kTile / kSlots; ++i) {
            const int ti = slot + i * kSlots;
            uint32_t words[kWordsPerPiece];
            if constexpr (kWordsPerPiece == 4) {
                const uint4 ch = lds_u4(vst + tile_off(ti, vc));
                words[0] = ch.x, words[1] = ch.y, words[2] = ch.z, words[3] = ch.w;
            } else {
                asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(words[0]), "=r"(words[1])
                             : "r"(vst + tile_off(ti, vc >> 1) + 8 * (vc & 1)));
            }
#pragma unroll
            for (int w = 0; w < kWordsPerPiece; ++w) {
                // word kWordsPerPiece vc + w of the row; its subgroup's factor (0 past the end)
                const int sub = (kWordsPerPiece * vc + w) / kWordsPerSub;
                const float pf = s_pf[sub][ti];
                const uint32_t ev = (words[w] & 0x0F0F0F0Fu) ^ 0x08080808u;         // codes 0, 2, 4, 6 as c + 8
                const uint32_t od = ((words[w] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;  // codes 1, 3, 5, 7
#pragma unroll
                for (int b = 0; b < 4; ++b)
                    fma_codes2(acc[8 * w + 2 * b], acc[8 * w + 2 * b + 1], pf, magic_float(ev, 0x7440u | b),
                               magic_float(od, 0x7440u | b));
            }
        }
        cur = nxt;
        __syncthreads();  // s_pf and this stage are rewritten later
    }
    cp_async_wait<0>();

    // ---- reduce over token slots, write this split's partial result -------
    // (the code ring is free now: thread (slot, vc) stores its kValDims sums
    // at (kPieces slot + vc) * (kValDims + 1), which keeps both the stores and
    // the column reads below free of bank conflicts)
    __syncthreads();
    float *s_red = reinterpret_cast<float *>(s_ring);
#pragma unroll
    for (int k = 0; k < kValDims; ++k) s_red[(slot * kPieces + vc) * (kValDims + 1) + k] = acc[k];
    float ws = l_thr;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ws += __shfl_xor_sync(0xffffffffu, ws, o);
    if ((tid & 31) == 0) s_wsum[tid >> 5] = ws;
    __syncthreads();
    float od = 0.f;
#pragma unroll 8
    for (int sl = 0; sl < kSlots; ++sl)
        od += s_red[(sl * kPieces + tid / kValDims) * (kValDims + 1) + (tid % kValDims)];
    float *part = a.part + (bh * a.n_split + split) * kPartStride;
    part[tid] = od;
    if (tid == 0) {
        float l = 0.f;
#pragma unroll
        for (int w = 0; w < kAttnThreads / 32; ++w) l += s_wsum[w];
        part[kD] = m_run;
        part[kD + 1] = l;
    }
}

template <int OUT>
__global__ void __launch_bounds__(kD) attn_combine_kernel(const float *__restrict__ part, int n_split, void *out)
{
    griddep_wait();
    const int64_t bh = blockIdx.x;
    const int d = threadIdx.x;
    const float *p = part + bh * n_split * kPartStride;
    float M = -INFINITY;
    for (int s = 0; s < n_split; ++s) M = fmaxf(M, p[s * kPartStride + kD]);
    float num = 0.f, den = 0.f;
    for (int s = 0; s < n_split; ++s) {
        const float w = exp2f(p[s * kPartStride + kD] - M);  // 0 for an empty split
        num = fmaf(w, p[s * kPartStride + d], num);
        den = fmaf(w, p[s * kPartStride + kD + 1], den);
    }
    const float v = num / den;
    const int64_t off = bh * kD + d;
    if (OUT == QUARTZ_OUT_F16) static_cast<__half *>(out)[off] = __float2half_rn(v);
    else if (OUT == QUARTZ_OUT_BF16) static_cast<__nv_bfloat16 *>(out)[off] = __float2bfloat16_rn(v);
    else static_cast<float *>(out)[off] = v;
}

// Splits of the L axis per head: chunks of about kSplitTiles tiles (1024
// tokens), and at least as many CTAs as fit the GPU at once.  Measured on the
// Table 6 settings against 1, 2, 3, 6, 8 and 16 splits and a wave-count
// model, this was the best or within 2% everywhere.
constexpr int64_t kSplitTiles = 8;
int attn_splits(int64_t BH, int64_t L, int64_t slots, int *chunk)
{
    const int64_t tiles = (L + kTile - 1) / kTile;
    int64_t n = (tiles + kSplitTiles - 1) / kSplitTiles;
    const int64_t fill = (slots + BH - 1) / BH;
    if (n < fill) n = fill;
    if (n > tiles) n = tiles;
    if (n > kMaxSplits) n = kMaxSplits;
    const int64_t per = (tiles + n - 1) / n;  // tiles per split
    *chunk = static_cast<int>(per * kTile);
    return static_cast<int>((tiles + per - 1) / per);
}

template <int GS>
cudaError_t launch_decode(int64_t BH, AttnArgs &a, cudaStream_t s)
{
    // resident CTAs per SM of this instance, looked up on first use (any
    // host thread; they all store the same value)
    static std::atomic<int> occ_cache{0};
    cudaError_t e = cudaFuncSetAttribute(attn_decode_kernel<GS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kAttnDynSmem);
    if (e != cudaSuccess) return e;
    int occ = occ_cache.load(std::memory_order_relaxed);
    if (occ == 0) {
        int n = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attn_decode_kernel<GS>, kAttnThreads, kAttnDynSmem);
        if (e != cudaSuccess) return e;
        occ = n > 0 ? n : 1;
        occ_cache.store(occ, std::memory_order_relaxed);
    }
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
    a.n_split = attn_splits(BH, a.L, static_cast<int64_t>(sms) * occ, &a.chunk);
    const dim3 grid(static_cast<unsigned>(a.n_split), static_cast<unsigned>(BH));
    launch_pdl(attn_decode_kernel<GS>, dim3(grid), dim3(kAttnThreads), kAttnDynSmem, s, a);
    return cudaGetLastError();
}

}  // namespace

size_t attention_workspace_bytes(int64_t BH, int64_t L)
{
    const int64_t tiles = (L + kTile - 1) / kTile;
    const int64_t splits = tiles < kMaxSplits ? tiles : kMaxSplits;
    return static_cast<size_t>(BH * splits * kPartStride) * sizeof(float);
}

cudaError_t launch_attention_decode(const quartz_encoded_t *q, const quartz_encoded_t *k, const quartz_encoded_t *v,
                                    int64_t L_max, int64_t L, float scale, void *o, int o_type, void *workspace,
                                    cudaStream_t s)
{
    const int64_t BH = q->rows;
    if (BH == 0) return cudaSuccess;
    AttnArgs a;
    a.q_codes = reinterpret_cast<const uint32_t *>(q->codes);
    a.q_flags = q->flags;
    a.q_scales = reinterpret_cast<const __half *>(q->scales);
    a.k_codes = reinterpret_cast<const uint32_t *>(k->codes);
    a.k_flags = k->flags;
    a.k_scales = reinterpret_cast<const __half *>(k->scales);
    a.v_codes = reinterpret_cast<const uint32_t *>(v->codes);
    a.v_flags = v->flags;
    a.v_scales = reinterpret_cast<const __half *>(v->scales);
    a.q_packed = q->p.flag_bits == 4;
    a.k_packed = k->p.flag_bits == 4;
    a.v_packed = v->p.flag_bits == 4;
    a.L_max = L_max;
    a.L = static_cast<int>(L);
    a.scale_log2 = scale * kLog2e;
    a.part = static_cast<float *>(workspace);
    cudaError_t e;
    switch (q->p.group_s) {
        case 8: e = launch_decode<8>(BH, a, s); break;
        case 16: e = launch_decode<16>(BH, a, s); break;
        case 32: e = launch_decode<32>(BH, a, s); break;
        default: e = launch_decode<64>(BH, a, s); break;
    }
    if (e != cudaSuccess) return e;
    const unsigned cb = static_cast<unsigned>(BH);
    if (o_type == QUARTZ_OUT_F16) launch_pdl(attn_combine_kernel<QUARTZ_OUT_F16>, dim3(cb), dim3(kD), 0, s, a.part, a.n_split, o);
    else if (o_type == QUARTZ_OUT_BF16) launch_pdl(attn_combine_kernel<QUARTZ_OUT_BF16>, dim3(cb), dim3(kD), 0, s, a.part, a.n_split, o);
    else launch_pdl(attn_combine_kernel<QUARTZ_OUT_F32>, dim3(cb), dim3(kD), 0, s, a.part, a.n_split, o);
    return cudaGetLastError();
}

}  // namespace quartz
