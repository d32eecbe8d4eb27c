// QuaRTZ W4A4 linear layer for sm_103a (Section 4.4; Appendix C scales).
//
// Pipeline of one quartz_linear call:
//   1. expand: the packed 4-bit codes and per-subgroup FLAGs of both operands
//      are decoded to v = sgn(c)(|c| << FLAG) and written as FP8 E4M3 (exact:
//      every decoded value is |c| <= 7 times a power of two up to 2^4, i.e.
//      at most 3 significant bits and |v| <= 112, inside E4M3's 4-bit
//      significand and 448 range), together with the group scales (and
//      zero-point side values) transposed to [G][rows] fp32 for contiguous
//      per-group access.  This pass is HBM-bound and touches each operand
//      element once, instead of once per output tile that reads it.
//   2. GEMM: a persistent warp-specialised tcgen05 kernel.  One TMA warp
//      streams 128x64 A and 256x64 W tiles (one 64-wide quantization group
//      per stage, 64-byte swizzle) into an 8-stage shared-memory ring and
//      each group's scales into a ring of its own; one thread issues
//      kind::f8f6f4 MMAs into a fresh fp32 TMEM accumulator for every group
//      (double-buffered, 2 x 256 columns), so each accumulator holds exactly
//      P_g = sum_{k in g} v_a v_w; sixteen epilogue warps read P_g with
//      tcgen05.ld and fold it into the register-resident output as
//      y += s_a * (s_w * P_g) with packed f32x2 arithmetic.
//
// Exactness of P_g: the products v_a * v_w are integers of magnitude at most
// 112^2 = 12544 and every partial sum over a group is an integer of
// magnitude at most 64 * 12544 < 2^20, all exactly representable in the fp32
// accumulator, so the tensor-core sum equals the integer sum.  (sm_103a has
// no integer tcgen05 MMA kind; this is why the integer GEMM runs on the
// floating-point pipe.)
//
// 16-bit stage-1 codes (Section 5 LLM variant): decoded values reach
// 7 * 2^12 and are expanded to E5M2 instead (exact, see lzs_e4m3.cuh).
// Each product is still exact, but a group sum can need more than fp32's 24
// significant bits (products from 2^0 to 49 * 2^24), so P_g is the fp32
// tensor-core sum of exact products rather than the exact integer; the
// accumulator-shift GEMM below is the exact path for those operands.
#include <cuda.h>
#include <cuda_fp16.h>
#include <atomic>
#include <type_traits>
#include <cuda_bf16.h>
#include <cuda_fp8.h>

#include "lzs_e4m3.cuh"
#include "ptx.cuh"
#include "quartz_internal.h"

namespace quartz {
namespace {

constexpr int kGroupQ = 64;

// ---------------------------------------------------------------------------
// 1. expand
// ---------------------------------------------------------------------------
// Row order of the expanded weight operand: inside every block of 16 rows,
// W row 4a + b is stored at position 4b + a (a 4x4 transposition; the map is
// its own inverse).  The GEMM's TMEM column j then holds output column
// perm16(j), which makes the four TMEM columns a thread reads with the
// 16x128b shape four consecutive output columns.
__host__ __device__ __forceinline__ int64_t perm16(int64_t r)
{
    return (r & ~int64_t(15)) | ((r & 3) << 2) | ((r >> 2) & 3);
}

// One launch prepares both GEMM operands (jobs selected by block index):
//   expand A, expand W: 16 codes per thread (8 bytes in, 16 E4M3 bytes out);
//     the weight operand is row-permuted (perm16) and zero-padded to a
//     multiple of 16 rows;
//   side A, side W: side[0][g][.] = s[r, g]; asymmetric adds side[1] = z and
//     side[2] = (is_a ? 64 z - gsum : gsum), so that the epilogue's integer
//     correction is P + z_w * (64 z_a - A_g) - z_a * W_g.  Rows in
//     [rows, rows_pad) are 0; weight rows are stored in natural order,
//     activation rows at perm32(r).  One thread per row and 8 groups: its
//     reads stay in L1 lines, consecutive threads write consecutive rows.
struct ExpandJob {
    const uint2 *codes;          // [rows, K/16] units of 16 codes
    const uint8_t *flags;        // [rows, K/G_s]
    uint4 *out;                  // [rows_out, K/16] units of 16 E4M3 values
    int64_t units, units_pad, units_per_row;
    int permute;
    int packed_flags;            // FLAGs two per byte
};
struct SideJob {
    const __half *scales;
    const int8_t *zeros;
    const int32_t *gsum;
    float *side;
    int64_t rows, rows_pad;
    int is_a;
};
struct PrepArgs {
    ExpandJob ex_a, ex_w;
    SideJob sd_a, sd_w;
    int64_t block_end[4];        // cumulative block counts: expand A, expand W, side A, side W
    int G, nside;
};
constexpr int kPrepThreads = 256;
constexpr int kSideGroupsPerThread = 8;

// kExpandPairs pairs of units per thread, a block apart (every load and
// store instruction of a warp is contiguous), one 16-byte code load per
// pair; all loads are issued before any decode so that several are in
// flight per thread (measured against 1, 4 and 8 single units and 1 and 4
// pairs per thread, and a grid-stride loop: 1.2-1.25x faster than 4 single
// units, the next best).
constexpr int kExpandPairs = 2;

template <int GS>
__device__ __forceinline__ void load_unit_flags(const ExpandJob &j, int64_t u, int &f0, int &f1)
{
    if (GS == 8) {
        if (j.packed_flags) {
            const uint32_t ff = j.flags[u];
            f0 = static_cast<int>(ff & 0xFu);
            f1 = static_cast<int>(ff >> 4);
        } else {
            const uint32_t ff = reinterpret_cast<const uint16_t *>(j.flags)[u];
            f0 = static_cast<int>(ff & 0xFFu);
            f1 = static_cast<int>(ff >> 8);
        }
    } else {
        f0 = f1 = load_flag(j.flags, (u * 16) / GS, j.packed_flags != 0);
    }
}

template <int GS, bool WIDE>
__device__ __forceinline__ void decode_unit(uint2 c, int f0, int f1, uint4 &o)
{
    if (WIDE) {
        e5m2_from_codes8(c.x, f0, o.x, o.y);
        e5m2_from_codes8(c.y, f1, o.z, o.w);
    } else {
        e4m3_from_codes8(c.x, f0, o.x, o.y);
        e4m3_from_codes8(c.y, f1, o.z, o.w);
    }
}

// kExpandPairs pairs of units per thread (one 16-byte code load per pair),
// a block apart; units and units_pad are multiples of 4 (K % 64 == 0), so a
// pair never straddles a row or the end.
template <int GS, bool WIDE>
__device__ __forceinline__ void run_expand(const ExpandJob &j, int64_t p0)
{
    uint4 c[kExpandPairs];
    int f[kExpandPairs][4];
#pragma unroll
    for (int q = 0; q < kExpandPairs; ++q) {
        const int64_t u = 2 * (p0 + q * kPrepThreads);
        c[q] = make_uint4(0u, 0u, 0u, 0u);
        f[q][0] = f[q][1] = f[q][2] = f[q][3] = 0;
        if (u < j.units) {
            c[q] = __ldcs(reinterpret_cast<const uint4 *>(j.codes) + (u >> 1));
            load_unit_flags<GS>(j, u, f[q][0], f[q][1]);
            load_unit_flags<GS>(j, u + 1, f[q][2], f[q][3]);
        }
    }
#pragma unroll
    for (int q = 0; q < kExpandPairs; ++q) {
        const int64_t u = 2 * (p0 + q * kPrepThreads);
        if (u >= j.units_pad) continue;
        int64_t dst = u;
        if (j.permute) {
            int64_t r;  // the row (32-bit division wherever the units fit)
            if (j.units_pad <= 0xFFFFFFFFll)
                r = static_cast<uint32_t>(u) / static_cast<uint32_t>(j.units_per_row);
            else
                r = u / j.units_per_row;
            dst = perm16(r) * j.units_per_row + (u - r * j.units_per_row);
        }
        uint4 o0 = make_uint4(0u, 0u, 0u, 0u), o1 = o0;  // padding rows stay zero
        if (u < j.units) {
            decode_unit<GS, WIDE>(make_uint2(c[q].x, c[q].y), f[q][0], f[q][1], o0);
            decode_unit<GS, WIDE>(make_uint2(c[q].z, c[q].w), f[q][2], f[q][3], o1);
        }
        j.out[dst] = o0;
        j.out[dst + 1] = o1;
    }
}

__device__ __forceinline__ void run_side(const SideJob &j, int64_t t, int G, int nside)
{
    const int64_t r = t % j.rows_pad;
    const int g0 = static_cast<int>(t / j.rows_pad) * kSideGroupsPerThread;
    if (g0 >= G) return;
    const int g1 = min(g0 + kSideGroupsPerThread, G);
    const int64_t total = j.rows_pad * G;
    const int64_t o = j.is_a ? perm32(r) : r;
    const bool in = r < j.rows;
    for (int g = g0; g < g1; ++g) {
        const int64_t i = static_cast<int64_t>(g) * j.rows_pad + o;
        j.side[i] = in ? __half2float(j.scales[r * G + g]) : 0.f;
        if (nside > 1) {
            const float z = in ? static_cast<float>(j.zeros[r * G + g]) : 0.f;
            const float gs = in ? static_cast<float>(j.gsum[r * G + g]) : 0.f;
            j.side[total + i] = z;
            j.side[2 * total + i] = j.is_a ? (static_cast<float>(kGroupQ) * z - gs) : gs;
        }
    }
}

template <int GS, bool WIDE>
__global__ void __launch_bounds__(kPrepThreads) prep_kernel(const __grid_constant__ PrepArgs args)
{
    griddep_wait();
    const int64_t bid = blockIdx.x;
    if (bid < args.block_end[0]) {
        run_expand<GS, WIDE>(args.ex_a, bid * (kPrepThreads * kExpandPairs) + threadIdx.x);
    } else if (bid < args.block_end[1]) {
        run_expand<GS, WIDE>(args.ex_w, (bid - args.block_end[0]) * (kPrepThreads * kExpandPairs) + threadIdx.x);
    } else if (bid < args.block_end[2]) {
        run_side(args.sd_a, (bid - args.block_end[1]) * kPrepThreads + threadIdx.x, args.G, args.nside);
    } else {
        run_side(args.sd_w, (bid - args.block_end[2]) * kPrepThreads + threadIdx.x, args.G, args.nside);
    }
}

// ---------------------------------------------------------------------------
// 2. tcgen05 GEMM
// ---------------------------------------------------------------------------
constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = kGroupQ;
constexpr int kStages = 8;
constexpr int kABytes = BM * BK;      // E4M3 operands: one byte per element
constexpr int kBBytes = BN * BK;
constexpr int kStageBytes = kABytes + kBBytes;
// Warpgroups 0-3 dequantise (16 warps: four per 32-lane TMEM quarter, 64
// columns each); warpgroup 4 holds the operand TMA producer, the MMA issuer,
// the scale copier and one idle warp.  The dequant epilogue is the
// throughput-critical part (two fp32 operations per output element per
// group), so it gets four warps per scheduler; the three control roles sit on
// three different schedulers (warp w runs on scheduler w % 4) because each
// slows the epilogue warps that share its scheduler.
constexpr int kEpiWarps = 16;
constexpr int kThreads = (kEpiWarps + 4) * 32;
constexpr int kProducerWarp = kEpiWarps;
constexpr int kMmaWarp = kEpiWarps + 1;
constexpr int kSideWarp = kEpiWarps + 2;
constexpr int kColsPerWarp = BN / 4;
// Register split (setmaxnreg): 640 threads launch with 96 registers each;
// warpgroup 4 drops to 32 so the epilogue warpgroups can hold 112
// (512*112 + 128*32 = 61440 = 640*96).
constexpr uint32_t kRegsLaunch = 96;
constexpr uint32_t kRegsEpilogue = 112;
constexpr uint32_t kRegsControl = 32;
static_assert(kEpiWarps * 32 * kRegsEpilogue + 128 * kRegsControl <= kThreads * kRegsLaunch,
              "register split exceeds the launch allocation");
constexpr uint32_t kTmemCols = 512;   // two fp32 accumulators of 256 columns
constexpr int kRasterM = 8;
constexpr int kRowRasterMaxN = 16;  // see tile_coords
// Per-row scales (group_q = K): the MMA accumulates kPerRowChunk stages (256
// of K) into one TMEM accumulator before the epilogue takes it; each such sum
// is an integer below 256 * 112^2 < 2^22, exact in fp32 and convertible with
// the 1.5 * 2^23 rounding addend, and the epilogue adds it to an int32.
constexpr int kPerRowChunk = 4;           // tiles are visited in bands of 8 M-tiles

struct GemmArgs {
    const float *a_side;  // [nside][G][m_pad]
    const float *w_side;  // [nside][G][n_pad]
    int64_t m_pad, n_pad;
    int M, N, G;
    int tiles_m, tiles_n, num_tiles;
    int raster_m;         // M-tiles per band of the visiting order: kRasterM or 1 (see tile_coords)
    const __half *bias;
    void *y;
    int y_type;
    int32_t *partials;
    int partials_group;
    int *dev_err;
    int per_row;          // scales per row (group_q = K) rather than per 64-group
    int wide;             // E5M2 operands (16-bit stage-1 codes) instead of E4M3
    // Split last wave: the first full_tiles tiles go round robin over the CTAs
    // (the same count each); each of the remaining tail_tiles is cut along K
    // into `split` group ranges taken by CTAs 0 .. tail_tiles * split - 1,
    // which leave fp32 partial tiles in tail_part; tail_combine_kernel adds
    // them in part order and writes the outputs.  Range forms (ls > 0): the
    // last tail_tiles tiles' tail_tiles * G group iterations (after at least
    // one wave of whole tiles, or every tile's when more than half but not
    // all of the SMs hold one) are cut into one contiguous range of ls per
    // CTA, one CTA per SM; a tile met by r ranges leaves parts 0 .. r - 1 in
    // group order (r <= 2 after whole tiles, where ls >= G; r <= 3 otherwise,
    // where ls >= G / 2), a tile inside one range is stored whole.
    int full_tiles, tail_tiles, split;
    int ls;
    float *tail_part;     // [tail_tiles][split][16][kEpiWarps * 32] float4 (fp32 pairs)
};

// Shared memory: the operand stages, then a ring of side-value slots (one
// group's NSIDE x BM activation and NSIDE x BN weight values each, copied by
// the producer and released by the epilogue), then the mbarriers.
template <int NSIDE>
struct Smem {
    static constexpr int kOperands = 0;
    static constexpr int kSide = kStages * kStageBytes;
    static constexpr int kSideSlots = NSIDE == 1 ? 8 : 4;
    static constexpr int kSideABytes = NSIDE * BM * 4;
    static constexpr int kSideSlotBytes = NSIDE * (BM + BN) * 4;
    static constexpr int kBars = kSide + kSideSlots * kSideSlotBytes;
    // full, empty, acc_full x2, acc_empty x2, drain, side_full, side_empty
    static constexpr int kNumBars = 2 * kStages + 4 + 1 + 2 * kSideSlots;
    static constexpr int kMisc = kBars + kNumBars * 8;
    static constexpr int kTotal = kMisc + 16;
    static constexpr int kAlloc = kTotal + 1024;  // slack to align the base to 1024 bytes
};

// Tile visiting order: bands of RM M-tiles, N-tiles inside a band (M
// fastest), so the CTAs resident at one time share few A row-blocks and W
// column-blocks and both stay in L2.  RM is kRasterM, or 1 (whole rows of
// tiles, one M-tile after the other) for layers at most kRowRasterMaxN
// tiles wide on the symmetric fast path: there a band of 8 M-tiles holds
// fewer tiles than one wave of CTAs, so the waves would cut bands and read
// an A row-block again in the next wave (measured 2.3x A reads for a
// 12-tile-wide, 192-group layer), while a row keeps each A row-block's
// consumers in one wave and the whole narrow W stays in L2.  RM is a
// template argument of the GEMM (a runtime band size measured 1.4% slower
// on the wide layers); a.raster_m holds it for the combine kernel.
template <int RM>
__device__ __forceinline__ void tile_coords(int tile, const GemmArgs &a, int &mt, int &nt)
{
    const int band = tile / (RM * a.tiles_n);
    const int m0 = band * RM;
    const int gm = min(RM, a.tiles_m - m0);
    const int r = tile - band * RM * a.tiles_n;
    mt = m0 + r % gm;
    nt = r / gm;
}

// This CTA's work: whole tiles, then (split last wave) one part of a tail tile.
struct WorkItem {
    int tile, g0, g1;  // tile index and group range [g0, g1)
    int part, tail;    // part of tail tile `tail` (part = -1: a whole tile)
};

__device__ __forceinline__ int work_items(const GemmArgs &a)
{
    const int c = blockIdx.x, P = gridDim.x;
    if (a.split <= 1) return (a.num_tiles - c + P - 1) / P;
    if (a.ls > 0) {  // (tail_tiles * G < 2^30: checked on the host)
        const int nf = a.full_tiles / P;
        const int U = a.tail_tiles * a.G, b = c * a.ls, e = min(b + a.ls, U);
        if (b >= e) return nf;
        return nf + (e - 1) / a.G - b / a.G + 1;
    }
    return a.full_tiles / P + (c < a.tail_tiles * a.split ? 1 : 0);
}

__device__ __forceinline__ WorkItem work_item(const GemmArgs &a, int k)
{
    WorkItem w;
    const int c = blockIdx.x, P = gridDim.x;
    if (a.ls > 0 && k >= a.full_tiles / P) {
        const int U = a.tail_tiles * a.G, b = c * a.ls, e = min(b + a.ls, U);
        const int t = b / a.G + (k - a.full_tiles / P);
        const int t0 = t * a.G;
        w.tile = a.full_tiles + t;
        w.g0 = max(b - t0, 0);
        w.g1 = min(e - t0, a.G);
        if (w.g0 == 0 && w.g1 == a.G) {
            w.part = -1;
            w.tail = 0;
        } else {
            w.part = c - t0 / a.ls;  // ranges before this one that meet the tile
            w.tail = t;
        }
        return w;
    }
    if (a.split <= 1 || k < a.full_tiles / P) {
        w.tile = c + k * P;
        w.g0 = 0;
        w.g1 = a.G;
        w.part = -1;
        w.tail = 0;
    } else {
        w.tail = c / a.split;
        w.part = c - w.tail * a.split;
        w.tile = a.full_tiles + w.tail;
        w.g0 = w.part * a.G / a.split;
        w.g1 = (w.part + 1) * a.G / a.split;
    }
    return w;
}

// (a.x, a.y) += (b.x, b.y) on a packed fp32 pair.
__device__ __forceinline__ void add2_rn(uint64_t &a, uint64_t b)
{
    asm("add.rn.f32x2 %0, %0, %1;" : "+l"(a) : "l"(b));
}

template <int OUT>
__device__ __forceinline__ void store_quad(void *y, int64_t off, float4 v)
{
    if (OUT == QUARTZ_OUT_F16) {
        const __half2 a = __floats2half2_rn(v.x, v.y), b = __floats2half2_rn(v.z, v.w);
        *reinterpret_cast<uint2 *>(static_cast<__half *>(y) + off) =
            make_uint2(*reinterpret_cast<const uint32_t *>(&a), *reinterpret_cast<const uint32_t *>(&b));
    } else if (OUT == QUARTZ_OUT_BF16) {
        const __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
        *reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(y) + off) =
            make_uint2(*reinterpret_cast<const uint32_t *>(&a), *reinterpret_cast<const uint32_t *>(&b));
    } else {
        *reinterpret_cast<float4 *>(static_cast<float *>(y) + off) = v;
    }
}

// v + bias[n .. n + 3] in fp32 (no bias: v).
__device__ __forceinline__ float4 add_bias4(const GemmArgs &args, int64_t n, float4 v)
{
    if (args.bias) {
        const uint2 braw = __ldg(reinterpret_cast<const uint2 *>(args.bias + n));
        const float2 b0 = __half22float2(*reinterpret_cast<const __half2 *>(&braw.x));
        const float2 b1 = __half22float2(*reinterpret_cast<const __half2 *>(&braw.y));
        v.x = __fadd_rn(v.x, b0.x);
        v.y = __fadd_rn(v.y, b0.y);
        v.z = __fadd_rn(v.z, b1.x);
        v.w = __fadd_rn(v.w, b1.y);
    }
    return v;
}

// Output of one 128 x 256 tile from the symmetric epilogue's registers:
// acc[c][4h + i] holds output column 16c + tq + i of this warp's slice, rows
// trow + 16h (low half) and trow + 16h + 8 (high half) of its quarter; the
// bias is added in fp32, then one rounding to the output type.
template <int OUT, int RM>
__device__ __forceinline__ void store_tile_sym(const GemmArgs &args, int tile, int quarter, int slot, int trow,
                                               int tq, const uint64_t (&acc)[4][8])
{
    int mt, nt;
    tile_coords<RM>(tile, args, mt, nt);
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int64_t m = static_cast<int64_t>(mt) * BM + quarter * 32 + 16 * h + 8 * e + trow;
            if (m >= args.M) continue;
#pragma unroll
            for (int chunk = 0; chunk < 4; ++chunk) {
                const int64_t n = static_cast<int64_t>(nt) * BN + slot * kColsPerWarp + 16 * chunk + tq;
                if (n >= args.N) continue;
                float vv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const uint64_t q = acc[chunk][4 * h + i];
                    vv[i] = __uint_as_float(static_cast<uint32_t>(e ? (q >> 32) : q));
                }
                store_quad<OUT>(args.y, m * args.N + n, add_bias4(args, n, make_float4(vv[0], vv[1], vv[2], vv[3])));
            }
        }
}

// Half of one 16-column chunk: one 16x128b.x4 TMEM load (16 lanes), then
// acc[i] += s_a * (s_w[i] * P_i) for the four pairs P_i = (row, row + 8) of
// column i, on explicit 64-bit register pairs (q: the loaded pairs, s: the
// column scale duplicated into both halves, t: s_w * P).
__device__ __forceinline__ void epi_half_chunk_sym(uint32_t taddr, float4 sw, uint64_t sa, uint64_t *acc)
{
    asm volatile(
        "{\n\t"
        ".reg .b32 p<8>;\n\t"
        ".reg .b64 q<4>, t<4>, s<4>;\n\t"
        "tcgen05.ld.sync.aligned.16x128b.x4.b32 {p0, p1, p2, p3, p4, p5, p6, p7}, [%4];\n\t"
        "tcgen05.wait::ld.sync.aligned;\n\t"
        "mov.b64 q0, {p0, p1};\n\t"
        "mov.b64 q1, {p2, p3};\n\t"
        "mov.b64 q2, {p4, p5};\n\t"
        "mov.b64 q3, {p6, p7};\n\t"
        "mov.b64 s0, {%5, %5};\n\t"
        "mov.b64 s1, {%6, %6};\n\t"
        "mov.b64 s2, {%7, %7};\n\t"
        "mov.b64 s3, {%8, %8};\n\t"
        "mul.rn.f32x2 t0, q0, s0;\n\t"
        "fma.rn.f32x2 %0, t0, %9, %0;\n\t"
        "mul.rn.f32x2 t1, q1, s1;\n\t"
        "fma.rn.f32x2 %1, t1, %9, %1;\n\t"
        "mul.rn.f32x2 t2, q2, s2;\n\t"
        "fma.rn.f32x2 %2, t2, %9, %2;\n\t"
        "mul.rn.f32x2 t3, q3, s3;\n\t"
        "fma.rn.f32x2 %3, t3, %9, %3;\n\t"
        "}"
        : "+l"(acc[0]), "+l"(acc[1]), "+l"(acc[2]), "+l"(acc[3])
        : "r"(taddr), "f"(sw.x), "f"(sw.y), "f"(sw.z), "f"(sw.w), "l"(sa)
        : "memory");
}

// Per-row-scale epilogue step for half of one 16-column chunk: one
// 16x128b.x4 TMEM load of an accumulator whose values are exact integers
// below 2^22, each turned into an int32 with the 1.5 * 2^23 rounding addend
// (the integer is the float's bit pattern minus 0x4B400000) and added to acc.
__device__ __forceinline__ void epi_half_chunk_int(uint32_t taddr, int32_t *acc)
{
    asm volatile(
        "{\n\t"
        ".reg .b32 p<8>;\n\t"
        ".reg .f32 f<8>;\n\t"
        "tcgen05.ld.sync.aligned.16x128b.x4.b32 {p0, p1, p2, p3, p4, p5, p6, p7}, [%8];\n\t"
        "tcgen05.wait::ld.sync.aligned;\n\t"
        "add.rn.f32 f0, p0, 0f4B400000;\n\t"
        "add.rn.f32 f1, p1, 0f4B400000;\n\t"
        "add.rn.f32 f2, p2, 0f4B400000;\n\t"
        "add.rn.f32 f3, p3, 0f4B400000;\n\t"
        "add.rn.f32 f4, p4, 0f4B400000;\n\t"
        "add.rn.f32 f5, p5, 0f4B400000;\n\t"
        "add.rn.f32 f6, p6, 0f4B400000;\n\t"
        "add.rn.f32 f7, p7, 0f4B400000;\n\t"
        "mov.b32 p0, f0;\n\t"
        "mov.b32 p1, f1;\n\t"
        "mov.b32 p2, f2;\n\t"
        "mov.b32 p3, f3;\n\t"
        "mov.b32 p4, f4;\n\t"
        "mov.b32 p5, f5;\n\t"
        "mov.b32 p6, f6;\n\t"
        "mov.b32 p7, f7;\n\t"
        "sub.s32 p0, p0, 0x4B400000;\n\t"
        "sub.s32 p1, p1, 0x4B400000;\n\t"
        "sub.s32 p2, p2, 0x4B400000;\n\t"
        "sub.s32 p3, p3, 0x4B400000;\n\t"
        "sub.s32 p4, p4, 0x4B400000;\n\t"
        "sub.s32 p5, p5, 0x4B400000;\n\t"
        "sub.s32 p6, p6, 0x4B400000;\n\t"
        "sub.s32 p7, p7, 0x4B400000;\n\t"
        "add.s32 %0, %0, p0;\n\t"
        "add.s32 %1, %1, p1;\n\t"
        "add.s32 %2, %2, p2;\n\t"
        "add.s32 %3, %3, p3;\n\t"
        "add.s32 %4, %4, p4;\n\t"
        "add.s32 %5, %5, p5;\n\t"
        "add.s32 %6, %6, p6;\n\t"
        "add.s32 %7, %7, p7;\n\t"
        "}"
        : "+r"(acc[0]), "+r"(acc[1]), "+r"(acc[2]), "+r"(acc[3]), "+r"(acc[4]), "+r"(acc[5]),
          "+r"(acc[6]), "+r"(acc[7])
        : "r"(taddr)
        : "memory");
}

// Two 64-bit words from shared memory (one 16-byte load).
__device__ __forceinline__ void lds_b64x2(uint32_t addr, uint64_t &a, uint64_t &b)
{
    asm volatile("ld.shared.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "r"(addr) : "memory");
}

template <int MODE, int OUT, bool DUMP, bool PERROW, int RM = kRasterM>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tcgen05_kernel(const __grid_constant__ CUtensorMap tmap_a,
                        const __grid_constant__ CUtensorMap tmap_w, const GemmArgs args)
{
    griddep_wait();
    constexpr int NSIDE = (MODE == QUARTZ_ASYMMETRIC) ? 3 : 1;
    using L = Smem<NSIDE>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t smem_base = smem_u32(smem);
    const uint32_t bar_base = smem_base + L::kBars;
    auto full_bar = [&](int s) { return bar_base + 8u * s; };
    auto empty_bar = [&](int s) { return bar_base + 8u * (kStages + s); };
    auto acc_full_bar = [&](int b) { return bar_base + 8u * (2 * kStages + b); };
    auto acc_empty_bar = [&](int b) { return bar_base + 8u * (2 * kStages + 2 + b); };
    const uint32_t drain_bar = bar_base + 8u * (2 * kStages + 4);
    auto side_full_bar = [&](int s) { return bar_base + 8u * (2 * kStages + 5 + s); };
    auto side_empty_bar = [&](int s) { return bar_base + 8u * (2 * kStages + 5 + L::kSideSlots + s); };
    uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(smem + L::kMisc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::kMisc + 4);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(acc_full_bar(b), 1);
            mbar_init(acc_empty_bar(b), kEpiWarps);
        }
        mbar_init(drain_bar, 1);
        for (int s = 0; s < L::kSideSlots; ++s) {
            mbar_init(side_full_bar(s), 1);
            mbar_init(side_empty_bar(s), kEpiWarps);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(smem_u32(tmem_holder), kTmemCols);
        tmem_relinquish();
    }
    if (warp == kProducerWarp && lane == 0) {
        tma_prefetch_desc(&tmap_a);
        tma_prefetch_desc(&tmap_w);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;
    const int G = args.G;

    if (warp >= kEpiWarps) {
      regs_decrease<kRegsControl>();
      if (warp == kProducerWarp) {
        // ------------------------------------------------------------------
        // TMA producer: one stage = one 64-wide group of A (128 rows) and W
        // (256 rows).  Rows past M or N are zero-filled by the tensor map.
        // ------------------------------------------------------------------
        if (lane == 0) {
            int it = 0;  // groups whose operand copies were issued
            bool ok = true;
            const int n_items = work_items(args);
            for (int k = 0; k < n_items && ok; ++k) {
                const WorkItem wi = work_item(args, k);
                int mt, nt;
                tile_coords<RM>(wi.tile, args, mt, nt);
                for (int g = wi.g0; g < wi.g1; ++g, ++it) {
                    const int s = it % kStages;
                    if (it >= kStages &&
                        !mbar_wait_bounded(empty_bar(s), ((it / kStages) - 1) & 1, abort_flag,
                                           args.dev_err, kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = smem_base + L::kOperands + s * kStageBytes;
                    mbar_arrive_expect_tx(full_bar(s), kStageBytes);
                    tma_load_2d(sa, &tmap_a, g * BK, mt * BM, full_bar(s));
                    tma_load_2d(sa + kABytes, &tmap_w, g * BK, nt * BN, full_bar(s));
                }
            }
            // Never leave the CTA with copies in flight: wait for the last
            // load issued into every stage (bounded, even after an abort).
            int zero = 0;
            for (int s = 0; s < kStages && s < it; ++s) {
                const int last = it - 1 - ((it - 1 - s) % kStages);
                mbar_wait_bounded(full_bar(s), (last / kStages) & 1, &zero, args.dev_err, kWaitLimitNs);
            }
        }
        __syncwarp();
      } else if (warp == kSideWarp) {
        // ------------------------------------------------------------------
        // Scale copier: each group's side values (scales; asymmetric also
        // zero-point terms) go by bulk copy into a ring slot that the
        // epilogue frees.
        // ------------------------------------------------------------------
        if (!PERROW && lane == 0) {
            constexpr int S = L::kSideSlots;
            const int64_t a_plane = args.m_pad * G;
            const int64_t w_plane = args.n_pad * G;
            int it = 0;  // groups whose side-value copies were issued
            bool ok = true;
            const int n_items = work_items(args);
            for (int k = 0; k < n_items && ok; ++k) {
                const WorkItem wi = work_item(args, k);
                int mt, nt;
                tile_coords<RM>(wi.tile, args, mt, nt);
                for (int g = wi.g0; g < wi.g1; ++g, ++it) {
                    const int ss = it % S;
                    if (it >= S && !mbar_wait_bounded(side_empty_bar(ss), ((it / S) - 1) & 1, abort_flag,
                                                      args.dev_err, kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    const uint32_t dst = smem_base + L::kSide + ss * L::kSideSlotBytes;
                    mbar_arrive_expect_tx(side_full_bar(ss), L::kSideSlotBytes);
                    const float *src_a = args.a_side + static_cast<int64_t>(g) * args.m_pad + static_cast<int64_t>(mt) * BM;
                    const float *src_w = args.w_side + static_cast<int64_t>(g) * args.n_pad + static_cast<int64_t>(nt) * BN;
#pragma unroll
                    for (int sd = 0; sd < NSIDE; ++sd) {
                        bulk_load(dst + sd * BM * 4, src_a + sd * a_plane, BM * 4, side_full_bar(ss));
                        bulk_load(dst + L::kSideABytes + sd * BN * 4, src_w + sd * w_plane, BN * 4, side_full_bar(ss));
                    }
                }
            }
            int zero = 0;
            for (int s = 0; s < S && s < it; ++s) {
                const int last = it - 1 - ((it - 1 - s) % S);
                mbar_wait_bounded(side_full_bar(s), (last / S) & 1, &zero, args.dev_err, kWaitLimitNs);
            }
        }
        __syncwarp();
      } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------------
        // MMA issuer: 2 x (M=128, N=256, K=32) kind::f8f6f4 MMAs per group into
        // a fresh accumulator (first MMA overwrites), then two commits: one
        // frees the operand stage, one hands P_g to the epilogue.
        // ------------------------------------------------------------------
        if (lane == 0) {
            const uint32_t idesc = args.wide ? idesc_e5m2_f32(BM, BN) : idesc_e4m3_f32(BM, BN);
            int it = 0;
            bool ok = true;
            constexpr int CH = PERROW ? kPerRowChunk : 1;  // stages per TMEM accumulator
            int ic = 0;                                    // accumulators handed to the epilogue
            const int n_items = work_items(args);
            for (int k = 0; k < n_items && ok; ++k) {
                const WorkItem wi = work_item(args, k);
                for (int g = wi.g0; g < wi.g1; ++g, ++it) {
                    const int s = it % kStages;
                    const int b = ic & 1;
                    const bool first = (g % CH) == 0;
                    const bool last = (g % CH) == CH - 1 || g == G - 1;
                    if (!mbar_wait_bounded(full_bar(s), (it / kStages) & 1, abort_flag, args.dev_err,
                                           kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    if (first && ic >= 2 && !mbar_wait_bounded(acc_empty_bar(b), ((ic >> 1) - 1) & 1,
                                                               abort_flag, args.dev_err, kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_base + L::kOperands + s * kStageBytes;
                    const uint32_t d = tmem_base + static_cast<uint32_t>(b * BN);
#pragma unroll
                    for (int kk = 0; kk < BK / 32; ++kk) {
                        const uint64_t adesc = sdesc_k_major_sw64(sa + kk * 32);
                        const uint64_t bdesc = sdesc_k_major_sw64(sa + kABytes + kk * 32);
                        mma_f8_ss(d, adesc, bdesc, idesc, (kk > 0 || !first) ? 1u : 0u);
                    }
                    mma_commit(empty_bar(s));
                    if (last) {
                        mma_commit(acc_full_bar(b));
                        ++ic;
                    }
                }
            }
            // Make sure no MMA is still writing TMEM before it is freed.
            mma_commit(drain_bar);
            int zero = 0;
            mbar_wait_bounded(drain_bar, 0, &zero, args.dev_err, kWaitLimitNs);
        }
        __syncwarp();
      }
    } else {
        regs_increase<kRegsEpilogue>();
        // ------------------------------------------------------------------
        // Epilogue.  Warp w reads TMEM lanes [32*(w%4), +32) (tile rows) and
        // TMEM columns [64*(w/4), +64) with the 16x128b shape: per 16-column
        // chunk, thread t holds TMEM columns t%4 + {0,4,8,12} of lanes t/4 and
        // t/4 + 8 (and t/4 + 16, t/4 + 24 from the second lane half).  With
        // the weight rows transposed inside each 16-row block, those four TMEM
        // columns are the four consecutive output columns 4*(t%4) + {0..3},
        // so one 16-byte shared load gives their scales (each used for four
        // rows) and the stores are 4-wide.  The thread's four row scales are
        // one 16-byte load as well (rows are permuted in the side values).
        // Per group, y += s_a * (s_w * P_g) on (row, row + 8) pairs with
        // f32x2 arithmetic (asymmetric first adds the exact integer
        // zero-point terms to P_g).
        // ------------------------------------------------------------------
        constexpr int S = L::kSideSlots;
        const int quarter = warp & 3;
        const int slot = warp >> 2;
        const int trow = lane >> 2;          // row offset inside each 8-row band
        const int tq = 4 * (lane & 3);       // first of this thread's 4 output columns in a 16-column chunk

        // acc[h][j]: output column 16*(j/4) + tq + j%4 of this warp's slice,
        // rows trow + 16h (.x) and trow + 16h + 8 (.y)
        if constexpr (PERROW) {
            // Per-row scales (group_q = K, symmetric): each TMEM accumulator
            // holds the exact integer sum of kPerRowChunk stages; the epilogue
            // adds it into int32 accumulators and scales once per tile:
            // y = s_a * (s_w * P).  acci[c][4h + i] = rows trow + 16h (i < 4:
            // pairs 2i / 2i + 1 are rows +0 / +8) of column 16c + tq + i%4.
            int32_t acci[4][16];
            int ic = 0;
            bool ok = true;
            const int nchunks = (G + kPerRowChunk - 1) / kPerRowChunk;
            for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int j = 0; j < 16; ++j) acci[c][j] = 0;
                for (int cc = 0; cc < nchunks; ++cc, ++ic) {
                    const int b = ic & 1;
                    if (!mbar_wait_bounded(acc_full_bar(b), (ic >> 1) & 1, abort_flag, args.dev_err,
                                           kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                                           static_cast<uint32_t>(b * BN + slot * kColsPerWarp);
#pragma unroll
                    for (int chunk = 0; chunk < 4; ++chunk) {
                        epi_half_chunk_int(tbase + 16 * chunk, acci[chunk]);
                        epi_half_chunk_int(tbase + (16u << 16) + 16 * chunk, acci[chunk] + 8);
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(acc_empty_bar(b));
                }
                if (!ok) break;
                int mt, nt;
                tile_coords<RM>(tile, args, mt, nt);
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const int64_t m = static_cast<int64_t>(mt) * BM + quarter * 32 + 16 * h + 8 * e + trow;
                        if (m >= args.M) continue;
                        const float s_a = args.a_side[perm32(m)];
#pragma unroll
                        for (int chunk = 0; chunk < 4; ++chunk) {
                            const int64_t n = static_cast<int64_t>(nt) * BN + slot * kColsPerWarp + 16 * chunk + tq;
                            if (n >= args.N) continue;
                            float vv[4];
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const int32_t P = acci[chunk][8 * h + 2 * i + e];
                                if (DUMP) args.partials[m * args.N + n + i] = P;
                                const float t = __fmul_rn(static_cast<float>(P), args.w_side[n + i]);
                                vv[i] = __fmul_rn(t, s_a);
                            }
                            float4 v = make_float4(vv[0], vv[1], vv[2], vv[3]);
                            if (args.bias) {
                                const uint2 braw = __ldg(reinterpret_cast<const uint2 *>(args.bias + n));
                                const float2 b0 = __half22float2(*reinterpret_cast<const __half2 *>(&braw.x));
                                const float2 b1 = __half22float2(*reinterpret_cast<const __half2 *>(&braw.y));
                                v.x = __fadd_rn(v.x, b0.x);
                                v.y = __fadd_rn(v.y, b0.y);
                                v.z = __fadd_rn(v.z, b1.x);
                                v.w = __fadd_rn(v.w, b1.y);
                            }
                            store_quad<OUT>(args.y, m * args.N + n, v);
                        }
                    }
            }
        } else if constexpr (MODE == QUARTZ_SYMMETRIC && !DUMP) {
            // Symmetric fast path: each half chunk (16 lanes x 16 columns: TMEM
            // load, wait and the scale arithmetic) is one PTX block on
            // explicit 64-bit pairs, which keeps the kernel free of spills.
            // acc64[c][4h + i]: output column 16c + tq + i, rows trow + 16h (low) and + 8 (high)
            uint64_t acc64[4][8];
            int it = 0;
            bool ok = true;
            const int n_items = work_items(args);
            for (int k = 0; k < n_items && ok; ++k) {
                const WorkItem wi = work_item(args, k);
#pragma unroll
                for (int c = 0; c < 4; ++c)
#pragma unroll
                    for (int j = 0; j < 8; ++j) acc64[c][j] = 0ull;
                for (int g = wi.g0; g < wi.g1; ++g, ++it) {
                    const int b = it & 1;
                    const int ss = it % S;
                    if (!mbar_wait_bounded(side_full_bar(ss), (it / S) & 1, abort_flag, args.dev_err,
                                           kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    const uint32_t side_a = smem_base + L::kSide + ss * L::kSideSlotBytes + (quarter * 32 + 4 * trow) * 4;
                    const uint32_t side_w = smem_base + L::kSide + ss * L::kSideSlotBytes + L::kSideABytes +
                                            (slot * kColsPerWarp + tq) * 4;
                    if (!mbar_wait_bounded(acc_full_bar(b), (it >> 1) & 1, abort_flag, args.dev_err,
                                           kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    uint64_t sa0, sa1;
                    lds_b64x2(side_a, sa0, sa1);
                    tc_fence_after();
                    const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                                           static_cast<uint32_t>(b * BN + slot * kColsPerWarp);
#pragma unroll
                    for (int chunk = 0; chunk < 4; ++chunk) {
                        const float4 sw = lds_f4(side_w + 16 * chunk * 4);
                        epi_half_chunk_sym(tbase + 16 * chunk, sw, sa0, acc64[chunk]);
                        epi_half_chunk_sym(tbase + (16u << 16) + 16 * chunk, sw, sa1, acc64[chunk] + 4);
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        mbar_arrive(acc_empty_bar(b));
                        mbar_arrive(side_empty_bar(ss));
                    }
                }
                if (!ok) break;
                if (wi.part >= 0) {
                    // split last wave: leave this part's fp32 partial tile for
                    // tail_combine_kernel: slot tail * split + part holds 16
                    // planes of one uint4 per epilogue thread (coalesced)
                    uint4 *dst = reinterpret_cast<uint4 *>(args.tail_part) +
                                 ((wi.tail * args.split + wi.part) * 16 * (kEpiWarps * 32) + warp * 32 + lane);
#pragma unroll
                    for (int c = 0; c < 4; ++c)
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            dst[(4 * c + j) * (kEpiWarps * 32)] = make_uint4(static_cast<uint32_t>(acc64[c][2 * j]),
                                                        static_cast<uint32_t>(acc64[c][2 * j] >> 32),
                                                        static_cast<uint32_t>(acc64[c][2 * j + 1]),
                                                        static_cast<uint32_t>(acc64[c][2 * j + 1] >> 32));
                    continue;
                }
                store_tile_sym<OUT, RM>(args, wi.tile, quarter, slot, trow, tq, acc64);
            }
        } else {
            float2 acc[2][16];
            int it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int j = 0; j < 16; ++j) acc[h][j] = make_float2(0.f, 0.f);
                for (int g = 0; g < G; ++g, ++it) {
                    const int b = it & 1;
                    const int ss = it % S;
                    if (!mbar_wait_bounded(side_full_bar(ss), (it / S) & 1, abort_flag, args.dev_err,
                                           kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    const uint32_t side_a = smem_base + L::kSide + ss * L::kSideSlotBytes + (quarter * 32 + 4 * trow) * 4;
                    const uint32_t side_w = smem_base + L::kSide + ss * L::kSideSlotBytes + L::kSideABytes +
                                            (slot * kColsPerWarp + tq) * 4;
                    if (!mbar_wait_bounded(acc_full_bar(b), (it >> 1) & 1, abort_flag, args.dev_err,
                                           kWaitLimitNs)) {
                        ok = false;
                        break;
                    }
                    // cur_a[sd][k]: side value sd of row trow + 8k of the quarter
                    float cur_a[NSIDE][4];
#pragma unroll
                    for (int sd = 0; sd < NSIDE; ++sd) {
                        const float4 v = lds_f4(side_a + sd * BM * 4);
                        cur_a[sd][0] = v.x;
                        cur_a[sd][1] = v.y;
                        cur_a[sd][2] = v.z;
                        cur_a[sd][3] = v.w;
                    }
                    tc_fence_after();
                    const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                                           static_cast<uint32_t>(b * BN + slot * kColsPerWarp);
#pragma unroll
                    for (int chunk = 0; chunk < 4; ++chunk) {    // 16-column chunks of the slice
                        uint32_t r[16];
                        tmem_ld_16x128b_x4_pair(tbase + 16 * chunk, tbase + (16u << 16) + 16 * chunk, r);
                        tmem_wait_ld(r);
                        const float4 sw = lds_f4(side_w + 16 * chunk * 4);
                        const float swv[4] = {sw.x, sw.y, sw.z, sw.w};
                        float4 zw4 = make_float4(0.f, 0.f, 0.f, 0.f), gw4 = zw4;
                        if (MODE == QUARTZ_ASYMMETRIC) {
                            zw4 = lds_f4(side_w + (BN + 16 * chunk) * 4);
                            gw4 = lds_f4(side_w + (2 * BN + 16 * chunk) * 4);
                        }
                        const float zwv[4] = {zw4.x, zw4.y, zw4.z, zw4.w};
                        const float gwv[4] = {gw4.x, gw4.y, gw4.z, gw4.w};
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                float2 p = make_float2(__uint_as_float(r[8 * h + 2 * i]), __uint_as_float(r[8 * h + 2 * i + 1]));
                                if (DUMP && g == args.partials_group) {
                                    int mt, nt;
                                    tile_coords<RM>(tile, args, mt, nt);
                                    const int64_t m = static_cast<int64_t>(mt) * BM + quarter * 32 + 16 * h + trow;
                                    const int64_t n = static_cast<int64_t>(nt) * BN + slot * kColsPerWarp + 16 * chunk + tq + i;
                                    if (n < args.N) {
                                        if (m < args.M) args.partials[m * args.N + n] = __float2int_rn(p.x);
                                        if (m + 8 < args.M) args.partials[(m + 8) * args.N + n] = __float2int_rn(p.y);
                                    }
                                }
                                if (MODE == QUARTZ_ASYMMETRIC) {
                                    const float2 ua = make_float2(cur_a[2][2 * h], cur_a[2][2 * h + 1]);
                                    const float2 nza = make_float2(-cur_a[1][2 * h], -cur_a[1][2 * h + 1]);
                                    p = __ffma2_rn(make_float2(zwv[i], zwv[i]), ua, p);
                                    p = __ffma2_rn(nza, make_float2(gwv[i], gwv[i]), p);
                                }
                                const float2 t = __fmul2_rn(p, make_float2(swv[i], swv[i]));
                                acc[h][4 * chunk + i] = __ffma2_rn(t, make_float2(cur_a[0][2 * h], cur_a[0][2 * h + 1]),
                                                                   acc[h][4 * chunk + i]);
                            }
                        }
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        mbar_arrive(acc_empty_bar(b));
                        mbar_arrive(side_empty_bar(ss));
                    }
                }
                if (!ok) break;
                int mt, nt;
                tile_coords<RM>(tile, args, mt, nt);
                // ---- store: 4 rows x 4 chunks of 4 consecutive columns per thread ----
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const int64_t m = static_cast<int64_t>(mt) * BM + quarter * 32 + 16 * h + 8 * e + trow;
                        if (m >= args.M) continue;
#pragma unroll
                        for (int chunk = 0; chunk < 4; ++chunk) {
                            const int64_t n = static_cast<int64_t>(nt) * BN + slot * kColsPerWarp + 16 * chunk + tq;
                            if (n >= args.N) continue;
                            float4 v;
                            v.x = e ? acc[h][4 * chunk + 0].y : acc[h][4 * chunk + 0].x;
                            v.y = e ? acc[h][4 * chunk + 1].y : acc[h][4 * chunk + 1].x;
                            v.z = e ? acc[h][4 * chunk + 2].y : acc[h][4 * chunk + 2].x;
                            v.w = e ? acc[h][4 * chunk + 3].y : acc[h][4 * chunk + 3].x;
                            if (args.bias) {
                                const uint2 braw = __ldg(reinterpret_cast<const uint2 *>(args.bias + n));
                                const float2 b0 = __half22float2(*reinterpret_cast<const __half2 *>(&braw.x));
                                const float2 b1 = __half22float2(*reinterpret_cast<const __half2 *>(&braw.y));
                                v.x = __fadd_rn(v.x, b0.x);
                                v.y = __fadd_rn(v.y, b0.y);
                                v.z = __fadd_rn(v.z, b1.x);
                                v.w = __fadd_rn(v.w, b1.y);
                            }
                            store_quad<OUT>(args.y, m * args.N + n, v);
                        }
                    }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}

// Split last wave (see GemmArgs): adds each tail tile's `split` fp32
// partial tiles in part order, then stores the sum as the epilogue would
// have.  Grid: (tail tile, 16-column chunk c of every warp's slice); block:
// one thread per epilogue thread, which owns the chunk's 8 column pairs.
template <int OUT>
__global__ void __launch_bounds__(kEpiWarps * 32) tail_combine_kernel(const __grid_constant__ GemmArgs args)
{
    griddep_wait();
    constexpr int T = kEpiWarps * 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tail = blockIdx.x >> 2, c = blockIdx.x & 3;
    // parts of this tile: every one of the split equal parts, or (range
    // forms) one per CTA range the tile's groups meet
    const int parts = args.ls > 0 ? ((tail + 1) * args.G - 1) / args.ls - (tail * args.G) / args.ls + 1
                                  : args.split;
    if (parts == 1) return;  // the tile lies in one CTA's range: stored whole by the GEMM
    const uint4 *src = reinterpret_cast<const uint4 *>(args.tail_part) +
                       static_cast<int64_t>(tail) * args.split * 16 * T + 4 * c * T + threadIdx.x;
    uint64_t acc[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const uint4 v = __ldcg(src + j * T);
        acc[2 * j] = (static_cast<uint64_t>(v.y) << 32) | v.x;
        acc[2 * j + 1] = (static_cast<uint64_t>(v.w) << 32) | v.z;
    }
    for (int p = 1; p < parts; ++p) {
        const uint4 *sp = src + static_cast<int64_t>(p) * 16 * T;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint4 v = __ldcg(sp + j * T);
            add2_rn(acc[2 * j], (static_cast<uint64_t>(v.y) << 32) | v.x);
            add2_rn(acc[2 * j + 1], (static_cast<uint64_t>(v.w) << 32) | v.z);
        }
    }
    int mt, nt;
    if (args.raster_m == 1)
        tile_coords<1>(args.full_tiles + tail, args, mt, nt);
    else
        tile_coords<kRasterM>(args.full_tiles + tail, args, mt, nt);
    const int quarter = warp & 3, slot = warp >> 2, trow = lane >> 2, tq = 4 * (lane & 3);
    const int64_t n = static_cast<int64_t>(nt) * BN + slot * kColsPerWarp + 16 * c + tq;
    if (n >= args.N) return;
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int64_t m = static_cast<int64_t>(mt) * BM + quarter * 32 + 16 * h + 8 * e + trow;
            if (m >= args.M) continue;
            float vv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i)
                vv[i] = __uint_as_float(static_cast<uint32_t>(e ? (acc[4 * h + i] >> 32) : acc[4 * h + i]));
            store_quad<OUT>(args.y, m * args.N + n, add_bias4(args, n, make_float4(vv[0], vv[1], vv[2], vv[3])));
        }
}

// ---------------------------------------------------------------------------
// 3. SIMT GEMM: same decoded operands, same epilogue arithmetic, CUDA cores.
//    64x64 output tile per 256-thread block, 4x4 outputs per thread.
// ---------------------------------------------------------------------------
template <int MODE, int OUT>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const __nv_fp8_e4m3 *__restrict__ a_op,
                                                        const __nv_fp8_e4m3 *__restrict__ w_op,
                                                        const GemmArgs args, int K)
{
    griddep_wait();
    __shared__ int16_t sa[64][kGroupQ + 2];
    __shared__ int16_t sw[64][kGroupQ + 2];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
    float y[4][4] = {};
    const int64_t a_plane = args.m_pad * args.G;
    const int64_t w_plane = args.n_pad * args.G;
    for (int g = 0; g < args.G; ++g) {
        for (int i = threadIdx.x; i < 64 * kGroupQ; i += 256) {
            const int r = i / kGroupQ, k = i % kGroupQ;
            const int64_t kk = static_cast<int64_t>(g) * kGroupQ + k;
            sa[r][k] = (m0 + r < args.M) ? static_cast<int16_t>(static_cast<float>(a_op[(int64_t)(m0 + r) * K + kk])) : 0;
            sw[r][k] = (n0 + r < args.N) ? static_cast<int16_t>(static_cast<float>(w_op[perm16(n0 + r) * K + kk])) : 0;
        }
        __syncthreads();
        int p[4][4] = {};
        for (int k = 0; k < kGroupQ; ++k)
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) p[i][j] += sa[ty * 4 + i][k] * sw[tx * 4 + j][k];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int m = m0 + ty * 4 + i;
            const float s_a = args.a_side[static_cast<int64_t>(g) * args.m_pad + perm32(m)];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int n = n0 + tx * 4 + j;
                if (m >= args.M || n >= args.N) continue;
                float P = static_cast<float>(p[i][j]);
                if (args.partials && g == args.partials_group) args.partials[(int64_t)m * args.N + n] = p[i][j];
                if (MODE == QUARTZ_ASYMMETRIC) {
                    const float za = args.a_side[a_plane + (int64_t)g * args.m_pad + perm32(m)];
                    const float ua = args.a_side[2 * a_plane + (int64_t)g * args.m_pad + perm32(m)];
                    const float zw = args.w_side[w_plane + (int64_t)g * args.n_pad + n];
                    const float gw = args.w_side[2 * w_plane + (int64_t)g * args.n_pad + n];
                    P = __fmaf_rn(zw, ua, P);
                    P = __fmaf_rn(-za, gw, P);
                }
                const float t = __fmul_rn(P, args.w_side[static_cast<int64_t>(g) * args.n_pad + n]);
                y[i][j] = __fmaf_rn(t, s_a, y[i][j]);
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + ty * 4 + i;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int n = n0 + tx * 4 + j;
            if (m >= args.M || n >= args.N) continue;
            float v = y[i][j];
            if (args.bias) v = __fadd_rn(v, __half2float(args.bias[n]));
            const int64_t off = (int64_t)m * args.N + n;
            if (OUT == QUARTZ_OUT_F16) static_cast<__half *>(args.y)[off] = __float2half_rn(v);
            else if (OUT == QUARTZ_OUT_BF16) static_cast<__nv_bfloat16 *>(args.y)[off] = __float2bfloat16_rn(v);
            else static_cast<float *>(args.y)[off] = v;
        }
    }
}

// ---------------------------------------------------------------------------
// 4. Accumulator-shift GEMM (the paper's own schedule, Section 4.4): works on
//    the packed 4-bit codes and FLAGs directly, with no decoded operand.  Per
//    subgroup j of G_s elements it forms the integer dot product of the codes
//    and shifts it by the two FLAGs: P_g = sum_j (sum_{k in j} c_a c_w)
//    << (F_a[j] + F_w[j]), which equals sum_k v_a v_w exactly.  The dot
//    products run on dp4a over the codes placed in the high nibble of each
//    byte (int8 value 16c, so a dot product is 256 x the code dot product).
//    The dequant arithmetic is the SIMT kernel's.  64x64 output tile per
//    256-thread block, 4x4 outputs per thread.  WIDE: operands with 16-bit
//    stage-1 codes (Section 5 LLM variant), FLAGs up to 12, so a shifted
//    subgroup product reaches 392 << 24 and the group sums are 64-bit.
// ---------------------------------------------------------------------------
template <int GS, int MODE, int OUT, bool WIDE>
__global__ void __launch_bounds__(256) gemm_shift_kernel(const uint32_t *__restrict__ a_codes,
                                                         const uint8_t *__restrict__ a_flags,
                                                         const uint32_t *__restrict__ w_codes,
                                                         const uint8_t *__restrict__ w_flags,
                                                         const GemmArgs args, int K, int a_packed, int w_packed)
{
    griddep_wait();
    constexpr int kSub = kGroupQ / GS;            // subgroups per group
    constexpr int kWordsPerSub = GS / 4;          // int8x4 words per subgroup
    __shared__ uint32_t sa[64][2 * kGroupQ / 8 + 1];
    __shared__ uint32_t sw[64][2 * kGroupQ / 8 + 1];
    __shared__ uint8_t fa[64][kSub];
    __shared__ uint8_t fw[64][kSub];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
    const int64_t words_per_row = K / 8, flags_per_row = K / GS;
    float y[4][4] = {};
    const int64_t a_plane = args.m_pad * args.G;
    const int64_t w_plane = args.n_pad * args.G;
    for (int g = 0; g < args.G; ++g) {
        for (int i = threadIdx.x; i < 64 * (kGroupQ / 8); i += 256) {
            const int r = i / (kGroupQ / 8), wi = i % (kGroupQ / 8);
            const int64_t col = static_cast<int64_t>(g) * (kGroupQ / 8) + wi;
            const uint32_t ca = (m0 + r < args.M) ? a_codes[(m0 + r) * words_per_row + col] : 0u;
            const uint32_t cw = (n0 + r < args.N) ? w_codes[(n0 + r) * words_per_row + col] : 0u;
            sa[r][2 * wi] = (ca << 4) & 0xF0F0F0F0u;  // even codes, as 16c
            sa[r][2 * wi + 1] = ca & 0xF0F0F0F0u;     // odd codes, as 16c
            sw[r][2 * wi] = (cw << 4) & 0xF0F0F0F0u;
            sw[r][2 * wi + 1] = cw & 0xF0F0F0F0u;
        }
        for (int i = threadIdx.x; i < 64 * kSub; i += 256) {
            const int r = i / kSub, j = i % kSub;
            const int64_t col = static_cast<int64_t>(g) * kSub + j;
            fa[r][j] = (m0 + r < args.M) ? load_flag(a_flags, (m0 + r) * flags_per_row + col, a_packed != 0) : 0;
            fw[r][j] = (n0 + r < args.N) ? load_flag(w_flags, (n0 + r) * flags_per_row + col, w_packed != 0) : 0;
        }
        __syncthreads();
        using Acc = typename std::conditional<WIDE, long long, int>::type;
        Acc p[4][4] = {};
#pragma unroll
        for (int j = 0; j < kSub; ++j) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int jj = 0; jj < 4; ++jj) {
                    int dot = 0;
#pragma unroll
                    for (int q = 0; q < kWordsPerSub; ++q)
                        dot = __dp4a(static_cast<int>(sa[ty * 4 + i][j * kWordsPerSub + q]),
                                     static_cast<int>(sw[tx * 4 + jj][j * kWordsPerSub + q]), dot);
                    p[i][jj] += static_cast<Acc>(dot >> 8) << (fa[ty * 4 + i][j] + fw[tx * 4 + jj][j]);
                }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int m = m0 + ty * 4 + i;
            if (m >= args.M) continue;
            const float s_a = args.a_side[static_cast<int64_t>(g) * args.m_pad + perm32(m)];
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
                const int n = n0 + tx * 4 + jj;
                if (n >= args.N) continue;
                float P = static_cast<float>(p[i][jj]);
                if (!WIDE && args.partials && g == args.partials_group)
                    args.partials[(int64_t)m * args.N + n] = static_cast<int32_t>(p[i][jj]);
                if (MODE == QUARTZ_ASYMMETRIC) {
                    const float za = args.a_side[a_plane + (int64_t)g * args.m_pad + perm32(m)];
                    const float ua = args.a_side[2 * a_plane + (int64_t)g * args.m_pad + perm32(m)];
                    const float zw = args.w_side[w_plane + (int64_t)g * args.n_pad + n];
                    const float gw = args.w_side[2 * w_plane + (int64_t)g * args.n_pad + n];
                    P = __fmaf_rn(zw, ua, P);
                    P = __fmaf_rn(-za, gw, P);
                }
                const float t = __fmul_rn(P, args.w_side[static_cast<int64_t>(g) * args.n_pad + n]);
                y[i][jj] = __fmaf_rn(t, s_a, y[i][jj]);
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + ty * 4 + i;
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
            const int n = n0 + tx * 4 + jj;
            if (m >= args.M || n >= args.N) continue;
            float v = y[i][jj];
            if (args.bias) v = __fadd_rn(v, __half2float(args.bias[n]));
            const int64_t off = (int64_t)m * args.N + n;
            if (OUT == QUARTZ_OUT_F16) static_cast<__half *>(args.y)[off] = __float2half_rn(v);
            else if (OUT == QUARTZ_OUT_BF16) static_cast<__nv_bfloat16 *>(args.y)[off] = __float2bfloat16_rn(v);
            else static_cast<float *>(args.y)[off] = v;
        }
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }
size_t align256(size_t v) { return (v + 255) & ~size_t(255); }

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn lookup_encode_tiled()
{
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
        return reinterpret_cast<EncodeTiledFn>(p);
    return nullptr;
}

// Looked up once (the initialisation of a function-local static is
// thread-safe, so concurrent first calls from several host threads are fine).
EncodeTiledFn encode_tiled_fn()
{
    static const EncodeTiledFn fn = lookup_encode_tiled();
    return fn;
}

// K-major E4M3 operand [rows, K] (one byte per element) read in boxes of
// [box_rows, 64] with the 64-byte swizzle; out-of-range rows read as zero.
bool make_operand_map(CUtensorMap *m, const void *base, int64_t rows, int64_t K, int box_rows)
{
    EncodeTiledFn fn = encode_tiled_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(K)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// SM count of the current device (0 if there is none), looked up once per device.
int device_sms_or_zero()
{
    constexpr int kMaxDevices = 64;
    static std::atomic<int> cached[kMaxDevices];  // 0: not looked up yet
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    const bool slot = dev >= 0 && dev < kMaxDevices;
    if (slot && (n = cached[dev].load(std::memory_order_relaxed)) > 0) return n;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 0;
    if (slot) cached[dev].store(n, std::memory_order_relaxed);
    return n;
}

int num_sms()
{
    const int n = device_sms_or_zero();
    return n > 0 ? n : 1;
}

template <int MODE, int OUT>
cudaError_t launch_tc(const CUtensorMap &ta, const CUtensorMap &tw, const GemmArgs &args,
                      cudaStream_t s)
{
    constexpr int NSIDE = (MODE == QUARTZ_ASYMMETRIC) ? 3 : 1;
    constexpr int smem = Smem<NSIDE>::kAlloc;
    static_assert(smem <= 227 * 1024, "shared memory budget");
    auto kern = args.partials ? gemm_tcgen05_kernel<MODE, OUT, true, false>
                              : gemm_tcgen05_kernel<MODE, OUT, false, false>;
    if constexpr (MODE == QUARTZ_SYMMETRIC) {
        if (!args.partials && !args.per_row && args.raster_m == 1) kern = gemm_tcgen05_kernel<MODE, OUT, false, false, 1>;
    }
    if constexpr (MODE == QUARTZ_SYMMETRIC) {
        if (args.per_row)
            kern = args.partials ? gemm_tcgen05_kernel<MODE, OUT, true, true>
                                 : gemm_tcgen05_kernel<MODE, OUT, false, true>;
    }
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int grid = args.num_tiles < num_sms() ? args.num_tiles : num_sms();
    if (args.split > 1 && args.ls == 0 && args.full_tiles == 0) grid = args.tail_tiles * args.split;
    if (args.ls > 0) grid = num_sms();  // one group range per SM
    launch_pdl(kern, dim3(grid), dim3(kThreads), smem, s, ta, tw, args);
    return cudaGetLastError();
}

template <int MODE>
cudaError_t launch_tc_out(const CUtensorMap &ta, const CUtensorMap &tw, const GemmArgs &args,
                          int y_type, cudaStream_t s)
{
    switch (y_type) {
        case QUARTZ_OUT_F16: return launch_tc<MODE, QUARTZ_OUT_F16>(ta, tw, args, s);
        case QUARTZ_OUT_BF16: return launch_tc<MODE, QUARTZ_OUT_BF16>(ta, tw, args, s);
        default: return launch_tc<MODE, QUARTZ_OUT_F32>(ta, tw, args, s);
    }
}

cudaError_t launch_tail_combine(const GemmArgs &args, int y_type, cudaStream_t s)
{
    const unsigned grid = static_cast<unsigned>(args.tail_tiles) * 4;
    switch (y_type) {
        case QUARTZ_OUT_F16: launch_pdl(tail_combine_kernel<QUARTZ_OUT_F16>, dim3(grid), dim3(kEpiWarps * 32), 0, s, args); break;
        case QUARTZ_OUT_BF16: launch_pdl(tail_combine_kernel<QUARTZ_OUT_BF16>, dim3(grid), dim3(kEpiWarps * 32), 0, s, args); break;
        default: launch_pdl(tail_combine_kernel<QUARTZ_OUT_F32>, dim3(grid), dim3(kEpiWarps * 32), 0, s, args); break;
    }
    return cudaGetLastError();
}

template <int MODE, int OUT>
cudaError_t launch_simt(const LinearWorkspace &ws, const GemmArgs &args, int K, cudaStream_t s)
{
    dim3 grid(static_cast<unsigned>((args.N + 63) / 64), static_cast<unsigned>((args.M + 63) / 64));
    launch_pdl(gemm_simt_kernel<MODE, OUT>, dim3(grid), dim3(256), 0, s, static_cast<const __nv_fp8_e4m3 *>(ws.a_op),
                                                     static_cast<const __nv_fp8_e4m3 *>(ws.w_op), args, K);
    return cudaGetLastError();
}

template <int MODE>
cudaError_t launch_simt_out(const LinearWorkspace &ws, const GemmArgs &args, int K, int y_type,
                            cudaStream_t s)
{
    switch (y_type) {
        case QUARTZ_OUT_F16: return launch_simt<MODE, QUARTZ_OUT_F16>(ws, args, K, s);
        case QUARTZ_OUT_BF16: return launch_simt<MODE, QUARTZ_OUT_BF16>(ws, args, K, s);
        default: return launch_simt<MODE, QUARTZ_OUT_F32>(ws, args, K, s);
    }
}

GemmArgs make_args(const LinearWorkspace &ws, int64_t M, int64_t N, int64_t K, const void *bias,
                   void *y, int y_type, int32_t *partials, int partials_group, int *dev_err)
{
    GemmArgs a;
    a.per_row = 0;
    a.wide = 0;
    a.split = 1;
    a.ls = 0;
    a.tail_tiles = 0;
    a.tail_part = ws.tail_part;
    a.a_side = ws.a_side;
    a.w_side = ws.w_side;
    a.m_pad = ws.m_pad;
    a.n_pad = ws.n_pad;
    a.M = static_cast<int>(M);
    a.N = static_cast<int>(N);
    a.G = static_cast<int>(K / kGroupQ);
    a.tiles_n = static_cast<int>((N + BN - 1) / BN);
    a.tiles_m = static_cast<int>((M + BM - 1) / BM);
    a.num_tiles = a.tiles_m * a.tiles_n;
    a.raster_m = kRasterM;
    a.full_tiles = a.num_tiles;
    a.bias = static_cast<const __half *>(bias);
    a.y = y;
    a.y_type = y_type;
    a.partials = partials;
    a.partials_group = partials_group;
    a.dev_err = dev_err;
    return a;
}

}  // namespace

// Split of the GEMM's last wave on this device (symmetric, group-64 fast
// path): when the tiles left after whole waves fill at most half of one,
// each of them is cut along K into `split` group ranges (at most
// kMaxTailSplit, at least two groups each) for otherwise idle CTAs; with
// fewer tiles than SMs (a first wave that is also the last), every tile is
// cut that way and the grid has tiles x split CTAs.  When
// they fill more than half, the last two waves' group iterations are spread
// evenly over the CTAs (two-wave form), but only where that shortens the
// critical path by at least kMinStreamSaving group iterations: it costs
// about the time of 25 (partial tiles written and read back, the combine
// launch), measured on the LLaMA-2-7B o (saves 20: 3% slower) and down
// (saves 54: 9% faster) projections.
constexpr int kMaxTailSplit = 4;
constexpr int kMinStreamSaving = 32;

void tail_split(int64_t M, int64_t N, int64_t K, int mode, int *tail, int *split, int *ls = nullptr)
{
    *tail = 0;
    *split = 1;
    if (ls) *ls = 0;
    const int sms = device_sms_or_zero();
    if (mode != QUARTZ_SYMMETRIC || sms <= 0 || M <= 0) return;
    const int64_t T = ((M + BM - 1) / BM) * ((N + BN - 1) / BN);
    const int64_t P = T < sms ? T : sms;
    const int64_t W = T / P, R = T % P, G = K / kGroupQ;
    if (W >= 1 && 2 * R > P) {
        const int64_t Ts = P + R, U = Ts * G;
        if (G * (P - R) < kMinStreamSaving * P || U >= (int64_t(1) << 30)) return;
        *tail = static_cast<int>(Ts);
        *split = 2;
        if (ls) *ls = static_cast<int>((U + P - 1) / P);
        return;
    }
    if (T < sms && 2 * T > sms) {
        // more than half the SMs hold a tile: the tiles' T * G group
        // iterations are cut into one contiguous range per SM (ls >= G / 2,
        // so a tile meets at most 3 ranges: 3 part slots per tile)
        const int64_t U = T * G;
        if (G * (sms - T) < kMinStreamSaving * sms || U >= (int64_t(1) << 30)) return;
        *tail = static_cast<int>(T);
        *split = 3;
        if (ls) *ls = static_cast<int>((U + sms - 1) / sms);
        return;
    }
    if (T < sms) {  // fewer tiles than SMs: every tile is cut along K for the idle SMs
        int64_t S = sms / T;
        if (S > kMaxTailSplit) S = kMaxTailSplit;
        if (S > G / 2) S = G / 2;
        if (S < 2) return;
        *tail = static_cast<int>(T);
        *split = static_cast<int>(S);
        return;
    }
    if (W < 1 || R == 0) return;
    int64_t S = P / R;
    if (S > kMaxTailSplit) S = kMaxTailSplit;
    if (S > G / 2) S = G / 2;
    if (S < 2) return;
    *tail = static_cast<int>(R);
    *split = static_cast<int>(S);
}

int linear_tail_parts(int64_t M, int64_t N, int64_t K, int mode)
{
    int tail = 0, split = 1;
    tail_split(M, N, K, mode, &tail, &split);
    return split;
}

size_t tail_part_bytes(int tail, int split) { return static_cast<size_t>(tail) * split * kEpiWarps * 32 * 64 * 4; }

size_t linear_workspace_bytes(int64_t M, int64_t N, int64_t K, int mode)
{
    const int nside = mode == QUARTZ_ASYMMETRIC ? 3 : 1;
    const int64_t G = K / kGroupQ;
    size_t b = align256(static_cast<size_t>(M) * K);
    b += align256(static_cast<size_t>(round_up(N, 16)) * K);
    b += align256(static_cast<size_t>(nside) * G * round_up(M > 0 ? M : 1, BM) * 4);
    b += align256(static_cast<size_t>(nside) * G * round_up(N, BN) * 4);
    int tail = 0, split = 1;
    tail_split(M, N, K, mode, &tail, &split);
    if (split > 1) b += align256(tail_part_bytes(tail, split));
    return b;
}

void linear_workspace_carve(void *base, int64_t M, int64_t N, int64_t K, int mode,
                            LinearWorkspace *ws)
{
    const int nside = mode == QUARTZ_ASYMMETRIC ? 3 : 1;
    const int64_t G = K / kGroupQ;
    uint8_t *p = static_cast<uint8_t *>(base);
    ws->nside = nside;
    ws->m_pad = round_up(M > 0 ? M : 1, BM);
    ws->n_pad = round_up(N, BN);
    ws->a_op = p;
    p += align256(static_cast<size_t>(M) * K);
    ws->w_op = p;
    p += align256(static_cast<size_t>(round_up(N, 16)) * K);
    ws->a_side = reinterpret_cast<float *>(p);
    p += align256(static_cast<size_t>(nside) * G * ws->m_pad * 4);
    ws->w_side = reinterpret_cast<float *>(p);
    p += align256(static_cast<size_t>(nside) * G * ws->n_pad * 4);
    tail_split(M, N, K, mode, &ws->tail_tiles, &ws->tail_split, &ws->tail_ls);
    ws->tail_part = ws->tail_split > 1 ? reinterpret_cast<float *>(p) : nullptr;
}

size_t prepared_weights_bytes(int64_t N, int64_t K, int mode)
{
    const int nside = mode == QUARTZ_ASYMMETRIC ? 3 : 1;
    const int64_t G = K / kGroupQ;
    return align256(static_cast<size_t>(round_up(N, 16)) * K) + align256(static_cast<size_t>(nside) * G * round_up(N, BN) * 4);
}

void prepared_weights_carve(const void *base, int64_t N, int64_t K, int mode, LinearWorkspace *ws)
{
    uint8_t *p = static_cast<uint8_t *>(const_cast<void *>(base));
    ws->w_op = p;
    ws->w_side = reinterpret_cast<float *>(p + align256(static_cast<size_t>(round_up(N, 16)) * K));
    ws->n_pad = round_up(N, BN);
    ws->nside = mode == QUARTZ_ASYMMETRIC ? 3 : 1;
}

cudaError_t launch_prepare(const quartz_encoded_t *a, const quartz_encoded_t *w, const LinearWorkspace &ws,
                           cudaStream_t s, bool expand, bool w_ready)
{
    const int64_t K = w->K;
    const int64_t upr = K / 16;
    PrepArgs p{};
    p.G = static_cast<int>(K / w->p.group_q);  // scale groups per row
    p.nside = ws.nside;
    if (a)
        p.ex_a = {reinterpret_cast<const uint2 *>(a->codes), a->flags, static_cast<uint4 *>(ws.a_op),
                  a->rows * upr, a->rows * upr, upr, 0, a->p.flag_bits == 4};
    // the weight operand is row-permuted and padded to a multiple of 16 rows
    p.ex_w = {reinterpret_cast<const uint2 *>(w->codes), w->flags, static_cast<uint4 *>(ws.w_op),
              w->rows * upr, round_up(w->rows, 16) * upr, upr, 1, w->p.flag_bits == 4};
    if (a)
        p.sd_a = {reinterpret_cast<const __half *>(a->scales), a->zeros, a->gsum, ws.a_side, a->rows, ws.m_pad, 1};
    p.sd_w = {reinterpret_cast<const __half *>(w->scales), w->zeros, w->gsum, ws.w_side, w->rows, ws.n_pad, 0};
    const int64_t side_chunks = (p.G + kSideGroupsPerThread - 1) / kSideGroupsPerThread;
    const int64_t items[4] = {expand ? p.ex_a.units_pad : 0, expand && !w_ready ? p.ex_w.units_pad : 0,
                              a ? ws.m_pad * side_chunks : 0, w_ready ? 0 : ws.n_pad * side_chunks};
    const int64_t per_block[4] = {2 * kPrepThreads * kExpandPairs, 2 * kPrepThreads * kExpandPairs, kPrepThreads,
                                  kPrepThreads};
    int64_t acc = 0;
    for (int i = 0; i < 4; ++i) {
        acc += (items[i] + per_block[i] - 1) / per_block[i];
        p.block_end[i] = acc;
    }
    if (acc == 0) return cudaSuccess;
    const unsigned blocks = static_cast<unsigned>(acc);
    if (w->p.code_bits == 16) {  // 16-bit stage-1 codes: E5M2 operands
        switch (w->p.group_s) {
            case 8: launch_pdl(prep_kernel<8, true>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
            case 16: launch_pdl(prep_kernel<16, true>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
            case 32: launch_pdl(prep_kernel<32, true>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
            default: launch_pdl(prep_kernel<64, true>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
        }
        return cudaGetLastError();
    }
    switch (w->p.group_s) {
        case 8: launch_pdl(prep_kernel<8, false>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
        case 16: launch_pdl(prep_kernel<16, false>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
        case 32: launch_pdl(prep_kernel<32, false>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
        default: launch_pdl(prep_kernel<64, false>, dim3(blocks), dim3(kPrepThreads), 0, s, p); break;
    }
    return cudaGetLastError();
}

cudaError_t launch_gemm_tcgen05(const LinearWorkspace &ws, int64_t M, int64_t N, int64_t K,
                                int mode, const void *bias, void *y, int y_type,
                                int32_t *partials, int partials_group, int *dev_err,
                                cudaStream_t s, bool per_row, bool wide)
{
    if (M == 0) return cudaSuccess;
    CUtensorMap ta, tw;
    if (!make_operand_map(&ta, ws.a_op, M, K, BM) || !make_operand_map(&tw, ws.w_op, round_up(N, 16), K, BN))
        return cudaErrorInvalidValue;
    GemmArgs args = make_args(ws, M, N, K, bias, y, y_type, partials, partials_group, dev_err);
    args.per_row = per_row ? 1 : 0;
    args.wide = wide ? 1 : 0;
    if (mode == QUARTZ_SYMMETRIC && !partials && !per_row && args.tiles_n <= kRowRasterMaxN) args.raster_m = 1;
    int tail = 0, split = 1, ls = 0;  // the workspace's split must still match this device's grid
    if (mode == QUARTZ_SYMMETRIC && !partials && !per_row && ws.tail_split > 1 && ws.tail_part)
        tail_split(M, N, K, mode, &tail, &split, &ls);
    if (split > 1 && split == ws.tail_split && tail == ws.tail_tiles && ls == ws.tail_ls) {
        args.split = ws.tail_split;
        args.ls = ls;
        args.tail_tiles = ws.tail_tiles;
        args.full_tiles = args.num_tiles - ws.tail_tiles;
        cudaError_t e = launch_tc_out<QUARTZ_SYMMETRIC>(ta, tw, args, y_type, s);
        if (e != cudaSuccess) return e;
        return launch_tail_combine(args, y_type, s);
    }
    if (per_row) return launch_tc_out<QUARTZ_SYMMETRIC>(ta, tw, args, y_type, s);
    return mode == QUARTZ_ASYMMETRIC ? launch_tc_out<QUARTZ_ASYMMETRIC>(ta, tw, args, y_type, s)
                                     : launch_tc_out<QUARTZ_SYMMETRIC>(ta, tw, args, y_type, s);
}

cudaError_t launch_gemm_simt(const LinearWorkspace &ws, int64_t M, int64_t N, int64_t K, int mode,
                             const void *bias, void *y, int y_type, int32_t *partials,
                             int partials_group, cudaStream_t s)
{
    if (M == 0) return cudaSuccess;
    const GemmArgs args = make_args(ws, M, N, K, bias, y, y_type, partials, partials_group, nullptr);
    return mode == QUARTZ_ASYMMETRIC
               ? launch_simt_out<QUARTZ_ASYMMETRIC>(ws, args, static_cast<int>(K), y_type, s)
               : launch_simt_out<QUARTZ_SYMMETRIC>(ws, args, static_cast<int>(K), y_type, s);
}

namespace {
template <int GS, int MODE, int OUT, bool WIDE>
cudaError_t launch_shift(const quartz_encoded_t *a, const quartz_encoded_t *w, const GemmArgs &args,
                         cudaStream_t s)
{
    dim3 grid(static_cast<unsigned>((args.N + 63) / 64), static_cast<unsigned>((args.M + 63) / 64));
    launch_pdl(gemm_shift_kernel<GS, MODE, OUT, WIDE>, dim3(grid), dim3(256), 0, s, 
        reinterpret_cast<const uint32_t *>(a->codes), a->flags, reinterpret_cast<const uint32_t *>(w->codes),
        w->flags, args, static_cast<int>(a->K), a->p.flag_bits == 4, w->p.flag_bits == 4);
    return cudaGetLastError();
}

template <int GS, int MODE, bool WIDE>
cudaError_t launch_shift_out(const quartz_encoded_t *a, const quartz_encoded_t *w, const GemmArgs &args,
                             int y_type, cudaStream_t s)
{
    switch (y_type) {
        case QUARTZ_OUT_F16: return launch_shift<GS, MODE, QUARTZ_OUT_F16, WIDE>(a, w, args, s);
        case QUARTZ_OUT_BF16: return launch_shift<GS, MODE, QUARTZ_OUT_BF16, WIDE>(a, w, args, s);
        default: return launch_shift<GS, MODE, QUARTZ_OUT_F32, WIDE>(a, w, args, s);
    }
}

template <int GS>
cudaError_t launch_shift_mode(const quartz_encoded_t *a, const quartz_encoded_t *w, const GemmArgs &args,
                              int y_type, bool wide, cudaStream_t s)
{
    if (wide) return launch_shift_out<GS, QUARTZ_SYMMETRIC, true>(a, w, args, y_type, s);
    return a->p.mode == QUARTZ_ASYMMETRIC ? launch_shift_out<GS, QUARTZ_ASYMMETRIC, false>(a, w, args, y_type, s)
                                          : launch_shift_out<GS, QUARTZ_SYMMETRIC, false>(a, w, args, y_type, s);
}
}  // namespace

cudaError_t launch_gemm_shift(const LinearWorkspace &ws, const quartz_encoded_t *a, const quartz_encoded_t *w,
                              const void *bias, void *y, int y_type, int32_t *partials, int partials_group,
                              cudaStream_t s, bool wide)
{
    const int64_t M = a->rows, N = w->rows, K = a->K;
    if (M == 0) return cudaSuccess;
    const GemmArgs args = make_args(ws, M, N, K, bias, y, y_type, partials, partials_group, nullptr);
    switch (a->p.group_s) {
        case 8: return launch_shift_mode<8>(a, w, args, y_type, wide, s);
        case 16: return launch_shift_mode<16>(a, w, args, y_type, wide, s);
        case 32: return launch_shift_mode<32>(a, w, args, y_type, wide, s);
        default: return launch_shift_mode<64>(a, w, args, y_type, wide, s);
    }
}

// ---------------------------------------------------------------------------
// failure-detection self-test: a wait that nothing ever satisfies
// ---------------------------------------------------------------------------
namespace {
__global__ void selftest_timeout_kernel(uint64_t limit_ns, int *dev_err)
{
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) mbar_wait_bounded(smem_u32(&bar), 0, &abort_flag, dev_err, limit_ns);
    __syncthreads();
}
}  // namespace

cudaError_t launch_selftest_timeout(int64_t limit_ns, int *dev_err, cudaStream_t s)
{
    selftest_timeout_kernel<<<1, 32, 0, s>>>(static_cast<uint64_t>(limit_ns), dev_err);
    return cudaGetLastError();
}

}  // namespace quartz
