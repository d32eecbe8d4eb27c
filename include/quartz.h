/*
 * quartz.h -- C ABI of the GB300 (sm_103a) QuaRTZ W4A4 linear hot path.
 *
 * QuaRTZ (arXiv 2509.26436) quantizes activations and weights in two stages:
 * per-group 8-bit min-max quantization (Section 3, Eq. 1) followed by
 * Leading Zero Suppression of each 8-bit code to a signed 4-bit code plus a
 * per-subgroup FLAG (Section 3, Eq. 2).  The linear layer multiplies two such
 * encoded operands with an integer MMA and applies the per-group 16-bit
 * scales afterwards (Section 4.4; Appendix C: groups of 64 along K, 16-bit
 * scales).
 *
 * Conventions shared by every entry point
 *   - All tensor pointers are DEVICE pointers owned by the caller.  The
 *     library never allocates, frees or synchronises (except
 *     quartz_device_status, which synchronises the given stream).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Every launch is asynchronous on that stream.
 *   - Every call returns a quartz_status_t (as int32_t).  Arguments are
 *     validated on the host before anything is launched; on any error
 *     nothing is launched and no output is touched.
 *   - Inputs containing NaN or Inf are unsupported (results undefined; the
 *     kernels do not fault on them).
 *   - Layouts are row-major and contiguous.  "fp16" means IEEE binary16.
 */
#ifndef QUARTZ_H
#define QUARTZ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    QUARTZ_OK = 0,
    QUARTZ_ERR_INVALID_ARG = 1,   /* bad size, group size, mode, type or NULL pointer */
    QUARTZ_ERR_ALIGNMENT = 2,     /* a pointer is not 16-byte aligned */
    QUARTZ_ERR_UNSUPPORTED = 3,   /* valid per the paper but not built (e.g. group_q != 64) */
    QUARTZ_ERR_CUDA = 4,          /* a CUDA runtime / driver call failed */
    QUARTZ_ERR_TIMEOUT = 5,       /* a kernel's bounded wait expired (reported by quartz_device_status) */
    QUARTZ_ERR_WORKSPACE = 6      /* workspace missing or smaller than quartz_linear_workspace_size */
} quartz_status_t;

/* Eq. 1 conventions.  The paper's printed Eq. 1 (s = (max-min)/255, clamp to
 * [-127,127], z = round(-min/s)) is not self-consistent; Appendix A analyses
 * the symmetric midtread quantizer, which is the default here.
 *   SYMMETRIC:  s = fp16(max|x| / 127), z = 0, q = clamp(round(x/s), -127, 127)
 *   ASYMMETRIC: [lo, hi] = [min(min x, 0), max(max x, 0)],
 *               s = fp16((hi - lo) / 255), z = round(-lo/s) - 128 (stored),
 *               q = clamp(round(x/s) + z, -127, 127)
 * round() is round-half-to-even; x/s is evaluated as x * r, r = RN(1/s) in
 * binary32; a group whose fp16 scale is 0 gets all-zero codes and z = 0. */
typedef enum { QUARTZ_SYMMETRIC = 0, QUARTZ_ASYMMETRIC = 1 } quartz_mode_t;

typedef enum { QUARTZ_OUT_F16 = 0, QUARTZ_OUT_BF16 = 1, QUARTZ_OUT_F32 = 2 } quartz_out_t;

/* GEMM implementations behind quartz_linear_ex.  TCGEN05 is the product
 * path (tcgen05 tensor cores, TMEM accumulators, operands decoded first);
 * SIMT is a plain CUDA-core kernel with the same arithmetic, kept as a second
 * on-device path; SHIFT is the paper's own schedule (Section 4.4): integer
 * dot products of the packed 4-bit codes per subgroup, each shifted by the
 * two operands' FLAGs, with no decoded operand (CUDA cores, dp4a).  All three
 * give the same exact group partials P_g (8-bit codes; see quartz_linear for
 * 16-bit codes). */
typedef enum { QUARTZ_ALGO_TCGEN05 = 0, QUARTZ_ALGO_SIMT = 1, QUARTZ_ALGO_SHIFT = 2 } quartz_algo_t;

typedef struct {
    int32_t group_q; /* min-max quantization group along K: 64 (Appendix C), or K
                      * (one scale per row: per-token activations / per-channel
                      * weights; SYMMETRIC only) */
    int32_t group_s; /* LZS subgroup G_s along K: 8, 16, 32 or 64 (Section 3, Table 1) */
    int32_t mode;    /* quartz_mode_t */
    int32_t flag_bits; /* FLAG storage: 0 or 8 = one byte per subgroup (Section
                        * 4.4); 4 = two FLAGs per byte (values 0..4, or 0..12
                        * with 16-bit codes, fit in 4 bits), 4 + 4/G_s +
                        * 16/group_q bits per element */
    int32_t code_bits; /* width of the stage-1 codes: 0 or 8 = Eq. 1's 8-bit
                        * codes; 16 = the LLM variant of Section 5 (16-bit
                        * activations compressed straight to 4 bits; the
                        * paper uses G_s = 8): s = fp16(max|x| / 32767),
                        * q = clamp(round(x/s), -32767, 32767), Eq. 2 gives
                        * FLAG in 0..12 and decoded values up to 7 << 12.
                        * 16 requires SYMMETRIC mode and group_q == 64. */
} quartz_params_t;

/* One encoded tensor of `rows` rows and `K` columns (Section 4.4's format:
 * signed 4-bit codes two per byte, one FLAG byte per subgroup).  Buffers are device
 * memory owned by the caller; sizes in elements:
 *   codes  uint8 [rows, K/2]        two's-complement 4-bit codes in [-7, 7],
 *                                   element 2j in the low nibble of byte j
 *   flags  uint8 [rows, K/group_s]  FLAG of Eq. 2, values 0..4 (0..12 with
 *                                   16-bit codes); with
 *                                   flag_bits = 4: uint8 [ceil(rows*K/group_s
 *                                   / 2)], FLAG of subgroup 2j (counted over
 *                                   the whole tensor, row after row) in the
 *                                   low nibble of byte j, 2j + 1 in the high
 *   scales fp16  [rows, K/group_q]  16-bit scale s of each group (bits)
 *   zeros  int8  [rows, K/group_q]  stored zero point z (ASYMMETRIC only;
 *                                   may be NULL in SYMMETRIC mode)
 *   gsum   int32 [rows, K/group_q]  sum of the decoded values of each group,
 *                                   sum_k sgn(c_k)(|c_k| << FLAG) (ASYMMETRIC
 *                                   only; used by the zero-point correction)
 * Every pointer must be 16-byte aligned. */
typedef struct {
    uint8_t *codes;
    uint8_t *flags;
    uint16_t *scales;
    int8_t *zeros;
    int32_t *gsum;
    int64_t rows;
    int64_t K;
    quartz_params_t p;
} quartz_encoded_t;

/* Human-readable name of a status code (static storage; never NULL). */
const char *quartz_status_string(int32_t status);

/* ABI version of this library: (major << 16) | minor. */
int32_t quartz_version(void);

/* Bytes of each buffer of an encoded [rows, K] tensor, for allocation:
 * out[0..4] = codes, flags, scales, zeros, gsum.  Returns QUARTZ_OK or
 * QUARTZ_ERR_INVALID_ARG. */
int32_t quartz_encoded_sizes(int64_t rows, int64_t K, const quartz_params_t *p, size_t out[5]);

/* Two-stage QuaRTZ encoder, run on activations as they are produced
 * (Appendix C compresses them to 4 bits at run time): Eq. 1 per group of p->group_q along
 * K, then Eq. 2 per subgroup of p->group_s, then nibble packing.
 *   x_f16  fp16 [out->rows, out->K] device, 16-byte aligned
 *   out    describes the destination: rows, K, p and the buffers above
 * Requirements: rows >= 0, K > 0, K % 64 == 0, group_q == 64 (or K: one
 * scale per row, symmetric), group_s in {8,16,32,64}.  With code_bits = 16
 * the stage-1 codes are 16 bits wide (the LLM variant above).  rows == 0 is
 * a no-op. */
int32_t quartz_quantize(const void *x_f16, const quartz_encoded_t *out, void *stream);

/* Static per-tensor quantization (Appendix C: the latent-diffusion models
 * quantize activations with one static, calibrated scale per tensor): Eq. 1
 * with the given fp16 scale `scale_f16` (bits; finite, >= 0) for every
 * element instead of a scale computed from the data, then Eq. 2.  Elements
 * beyond 127 * scale saturate to +-127 before LZS.  SYMMETRIC mode, 8-bit
 * codes (else QUARTZ_ERR_UNSUPPORTED); any group_q; every stored scale of
 * `out` is `scale_f16`.  A zero scale gives all-zero codes. */
int32_t quartz_quantize_static(const void *x_f16, uint16_t scale_f16, const quartz_encoded_t *out, void *stream);

/* The same encoder applied to nn.Linear weights [N, K] (one quantization
 * row per output channel, groups along K).  Weights are encoded once,
 * offline; the arithmetic is identical to quartz_quantize. */
int32_t quartz_encode_weights(const void *w_f16, const quartz_encoded_t *out, void *stream);

/* Dequantise an encoded tensor: x_hat = s * (v - z) with the decoded LZS
 * value v = sgn(c)(|c| << FLAG) (Section 3: one FLAG shift for every value
 * of a subgroup), computed in binary32 and rounded once to fp16.
 *   x_hat_f16  fp16 [e->rows, e->K] device output. */
int32_t quartz_dequantize(const quartz_encoded_t *e, void *x_hat_f16, void *stream);

/* Workspace bytes quartz_linear needs for an [M, K] x [N, K]^T product
 * (the operands expanded to the tensor-core input format, transposed group
 * scales and, where the symmetric tcgen05 GEMM splits its last wave of
 * tiles along K, the fp32 partial tiles of that wave: 128 KB per part and
 * tile, up to 4 parts per tail tile; when the last two waves are spread
 * over all SMs, 2 parts are reserved for each of their tiles although only
 * the tiles cut by a CTA's range boundary, fewer than the SM count, use
 * them, e.g. 64 MiB of which at most 37.75 MiB is written for a
 * 2048 x 11008 -> 4096 layer; when more than half but not all of the SMs
 * hold a tile and every tile's groups are spread over all SMs, 3 parts
 * are reserved per tile).  The last part depends on the current
 * device's SM count: query it on the device that will run the call.
 * Returns 0 for invalid arguments. */
size_t quartz_linear_workspace_size(int64_t M, int64_t N, int64_t K, const quartz_params_t *p);

/* Kernels one quartz_linear_ex call with these sizes, algorithm and
 * partials setting launches on the current device: operand preparation,
 * the GEMM and, when the symmetric group-64 tcgen05 GEMM (no partials)
 * splits its last wave of tiles along K, the kernel that adds the parts in
 * a fixed order and writes those tiles.  Returns 0 for invalid arguments
 * or M = 0 (no launch). */
int32_t quartz_linear_launch_count(int64_t M, int64_t N, int64_t K, const quartz_params_t *p, int32_t algo,
                                   int32_t with_partials);

/* W4A4 QuaRTZ linear (Section 4.4 with Appendix C's group scales):
 *   y[m, n] = sum_g s_a[m,g] s_w[n,g] (P_g[m,n] - z_w[n,g] A_g[m] - z_a[m,g] W_g[n]
 *                                      + 64 z_a[m,g] z_w[n,g])  (+ bias[n])
 *   P_g[m, n] = sum_{k in group g} v_a[m,k] v_w[n,k]   (exact integer sum)
 * where A_g / W_g are the gsum side values (zero in SYMMETRIC mode).
 *   a          encoded activations [M, K]
 *   w          encoded weights [N, K] (same K, group_q, group_s and mode)
 *   bias_f16   fp16 [N] or NULL
 *   y          [M, N] of y_type (quartz_out_t), 16-byte aligned
 *   workspace  device scratch of at least quartz_linear_workspace_size bytes,
 *              16-byte aligned, owned by the caller; contents are scratch
 * Requirements: N % 8 == 0, K % 64 == 0, M >= 0.  The per-group partials
 * P_g are exact; the scaled sum is accumulated in binary32 in group order
 * and rounded once to y_type.  Where the symmetric TCGEN05 GEMM (no
 * partials) splits its last wave(s) of tiles along K (see
 * quartz_linear_launch_count), those tiles sum up to 4 consecutive runs of
 * groups separately and then add the runs in order: no chain is longer than
 * K/64 terms, and results are the same on every call on the same device.  Operands with 16-bit stage-1 codes (code_bits = 16, both
 * operands; decoded values up to 7 << 12, a group sum up to
 * 64 * 28672^2 > 2^31): QUARTZ_ALGO_SHIFT keeps P_g exact in 64-bit
 * integers; TCGEN05 (E5M2 operands) multiplies exactly but sums each group
 * in the tensor cores' fp32 accumulator, so P_g is then rounded like any
 * fp32 sum; SIMT returns QUARTZ_ERR_UNSUPPORTED. */
int32_t quartz_linear(const quartz_encoded_t *a, const quartz_encoded_t *w, const void *bias_f16,
                      void *y, int32_t y_type, void *workspace, size_t workspace_bytes,
                      void *stream);

/* Extra controls of quartz_linear_ex (all optional; zero-initialise):
 *   partials          NULL, or int32 [M, N] device buffer that receives
 *                     P_g[m, n] of group `partials_group` (0 <= g < K/64), the
 *                     raw integer MMA result before any scale or zero point
 *                     (8-bit codes only: QUARTZ_ERR_UNSUPPORTED with 16-bit
 *                     codes, whose partials need 64 bits)
 *   algo              quartz_algo_t: which GEMM kernel runs
 *   w_prepared        NULL, or prepared weights (below)
 *   gemm_event_begin  NULL, or a cudaEvent_t recorded on `stream` right before
 *   gemm_event_end    / right after the GEMM kernel and its tail combine, if
 *                     any (after operand expansion), so a caller can time the
 *                     GEMM alone */
typedef struct {
    int32_t *partials;
    int32_t partials_group;
    int32_t algo;
    void *gemm_event_begin;
    void *gemm_event_end;
    const void *w_prepared;  /* NULL, or the weights prepared by quartz_prepare_weights
                              * from the same encoded `w`: the call then prepares the
                              * activations only (same results) */
} quartz_linear_opts_t;

/* Bytes of a prepared weight operand for quartz_prepare_weights; 0 for
 * invalid arguments (the shape rules of quartz_linear's weights). */
size_t quartz_prepared_weights_size(int64_t N, int64_t K, const quartz_params_t *p);

/* Prepare encoded weights [N, K] once (offline, like their encoding): their
 * tensor-core operand (the decoded values, E4M3, or E5M2 for 16-bit codes)
 * and transposed group scales, written to `prepared` (device memory owned by
 * the caller, >= quartz_prepared_weights_size bytes, 16-byte aligned).  A
 * later quartz_linear_ex with opts->w_prepared = prepared and the same `w`
 * skips that work on every call; the buffer is only valid for that `w`
 * (its codes, FLAGs, scales and params) and becomes stale if `w` changes. */
int32_t quartz_prepare_weights(const quartz_encoded_t *w, void *prepared, size_t prepared_bytes, void *stream);

/* quartz_linear with the controls above (opts may be NULL = defaults). */
int32_t quartz_linear_ex(const quartz_encoded_t *a, const quartz_encoded_t *w,
                         const void *bias_f16, void *y, int32_t y_type, void *workspace,
                         size_t workspace_bytes, const quartz_linear_opts_t *opts, void *stream);

/* Fused activation path: the W4A4 linear layer straight from fp16
 * activations, encoding them at run time (Appendix C's run-time activation
 * compression).  One pass over x does Eq. 1 and Eq. 2 and
 * writes the tensor-core operand directly, instead of writing the encoded
 * activations and reading them back; results are bit-identical to
 * quartz_quantize followed by quartz_linear with the same parameters.
 *   x_f16      fp16 [M, K] device, 16-byte aligned
 *   w          encoded weights [N, K]; its params (group_s, mode, code_bits)
 *              are used for the activations; SYMMETRIC mode and
 *              group_q == 64 only (else QUARTZ_ERR_UNSUPPORTED).  With
 *              16-bit codes (Section 5 LLM variant) the activations are
 *              encoded with 32767 levels and FLAGs 0..12 and written as the
 *              E5M2 operand, bit-identical to quartz_quantize followed by
 *              quartz_linear with QUARTZ_ALGO_TCGEN05
 *   bias_f16, y, y_type, workspace, workspace_bytes: as quartz_linear
 *              (quartz_linear_workspace_size(M, N, K, &w->p) bytes)
 *   a_out      NULL, or an encoded [M, K] tensor with w's params that also
 *              receives the activations' encoding (codes, FLAGs, scales) */
int32_t quartz_linear_f16(const void *x_f16, int64_t M, const quartz_encoded_t *w, const void *bias_f16,
                          void *y, int32_t y_type, const quartz_encoded_t *a_out, void *workspace,
                          size_t workspace_bytes, void *stream);

/* quartz_linear_f16 with the weights prepared once by quartz_prepare_weights
 * (`w_prepared`, from the same `w`; NULL = quartz_linear_f16): the call is
 * then one encoder launch and the GEMM (plus the tail combine where
 * quartz_linear_launch_count counts one). */
int32_t quartz_linear_f16_ex(const void *x_f16, int64_t M, const quartz_encoded_t *w, const void *w_prepared,
                             const void *bias_f16, void *y, int32_t y_type, const quartz_encoded_t *a_out,
                             void *workspace, size_t workspace_bytes, void *stream);

/* Scratch-free variant of quartz_linear, for callers that cannot allocate
 * device memory (for example a plugin inside a host framework that owns all
 * device memory through its own pool and forbids side allocations, or code on
 * a latency-critical path where a cudaMalloc could synchronise the device).
 * The paper has no counterpart to this entry point; it only changes where
 * the scratch workspace lives.
 *
 * Same arguments, arithmetic and results as quartz_linear without the
 * workspace arguments.  The workspace is a library-owned device array of
 * QUARTZ_NOALLOC_SCRATCH_BYTES that every GPU loading the library holds until
 * the process exits; the call allocates and frees nothing.
 *   - Problems whose quartz_linear_workspace_size exceeds the array are
 *     rejected with QUARTZ_ERR_WORKSPACE before anything is launched.
 *   - The first call on a device looks up the array's device address with
 *     that device current; make that first call before any stream capture.
 *   - All calls on a device share the array and it keeps the last call's
 *     contents.  Calls that overlap on the GPU (e.g. on two unordered
 *     streams) race on it; serialise them. */
#define QUARTZ_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)
int32_t quartz_linear_noalloc(const quartz_encoded_t *a, const quartz_encoded_t *w,
                              const void *bias_f16, void *y, int32_t y_type, void *stream);

/* ---------------------------------------------------------------------------
 * QuaRTZ attention, one decode step (Appendix D, Table 6: attention kernels
 * for heads x 128 dimensions with LZS groups of 8 / 16 / 32).  The paper
 * gives no formula; here the query and a key / value cache are QuaRTZ-encoded
 * per token (Eq. 1 + Eq. 2 along the head dimension, 64-groups, symmetric
 * 8-bit codes), and for each of BH = batch x heads rows
 *     score_t = scale * sum_g s_q[g] s_k[t,g] P_g[t],
 *     P_g[t] = sum_{k in g} v_q[k] v_k[t,k]  (exact integer, as in the linear)
 *     o = sum_t softmax(score)_t s_v[t,g] v_v[t,.]
 * over the first L tokens of the head, softmax and value sum in binary32.
 * Cache layout: an encoded tensor of BH * L_max rows and K = 128 columns;
 * token t of head bh is row bh * L_max + t.
 * ------------------------------------------------------------------------- */

/* Workspace bytes of quartz_attention_decode (split-L partial results);
 * 0 for invalid sizes (BH outside [1, 65535], L outside [1, 2^30]). */
size_t quartz_attention_workspace_size(int64_t BH, int64_t L);

/* Encode new tokens into a cache: x_f16 fp16 [BH, T, K] (16-byte aligned)
 * goes to rows bh * L_max + t0 + j (j < T) of `cache` (BH * L_max rows,
 * K % 128 == 0, group_q 64, SYMMETRIC, 8-bit codes, any G_s and FLAG
 * storage), with the arithmetic of quartz_quantize.  Requires
 * 0 <= t0, t0 + T <= L_max.  T == 0 or BH == 0 is a no-op. */
int32_t quartz_kv_append(const void *x_f16, int64_t BH, int64_t T, const quartz_encoded_t *cache, int64_t L_max,
                         int64_t t0, void *stream);

/* One decode step of attention.
 *   q              encoded queries [BH, 128] (one per batch x head)
 *   k_cache        encoded keys   [BH * L_max, 128]
 *   v_cache        encoded values [BH * L_max, 128]
 *                  (all three: group_q 64, SYMMETRIC, 8-bit codes, the same
 *                  G_s; each may store its FLAGs in bytes or packed)
 *   L              tokens attended per head, 1 <= L <= L_max
 *   scale          softmax scale (finite; typically 1/sqrt(128))
 *   o              [BH, 128] of o_type (quartz_out_t), 16-byte aligned
 *   workspace      >= quartz_attention_workspace_size(BH, L) bytes, 16-byte
 *                  aligned, scratch owned by the caller
 * BH <= 65535. */
int32_t quartz_attention_decode(const quartz_encoded_t *q, const quartz_encoded_t *k_cache,
                                const quartz_encoded_t *v_cache, int64_t L_max, int64_t L, float scale, void *o,
                                int32_t o_type, void *workspace, size_t workspace_bytes, void *stream);

/* Synchronise `stream`, then read and clear the library's device error word.
 * Returns QUARTZ_OK, QUARTZ_ERR_TIMEOUT if a kernel gave up on a bounded
 * wait since the last call (its outputs are then invalid), or
 * QUARTZ_ERR_CUDA if the stream reports an error. */
int32_t quartz_device_status(void *stream);

/* Failure-detection self-test: launches one CTA that waits on an mbarrier
 * nothing ever arrives at, with a bound of `limit_ns` nanoseconds
 * (1e3 <= limit_ns <= 1e10).  The kernel gives up, records the timeout in
 * the device error word and returns; quartz_device_status then reports
 * QUARTZ_ERR_TIMEOUT.  The same bounded-wait routine guards every wait in
 * the GEMM pipeline. */
int32_t quartz_selftest_timeout(int64_t limit_ns, void *stream);

/* ---------------------------------------------------------------------------
 * Measurement aids.  The paper has no counterpart to these: they run one
 * execution pipe of the SM at full rate so that a benchmark can state the
 * linear layer's roofline against rates measured on the device at hand.
 * Their results are timing only; time them with events on `stream`.
 * ------------------------------------------------------------------------- */

/* `blocks` CTAs of 256 threads; every thread runs `iters` rounds of 8
 * independent fma.rn.f32x2 followed by 8 mul.rn.f32x2 (the paired fp32
 * operations of the GEMM's dequant epilogue): blocks * 256 * iters * 32
 * fp32 lane operations in total.  `sink` is a device float buffer of
 * blocks * 256 elements that receives one value per thread (keeps the work
 * observable).  1 <= blocks <= 2^20, 1 <= iters <= 2^32. */
int32_t quartz_probe_fp32_pipe(int32_t blocks, int64_t iters, float *sink, void *stream);

/* `blocks` CTAs (one per SM: each requests 200 KB of shared memory), each
 * issuing 2 * iters back-to-back tcgen05.mma.cta_group::1.kind::f8f6f4
 * M128 N256 K32 (E4M3 x E4M3 -> fp32 in TMEM) from one shared-memory stage:
 * blocks * iters * 2 * (2 * 128 * 256 * 32) flops.  Every wait is bounded;
 * a timeout is reported by quartz_device_status.  1 <= blocks <= 65535,
 * 1 <= iters <= 2^24. */
int32_t quartz_probe_mma_f8(int32_t blocks, int64_t iters, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* QUARTZ_H */
