// Host side of the C ABI declared in include/quartz.h: argument validation,
// workspace carving and kernel launches.  Nothing here allocates device
// memory or synchronises, except quartz_device_status.
#include <atomic>
#include <cstring>

#include "quartz_internal.h"

namespace quartz {
namespace {

__device__ int g_device_error;

constexpr int kMaxDevices = 64;
// per device, looked up on first use (any host thread; they all store the same value)
std::atomic<int *> g_error_ptr[kMaxDevices] = {};

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int32_t check_params(const quartz_params_t *p)
{
    if (!p) return QUARTZ_ERR_INVALID_ARG;
    if (p->mode != QUARTZ_SYMMETRIC && p->mode != QUARTZ_ASYMMETRIC) return QUARTZ_ERR_INVALID_ARG;
    if (p->flag_bits != 0 && p->flag_bits != 4 && p->flag_bits != 8) return QUARTZ_ERR_INVALID_ARG;
    if (p->group_s != 8 && p->group_s != 16 && p->group_s != 32 && p->group_s != 64)
        return QUARTZ_ERR_INVALID_ARG;
    if (p->group_q <= 0 || p->group_q % p->group_s != 0) return QUARTZ_ERR_INVALID_ARG;
    if (p->group_q % 64 != 0) return QUARTZ_ERR_UNSUPPORTED;
    if (p->code_bits != 0 && p->code_bits != 8 && p->code_bits != 16) return QUARTZ_ERR_INVALID_ARG;
    // 16-bit stage-1 codes (Section 5 LLM variant): symmetric groups of 64
    if (p->code_bits == 16 && (p->mode != QUARTZ_SYMMETRIC || p->group_q != 64)) return QUARTZ_ERR_UNSUPPORTED;
    return QUARTZ_OK;
}

bool wide_codes(const quartz_params_t &p) { return p.code_bits == 16; }

int32_t check_shape(int64_t rows, int64_t K, const quartz_params_t *p)
{
    const int32_t rc = check_params(p);
    if (rc) return rc;
    if (rows < 0 || K <= 0 || K % p->group_q != 0) return QUARTZ_ERR_INVALID_ARG;
    if (rows > (int64_t(1) << 31) || K > (int64_t(1) << 24)) return QUARTZ_ERR_UNSUPPORTED;
    // groups of 64 along K (Appendix C), or one group per row (per-token /
    // per-channel scales, symmetric)
    if (p->group_q != 64 && (p->group_q != K || p->mode != QUARTZ_SYMMETRIC)) return QUARTZ_ERR_UNSUPPORTED;
    return QUARTZ_OK;
}

int32_t check_encoded(const quartz_encoded_t *e)
{
    if (!e) return QUARTZ_ERR_INVALID_ARG;
    const int32_t rc = check_shape(e->rows, e->K, &e->p);
    if (rc) return rc;
    if (e->rows == 0) return QUARTZ_OK;
    if (!e->codes || !e->flags || !e->scales) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(e->codes) || !aligned16(e->flags) || !aligned16(e->scales))
        return QUARTZ_ERR_ALIGNMENT;
    if (e->p.mode == QUARTZ_ASYMMETRIC) {
        if (!e->zeros || !e->gsum) return QUARTZ_ERR_INVALID_ARG;
        if (!aligned16(e->zeros) || !aligned16(e->gsum)) return QUARTZ_ERR_ALIGNMENT;
    }
    return QUARTZ_OK;
}

int32_t map_cuda(cudaError_t e) { return e == cudaSuccess ? QUARTZ_OK : QUARTZ_ERR_CUDA; }

}  // namespace

int *device_error_word()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    int *ptr = g_error_ptr[dev].load(std::memory_order_acquire);
    if (!ptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) return nullptr;
        ptr = static_cast<int *>(p);
        g_error_ptr[dev].store(ptr, std::memory_order_release);
    }
    return ptr;
}

}  // namespace quartz

using namespace quartz;

extern "C" {

const char *quartz_status_string(int32_t status)
{
    switch (status) {
        case QUARTZ_OK: return "QUARTZ_OK";
        case QUARTZ_ERR_INVALID_ARG: return "QUARTZ_ERR_INVALID_ARG";
        case QUARTZ_ERR_ALIGNMENT: return "QUARTZ_ERR_ALIGNMENT";
        case QUARTZ_ERR_UNSUPPORTED: return "QUARTZ_ERR_UNSUPPORTED";
        case QUARTZ_ERR_CUDA: return "QUARTZ_ERR_CUDA";
        case QUARTZ_ERR_TIMEOUT: return "QUARTZ_ERR_TIMEOUT";
        case QUARTZ_ERR_WORKSPACE: return "QUARTZ_ERR_WORKSPACE";
        default: return "QUARTZ_ERR_UNKNOWN";
    }
}

int32_t quartz_version(void) { return (1 << 16) | 7; }

int32_t quartz_encoded_sizes(int64_t rows, int64_t K, const quartz_params_t *p, size_t out[5])
{
    if (!out) return QUARTZ_ERR_INVALID_ARG;
    const int32_t rc = check_shape(rows, K, p);
    if (rc) return rc;
    const int64_t G = K / p->group_q;
    out[0] = static_cast<size_t>(rows * (K / 2));
    out[1] = static_cast<size_t>(p->flag_bits == 4 ? (rows * (K / p->group_s) + 1) / 2 : rows * (K / p->group_s));
    out[2] = static_cast<size_t>(rows * G * 2);
    out[3] = static_cast<size_t>(rows * G);
    out[4] = static_cast<size_t>(rows * G * 4);
    return QUARTZ_OK;
}

int32_t quartz_quantize(const void *x_f16, const quartz_encoded_t *out, void *stream)
{
    int32_t rc = check_encoded(out);
    if (rc) return rc;
    if (out->rows == 0) return QUARTZ_OK;
    if (!x_f16) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(x_f16)) return QUARTZ_ERR_ALIGNMENT;
    return map_cuda(launch_quantize(x_f16, out, static_cast<cudaStream_t>(stream)));
}

int32_t quartz_quantize_static(const void *x_f16, uint16_t scale_f16, const quartz_encoded_t *out, void *stream)
{
    int32_t rc = check_encoded(out);
    if (rc) return rc;
    if (out->p.mode != QUARTZ_SYMMETRIC || wide_codes(out->p)) return QUARTZ_ERR_UNSUPPORTED;
    // a finite, non-negative fp16 scale
    if ((scale_f16 & 0x8000u) && scale_f16 != 0x8000u) return QUARTZ_ERR_INVALID_ARG;
    if ((scale_f16 & 0x7C00u) == 0x7C00u) return QUARTZ_ERR_INVALID_ARG;
    if (out->rows == 0) return QUARTZ_OK;
    if (!x_f16) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(x_f16)) return QUARTZ_ERR_ALIGNMENT;
    return map_cuda(launch_quantize_static(x_f16, out, static_cast<uint16_t>(scale_f16 & 0x7FFFu),
                                           static_cast<cudaStream_t>(stream)));
}

int32_t quartz_encode_weights(const void *w_f16, const quartz_encoded_t *out, void *stream)
{
    return quartz_quantize(w_f16, out, stream);
}

int32_t quartz_dequantize(const quartz_encoded_t *e, void *x_hat_f16, void *stream)
{
    int32_t rc = check_encoded(e);
    if (rc) return rc;
    if (e->rows == 0) return QUARTZ_OK;
    if (!x_hat_f16) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(x_hat_f16)) return QUARTZ_ERR_ALIGNMENT;
    return map_cuda(launch_dequantize(e, x_hat_f16, static_cast<cudaStream_t>(stream)));
}

size_t quartz_linear_workspace_size(int64_t M, int64_t N, int64_t K, const quartz_params_t *p)
{
    if (check_shape(M, K, p) != QUARTZ_OK || N <= 0 || N % 8 != 0) return 0;
    return linear_workspace_bytes(M, N, K, p->mode);
}

int32_t quartz_linear_launch_count(int64_t M, int64_t N, int64_t K, const quartz_params_t *p, int32_t algo,
                                   int32_t with_partials)
{
    if (check_shape(M, K, p) != QUARTZ_OK || N <= 0 || N % 8 != 0) return 0;
    if (algo != QUARTZ_ALGO_TCGEN05 && algo != QUARTZ_ALGO_SIMT && algo != QUARTZ_ALGO_SHIFT) return 0;
    if (M == 0) return 0;
    const bool split = algo == QUARTZ_ALGO_TCGEN05 && p->mode == QUARTZ_SYMMETRIC && !with_partials &&
                       p->group_q == 64 && linear_tail_parts(M, N, K, p->mode) > 1;
    return split ? 3 : 2;
}

int32_t quartz_linear_ex(const quartz_encoded_t *a, const quartz_encoded_t *w,
                         const void *bias_f16, void *y, int32_t y_type, void *workspace,
                         size_t workspace_bytes, const quartz_linear_opts_t *opts, void *stream)
{
    quartz_linear_opts_t o;
    std::memset(&o, 0, sizeof(o));
    if (opts) o = *opts;
    int32_t *partials = o.partials;
    const int32_t partials_group = o.partials_group;
    const int32_t algo = o.algo;
    int32_t rc = check_encoded(a);
    if (rc) return rc;
    rc = check_encoded(w);
    if (rc) return rc;
    if (a->K != w->K || a->p.group_q != w->p.group_q || a->p.group_s != w->p.group_s ||
        a->p.mode != w->p.mode || wide_codes(a->p) != wide_codes(w->p))
        return QUARTZ_ERR_INVALID_ARG;
    const bool wide = wide_codes(a->p);
    // 16-bit codes: decoded values up to 7 << 12 (E5M2 operands for the
    // tensor cores, no E4M3 SIMT path) and group sums beyond int32
    if (wide && (o.algo == QUARTZ_ALGO_SIMT || partials)) return QUARTZ_ERR_UNSUPPORTED;
    const bool per_row = a->p.group_q != 64;  // group_q == K (check_shape allows nothing else)
    if (per_row && o.algo != QUARTZ_ALGO_TCGEN05) return QUARTZ_ERR_UNSUPPORTED;
    const int64_t M = a->rows, N = w->rows, K = a->K;
    if (N <= 0 || N % 8 != 0 || N > (int64_t(1) << 24)) return QUARTZ_ERR_INVALID_ARG;
    if (y_type != QUARTZ_OUT_F16 && y_type != QUARTZ_OUT_BF16 && y_type != QUARTZ_OUT_F32)
        return QUARTZ_ERR_INVALID_ARG;
    if (algo != QUARTZ_ALGO_TCGEN05 && algo != QUARTZ_ALGO_SIMT && algo != QUARTZ_ALGO_SHIFT)
        return QUARTZ_ERR_INVALID_ARG;
    if (partials && (partials_group < 0 || partials_group >= K / a->p.group_q))
        return QUARTZ_ERR_INVALID_ARG;
    if (M * N >= (int64_t(1) << 40)) return QUARTZ_ERR_UNSUPPORTED;
    if (M == 0) return QUARTZ_OK;
    if (!y) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(y) || (bias_f16 && !aligned16(bias_f16)) || (partials && !aligned16(partials)))
        return QUARTZ_ERR_ALIGNMENT;
    const size_t need = linear_workspace_bytes(M, N, K, a->p.mode);
    if (!workspace || workspace_bytes < need) return QUARTZ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return QUARTZ_ERR_ALIGNMENT;
    if (o.w_prepared && !aligned16(o.w_prepared)) return QUARTZ_ERR_ALIGNMENT;
    int *dev_err = device_error_word();
    if (!dev_err) return QUARTZ_ERR_CUDA;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    LinearWorkspace ws;
    linear_workspace_carve(workspace, M, N, K, a->p.mode, &ws);
    if (o.w_prepared) prepared_weights_carve(o.w_prepared, N, K, a->p.mode, &ws);
    cudaError_t e = launch_prepare(a, w, ws, s, algo != QUARTZ_ALGO_SHIFT, o.w_prepared != nullptr);
    if (e != cudaSuccess) return QUARTZ_ERR_CUDA;
    if (o.gemm_event_begin && cudaEventRecord(static_cast<cudaEvent_t>(o.gemm_event_begin), s) != cudaSuccess)
        return QUARTZ_ERR_CUDA;
    if (algo == QUARTZ_ALGO_SIMT)
        e = launch_gemm_simt(ws, M, N, K, a->p.mode, bias_f16, y, y_type, partials, partials_group, s);
    else if (algo == QUARTZ_ALGO_SHIFT)
        e = launch_gemm_shift(ws, a, w, bias_f16, y, y_type, partials, partials_group, s, wide);
    else
        e = launch_gemm_tcgen05(ws, M, N, K, a->p.mode, bias_f16, y, y_type, partials,
                                partials_group, dev_err, s, per_row, wide);
    if (e == cudaSuccess && o.gemm_event_end)
        e = cudaEventRecord(static_cast<cudaEvent_t>(o.gemm_event_end), s);
    return map_cuda(e);
}

size_t quartz_prepared_weights_size(int64_t N, int64_t K, const quartz_params_t *p)
{
    if (check_shape(N, K, p) != QUARTZ_OK || N <= 0 || N % 8 != 0 || N > (int64_t(1) << 24)) return 0;
    return prepared_weights_bytes(N, K, p->mode);
}

int32_t quartz_prepare_weights(const quartz_encoded_t *w, void *prepared, size_t prepared_bytes, void *stream)
{
    int32_t rc = check_encoded(w);
    if (rc) return rc;
    const int64_t N = w->rows, K = w->K;
    if (N <= 0 || N % 8 != 0 || N > (int64_t(1) << 24)) return QUARTZ_ERR_INVALID_ARG;
    if (!prepared || prepared_bytes < prepared_weights_bytes(N, K, w->p.mode)) return QUARTZ_ERR_WORKSPACE;
    if (!aligned16(prepared)) return QUARTZ_ERR_ALIGNMENT;
    LinearWorkspace ws{};
    prepared_weights_carve(prepared, N, K, w->p.mode, &ws);
    return map_cuda(launch_prepare(nullptr, w, ws, static_cast<cudaStream_t>(stream)));
}

int32_t quartz_linear(const quartz_encoded_t *a, const quartz_encoded_t *w, const void *bias_f16,
                      void *y, int32_t y_type, void *workspace, size_t workspace_bytes,
                      void *stream)
{
    return quartz_linear_ex(a, w, bias_f16, y, y_type, workspace, workspace_bytes, nullptr, stream);
}

int32_t quartz_linear_f16(const void *x_f16, int64_t M, const quartz_encoded_t *w, const void *bias_f16,
                          void *y, int32_t y_type, const quartz_encoded_t *a_out, void *workspace,
                          size_t workspace_bytes, void *stream)
{
    return quartz_linear_f16_ex(x_f16, M, w, nullptr, bias_f16, y, y_type, a_out, workspace, workspace_bytes,
                                stream);
}

int32_t quartz_linear_f16_ex(const void *x_f16, int64_t M, const quartz_encoded_t *w, const void *w_prepared,
                             const void *bias_f16, void *y, int32_t y_type, const quartz_encoded_t *a_out,
                             void *workspace, size_t workspace_bytes, void *stream)
{
    int32_t rc = check_encoded(w);
    if (rc) return rc;
    if (w->p.mode != QUARTZ_SYMMETRIC || w->p.group_q != 64) return QUARTZ_ERR_UNSUPPORTED;
    const bool wide = wide_codes(w->p);  // 16-bit stage-1 codes: E5M2 operands
    const int64_t N = w->rows, K = w->K;
    rc = check_shape(M, K, &w->p);
    if (rc) return rc;
    if (N <= 0 || N % 8 != 0 || N > (int64_t(1) << 24)) return QUARTZ_ERR_INVALID_ARG;
    if (y_type != QUARTZ_OUT_F16 && y_type != QUARTZ_OUT_BF16 && y_type != QUARTZ_OUT_F32)
        return QUARTZ_ERR_INVALID_ARG;
    if (a_out) {
        rc = check_encoded(a_out);
        if (rc) return rc;
        if (a_out->rows != M || a_out->K != K || a_out->p.group_q != w->p.group_q ||
            a_out->p.group_s != w->p.group_s || a_out->p.mode != w->p.mode || wide_codes(a_out->p) != wide)
            return QUARTZ_ERR_INVALID_ARG;
    }
    if (M * N >= (int64_t(1) << 40)) return QUARTZ_ERR_UNSUPPORTED;
    if (M == 0) return QUARTZ_OK;
    if (!x_f16 || !y) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(x_f16) || !aligned16(y) || (bias_f16 && !aligned16(bias_f16)) ||
        (w_prepared && !aligned16(w_prepared)))
        return QUARTZ_ERR_ALIGNMENT;
    const size_t need = linear_workspace_bytes(M, N, K, w->p.mode);
    if (!workspace || workspace_bytes < need) return QUARTZ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return QUARTZ_ERR_ALIGNMENT;
    int *dev_err = device_error_word();
    if (!dev_err) return QUARTZ_ERR_CUDA;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    LinearWorkspace ws;
    linear_workspace_carve(workspace, M, N, K, w->p.mode, &ws);
    if (w_prepared) prepared_weights_carve(w_prepared, N, K, w->p.mode, &ws);
    cudaError_t e = launch_encode_operand(x_f16, M, K, &w->p, ws, a_out, s);
    if (e == cudaSuccess && !w_prepared) e = launch_prepare(nullptr, w, ws, s);
    if (e == cudaSuccess)
        e = launch_gemm_tcgen05(ws, M, N, K, w->p.mode, bias_f16, y, y_type, nullptr, 0, dev_err, s, false, wide);
    return map_cuda(e);
}

namespace {
// Encoded tensors of the attention step: 128 columns (the head dimension),
// 64-groups, symmetric 8-bit codes, the same G_s.
int32_t check_attention_operand(const quartz_encoded_t *e, int group_s)
{
    const int32_t rc = check_encoded(e);
    if (rc) return rc;
    if (e->K != 128 || e->p.group_s != group_s) return QUARTZ_ERR_INVALID_ARG;
    if (e->p.group_q != 64 || e->p.mode != QUARTZ_SYMMETRIC || wide_codes(e->p)) return QUARTZ_ERR_UNSUPPORTED;
    return QUARTZ_OK;
}
}  // namespace

size_t quartz_attention_workspace_size(int64_t BH, int64_t L)
{
    if (BH <= 0 || BH > 65535 || L <= 0 || L > (int64_t(1) << 30)) return 0;
    return attention_workspace_bytes(BH, L);
}

int32_t quartz_kv_append(const void *x_f16, int64_t BH, int64_t T, const quartz_encoded_t *cache, int64_t L_max,
                         int64_t t0, void *stream)
{
    if (!cache) return QUARTZ_ERR_INVALID_ARG;
    int32_t rc = check_encoded(cache);
    if (rc) return rc;
    if (cache->p.mode != QUARTZ_SYMMETRIC || cache->p.group_q != 64 || wide_codes(cache->p))
        return QUARTZ_ERR_UNSUPPORTED;
    if (cache->K % 128 != 0) return QUARTZ_ERR_UNSUPPORTED;
    if (BH < 0 || T < 0 || L_max <= 0 || t0 < 0 || t0 + T > L_max || cache->rows != BH * L_max)
        return QUARTZ_ERR_INVALID_ARG;
    if (BH == 0 || T == 0) return QUARTZ_OK;
    if (!x_f16) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(x_f16)) return QUARTZ_ERR_ALIGNMENT;
    return map_cuda(launch_kv_append(x_f16, BH, T, cache, L_max, t0, static_cast<cudaStream_t>(stream)));
}

int32_t quartz_attention_decode(const quartz_encoded_t *q, const quartz_encoded_t *k_cache,
                                const quartz_encoded_t *v_cache, int64_t L_max, int64_t L, float scale, void *o,
                                int32_t o_type, void *workspace, size_t workspace_bytes, void *stream)
{
    if (!q || !k_cache || !v_cache) return QUARTZ_ERR_INVALID_ARG;
    int32_t rc = check_attention_operand(q, q->p.group_s);
    if (rc) return rc;
    if ((rc = check_attention_operand(k_cache, q->p.group_s)) != QUARTZ_OK) return rc;
    if ((rc = check_attention_operand(v_cache, q->p.group_s)) != QUARTZ_OK) return rc;
    const int64_t BH = q->rows;
    if (BH > 65535 || L_max <= 0 || L <= 0 || L > L_max || L > (int64_t(1) << 30) ||
        BH * ((L + 127) / 128) > (int64_t(1) << 31) ||
        k_cache->rows != BH * L_max || v_cache->rows != BH * L_max)
        return QUARTZ_ERR_INVALID_ARG;
    if (!(scale == scale) || scale > 3.0e38f || scale < -3.0e38f) return QUARTZ_ERR_INVALID_ARG;  // finite
    if (o_type != QUARTZ_OUT_F16 && o_type != QUARTZ_OUT_BF16 && o_type != QUARTZ_OUT_F32)
        return QUARTZ_ERR_INVALID_ARG;
    if (BH == 0) return QUARTZ_OK;
    if (!o) return QUARTZ_ERR_INVALID_ARG;
    if (!aligned16(o)) return QUARTZ_ERR_ALIGNMENT;
    if (!workspace || workspace_bytes < attention_workspace_bytes(BH, L)) return QUARTZ_ERR_WORKSPACE;
    if (!aligned16(workspace)) return QUARTZ_ERR_ALIGNMENT;
    return map_cuda(launch_attention_decode(q, k_cache, v_cache, L_max, L, scale, o, o_type, workspace,
                                            static_cast<cudaStream_t>(stream)));
}

int32_t quartz_device_status(void *stream)
{
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return QUARTZ_ERR_CUDA;
    int *p = device_error_word();
    if (!p) return QUARTZ_ERR_CUDA;
    int v = 0;
    const int zero = 0;
    if (cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return QUARTZ_ERR_CUDA;
    if (cudaMemcpy(p, &zero, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess) return QUARTZ_ERR_CUDA;
    return v == QUARTZ_DEV_TIMEOUT ? QUARTZ_ERR_TIMEOUT : QUARTZ_OK;
}

int32_t quartz_selftest_timeout(int64_t limit_ns, void *stream)
{
    if (limit_ns < 1000 || limit_ns > 10000000000ll) return QUARTZ_ERR_INVALID_ARG;
    int *dev_err = device_error_word();
    if (!dev_err) return QUARTZ_ERR_CUDA;
    return map_cuda(launch_selftest_timeout(limit_ns, dev_err, static_cast<cudaStream_t>(stream)));
}

int32_t quartz_probe_fp32_pipe(int32_t blocks, int64_t iters, float *sink, void *stream)
{
    if (blocks < 1 || blocks > (1 << 20) || iters < 1 || iters > (int64_t(1) << 32) || !sink)
        return QUARTZ_ERR_INVALID_ARG;
    return map_cuda(launch_probe_fp32(blocks, iters, sink, static_cast<cudaStream_t>(stream)));
}

int32_t quartz_probe_mma_f8(int32_t blocks, int64_t iters, void *stream)
{
    if (blocks < 1 || blocks > (1 << 16) || iters < 1 || iters > (int64_t(1) << 24)) return QUARTZ_ERR_INVALID_ARG;
    int *dev_err = device_error_word();
    if (!dev_err) return QUARTZ_ERR_CUDA;
    return map_cuda(launch_probe_mma_f8(blocks, iters, dev_err, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
