// Declarations shared by the translation units of libquartz (not installed).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "quartz.h"

namespace quartz {

// Values of the library's device error word (0 = no error).
constexpr int QUARTZ_DEV_OK = 0;
constexpr int QUARTZ_DEV_TIMEOUT = 1;

// Upper bound on any single mbarrier wait inside a kernel.  No legitimate
// wait on a healthy GPU comes near it; it only turns a would-be hang into an
// error status.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// Device error word of the current device (see api.cu).
int *device_error_word();

// Programmatic dependent launch.  The library's kernels are launched with
// launch_pdl, which lets the launch of a kernel overlap the end of the
// previous kernel in the stream.  Every such kernel calls griddep_wait()
// before it reads or writes global memory: the wait returns once the
// previous kernel has completed and its writes are visible (at once under
// an ordinary launch), so stream order holds, and holds transitively,
// because that kernel waited in turn before its own first access.  No
// kernel triggers its dependents early (griddepcontrol.launch_dependents):
// measured on whole steps, an early trigger made the FLUX block 2% slower
// (dependent CTAs parked on the SMs ahead of the primary's last blocks),
// while the plain form is 1-8% faster than ordinary launches.
#ifdef __CUDACC__
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}
#endif

// Encoder / decoder launches (quantize.cu).  Arguments are pre-validated.
cudaError_t launch_quantize(const void *x, const quartz_encoded_t *out, cudaStream_t s);
// Attention decode step (attention.cu): encode x [BH, T, d] into cache rows
// bh * L_max + t0 + j (quantize.cu), and one query per bh row over the first
// L cached tokens of that head.
cudaError_t launch_kv_append(const void *x, int64_t BH, int64_t T, const quartz_encoded_t *cache, int64_t L_max,
                             int64_t t0, cudaStream_t s);
size_t attention_workspace_bytes(int64_t BH, int64_t L);
cudaError_t launch_attention_decode(const quartz_encoded_t *q, const quartz_encoded_t *k, const quartz_encoded_t *v,
                                    int64_t L_max, int64_t L, float scale, void *o, int o_type, void *workspace,
                                    cudaStream_t s);
cudaError_t launch_dequantize(const quartz_encoded_t *e, void *y, cudaStream_t s);
// Symmetric encoding with a static (calibrated) fp16 scale `s16` for every group.
cudaError_t launch_quantize_static(const void *x, const quartz_encoded_t *out, uint16_t s16, cudaStream_t s);

// Position of activation row r in its group's side-value row: inside every
// block of 32 rows, row 8a + b sits at 4b + a, so that the four rows
// b + {0, 8, 16, 24} one epilogue thread scales are one 16-byte vector.
__host__ __device__ __forceinline__ int64_t perm32(int64_t r)
{
    return (r & ~int64_t(31)) | ((r & 7) << 2) | ((r >> 3) & 3);
}

// Linear-layer workspace and launches (linear.cu).
struct LinearWorkspace {
    void *a_op;      // E4M3 [M, K]  decoded activations
    void *w_op;      // E4M3 [round_up(N, 16), K]  decoded weights, rows transposed 4x4 inside 16-row blocks
    float *a_side;   // fp32 [nside][G][Mpad]  scale (and z, gsum when asymmetric)
    float *w_side;   // fp32 [nside][G][Npad]
    float *tail_part;  // fp32 partial tiles of the split last wave (may be NULL)
    int64_t m_pad, n_pad;
    int nside;
    int tail_tiles, tail_split;  // tiles of the split last wave(s) and parts per tile (1 = no split)
    int tail_ls;                 // two-wave form: group iterations per CTA (0: one-wave form)
};
size_t linear_workspace_bytes(int64_t M, int64_t N, int64_t K, int mode);
// Parts each tile of the symmetric tcgen05 GEMM's split last wave is cut
// into on the current device (1: no split).
int linear_tail_parts(int64_t M, int64_t N, int64_t K, int mode);
void linear_workspace_carve(void *base, int64_t M, int64_t N, int64_t K, int mode,
                            LinearWorkspace *ws);
// Expands the operands to E4M3 and transposes their scales into the
// workspace (one launch).  `a` may be NULL: then only the weight operand is
// prepared (the fused encoder below has written the activation side).  With
// `expand` false only the scales are transposed (accumulator-shift GEMM).
// With `w_ready` the weight operand and its side values are already in
// ws.w_op / ws.w_side (prepared once, quartz_prepare_weights) and only the
// activation jobs run.
cudaError_t launch_prepare(const quartz_encoded_t *a, const quartz_encoded_t *w, const LinearWorkspace &ws,
                           cudaStream_t s, bool expand = true, bool w_ready = false);
// Layout of a prepared weight operand: the expanded operand [round_up(N, 16),
// K] bytes, then the side values [nside][K/64][round_up(N, 256)] fp32.
size_t prepared_weights_bytes(int64_t N, int64_t K, int mode);
void prepared_weights_carve(const void *base, int64_t N, int64_t K, int mode, LinearWorkspace *ws);
// The paper's accumulator-shift schedule on CUDA cores, from the packed codes;
// `wide`: 16-bit stage-1 codes (FLAGs up to 12, 64-bit group sums).
cudaError_t launch_gemm_shift(const LinearWorkspace &ws, const quartz_encoded_t *a, const quartz_encoded_t *w,
                              const void *bias, void *y, int y_type, int32_t *partials, int partials_group,
                              cudaStream_t s, bool wide = false);
// Fused activation path (quantize.cu, symmetric mode): Eq. 1 + Eq. 2 on fp16
// x [M, K] written straight into the workspace as E4M3 operand and scale
// side values; `enc` (may be NULL) also receives the encoded tensor.
cudaError_t launch_encode_operand(const void *x, int64_t M, int64_t K, const quartz_params_t *p,
                                  const LinearWorkspace &ws, const quartz_encoded_t *enc, cudaStream_t s);
// per_row: one scale per row of both operands (group_q = K, symmetric).
cudaError_t launch_gemm_tcgen05(const LinearWorkspace &ws, int64_t M, int64_t N, int64_t K,
                                int mode, const void *bias, void *y, int y_type,
                                int32_t *partials, int partials_group, int *dev_err,
                                cudaStream_t s, bool per_row = false, bool wide = false);
cudaError_t launch_gemm_simt(const LinearWorkspace &ws, int64_t M, int64_t N, int64_t K, int mode,
                             const void *bias, void *y, int y_type, int32_t *partials,
                             int partials_group, cudaStream_t s);
cudaError_t launch_selftest_timeout(int64_t limit_ns, int *dev_err, cudaStream_t s);
// Pipe-rate probes (probe.cu).
cudaError_t launch_probe_fp32(int blocks, int64_t iters, float *sink, cudaStream_t s);
cudaError_t launch_probe_mma_f8(int blocks, int64_t iters, int *dev_err, cudaStream_t s);

}  // namespace quartz
