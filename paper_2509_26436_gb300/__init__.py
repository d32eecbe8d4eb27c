"""QuaRTZ W4A4 linear hot path for GB300 (sm_103a).

Python front end of libquartz.so: it only marshals torch CUDA tensors into
the C ABI of include/quartz.h (device pointers, sizes, the current CUDA
stream).  Every step of the path (Eq. 1 quantization, Eq. 2 LZS encoding,
decode, the integer GEMM and the dequant epilogue) runs in the library's
CUDA kernels.

    e_a = quantize(x)                 # fp16 [M, K] -> encoded activations
    e_w = encode_weights(w)           # fp16 [N, K] -> encoded weights (offline)
    y = linear(e_a, e_w, bias)        # fp16 [M, N]

`inputs` (seeded synthetic data) imports nothing from here.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass

from . import _native as N
from ._native import (ALGO_SHIFT, ALGO_SIMT, ALGO_TCGEN05, ASYMMETRIC, OUT_BF16, OUT_F16, OUT_F32,  # noqa: F401
                      SYMMETRIC, QuartzError)

__all__ = ["Params", "Encoded", "quantize", "encode_weights", "dequantize", "linear",
           "linear_workspace_size", "empty_encoded", "device_status", "selftest_timeout",
           "kv_append", "attention_decode", "attention_workspace_size", "prepare_weights",
           "SYMMETRIC", "ASYMMETRIC", "QuartzError"]


def _torch():
    import torch
    return torch


@dataclass(frozen=True)
class Params:
    """group_q: min-max group along K (64, Appendix C, or K for one scale per
    row); group_s: LZS subgroup G_s (8/16/32/64, Section 3); mode: SYMMETRIC
    or ASYMMETRIC; flag_bits: 8 (one FLAG byte per subgroup) or 4 (two FLAGs
    per byte); code_bits: 8 (Eq. 1's codes) or 16 (the LLM variant of
    Section 5: 16-bit codes compressed straight to 4 bits, symmetric)."""
    group_q: int = 64
    group_s: int = 16
    mode: int = SYMMETRIC
    flag_bits: int = 8
    code_bits: int = 8

    def c(self) -> N.QuartzParams:
        return N.QuartzParams(self.group_q, self.group_s, self.mode, self.flag_bits, self.code_bits)


class Encoded:
    """An encoded [rows, K] tensor on the GPU (Section 4.4 storage format):
    codes uint8 [rows, K/2], flags uint8 [rows, K/G_s], scales fp16
    [rows, K/64], zeros int8 / gsum int32 [rows, K/64] (asymmetric only)."""

    def __init__(self, codes, flags, scales, zeros, gsum, rows, K, params: Params):
        self.codes, self.flags, self.scales = codes, flags, scales
        self.zeros, self.gsum = zeros, gsum
        self.rows, self.K, self.params = rows, K, params

    def c(self) -> N.QuartzEncoded:
        ptr = lambda t: None if t is None else t.data_ptr()  # noqa: E731
        return N.QuartzEncoded(ptr(self.codes), ptr(self.flags), ptr(self.scales), ptr(self.zeros),
                               ptr(self.gsum), self.rows, self.K, self.params.c())

    @property
    def nbytes(self) -> int:
        ts = [self.codes, self.flags, self.scales, self.zeros, self.gsum]
        return sum(t.numel() * t.element_size() for t in ts if t is not None)


def empty_encoded(rows: int, K: int, params: Params = Params(), device="cuda") -> Encoded:
    torch = _torch()
    sizes = (C.c_size_t * 5)()
    p = params.c()
    N.check(N.load().quartz_encoded_sizes(rows, K, C.byref(p), sizes), "quartz_encoded_sizes")
    G = K // params.group_q
    codes = torch.empty((rows, K // 2), dtype=torch.uint8, device=device)
    if params.flag_bits == 4:
        flags = torch.empty((max(int(sizes[1]), 1),), dtype=torch.uint8, device=device)
    else:
        flags = torch.empty((rows, K // params.group_s), dtype=torch.uint8, device=device)
    scales = torch.empty((rows, G), dtype=torch.float16, device=device)
    zeros = gsum = None
    if params.mode == ASYMMETRIC:
        zeros = torch.empty((rows, G), dtype=torch.int8, device=device)
        gsum = torch.empty((rows, G), dtype=torch.int32, device=device)
    return Encoded(codes, flags, scales, zeros, gsum, rows, K, params)


def _stream(stream=None) -> int:
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _check_f16(x, name):
    torch = _torch()
    if not (x.is_cuda and x.dtype == torch.float16 and x.dim() == 2 and x.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous 2-D float16 CUDA tensor")


def quantize(x, group_s: int = 16, mode: int = SYMMETRIC, out: Encoded | None = None,
             stream=None, _entry="quartz_quantize", group_q: int = 64, flag_bits: int = 8,
             code_bits: int = 8) -> Encoded:
    """Eq. 1 + Eq. 2 on fp16 activations [M, K] (K % 64 == 0); group_q = 64
    or K (one scale per row); code_bits = 16 for Section 5's LLM variant."""
    _check_f16(x, "x")
    rows, K = x.shape
    e = out if out is not None else empty_encoded(rows, K, Params(group_q, group_s, mode, flag_bits, code_bits),
                                                  x.device)
    ec = e.c()
    N.check(getattr(N.load(), _entry)(x.data_ptr(), C.byref(ec), _stream(stream)), _entry)
    return e


def encode_weights(w, group_s: int = 16, mode: int = SYMMETRIC, out: Encoded | None = None,
                   stream=None, group_q: int = 64, flag_bits: int = 8, code_bits: int = 8) -> Encoded:
    """The same encoder applied to nn.Linear weights [N, K], run offline
    (group_q = K gives per-output-channel scales)."""
    return quantize(w, group_s, mode, out, stream, _entry="quartz_encode_weights", group_q=group_q,
                    flag_bits=flag_bits, code_bits=code_bits)


def quantize_static(x, scale, group_s: int = 16, group_q: int = 64, out: Encoded | None = None,
                    stream=None, flag_bits: int = 8) -> Encoded:
    """Static per-tensor quantization: Eq. 1 with the given calibrated fp16
    scale for every element (symmetric), then Eq. 2."""
    import numpy as np
    _check_f16(x, "x")
    rows, K = x.shape
    e = out if out is not None else empty_encoded(rows, K, Params(group_q, group_s, SYMMETRIC, flag_bits), x.device)
    ec = e.c()
    bits = int(np.float16(scale).view(np.uint16))
    N.check(N.load().quartz_quantize_static(x.data_ptr(), bits, C.byref(ec), _stream(stream)),
            "quartz_quantize_static")
    return e


def dequantize(e: Encoded, stream=None, out=None):
    """x_hat = s (v - z) as fp16 [rows, K] (into `out` if given)."""
    torch = _torch()
    y = out if out is not None else torch.empty((e.rows, e.K), dtype=torch.float16, device=e.codes.device)
    if not (y.is_cuda and y.dtype == torch.float16 and y.is_contiguous() and y.numel() == e.rows * e.K):
        raise ValueError("out must be a contiguous float16 CUDA tensor of rows x K elements")
    ec = e.c()
    N.check(N.load().quartz_dequantize(C.byref(ec), y.data_ptr(), _stream(stream)), "quartz_dequantize")
    return y


def linear_workspace_size(M: int, N_: int, K: int, params: Params = Params()) -> int:
    p = params.c()
    return int(N.load().quartz_linear_workspace_size(M, N_, K, C.byref(p)))


def linear_launch_count(M: int, N_: int, K: int, params: Params = Params(), algo: int = ALGO_TCGEN05,
                        partials: bool = False) -> int:
    """Kernels one linear() call with these sizes launches on the current
    device (0: invalid arguments or M = 0)."""
    p = params.c()
    return int(N.load().quartz_linear_launch_count(M, N_, K, C.byref(p), algo, 1 if partials else 0))


_OUT = {"float16": OUT_F16, "bfloat16": OUT_BF16, "float32": OUT_F32}


def prepare_weights(w: Encoded, stream=None):
    """The weights' tensor-core operand and scale side values, prepared once
    (offline, like the encoding) for linear(..., w_prepared=...)."""
    torch = _torch()
    p = w.params.c()
    n = int(N.load().quartz_prepared_weights_size(w.rows, w.K, C.byref(p)))
    if n == 0:
        raise ValueError("invalid weight shape for preparation")
    buf = torch.empty(n, dtype=torch.uint8, device=w.codes.device)
    wc = w.c()
    N.check(N.load().quartz_prepare_weights(C.byref(wc), buf.data_ptr(), n, _stream(stream)),
            "quartz_prepare_weights")
    return buf


def linear(a: Encoded, w: Encoded, bias=None, out_dtype=None, out=None, workspace=None,
           partials_group: int | None = None, algo: int = ALGO_TCGEN05, stream=None,
           gemm_events=None, w_prepared=None):
    """W4A4 QuaRTZ linear: y = dequant(a) @ dequant(w)^T (+ bias), computed as
    exact integer group partials scaled by the 16-bit group scales.

    Returns y, or (y, partials) when `partials_group` is given (int32 [M, N]
    raw integer MMA sums of that 64-wide K group).  `gemm_events` = a pair
    of torch.cuda.Event recorded around the GEMM kernel alone.  Operands
    with 16-bit codes (Section 5 LLM variant) run on ALGO_TCGEN05 (E5M2
    operands, fp32 group sums) or ALGO_SHIFT (exact 64-bit group sums)."""
    torch = _torch()
    out_dtype = out_dtype or torch.float16
    M, Nn = a.rows, w.rows
    dev = a.codes.device
    y = out if out is not None else torch.empty((M, Nn), dtype=out_dtype, device=dev)
    y_type = _OUT[str(y.dtype).replace("torch.", "")]
    if workspace is None:
        workspace = torch.empty(max(linear_workspace_size(M, Nn, a.K, a.params), 16),
                                dtype=torch.uint8, device=dev)
    part = None
    if partials_group is not None:
        part = torch.empty((M, Nn), dtype=torch.int32, device=dev)
    if bias is not None and not (bias.dtype == torch.float16 and bias.is_cuda and bias.numel() == Nn):
        raise ValueError("bias must be a float16 CUDA tensor of N elements")
    ac, wc = a.c(), w.c()
    if gemm_events is not None:
        # torch creates events lazily and tracks their recording itself: a
        # first record through torch creates them; the library then
        # re-records them around the GEMM launch on the same stream.
        s_ = stream if stream is not None else torch.cuda.current_stream()
        for e in gemm_events:
            e.record(s_)
    opts = N.QuartzLinearOpts(None if part is None else part.data_ptr(),
                              0 if partials_group is None else partials_group, algo,
                              None if gemm_events is None else gemm_events[0].cuda_event,
                              None if gemm_events is None else gemm_events[1].cuda_event,
                              None if w_prepared is None else w_prepared.data_ptr())
    rc = N.load().quartz_linear_ex(
        C.byref(ac), C.byref(wc), None if bias is None else bias.data_ptr(), y.data_ptr(), y_type,
        workspace.data_ptr(), workspace.numel() * workspace.element_size(), C.byref(opts),
        _stream(stream))
    N.check(rc, "quartz_linear_ex")
    return y if part is None else (y, part)


def linear_f16(x, w: Encoded, bias=None, out_dtype=None, out=None, workspace=None,
               a_out: Encoded | None = None, stream=None, w_prepared=None):
    """Fused activation path: y = linear(quantize(x), w) from fp16 x [M, K]
    in one pass over x (the activations are encoded straight into the GEMM
    operand; symmetric mode, 8- or 16-bit codes as in w.params).  `a_out`
    optionally receives the encoding;
    `w_prepared` = prepare_weights(w) skips the per-call weight preparation."""
    torch = _torch()
    _check_f16(x, "x")
    out_dtype = out_dtype or torch.float16
    M, K = x.shape
    Nn = w.rows
    y = out if out is not None else torch.empty((M, Nn), dtype=out_dtype, device=x.device)
    y_type = _OUT[str(y.dtype).replace("torch.", "")]
    if workspace is None:
        workspace = torch.empty(max(linear_workspace_size(M, Nn, K, w.params), 16),
                                dtype=torch.uint8, device=x.device)
    if bias is not None and not (bias.dtype == torch.float16 and bias.is_cuda and bias.numel() == Nn):
        raise ValueError("bias must be a float16 CUDA tensor of N elements")
    wc = w.c()
    ac = a_out.c() if a_out is not None else None
    rc = N.load().quartz_linear_f16_ex(
        x.data_ptr(), M, C.byref(wc), None if w_prepared is None else w_prepared.data_ptr(),
        None if bias is None else bias.data_ptr(), y.data_ptr(), y_type,
        None if ac is None else C.byref(ac), workspace.data_ptr(),
        workspace.numel() * workspace.element_size(), _stream(stream))
    N.check(rc, "quartz_linear_f16_ex")
    return y


def device_status(stream=None) -> int:
    """Synchronise the stream; return (and clear) the library's device status."""
    return int(N.load().quartz_device_status(_stream(stream)))


def selftest_timeout(limit_ns: int, stream=None) -> int:
    return int(N.load().quartz_selftest_timeout(limit_ns, _stream(stream)))


# --- measurement aids (pipe-rate probes; no counterpart in the paper) -------

def probe_fp32_pipe(blocks: int, iters: int, sink, stream=None) -> int:
    """Launch the paired-fp32 probe; returns the fp32 lane operations it does
    (blocks * 256 * iters * 32).  `sink`: float32 CUDA tensor of >= blocks * 256."""
    if sink.numel() < blocks * 256 or not sink.is_cuda:
        raise ValueError("sink must be a float32 CUDA tensor of at least blocks * 256 elements")
    N.check(N.load().quartz_probe_fp32_pipe(blocks, iters, sink.data_ptr(), _stream(stream)),
            "quartz_probe_fp32_pipe")
    return blocks * 256 * iters * 32


def probe_mma_f8(blocks: int, iters: int, stream=None) -> int:
    """Launch the FP8 tcgen05 MMA probe; returns the flops it does
    (blocks * iters * 2 MMAs of 2 * 128 * 256 * 32)."""
    N.check(N.load().quartz_probe_mma_f8(blocks, iters, _stream(stream)), "quartz_probe_mma_f8")
    return blocks * iters * 2 * 2 * 128 * 256 * 32


# --- attention decode step (Appendix D, Table 6) ----------------------------

def attention_workspace_size(BH: int, L: int) -> int:
    return int(N.load().quartz_attention_workspace_size(BH, L))


def kv_append(x, cache: Encoded, L_max: int, t0: int, stream=None) -> None:
    """Encode fp16 x [BH, T, d] into cache rows bh * L_max + t0 + j."""
    torch = _torch()
    if not (x.is_cuda and x.dtype == torch.float16 and x.dim() == 3 and x.is_contiguous()):
        raise ValueError("x must be a contiguous [BH, T, d] float16 CUDA tensor")
    BH, T, _ = x.shape
    cc = cache.c()
    N.check(N.load().quartz_kv_append(x.data_ptr(), BH, T, C.byref(cc), L_max, t0, _stream(stream)),
            "quartz_kv_append")


def attention_decode(q: Encoded, k_cache: Encoded, v_cache: Encoded, L_max: int, L: int, scale: float,
                     out_dtype=None, out=None, workspace=None, stream=None):
    """o [BH, 128]: one encoded query per (batch x head) row attending over
    the first L tokens of that head's encoded key / value cache."""
    torch = _torch()
    out_dtype = out_dtype or torch.float16
    dev = q.codes.device
    o = out if out is not None else torch.empty((q.rows, q.K), dtype=out_dtype, device=dev)
    o_type = _OUT[str(o.dtype).replace("torch.", "")]
    if workspace is None:
        workspace = torch.empty(max(attention_workspace_size(q.rows, L), 16), dtype=torch.uint8, device=dev)
    qc, kc, vc = q.c(), k_cache.c(), v_cache.c()
    N.check(N.load().quartz_attention_decode(C.byref(qc), C.byref(kc), C.byref(vc), L_max, L, float(scale),
                                             o.data_ptr(), o_type, workspace.data_ptr(),
                                             workspace.numel() * workspace.element_size(), _stream(stream)),
            "quartz_attention_decode")
    return o
