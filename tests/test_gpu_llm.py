"""GPU parity of the LLM variant (Section 5: 16-bit activations compressed
straight to 4 bits, G_s = 8) against the CPU oracle.

* Encoder: codes, FLAGs (0..12) and fp16 scale bits bit-exact against
  oracle.encode16, including saturated groups, subnormal scales and packed
  FLAG storage; the dequantiser bit-exact against the oracle's binary64
  value rounded once to fp16.
* Linear, accumulator-shift GEMM (64-bit group sums): outputs against the
  oracle's binary64 y.  Tolerance from the kernel's arithmetic: P_g is exact
  in 64 bits and is rounded once to binary32; s_a*(s_w*P_g) adds two more
  roundings and the G-term running sum G more, so |y_gpu - y| <=
  (G + 5) 2^-24 sum_g |s_a s_w D_g| before the output conversion (relative
  2^-11 for fp16, 2^-8 for bf16).
* Linear, tcgen05 GEMM on E5M2 operands: every product is exact, but the
  64 products of a group are summed in the tensor cores' fp32 accumulator;
  at most one rounding per product gives a further 64 2^-24
  sum_g s_a s_w sum_k |v_a v_w| (the magnitude of the group's products).
"""
import numpy as np
import pytest

import oracle as O
from paper_2509_26436_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

REL = {"float16": 1e-3, "bfloat16": 4e-3, "float32": 1e-5}


@pytest.fixture(scope="module")
def Q():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2509_26436_gb300 as Q
    return Q


def _enc(Q, x16, gs=8, flag_bits=8):
    e = Q.quantize(torch.from_numpy(x16).cuda(), group_s=gs, code_bits=16, flag_bits=flag_bits)
    torch.cuda.synchronize()
    return e


def _assert_equal(e, ref):
    assert np.array_equal(e.codes.cpu().numpy(), ref.codes)
    assert np.array_equal(e.flags.cpu().numpy(), ref.flags)
    assert np.array_equal(e.scales.cpu().numpy().view(np.uint16), ref.scales.view(np.uint16))


def _pack_flags(flags):
    f = flags.reshape(-1).astype(np.uint8)
    if f.size % 2:
        f = np.concatenate([f, np.zeros(1, np.uint8)])
    return f[0::2] | (f[1::2] << 4)


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("shape", [(1, 64), (3, 128), (37, 1152), (129, 4096), (1000, 640)])
def test_encode16_bit_exact(Q, gs, shape):
    x = inputs.mixture_activations(*shape, seed=5000 + shape[0] + gs)
    _assert_equal(_enc(Q, x, gs), O.encode16(x, 64, gs))


def test_encode16_edge_values(Q):
    """Zero groups, scale underflow, subnormal scales (max|x| < 2), fp16
    extremes (x r lands on 32768 and saturates), ties and all-equal groups."""
    rows = [np.zeros(256), np.full(256, 1e-7), np.linspace(-3e-4, 3e-4, 256),
            np.concatenate([np.full(64, 65504.0), -np.full(64, 65504.0), np.full(64, 4.0),
                            np.linspace(-4, 4, 64)]),
            np.concatenate([np.full(64, 0.5), np.arange(64) * 2.0 ** -13, np.arange(64) * 1.5 * 2.0 ** -14,
                            -np.arange(64) * 2.0 ** -10]),
            np.tile([1.0, -1.0, 1e-3, -1e-3], 64)]
    x = np.stack(rows).astype(np.float16)
    for gs in (8, 16, 32, 64):
        ref = O.encode16(x, 64, gs)
        _assert_equal(_enc(Q, x, gs), ref)
    assert ref.flags.max() == 12


def test_encode16_cap_every_fp16_maximum(Q):
    """The 32767 cap at every scale: one 64-element group per positive finite
    fp16 maximum (31743 rows, normal and subnormal scales), holding that
    maximum and the 63 fp16 values just below it with seeded signs.  The
    fp16 scale rounds down for about half of the maxima, so rne(|x| r)
    passes 32767 (up to about 1.5 x 32767 for the smallest subnormal scales)
    for the values nearest the maximum; codes, FLAGs and scales must still be
    Eq. 1 + Eq. 2's with the cap, at every G_s."""
    top = np.arange(1, 0x7C00, dtype=np.int64)
    bits = np.clip(top[:, None] - np.arange(64)[None, :], 0, None).astype(np.uint16)
    x = bits.view(np.float16).copy()
    signs = np.random.default_rng(2509).integers(0, 2, size=x.shape).astype(bool)
    x[signs] = -x[signs]
    for gs in (8, 16, 32, 64):
        ref = O.encode16(x, 64, gs)
        _assert_equal(_enc(Q, x, gs), ref)
    assert ref.flags.max() == 12


@pytest.mark.parametrize("gs", [8, 16, 64])
@pytest.mark.parametrize("shape", [(1, 64), (3, 576), (129, 4096)])
def test_encode16_packed_flags(Q, gs, shape):
    x = inputs.mixture_activations(*shape, seed=5100 + gs)
    ref = O.encode16(x, 64, gs)
    e = _enc(Q, x, gs, flag_bits=4)
    assert np.array_equal(e.codes.cpu().numpy(), ref.codes)
    assert np.array_equal(e.flags.cpu().numpy(), _pack_flags(ref.flags))
    assert np.array_equal(e.scales.cpu().numpy().view(np.uint16), ref.scales.view(np.uint16))


@pytest.mark.parametrize("gs", [8, 32])
def test_dequantize16_bit_exact(Q, gs):
    x = inputs.laplace_activations(77, 1152, seed=5200 + gs, outlier_frac=0.002, outlier_scale=100.0)
    e = _enc(Q, x, gs)
    y = Q.dequantize(e)
    torch.cuda.synchronize()
    ref = O.dequantize(O.encode16(x, 64, gs)).astype(np.float16)
    assert np.array_equal(y.cpu().numpy().view(np.uint16), ref.view(np.uint16))


def _tol_check(y_gpu, y_ref, y_abs, G, dtype_name):
    y_gpu = y_gpu.astype(np.float64)
    tol = REL[dtype_name] * np.abs(y_ref) + (G + 5) * 2.0 ** -24 * y_abs + 2.0 ** -24
    err = np.abs(y_gpu - y_ref)
    bad = err > tol
    assert not bad.any(), (f"{bad.sum()} of {bad.size} outside tolerance; worst "
                           f"{(err / np.maximum(tol, 1e-30)).max():.3g}x")


def _products_magnitude(ea, ew):
    """sum_g s_a s_w sum_{k in g} |v_a v_w| for every output (binary64)."""
    va = np.abs(O.decode_values(ea).astype(np.float64))
    vw = np.abs(O.decode_values(ew).astype(np.float64))
    sa, sw = ea.scales.astype(np.float64), ew.scales.astype(np.float64)
    out = np.zeros((va.shape[0], vw.shape[0]))
    for g in range(va.shape[1] // 64):
        blk = va[:, 64 * g:64 * g + 64] @ vw[:, 64 * g:64 * g + 64].T
        out += sa[:, g:g + 1] * sw[:, g][None, :] * blk
    return out


def _tc_tol_check(y_gpu, ea, ew, bias, G, dtype_name):
    ref, rabs = O.linear(ea, ew, bias, with_abs=True)
    _tol_check(y_gpu, ref, rabs + 64 * _products_magnitude(ea, ew), G, dtype_name)


def _linear16(Q, xa, xw, gs, bias=None, out_dtype="float16", flag_bits=8, algo=None):
    a = _enc(Q, xa, gs, flag_bits)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=gs, code_bits=16, flag_bits=flag_bits)
    b = None if bias is None else torch.from_numpy(bias).cuda()
    y = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype), algo=Q.ALGO_SHIFT if algo is None else algo)
    assert Q.device_status() == 0
    return y.float().cpu().numpy()


@pytest.mark.parametrize("gs", [8, 16, 64])
@pytest.mark.parametrize("M,N,K", [(1, 8, 64), (200, 264, 640), (129, 520, 1216)])
def test_linear16_ragged_shapes(Q, gs, M, N, K):
    xa = inputs.laplace_activations(M, K, seed=5300 + M, outlier_frac=0.002, outlier_scale=100.0)
    xw = inputs.gaussian_weights(N, K, seed=5301 + N)
    bias = np.random.default_rng(M).normal(0, 0.1, N).astype(np.float16)
    y = _linear16(Q, xa, xw, gs, bias)
    ref, rabs = O.linear(O.encode16(xa, 64, gs), O.encode16(xw, 64, gs), bias, with_abs=True)
    _tol_check(y, ref, rabs, K // 64, "float16")


@pytest.mark.parametrize("out_dtype", ["float16", "bfloat16", "float32"])
def test_linear16_out_dtypes_and_packed_flags(Q, out_dtype):
    xa = inputs.laplace_activations(256, 1152, seed=5400, outlier_frac=0.002, outlier_scale=100.0)
    xw = inputs.gaussian_weights(384, 1152, seed=5401)
    ref, rabs = O.linear(O.encode16(xa, 64, 8), O.encode16(xw, 64, 8), with_abs=True)
    y = _linear16(Q, xa, xw, 8, out_dtype=out_dtype)
    _tol_check(y, ref, rabs, 18, out_dtype)
    y4 = _linear16(Q, xa, xw, 8, out_dtype=out_dtype, flag_bits=4)
    assert np.array_equal(y4, y)


def test_linear16_group_sums_beyond_int32(Q):
    """Saturated rows decode to +-28672 everywhere, so a 64-wide group sum is
    64 x 28672^2 > 2^31; rows with mixed FLAG 0..12 subgroups interleave."""
    xa = inputs.mixture_activations(40, 512, seed=5500)
    xw = inputs.gaussian_weights(64, 512, seed=5501)
    xa[0, :] = 8.0
    xa[1, ::2], xa[1, 1::2] = -3.0, 3.0
    xw[0, :] = -2.0
    xw[1, :] = 0.5
    xa[2, :] = (np.arange(512) % 8 - 3.5).astype(np.float16) * np.float16(2.0 ** -12)
    ea, ew = O.encode16(xa, 64, 8), O.encode16(xw, 64, 8)
    P = O.group_partials(O.decode_values(ea), O.decode_values(ew), 64)
    assert np.abs(P).max() > 2 ** 31
    y = _linear16(Q, xa, xw, 8, out_dtype="float32")
    ref, rabs = O.linear(ea, ew, with_abs=True)
    _tol_check(y, ref, rabs, 8, "float32")


def test_linear16_other_algorithms_rejected(Q):
    """No SIMT GEMM and no int32 partials for 16-bit codes; mixing 8-bit and
    16-bit operands is an argument error."""
    x = torch.from_numpy(inputs.mixture_activations(16, 128, seed=5600)).cuda()
    a = Q.quantize(x, group_s=8, code_bits=16)
    w = Q.encode_weights(x[:8].contiguous(), group_s=8, code_bits=16)
    w8 = Q.encode_weights(x[:8].contiguous(), group_s=8)
    with pytest.raises(Q.QuartzError, match="UNSUPPORTED"):
        Q.linear(a, w, algo=Q.ALGO_SIMT)
    for algo in (Q.ALGO_SHIFT, Q.ALGO_TCGEN05):
        with pytest.raises(Q.QuartzError, match="UNSUPPORTED"):
            Q.linear(a, w, algo=algo, partials_group=0)
    with pytest.raises(Q.QuartzError, match="INVALID_ARG"):
        Q.linear(a, w8, algo=Q.ALGO_SHIFT)
    torch.cuda.synchronize()
    assert Q.device_status() == 0


@pytest.mark.parametrize("layer", inputs.CONFIG_LLM, ids=[l.name for l in inputs.CONFIG_LLM])
def test_linear16_llama_layers_sampled(Q, layer):
    """Full-size LLaMA-2-7B block linears (G_s = 8, fp16 out) in the
    benchmark's launch configuration: codes of sampled rows bit-exact and
    their outputs within tolerance of the oracle."""
    xa, xw = layer.activations(), layer.weights()
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=8, code_bits=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=8, code_bits=16)
    y = Q.linear(a, w, algo=Q.ALGO_SHIFT)
    assert Q.device_status() == 0
    rows = np.unique(np.concatenate([np.arange(3), np.arange(layer.M - 3, layer.M),
                                     np.linspace(3, layer.M - 4, 6).astype(np.int64)]))
    rt = torch.from_numpy(rows).cuda()
    ea, ew = O.encode16(xa[rows], 64, 8), O.encode16(xw, 64, 8)
    assert np.array_equal(a.codes[rt].cpu().numpy(), ea.codes)
    assert np.array_equal(a.flags[rt].cpu().numpy(), ea.flags)
    assert np.array_equal(w.codes.cpu().numpy(), ew.codes)
    ref, rabs = O.linear(ea, ew, with_abs=True)
    _tol_check(y[rt].float().cpu().numpy(), ref, rabs, layer.K // 64, "float16")


# --- tcgen05 GEMM on E5M2 operands ------------------------------------------

@pytest.mark.parametrize("gs", [8, 16, 64])
@pytest.mark.parametrize("M,N,K", [(1, 8, 64), (200, 264, 640), (129, 520, 1216), (300, 1024, 4096)])
def test_linear16_tcgen05_ragged_shapes(Q, gs, M, N, K):
    xa = inputs.laplace_activations(M, K, seed=5700 + M, outlier_frac=0.002, outlier_scale=100.0)
    xw = inputs.gaussian_weights(N, K, seed=5701 + N)
    bias = np.random.default_rng(M).normal(0, 0.1, N).astype(np.float16)
    y = _linear16(Q, xa, xw, gs, bias, algo=Q.ALGO_TCGEN05)
    _tc_tol_check(y, O.encode16(xa, 64, gs), O.encode16(xw, 64, gs), bias, K // 64, "float16")


def test_linear16_tcgen05_extremes_and_packed_flags(Q):
    """Saturated rows (group sums 64 x 28672^2) and mixed FLAG 0..12 rows
    through the E5M2 operands; packed FLAGs give the identical output."""
    xa = inputs.mixture_activations(130, 512, seed=5800)
    xw = inputs.gaussian_weights(264, 512, seed=5801)
    xa[0, :] = 8.0
    xa[1, ::2], xa[1, 1::2] = -3.0, 3.0
    xw[0, :] = -2.0
    xa[2, :] = (np.arange(512) % 8 - 3.5).astype(np.float16) * np.float16(2.0 ** -12)
    y = _linear16(Q, xa, xw, 8, out_dtype="float32", algo=Q.ALGO_TCGEN05)
    _tc_tol_check(y, O.encode16(xa, 64, 8), O.encode16(xw, 64, 8), None, 8, "float32")
    y4 = _linear16(Q, xa, xw, 8, out_dtype="float32", flag_bits=4, algo=Q.ALGO_TCGEN05)
    assert np.array_equal(y4, y)


@pytest.mark.parametrize("layer", inputs.CONFIG_LLM, ids=[l.name for l in inputs.CONFIG_LLM])
def test_linear16_tcgen05_llama_layers_sampled(Q, layer):
    xa, xw = layer.activations(), layer.weights()
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=8, code_bits=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=8, code_bits=16)
    y = Q.linear(a, w, algo=Q.ALGO_TCGEN05)
    assert Q.device_status() == 0
    rows = np.unique(np.concatenate([np.arange(3), np.arange(layer.M - 3, layer.M),
                                     np.linspace(3, layer.M - 4, 6).astype(np.int64)]))
    rt = torch.from_numpy(rows).cuda()
    _tc_tol_check(y[rt].float().cpu().numpy(), O.encode16(xa[rows], 64, 8), O.encode16(xw, 64, 8), None,
                  layer.K // 64, "float16")


def test_linear16_tcgen05_range_split(Q):
    """16-bit codes through the range plan (90 tiles on 152 SMs, 100 groups,
    tiles in up to 3 parts added by the combine kernel): rows sampled from
    every M tile, a bias, against the oracle with the E5M2 sum bound."""
    M, N, K = 1200, 2296, 6400
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    T = -(-M // 128) * -(-N // 256)
    if not (T < sms < 2 * T and (K // 64) * (sms - T) >= 32 * sms):
        pytest.skip("this device's SM count does not take the range plan here")
    assert Q.linear_launch_count(M, N, K, Q.Params(64, 8, code_bits=16)) == 3
    xa = inputs.laplace_activations(M, K, seed=5900, outlier_frac=0.002, outlier_scale=100.0)
    xw = inputs.gaussian_weights(N, K, seed=5901)
    bias = np.random.default_rng(5902).normal(0, 0.1, N).astype(np.float16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=8, code_bits=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=8, code_bits=16)
    y = Q.linear(a, w, torch.from_numpy(bias).cuda(), algo=Q.ALGO_TCGEN05)
    assert Q.device_status() == 0
    rows = np.unique([min(m0 + d, M - 1) for m0 in range(0, M, 128) for d in (0, 5, 63, 127)])
    rt = torch.from_numpy(rows).cuda()
    _tc_tol_check(y[rt].float().cpu().numpy(), O.encode16(xa[rows], 64, 8), O.encode16(xw, 64, 8), bias,
                  K // 64, "float16")


# --- fused activation path with 16-bit codes ---------------------------------

@pytest.mark.parametrize("flag_bits", [8, 4])
@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("M,N,K", [(1, 8, 64), (200, 264, 640), (129, 520, 1216)])
def test_linear16_f16_fused_identical(Q, M, N, K, gs, flag_bits):
    """quartz_linear_f16 on 16-bit codes: the activations' encoding written
    beside the E5M2 operand equals quartz_quantize's bit for bit, and so does
    y against quantize + the tcgen05 linear; y also within tolerance of the
    oracle."""
    xa = inputs.laplace_activations(M, K, seed=6100 + M + gs, outlier_frac=0.002, outlier_scale=100.0)
    xw = inputs.gaussian_weights(N, K, seed=6101 + N + gs)
    xa[0, :64] = 0.0                                        # an all-zero group
    bias = torch.from_numpy(np.random.default_rng(N).normal(0, 0.1, N).astype(np.float16)).cuda()
    x = torch.from_numpy(xa).cuda()
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=gs, code_bits=16, flag_bits=flag_bits)
    a = Q.quantize(x, group_s=gs, code_bits=16, flag_bits=flag_bits)
    ref = Q.linear(a, w, bias, out_dtype=torch.float32, algo=Q.ALGO_TCGEN05)
    a_out = Q.empty_encoded(M, K, w.params, x.device)
    y = Q.linear_f16(x, w, bias, out_dtype=torch.float32, a_out=a_out)
    y_prep = Q.linear_f16(x, w, bias, out_dtype=torch.float32, w_prepared=Q.prepare_weights(w))
    assert Q.device_status() == 0
    assert torch.equal(a_out.codes, a.codes) and torch.equal(a_out.flags, a.flags)
    assert torch.equal(a_out.scales.view(torch.int16), a.scales.view(torch.int16))
    assert torch.equal(y, ref) and torch.equal(y_prep, ref)
    ea, ew = O.encode16(xa, 64, gs), O.encode16(xw, 64, gs)
    _tc_tol_check(y.cpu().numpy(), ea, ew, bias.cpu().numpy(), K // 64, "float32")


def test_linear16_f16_fused_llama_qkv(Q):
    """Full-size LLaMA-2-7B qkv (its last wave split along K) through the
    fused path: identical to quantize + linear."""
    layer = [l for l in inputs.CONFIG_LLM if l.name == "llama2_qkv"][0]
    x = torch.from_numpy(layer.activations()).cuda()
    w = Q.encode_weights(torch.from_numpy(layer.weights()).cuda(), group_s=8, code_bits=16)
    ref = Q.linear(Q.quantize(x, group_s=8, code_bits=16), w, algo=Q.ALGO_TCGEN05)
    y = Q.linear_f16(x, w, w_prepared=Q.prepare_weights(w))
    assert Q.device_status() == 0
    assert torch.equal(y, ref)
