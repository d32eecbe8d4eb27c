"""GPU encoder / dequantiser parity against the CPU oracle (bit-exact).

Codes, FLAGs, fp16 scale bits, zero points and group sums from the CUDA
kernels must equal the oracle's on the same seeded fp16 inputs; the
dequantised fp16 tensor must equal the oracle's binary64 value rounded once
to fp16 (the product s*(v-z) is exact in both precisions).
"""
import numpy as np
import pytest

import oracle as O
from paper_2509_26436_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def Q():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2509_26436_gb300 as Q
    return Q


def _gpu_encode(Q, x16, gs, mode):
    x = torch.from_numpy(x16).cuda()
    e = Q.quantize(x, group_s=gs, mode=mode)
    torch.cuda.synchronize()
    return e


def _assert_encoded_equal(e, ref, mode, rows=None):
    sel = slice(None) if rows is None else rows
    assert np.array_equal(e.codes.cpu().numpy()[sel], ref.codes)
    assert np.array_equal(e.flags.cpu().numpy()[sel], ref.flags)
    assert np.array_equal(e.scales.cpu().numpy().view(np.uint16)[sel], ref.scales.view(np.uint16))
    if mode == O.ASYMMETRIC:
        assert np.array_equal(e.zeros.cpu().numpy()[sel], ref.zeros)
        assert np.array_equal(e.gsum.cpu().numpy()[sel], ref.gsum)


@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("shape", [(1, 64), (3, 128), (37, 1152), (129, 4096), (1000, 640)])
def test_encode_bit_exact(Q, mode, gs, shape):
    x = inputs.mixture_activations(*shape, seed=1000 + shape[0] + gs)
    e = _gpu_encode(Q, x, gs, mode)
    _assert_encoded_equal(e, O.encode(x, 64, gs, mode), mode)


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
def test_encode_all_int8_codes(Q, gs):
    """Every code -127..127 reaches the LZS stage: groups whose max |x| is
    127 have scale exactly 1, so integer inputs quantize to themselves."""
    vals = np.arange(-127, 128, dtype=np.float32)
    x = np.zeros((1, 320), np.float32)
    for g in range(5):  # each 64-group: 127 followed by 63 of the 255 codes
        x[0, 64 * g] = 127
        x[0, 64 * g + 1:64 * g + 64] = vals[63 * g:63 * g + 63] if g < 4 else np.concatenate(
            [vals[252:], np.zeros(60, np.float32)])
    x = np.concatenate([x, -x], axis=0)
    x16 = x.astype(np.float16)
    for mode in (O.SYMMETRIC, O.ASYMMETRIC):
        e = _gpu_encode(Q, x16, gs, mode)
        ref = O.encode(x16, 64, gs, mode)
        _assert_encoded_equal(e, ref, mode)
    q, s, _ = O.quantize(x16, 64, O.SYMMETRIC)
    assert set(np.unique(q[0])) == set(range(-127, 128))


def test_encode_edge_values(Q):
    """All-zero groups, scale underflow, subnormal scales (including ones
    rounded so far down that |x| r exceeds 127), fp16 extremes, exact ties,
    all-equal and one-sided groups."""
    rows = []
    rows.append(np.zeros(256))
    rows.append(np.full(256, 1e-7))
    rows.append(np.linspace(-3e-4, 3e-4, 256))
    rows.append(np.concatenate([np.full(64, 65504.0), -np.full(64, 65504.0),
                                np.linspace(-65504, 65504, 128)]))
    t = np.zeros(256)
    t[:7] = np.array([127, 2.5, 3.5, -2.5, -0.5, 0.5, 1.5]) * 2.0 ** -10
    rows.append(t)
    t = np.zeros(256)  # subnormal scales rounded far down: |x| r exceeds 127 and is clamped
    t[:64] = np.linspace(-189, 189, 64).round() * 2.0 ** -24
    t[64:128] = np.arange(64) * 3 * 2.0 ** -24
    t[128:192] = (np.arange(64) - 32) * 5 * 2.0 ** -24
    rows.append(t)
    rows.append(np.full(256, 0.5))
    rows.append(np.abs(np.random.default_rng(4).laplace(0, 1, 256)) + 1)
    rows.append(-np.abs(np.random.default_rng(5).laplace(0, 1, 256)))
    x16 = np.stack(rows).astype(np.float16)
    for mode in (O.SYMMETRIC, O.ASYMMETRIC):
        for gs in (8, 16, 32, 64):
            e = _gpu_encode(Q, x16, gs, mode)
            _assert_encoded_equal(e, O.encode(x16, 64, gs, mode), mode)


def test_encode_zero_rows_is_noop(Q):
    x = torch.empty((0, 128), dtype=torch.float16, device="cuda")
    e = Q.quantize(x)
    torch.cuda.synchronize()
    assert e.codes.shape == (0, 64)


@pytest.mark.parametrize("rows,K", inputs.ENCODE_SWEEP)
@pytest.mark.parametrize("gs", [8, 16, 32])
def test_encode_sweep_sizes(Q, rows, K, gs):
    """The 1M / 16M / 128M-element encode workloads, in the launch the
    benchmark times; 128M is compared on a deterministic sample of rows."""
    x = inputs.mixture_activations(rows, K, seed=inputs.seed_for(1, gs))
    e = _gpu_encode(Q, x, gs, O.SYMMETRIC)
    if rows * K <= 16 * 2 ** 20:
        _assert_encoded_equal(e, O.encode(x, 64, gs, O.SYMMETRIC), O.SYMMETRIC)
    else:
        sel = np.unique(np.concatenate([np.arange(0, rows, 37), np.arange(rows - 64, rows)]))
        _assert_encoded_equal(e, O.encode(x[sel], 64, gs, O.SYMMETRIC), O.SYMMETRIC, rows=sel)


@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
@pytest.mark.parametrize("gs", [8, 16, 32, 64])
def test_dequantize_bit_exact(Q, mode, gs):
    x = inputs.laplace_activations(77, 1152, seed=77 + gs)
    e = _gpu_encode(Q, x, gs, mode)
    y = Q.dequantize(e)
    torch.cuda.synchronize()
    ref = O.dequantize(O.encode(x, 64, gs, mode)).astype(np.float16)
    assert np.array_equal(y.cpu().numpy().view(np.uint16), ref.view(np.uint16))


def test_weights_encoder_is_the_same_arithmetic(Q):
    w = inputs.gaussian_weights(300, 1152, seed=5)
    e = Q.encode_weights(torch.from_numpy(w).cuda(), group_s=16)
    torch.cuda.synchronize()
    _assert_encoded_equal(e, O.encode(w, 64, 16, O.SYMMETRIC), O.SYMMETRIC)
    assert Q.device_status() == 0


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("shape", [(1, 64), (37, 1152), (5, 12288), (300, 3072)])
def test_encode_per_row_scale_bit_exact(Q, gs, shape):
    """group_q = K: one scale per row (per-token activations / per-channel
    weights), bit-exact against the oracle."""
    rows, K = shape
    x = inputs.mixture_activations(rows, K, seed=2000 + rows + gs)
    e = Q.quantize(torch.from_numpy(x).cuda(), group_s=gs, group_q=K)
    torch.cuda.synchronize()
    ref = O.encode(x, K, gs)
    _assert_encoded_equal(e, ref, O.SYMMETRIC)
    xh = Q.dequantize(e)
    assert torch.equal(xh.cpu(), torch.from_numpy(O.dequantize(ref).astype(np.float16)))


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("group_q", [64, "K"])
def test_encode_static_scale_bit_exact(Q, gs, group_q):
    """Static per-tensor scale (calibrated elsewhere): bit-exact against the
    oracle, including saturation of values beyond 127 * scale."""
    rows, K = 40, 1152
    gq = K if group_q == "K" else 64
    x = inputs.mixture_activations(rows, K, seed=3000 + gs)
    for scale in (np.float16(0.06), np.float16(0.004), np.float16(2.0 ** -20), np.float16(0)):
        e = Q.quantize_static(torch.from_numpy(x).cuda(), scale, group_s=gs, group_q=gq)
        torch.cuda.synchronize()
        _assert_encoded_equal(e, O.encode_static(x, scale, gq, gs), O.SYMMETRIC)


@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("shape", [(1, 64), (3, 576), (37, 1152), (129, 4096)])
def test_encode_packed_flags(Q, mode, gs, shape):
    """flag_bits = 4: FLAGs two per byte, subgroup 2j in the low nibble of
    byte j over the whole tensor; codes and scales unchanged."""
    x = inputs.mixture_activations(*shape, seed=4000 + shape[0] + gs)
    e = Q.quantize(torch.from_numpy(x).cuda(), group_s=gs, mode=mode, flag_bits=4)
    torch.cuda.synchronize()
    ref = O.encode(x, 64, gs, mode)
    assert np.array_equal(e.flags.cpu().numpy(), O.pack_nibbles(ref.flags.reshape(-1).astype(np.int8)))
    assert np.array_equal(e.codes.cpu().numpy(), ref.codes)
    assert np.array_equal(e.scales.cpu().numpy().view(np.uint16), ref.scales.view(np.uint16))
    xh = Q.dequantize(e)
    assert torch.equal(xh.cpu(), torch.from_numpy(O.dequantize(ref).astype(np.float16)))


@pytest.mark.parametrize("gs", [8, 16, 64])
def test_encode_packed_flags_per_row_and_static(Q, gs):
    x = inputs.mixture_activations(33, 3072, seed=5000 + gs)
    xt = torch.from_numpy(x).cuda()
    e = Q.quantize(xt, group_s=gs, group_q=3072, flag_bits=4)
    ref = O.encode(x, 3072, gs)
    assert np.array_equal(e.flags.cpu().numpy(), O.pack_nibbles(ref.flags.reshape(-1).astype(np.int8)))
    assert np.array_equal(e.codes.cpu().numpy(), ref.codes)
    s = np.float16(0.01)
    e = Q.quantize_static(xt, s, group_s=gs, flag_bits=4)
    ref = O.encode_static(x, s, 64, gs)
    assert np.array_equal(e.flags.cpu().numpy(), O.pack_nibbles(ref.flags.reshape(-1).astype(np.int8)))
    assert np.array_equal(e.codes.cpu().numpy(), ref.codes)
