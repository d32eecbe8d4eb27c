"""GPU W4A4 linear parity against the CPU oracle.

* Integer group partials P_g (the MMA result of one 64-wide K group) are
  compared bit-exactly with the oracle's int64 sums.
* Outputs are compared with the oracle's binary64 y.  Tolerance, derived
  from the kernel's arithmetic: P_g is exact; each group term s_a*(s_w*P_g)
  adds at most two binary32 roundings and the G-term running sum at most G
  more, so |y_gpu - y| <= (G + 4) * 2^-24 * sum_g |s_a s_w D_g| before the
  output conversion, which adds a relative 2^-11 (fp16), 2^-8 (bf16) or
  nothing (fp32).  The test allows the stated relative bounds 1e-3 (fp16),
  4e-3 (bf16), 1e-5 (fp32) plus that cancellation-aware absolute term.
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


def _tol_check(y_gpu, y_ref, y_abs, G, dtype_name):
    y_gpu = y_gpu.astype(np.float64)
    tol = REL[dtype_name] * np.abs(y_ref) + (G + 4) * 2.0 ** -24 * y_abs + 2.0 ** -24
    err = np.abs(y_gpu - y_ref)
    bad = err > tol
    assert not bad.any(), (f"{bad.sum()} of {bad.size} outside tolerance; worst "
                           f"{(err / np.maximum(tol, 1e-30)).max():.3g}x")


def _run(Q, xa, xw, gs, mode, bias=None, out_dtype="float16", algo=None, partials_group=None):
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=gs, mode=mode)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=gs, mode=mode)
    b = None if bias is None else torch.from_numpy(bias).cuda()
    kw = {}
    if algo is not None:
        kw["algo"] = algo
    r = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype), partials_group=partials_group, **kw)
    assert Q.device_status() == 0
    return r


ALGOS = {"tcgen05": 0, "simt": 1, "shift": 2}


@pytest.mark.parametrize("algo", list(ALGOS))
@pytest.mark.parametrize("out_dtype", ["float16", "bfloat16", "float32"])
def test_linear_single_layer(Q, algo, out_dtype):
    """256 tokens x 1152 -> 1152, G_s = 16, symmetric, with bias."""
    layer = inputs.CONFIG0[0]
    xa, xw = layer.activations(), layer.weights()
    bias = inputs.gaussian_weights(1, layer.N, seed=3)[0]
    y = _run(Q, xa, xw, 16, O.SYMMETRIC, bias, out_dtype, ALGOS[algo])
    a, w = O.encode(xa, 64, 16), O.encode(xw, 64, 16)
    ref, rabs = O.linear(a, w, bias, with_abs=True)
    _tol_check(y.float().cpu().numpy(), ref, rabs, layer.K // 64, out_dtype)


@pytest.mark.parametrize("algo", list(ALGOS))
@pytest.mark.parametrize("group", [0, 9, 17])
def test_group_partials_bit_exact(Q, algo, group):
    """The integer MMA result of one group equals the oracle's int64 sum."""
    layer = inputs.CONFIG0[0]
    xa, xw = layer.activations(), layer.weights()
    _, part = _run(Q, xa, xw, 16, O.SYMMETRIC, algo=ALGOS[algo], partials_group=group)
    va = O.decode_values(O.encode(xa, 64, 16))[:, group * 64:(group + 1) * 64]
    vw = O.decode_values(O.encode(xw, 64, 16))[:, group * 64:(group + 1) * 64]
    ref = O.group_partials(va, vw, 64)[0]
    assert np.array_equal(part.cpu().numpy().astype(np.int64), ref)


@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
@pytest.mark.parametrize("gs", [8, 32])
@pytest.mark.parametrize("M,N,K", [(1, 8, 64), (200, 264, 192), (300, 520, 640), (129, 256, 64),
                                   (1000, 776, 1216), (384, 1024, 256)])
def test_linear_ragged_shapes(Q, mode, gs, M, N, K):
    """Several tiles with ragged M and N tails, one-group K, all G_s."""
    xa = inputs.laplace_activations(M, K, seed=M + N + K)
    xw = inputs.gaussian_weights(N, K, seed=M * 7 + N)
    bias = inputs.gaussian_weights(1, N, seed=N)[0]
    g = (K // 64) // 2
    y, part = _run(Q, xa, xw, gs, mode, bias, "float32", partials_group=g)
    a, w = O.encode(xa, 64, gs, mode), O.encode(xw, 64, gs, mode)
    ref, rabs = O.linear(a, w, bias, with_abs=True)
    _tol_check(y.cpu().numpy(), ref, rabs, K // 64, "float32")
    va = O.decode_values(a)[:, g * 64:(g + 1) * 64]
    vw = O.decode_values(w)[:, g * 64:(g + 1) * 64]
    assert np.array_equal(part.cpu().numpy().astype(np.int64), O.group_partials(va, vw, 64)[0])


def test_linear_asymmetric_conv_activations(Q):
    """Zero-point path on one-sided post-SiLU im2col activations."""
    xa = inputs.silu_im2col(1, 64, 16, 16, seed=8)        # [256, 576]
    xw = inputs.gaussian_weights(320, 576, seed=9)
    for out_dtype in ("float16", "float32"):
        y = _run(Q, xa, xw, 16, O.ASYMMETRIC, None, out_dtype)
        ref, rabs = O.linear(O.encode(xa, 64, 16, O.ASYMMETRIC), O.encode(xw, 64, 16, O.ASYMMETRIC),
                             with_abs=True)
        _tol_check(y.float().cpu().numpy(), ref, rabs, 9, out_dtype)


def test_linear_zero_rows(Q):
    a = Q.quantize(torch.empty((0, 128), dtype=torch.float16, device="cuda"))
    w = Q.encode_weights(torch.randn(16, 128, device="cuda").half())
    y = Q.linear(a, w)
    torch.cuda.synchronize()
    assert y.shape == (0, 16)


def _sample_rows(M):
    return np.unique(np.concatenate([np.arange(4), np.arange(M - 4, M),
                                     np.linspace(4, M - 5, 8).astype(np.int64)]))


FULL_LAYERS = inputs.CONFIG2 + inputs.CONFIG3 + inputs.CONFIG4


@pytest.mark.parametrize("layer", FULL_LAYERS, ids=[l.name for l in FULL_LAYERS])
def test_linear_full_size_sampled(Q, layer):
    """Full-size layers in the benchmark's launch configuration (G_s = 16,
    symmetric, fp16 out): codes, one group's integer partials and outputs
    compared with the oracle on a deterministic sample of token rows."""
    xa, xw = layer.activations(), layer.weights()
    G = layer.K // 64
    g = G // 2
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    y, part = Q.linear(a, w, partials_group=g)
    assert Q.device_status() == 0
    rows = _sample_rows(layer.M)
    rows_t = torch.from_numpy(rows).cuda()
    ea = O.encode(xa[rows], 64, 16)
    ew = O.encode(xw, 64, 16)
    assert np.array_equal(a.codes[rows_t].cpu().numpy(), ea.codes)
    assert np.array_equal(a.flags[rows_t].cpu().numpy(), ea.flags)
    assert np.array_equal(w.codes.cpu().numpy(), ew.codes)
    ref, rabs = O.linear(ea, ew, with_abs=True)
    _tol_check(y[rows_t].float().cpu().numpy(), ref, rabs, G, "float16")
    va = O.decode_values(ea)[:, g * 64:(g + 1) * 64]
    vw = O.decode_values(ew)[:, g * 64:(g + 1) * 64]
    assert np.array_equal(part[rows_t].cpu().numpy().astype(np.int64), O.group_partials(va, vw, 64)[0])
    # without group partials the symmetric launch may split its last wave of
    # tiles along K (sums in another order, same bound)
    y2 = Q.linear(a, w)
    assert Q.device_status() == 0
    _tol_check(y2[rows_t].float().cpu().numpy(), ref, rabs, G, "float16")


# Shapes whose last wave of 128 x 256 tiles, on a 152-SM GB300, is cut along K:
# 9 x 18 tiles = 152 + 10 (4 parts of 2-3 groups), 13 x 15 = 152 + 43
# (3 parts), 12 x 18 = 152 + 64 with 4 groups (2 parts of 2), and 4 x 39 =
# 152 + 4 with 5 groups (2 parts of 2 and 3).  Every m-tile is sampled.
SPLIT_SHAPES = [(1100, 4400, 640), (1614, 3816, 640), (1472, 4408, 256), (449, 9904, 320)]


@pytest.mark.parametrize("out_dtype", ["float16", "bfloat16", "float32"])
@pytest.mark.parametrize("M,N,K", SPLIT_SHAPES)
def test_linear_split_last_wave(Q, M, N, K, out_dtype):
    xa = inputs.laplace_activations(M, K, seed=9100 + M)
    xw = inputs.gaussian_weights(N, K, seed=9101 + N)
    bias = np.random.default_rng(N).normal(0, 0.1, N).astype(np.float16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    b = torch.from_numpy(bias).cuda()
    y = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype))
    y_again = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype), w_prepared=Q.prepare_weights(w))
    assert Q.device_status() == 0
    assert torch.equal(y, y_again)
    rows = np.unique(np.concatenate([np.arange(0, M, 5), [M - 1]]))
    ref, rabs = O.linear(O.encode(xa[rows], 64, 16), O.encode(xw, 64, 16), bias, with_abs=True)
    _tol_check(y[torch.from_numpy(rows).cuda()].float().cpu().numpy(), ref, rabs, K // 64, out_dtype)


# Fewer tiles than SMs: every tile is cut along K into up to 4 parts (one
# CTA each): 2 x 5 tiles of 18 groups (the 256 x 1152 single layer, 4
# parts), 1 tile of 10 groups (4 parts), 3 x 3 ragged tiles of 5 groups (2
# parts), 40 tiles of 3 groups (stays whole: parts keep at least two groups).
SMALL_SHAPES = [(256, 1152, 1152), (100, 200, 640), (300, 520, 320), (1000, 1200, 192)]


@pytest.mark.parametrize("out_dtype", ["float16", "bfloat16", "float32"])
@pytest.mark.parametrize("M,N,K", SMALL_SHAPES)
def test_linear_split_small_problems(Q, M, N, K, out_dtype):
    """Split along K of every tile when the problem has fewer tiles than SMs:
    all outputs against the oracle, with a bias; the prepared-weights call is
    bit-identical."""
    xa = inputs.laplace_activations(M, K, seed=9300 + M)
    xw = inputs.gaussian_weights(N, K, seed=9301 + N)
    bias = np.random.default_rng(N + 2).normal(0, 0.1, N).astype(np.float16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    b = torch.from_numpy(bias).cuda()
    y = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype))
    y_again = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype), w_prepared=Q.prepare_weights(w))
    assert Q.device_status() == 0
    assert torch.equal(y, y_again)
    ref, rabs = O.linear(O.encode(xa, 64, 16), O.encode(xw, 64, 16), bias, with_abs=True)
    _tol_check(y.float().cpu().numpy(), ref, rabs, K // 64, out_dtype)


# Shapes whose last wave is more than half full, so that the last P + R tiles'
# group iterations are spread over all CTAs after one wave of whole tiles
# (two-wave form), with 8-bit codes (exact P_g): 9 x 45 = 405 tiles = 2 x 152
# + 101 with 96 groups, and 12 x 32 = 384 = 2 x 152 + 80 with 68 groups.  Both
# mix whole tiles, whole tail tiles and tail tiles cut into two parts; M and
# N are ragged, so the combine kernel stores partial edge tiles.
TWO_WAVE_SHAPES = [(1100, 11400, 6144), (1500, 8000, 4352)]
_two_wave_ref = {}


def _two_wave_predicate(M, N, K, sms):
    T = -(-M // 128) * -(-N // 256)
    P = min(T, sms)
    W, R = divmod(T, P)
    return W >= 1 and 2 * R > P and (K // 64) * (P - R) >= 32 * P


def _rows_every_m_tile(M):
    rows = []
    for m0 in range(0, M, 128):
        m1 = min(m0 + 128, M)
        rows += [m0, m0 + 1, m0 + 8, m0 + 37, m0 + 64, m1 - 9, m1 - 1]
    return np.unique(np.clip(np.array(rows), 0, M - 1))


@pytest.mark.parametrize("out_dtype", ["float16", "bfloat16", "float32"])
@pytest.mark.parametrize("M,N,K", TWO_WAVE_SHAPES)
def test_linear_two_wave_split_8bit(Q, M, N, K, out_dtype):
    """Two-wave form on 8-bit codes against the oracle: all output columns of
    rows sampled from every M tile, with a bias, three output types; the
    prepared-weights call is bit-identical; the host really takes the form."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    if not _two_wave_predicate(M, N, K, sms):
        pytest.skip(f"{sms} SMs: this shape does not take the two-wave form")
    assert Q.linear_launch_count(M, N, K) == 3
    xa = inputs.laplace_activations(M, K, seed=9200 + M)
    xw = inputs.gaussian_weights(N, K, seed=9201 + N)
    bias = np.random.default_rng(N + 1).normal(0, 0.1, N).astype(np.float16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    b = torch.from_numpy(bias).cuda()
    y = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype))
    y_again = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype), w_prepared=Q.prepare_weights(w))
    assert Q.device_status() == 0
    assert torch.equal(y, y_again)
    rows = _rows_every_m_tile(M)
    if (M, N, K) not in _two_wave_ref:
        _two_wave_ref[(M, N, K)] = O.linear(O.encode(xa[rows], 64, 16), O.encode(xw, 64, 16), bias,
                                            with_abs=True)
    ref, rabs = _two_wave_ref[(M, N, K)]
    _tol_check(y[torch.from_numpy(rows).cuda()].float().cpu().numpy(), ref, rabs, K // 64, out_dtype)


# More than half but not all of the 152 SMs hold a tile: every tile's group
# iterations are spread in one range per SM, a tile in up to 3 parts.
# 90 tiles (ragged M and N, 100 groups, ls 60) and SDXL's 3x3 conv on 1280
# channels at 32x32 (80 tiles, 180 groups, ls 95).
RANGE_SHAPES = [(1200, 2296, 6400), (2048, 1280, 11520)]


def _range_predicate(M, N, K, sms):
    T = -(-M // 128) * -(-N // 256)
    return T < sms < 2 * T and (K // 64) * (sms - T) >= 32 * sms


@pytest.mark.parametrize("out_dtype", ["float16", "bfloat16", "float32"])
@pytest.mark.parametrize("M,N,K", RANGE_SHAPES)
def test_linear_range_split_fewer_tiles_than_sms(Q, M, N, K, out_dtype):
    """Range plan over all tiles (up to three parts per tile, added by the
    combine kernel in group order): rows sampled from every M tile, all
    columns, with a bias, three output types; prepared weights give the
    same bits."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    if not _range_predicate(M, N, K, sms):
        pytest.skip("this device's SM count does not take the range plan here")
    assert Q.linear_launch_count(M, N, K) == 3
    xa = inputs.laplace_activations(M, K, seed=M + K + 3)
    xw = inputs.gaussian_weights(N, K, seed=N + K + 4)
    bias = np.random.default_rng(N + 5).normal(0, 0.1, N).astype(np.float16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    b = torch.from_numpy(bias).cuda()
    y = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype))
    y_again = Q.linear(a, w, b, out_dtype=getattr(torch, out_dtype), w_prepared=Q.prepare_weights(w))
    assert Q.device_status() == 0
    assert torch.equal(y, y_again)
    rows = _rows_every_m_tile(M)
    if (M, N, K) not in _two_wave_ref:
        _two_wave_ref[(M, N, K)] = O.linear(O.encode(xa[rows], 64, 16), O.encode(xw, 64, 16), bias,
                                            with_abs=True)
    ref, rabs = _two_wave_ref[(M, N, K)]
    _tol_check(y[torch.from_numpy(rows).cuda()].float().cpu().numpy(), ref, rabs, K // 64, out_dtype)


def test_split_last_wave_launch_count(Q):
    """The host splits the last wave when the tiles after whole waves fill at
    most half a wave and each part keeps at least two groups, and spreads the
    last two waves over all CTAs when they fill more than half and that saves
    at least 32 group iterations on the critical path; the launch count and
    the workspace report it."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    shapes = SPLIT_SHAPES + SMALL_SHAPES + RANGE_SHAPES + [(2048, 4096, 4096), (2048, 4096, 11008),
                                                           (1100, 4400, 128), (128, 256, 640), (128, 256, 64),
                                                           (1200, 2296, 640)]
    for M, N, K in shapes:
        T = -(-M // 128) * -(-N // 256)
        P = min(T, sms)
        W, R = divmod(T, P)
        G = K // 64
        if T < sms and 2 * T > sms:
            split, part_tiles = G * (sms - T) >= 32 * sms, 3 * T
        elif T < sms:
            split = min(sms // T, 4, G // 2) >= 2
            part_tiles = T * min(sms // T, 4, G // 2) if split else 0
        elif W >= 1 and 2 * R > P:
            split, part_tiles = G * (P - R) >= 32 * P, 2 * (P + R)
        else:
            split = W >= 1 and R > 0 and min(P // R, 4, G // 2) >= 2
            part_tiles = R * min(P // R, 4, G // 2) if split else 0
        if sms == 152 and (M, N, K) in SPLIT_SHAPES + [(2048, 4096, 11008)]:
            assert split
        assert Q.linear_launch_count(M, N, K) == (3 if split else 2)
        assert Q.linear_launch_count(M, N, K, partials=True) == 2
        assert Q.linear_launch_count(M, N, K, algo=Q.ALGO_SIMT) == 2
        if split:
            assert Q.linear_workspace_size(M, N, K) >= part_tiles * 128 * 256 * 4


def test_bounded_wait_reports_timeout(Q):
    """Failure detection without a fault: a kernel waits on an mbarrier that
    nothing arrives at, gives up after 1 ms and the host reads the status;
    the context stays usable."""
    assert Q.device_status() == 0
    assert Q.selftest_timeout(1_000_000) == 0
    assert Q.device_status() == 5          # QUARTZ_ERR_TIMEOUT
    assert Q.device_status() == 0          # cleared
    x = torch.randn(4, 64, device="cuda").half()
    Q.quantize(x)
    assert Q.device_status() == 0


def test_gemm_events_bracket_the_gemm_kernel(Q):
    """The events quartz_linear_ex records sit around the GEMM launch only:
    they measure a positive time no longer than the whole call."""
    layer = inputs.CONFIG0[0]
    a = Q.quantize(torch.from_numpy(layer.activations()).cuda())
    w = Q.encode_weights(torch.from_numpy(layer.weights()).cuda())
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for _ in range(3):
        c0.record()
        Q.linear(a, w, gemm_events=(g0, g1))
        c1.record()
    torch.cuda.synchronize()
    t_gemm, t_call = g0.elapsed_time(g1), c0.elapsed_time(c1)
    assert 0 < t_gemm <= t_call
    assert Q.device_status() == 0


def _lzs_extreme(rows, K, seed):
    """Rows whose 16-wide subgroups alternate between the two ends of the LZS
    range: even subgroups hold +-1.0 (the group maximum, q = +-127, FLAG 4,
    decoded +-112) and odd subgroups hold q/127 with |q| <= 7 (FLAG 0,
    decoded q).  One group partial then mixes products of 12544 with
    products of 1, so any loss of low-order bits in the tensor-core sums
    shows up as a wrong integer."""
    rng = np.random.default_rng(seed)
    x = np.where(rng.random((rows, K)) < 0.5, -1.0, 1.0)
    small = rng.integers(-7, 8, size=(rows, K)) / 127.0
    odd = (np.arange(K) // 16) % 2 == 1
    x[:, odd] = small[:, odd]
    return x.astype(np.float16)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_group_partials_lzs_extremes_bit_exact(Q, seed):
    M, N, K = 256, 272, 512
    xa, xw = _lzs_extreme(M, K, 100 + seed), _lzs_extreme(N, K, 200 + seed)
    ea, ew = O.encode(xa, 64, 16), O.encode(xw, 64, 16)
    va, vw = O.decode_values(ea), O.decode_values(ew)
    assert np.abs(va).max() == 112 and np.abs(vw).max() == 112
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    for g in range(K // 64):
        y, part = Q.linear(a, w, out_dtype=torch.float32, partials_group=g)
        assert Q.device_status() == 0
        ref = O.group_partials(va[:, g * 64:(g + 1) * 64], vw[:, g * 64:(g + 1) * 64], 64)[0]
        assert (np.abs(ref) > 2 ** 17).any() and (ref % 2 == 1).any()
        assert np.array_equal(part.cpu().numpy().astype(np.int64), ref), f"group {g}"
    ref, rabs = O.linear(ea, ew, with_abs=True)
    _tol_check(y.cpu().numpy(), ref, rabs, K // 64, "float32")


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("M,N,K", [(200, 264, 640), (1, 8, 64), (300, 1024, 1216)])
def test_linear_f16_fused_is_bit_identical(Q, gs, M, N, K):
    """quartz_linear_f16 (encode on the fly into the GEMM operand) gives the
    same bits as quartz_quantize + quartz_linear, and its optional encoded
    output equals quartz_quantize's."""
    x16 = inputs.mixture_activations(M, K, seed=M + 3 * N + gs)
    w16 = inputs.gaussian_weights(N, K, seed=N + gs)
    x = torch.from_numpy(x16).cuda()
    w = Q.encode_weights(torch.from_numpy(w16).cuda(), group_s=gs)
    bias = torch.from_numpy(inputs.gaussian_weights(1, N, seed=5)[0]).cuda()
    a = Q.quantize(x, group_s=gs)
    for dt in (torch.float16, torch.float32):
        ref = Q.linear(a, w, bias, out_dtype=dt)
        a_out = Q.empty_encoded(M, K, Q.Params(64, gs, O.SYMMETRIC), x.device)
        y = Q.linear_f16(x, w, bias, out_dtype=dt, a_out=a_out)
        assert Q.device_status() == 0
        assert torch.equal(y, ref)
        assert torch.equal(a_out.codes, a.codes) and torch.equal(a_out.flags, a.flags)
        assert torch.equal(a_out.scales.view(torch.int16), a.scales.view(torch.int16))
    # and against the oracle directly (same tolerance as the other linear tests)
    ref, rabs = O.linear(O.encode(x16, 64, gs), O.encode(w16, 64, gs), bias.cpu().numpy(), with_abs=True)
    y = Q.linear_f16(x, w, bias, out_dtype=torch.float32)
    _tol_check(y.cpu().numpy(), ref, rabs, K // 64, "float32")


def test_linear_f16_flux_layer_matches_two_call_path(Q):
    """Full-size FLUX fc1 activations, fused path vs quantize + linear."""
    layer = [l for l in inputs.CONFIG4 if l.name == "flux_fc1"][0]
    x = torch.from_numpy(layer.activations()).cuda()
    w = Q.encode_weights(torch.from_numpy(layer.weights()).cuda(), group_s=16)
    ref = Q.linear(Q.quantize(x, group_s=16), w)
    y = Q.linear_f16(x, w)
    assert Q.device_status() == 0
    assert torch.equal(y, ref)


@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("M,N,K", [(1, 8, 64), (200, 264, 640), (129, 520, 1216)])
def test_shift_schedule_matches_decode_before_mma(Q, mode, gs, M, N, K):
    """The paper's accumulator-shift schedule (integer code dot products per
    subgroup, shifted by both FLAGs) gives the same exact group partials as
    decode-before-MMA on the tensor cores, and outputs within tolerance."""
    xa = inputs.mixture_activations(M, K, seed=7 * M + K + gs)
    xw = inputs.gaussian_weights(N, K, seed=N + K + gs)
    g = (K // 64) // 2
    y_s, p_s = _run(Q, xa, xw, gs, mode, None, "float32", Q.ALGO_SHIFT, partials_group=g)
    y_t, p_t = _run(Q, xa, xw, gs, mode, None, "float32", Q.ALGO_TCGEN05, partials_group=g)
    assert torch.equal(p_s, p_t)
    a, w = O.encode(xa, 64, gs, mode), O.encode(xw, 64, gs, mode)
    ref, rabs = O.linear(a, w, with_abs=True)
    _tol_check(y_s.cpu().numpy(), ref, rabs, K // 64, "float32")
    va = O.decode_values(a)[:, g * 64:(g + 1) * 64]
    vw = O.decode_values(w)[:, g * 64:(g + 1) * 64]
    assert np.array_equal(p_s.cpu().numpy().astype(np.int64), O.group_partials(va, vw, 64)[0])


@pytest.mark.parametrize("seed", [0, 1])
def test_shift_schedule_lzs_extremes(Q, seed):
    """Groups mixing decoded +-112 and +-1..7 through the shift schedule."""
    M, N, K = 128, 136, 256
    xa, xw = _lzs_extreme(M, K, 300 + seed), _lzs_extreme(N, K, 400 + seed)
    va, vw = O.decode_values(O.encode(xa, 64, 16)), O.decode_values(O.encode(xw, 64, 16))
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    for g in range(K // 64):
        _, part = Q.linear(a, w, out_dtype=torch.float32, partials_group=g, algo=Q.ALGO_SHIFT)
        ref = O.group_partials(va[:, g * 64:(g + 1) * 64], vw[:, g * 64:(g + 1) * 64], 64)[0]
        assert np.array_equal(part.cpu().numpy().astype(np.int64), ref), f"group {g}"


@pytest.mark.parametrize("gs", [8, 16, 64])
@pytest.mark.parametrize("M,N,K", [(1, 8, 64), (200, 264, 640), (300, 520, 3072), (129, 256, 12288)])
def test_per_row_scales_linear(Q, gs, M, N, K):
    """group_q = K on both operands (per-token activations, per-channel
    weights): the whole-K integer partial sum is exact (it is accumulated in
    exact 256-wide pieces) and y matches the oracle."""
    xa = inputs.laplace_activations(M, K, seed=M + N + K + gs)
    xw = inputs.gaussian_weights(N, K, seed=3 * N + K)
    bias = inputs.gaussian_weights(1, N, seed=N + 1)[0]
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=gs, group_q=K)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=gs, group_q=K)
    y, part = Q.linear(a, w, torch.from_numpy(bias).cuda(), out_dtype=torch.float32, partials_group=0)
    assert Q.device_status() == 0
    ea, ew = O.encode(xa, K, gs), O.encode(xw, K, gs)
    ref, rabs = O.linear(ea, ew, bias, with_abs=True)
    _tol_check(y.cpu().numpy(), ref, rabs, 1, "float32")
    P = O.group_partials(O.decode_values(ea), O.decode_values(ew), K)[0]
    assert np.array_equal(part.cpu().numpy().astype(np.int64), P)
    y16 = Q.linear(a, w, torch.from_numpy(bias).cuda())
    _tol_check(y16.float().cpu().numpy(), ref, rabs, 1, "float16")


def test_per_row_scales_extreme_partials(Q):
    """Whole-K partials far beyond 2^24 (every decoded value +-112): exact."""
    M, N, K = 128, 64, 12288
    xa = np.where(np.random.default_rng(1).random((M, K)) < 0.9, 1.0, -1.0).astype(np.float16)
    xw = np.ones((N, K), np.float16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16, group_q=K)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16, group_q=K)
    _, part = Q.linear(a, w, out_dtype=torch.float32, partials_group=0)
    P = O.group_partials(O.decode_values(O.encode(xa, K, 16)), O.decode_values(O.encode(xw, K, 16)), K)[0]
    assert np.abs(P).max() > 2 ** 24
    assert np.array_equal(part.cpu().numpy().astype(np.int64), P)


def test_static_activation_per_channel_weight_linear(Q):
    """Appendix C's latent-diffusion setting: activations quantized with one
    static calibrated scale, weights per output channel."""
    M, N, K = 256, 320, 1152
    xa = inputs.laplace_activations(M, K, seed=17)
    xw = inputs.gaussian_weights(N, K, seed=18)
    scale = np.float16(np.abs(xa.astype(np.float32)).max() / 127 * 0.8)   # clips the largest 20%
    a = Q.quantize_static(torch.from_numpy(xa).cuda(), scale, group_s=16, group_q=K)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16, group_q=K)
    y = Q.linear(a, w, out_dtype=torch.float32)
    assert Q.device_status() == 0
    ref, rabs = O.linear(O.encode_static(xa, scale, K, 16), O.encode(xw, K, 16), with_abs=True)
    _tol_check(y.cpu().numpy(), ref, rabs, 1, "float32")


@pytest.mark.parametrize("algo", list(ALGOS))
@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
@pytest.mark.parametrize("gs", [8, 16, 64])
def test_linear_packed_flags_identical(Q, algo, mode, gs):
    """Operands stored with FLAGs two per byte give the same bits as with
    one FLAG byte per subgroup (each operand independently)."""
    M, N, K = 200, 264, 576
    xa = inputs.mixture_activations(M, K, seed=M + gs)
    xw = inputs.gaussian_weights(N, K, seed=N + gs)
    a8 = Q.quantize(torch.from_numpy(xa).cuda(), group_s=gs, mode=mode)
    w8 = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=gs, mode=mode)
    a4 = Q.quantize(torch.from_numpy(xa).cuda(), group_s=gs, mode=mode, flag_bits=4)
    w4 = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=gs, mode=mode, flag_bits=4)
    ref = Q.linear(a8, w8, out_dtype=torch.float32, algo=ALGOS[algo])
    for a, w in ((a4, w4), (a4, w8), (a8, w4)):
        y = Q.linear(a, w, out_dtype=torch.float32, algo=ALGOS[algo])
        assert Q.device_status() == 0
        assert torch.equal(y, ref)


def test_linear_f16_packed_flag_output(Q):
    M, N, K = 128, 256, 1152
    x = torch.from_numpy(inputs.mixture_activations(M, K, seed=11)).cuda()
    w = Q.encode_weights(torch.from_numpy(inputs.gaussian_weights(N, K, seed=12)).cuda(), flag_bits=4)
    a_out = Q.empty_encoded(M, K, Q.Params(64, 16, O.SYMMETRIC, 4), x.device)
    y = Q.linear_f16(x, w, a_out=a_out)
    a = Q.quantize(x, flag_bits=4)
    assert torch.equal(a_out.flags, a.flags) and torch.equal(a_out.codes, a.codes)
    assert torch.equal(y, Q.linear(a, w))


@pytest.mark.parametrize("algo", list(ALGOS))
@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
def test_prepared_weights_identical(Q, algo, mode):
    """Weights prepared once give the same bits as preparing them per call."""
    xa = inputs.laplace_activations(200, 640, seed=8100)
    xw = inputs.gaussian_weights(264, 640, seed=8101)
    bias = np.random.default_rng(3).normal(0, 0.1, 264).astype(np.float16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=16, mode=mode)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16, mode=mode)
    b = torch.from_numpy(bias).cuda()
    prep = Q.prepare_weights(w)
    y0, p0 = Q.linear(a, w, b, algo=ALGOS[algo], partials_group=3)
    y1, p1 = Q.linear(a, w, b, algo=ALGOS[algo], w_prepared=prep, partials_group=3)
    # without partials the tcgen05 launch cuts these 4 tiles along K (another
    # summation order): compare like with like
    y2 = Q.linear(a, w, b, algo=ALGOS[algo], w_prepared=prep)   # reusable
    y3 = Q.linear(a, w, b, algo=ALGOS[algo])
    assert Q.device_status() == 0
    assert torch.equal(y0, y1) and torch.equal(y2, y3) and torch.equal(p0, p1)


@pytest.mark.parametrize("kind", ["per_row", "wide", "packed"])
def test_prepared_weights_other_formats(Q, kind):
    xa = inputs.laplace_activations(130, 1152, seed=8200)
    xw = inputs.gaussian_weights(136, 1152, seed=8201)
    kw = {"per_row": dict(group_q=1152), "wide": dict(group_s=8, code_bits=16),
          "packed": dict(flag_bits=4)}[kind]
    gs = kw.pop("group_s", 16)
    a = Q.quantize(torch.from_numpy(xa).cuda(), group_s=gs, **kw)
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=gs, **kw)
    prep = Q.prepare_weights(w)
    y0 = Q.linear(a, w)
    y1 = Q.linear(a, w, w_prepared=prep)
    assert Q.device_status() == 0
    assert torch.equal(y0, y1)


def test_prepared_weights_flux_fc1(Q):
    layer = inputs.CONFIG4[2]
    a = Q.quantize(torch.from_numpy(layer.activations()).cuda(), group_s=16)
    w = Q.encode_weights(torch.from_numpy(layer.weights()).cuda(), group_s=16)
    y0 = Q.linear(a, w)
    y1 = Q.linear(a, w, w_prepared=Q.prepare_weights(w))
    assert Q.device_status() == 0
    assert torch.equal(y0, y1)


def test_linear_f16_prepared_weights_identical(Q):
    xa = inputs.laplace_activations(300, 1216, seed=8300)
    xw = inputs.gaussian_weights(520, 1216, seed=8301)
    x = torch.from_numpy(xa).cuda()
    w = Q.encode_weights(torch.from_numpy(xw).cuda(), group_s=16)
    y0 = Q.linear_f16(x, w)
    a_out = Q.empty_encoded(300, 1216, Q.Params(64, 16), "cuda")
    y1 = Q.linear_f16(x, w, w_prepared=Q.prepare_weights(w), a_out=a_out)
    a = Q.quantize(x, group_s=16)
    y2 = Q.linear(a, w)
    assert Q.device_status() == 0
    assert torch.equal(y0, y1) and torch.equal(y0, y2)
    assert torch.equal(a_out.codes, a.codes) and torch.equal(a_out.flags, a.flags)
    assert torch.equal(a_out.scales, a.scales)


def test_back_to_back_calls_share_buffers(Q):
    """The kernels are launched with programmatic dependent launch and each
    waits for its predecessor before touching memory.  Calls issued back to
    back on one stream that share one encoded-activation buffer and one
    workspace (each encoder overwrites what the previous GEMM reads; split
    and unsplit GEMMs, two-call and fused paths) give bit-identical results
    to the same calls run one at a time with a synchronisation between."""
    M, K = 1100, 640
    Ns = [4400, 1200, 4096, 520]  # 4096: 144 tiles, unsplit; the others split
    xs = [torch.from_numpy(inputs.laplace_activations(M, K, seed=8400 + i)).cuda() for i in range(len(Ns))]
    ws = [Q.encode_weights(torch.from_numpy(inputs.gaussian_weights(n, K, seed=8500 + i)).cuda(), group_s=16)
          for i, n in enumerate(Ns)]
    a_buf = Q.empty_encoded(M, K, Q.Params(64, 16), "cuda")
    work = torch.empty(max(Q.linear_workspace_size(M, n, K) for n in Ns), dtype=torch.uint8, device="cuda")

    def run(sync):
        ys = []
        for _ in range(2):
            for x, w in zip(xs, ws):
                a = Q.quantize(x, group_s=16, out=a_buf)
                ys.append(Q.linear(a, w, workspace=work))
                if sync:
                    torch.cuda.synchronize()
                ys.append(Q.linear_f16(x, w, workspace=work))
                if sync:
                    torch.cuda.synchronize()
        torch.cuda.synchronize()
        return ys

    ref = run(True)
    got = run(False)
    assert Q.device_status() == 0
    for i, (r, g) in enumerate(zip(ref, got)):
        assert torch.equal(r, g), f"call {i} differs when issued back to back"
    for i in range(len(Ns)):
        assert torch.equal(ref[2 * i], ref[2 * i + 1])  # two-call and fused paths agree


def test_three_stream_pipeline_matches_synchronous(Q):
    """Host-to-device copies on one stream, quantize + linear on another and
    device-to-host copies on a third, ordered only by events, with each
    device buffer reused two units later (the end-to-end pattern of the
    benchmark): every host output equals the one a synchronous run gives."""
    M, K = 700, 1152
    Ns = [1152, 4608, 3456]
    xs = [torch.from_numpy(inputs.laplace_activations(M, K, seed=8600 + i)).pin_memory() for i in range(len(Ns))]
    ws = [Q.encode_weights(torch.from_numpy(inputs.gaussian_weights(n, K, seed=8700 + i)).cuda(), group_s=16)
          for i, n in enumerate(Ns)]
    preps = [Q.prepare_weights(w) for w in ws]
    work = torch.empty(max(Q.linear_workspace_size(M, n, K) for n in Ns), dtype=torch.uint8, device="cuda")
    enc = Q.empty_encoded(M, K, Q.Params(64, 16), "cuda")
    steps = 3
    units = [(k, i) for k in range(steps) for i in range(len(Ns))]

    ref = []
    for k, i in units:
        a = Q.quantize(xs[i].cuda(), group_s=16)
        ref.append(Q.linear(a, ws[i], w_prepared=preps[i]).cpu())

    x_buf = [torch.empty((M, K), dtype=torch.float16, device="cuda") for _ in range(2)]
    y_buf = [[torch.empty((M, n), dtype=torch.float16, device="cuda") for n in Ns] for _ in range(2)]
    y_host = [torch.empty((M, Ns[i]), dtype=torch.float16).pin_memory() for _, i in units]
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    main = torch.cuda.current_stream()
    loaded, consumed, computed, drained = {}, {}, {}, {}
    for u, (k, i) in enumerate(units):
        p = u % 2
        with torch.cuda.stream(s_in):
            if u >= 2:
                s_in.wait_event(consumed[u - 2])
            x_buf[p].copy_(xs[i], non_blocking=True)
            loaded[u] = torch.cuda.Event(); loaded[u].record(s_in)
        main.wait_event(loaded[u])
        Q.quantize(x_buf[p], out=enc, group_s=16)
        consumed[u] = torch.cuda.Event(); consumed[u].record(main)
        if u >= 2:
            main.wait_event(drained[u - 2])
        Q.linear(enc, ws[i], out=y_buf[p][i], workspace=work, w_prepared=preps[i])
        computed[u] = torch.cuda.Event(); computed[u].record(main)
        with torch.cuda.stream(s_out):
            s_out.wait_event(computed[u])
            y_host[u].copy_(y_buf[p][i], non_blocking=True)
            drained[u] = torch.cuda.Event(); drained[u].record(s_out)
    torch.cuda.synchronize()
    assert Q.device_status() == 0
    for u in range(len(units)):
        assert torch.equal(y_host[u], ref[u]), f"unit {u} differs"


def test_graph_replay_matches_eager(Q):
    """quantize + linear and the fused path captured into one CUDA graph
    (kernels with programmatic dependent launch keep their ordering inside
    a graph) and replayed twice give the eager results bit for bit."""
    M, K = 1100, 640
    Ns = [4400, 4096]  # split last wave / whole tiles
    xs = [torch.from_numpy(inputs.laplace_activations(M, K, seed=8800 + i)).cuda() for i in range(len(Ns))]
    ws = [Q.encode_weights(torch.from_numpy(inputs.gaussian_weights(n, K, seed=8900 + i)).cuda(), group_s=16)
          for i, n in enumerate(Ns)]
    preps = [Q.prepare_weights(w) for w in ws]
    work = torch.empty(max(Q.linear_workspace_size(M, n, K) for n in Ns), dtype=torch.uint8, device="cuda")
    enc = Q.empty_encoded(M, K, Q.Params(64, 16), "cuda")
    ys = [torch.empty((M, n), dtype=torch.float16, device="cuda") for n in Ns]
    yf = [torch.empty((M, n), dtype=torch.float16, device="cuda") for n in Ns]

    def body(stream):
        for i in range(len(Ns)):
            Q.quantize(xs[i], out=enc, group_s=16, stream=stream)
            Q.linear(enc, ws[i], out=ys[i], workspace=work, w_prepared=preps[i], stream=stream)
            Q.linear_f16(xs[i], ws[i], out=yf[i], workspace=work, w_prepared=preps[i], stream=stream)

    body(None)
    torch.cuda.synchronize()
    ref = [y.clone() for y in ys] + [y.clone() for y in yf]
    for y in ys + yf:
        y.zero_()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side):
            body(side)
    torch.cuda.current_stream().wait_stream(side)
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        assert Q.device_status() == 0
        for r, y in zip(ref, ys + yf):
            assert torch.equal(r, y)
        for y in ys + yf:
            y.zero_()


def test_two_host_threads(Q):
    """Two host threads, each with its own stream, workspace and buffers,
    issue quantize + linear and the fused path concurrently (the ctypes
    calls release the GIL): every result equals the one a single thread
    gives."""
    import threading

    M, K = 700, 1152
    Ns = [4608, 1152]
    xs = [torch.from_numpy(inputs.laplace_activations(M, K, seed=9000 + i)).cuda() for i in range(2)]
    ws = [Q.encode_weights(torch.from_numpy(inputs.gaussian_weights(n, K, seed=9100 + i)).cuda(), group_s=16)
          for i, n in enumerate(Ns)]
    preps = [Q.prepare_weights(w) for w in ws]
    torch.cuda.synchronize()

    def job(i, stream, out):
        work = torch.empty(Q.linear_workspace_size(M, Ns[i], K), dtype=torch.uint8, device="cuda")
        with torch.cuda.stream(stream):
            for _ in range(5):
                a = Q.quantize(xs[i], group_s=16, stream=stream)
                out.append(Q.linear(a, ws[i], workspace=work, w_prepared=preps[i], stream=stream))
                out.append(Q.linear_f16(xs[i], ws[i], workspace=work, w_prepared=preps[i], stream=stream))
        stream.synchronize()

    ref = [[], []]
    for i in range(2):
        job(i, torch.cuda.Stream(), ref[i])
    got = [[], []]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    threads = [threading.Thread(target=job, args=(i, streams[i], got[i])) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    torch.cuda.synchronize()
    assert Q.device_status() == 0
    for i in range(2):
        assert len(got[i]) == len(ref[i])
        for r, g in zip(ref[i], got[i]):
            assert torch.equal(r, g)
