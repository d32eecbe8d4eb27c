"""Pins of the CPU oracle against what the paper and mathematics fix.

These tests never compare the oracle with itself: each check is a closed
form, an invariant, an exhaustive enumeration against an independent
characterisation, a library routine for a special case, a hand-worked
example (tests/golden) or exact rational arithmetic.
"""
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as O
from paper_2509_26436_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# IEEE binary16 conversions: special case that reduces to a library routine
# --------------------------------------------------------------------------

def test_half_to_float_all_bit_patterns():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ref = bits.view(np.float16).astype(np.float32)
    got = np.array([O.half_to_float(int(b)) for b in bits], dtype=np.float32)
    finite = np.isfinite(ref)
    assert np.array_equal(got[finite].view(np.uint32), ref[finite].view(np.uint32))
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    assert np.array_equal(np.isinf(got), np.isinf(ref))


def test_float_to_half_matches_numpy_rne():
    rng = np.random.default_rng(1)
    vals = [rng.standard_normal(4000).astype(np.float32) * np.float32(10.0) ** rng.integers(-9, 5, 4000)]
    # every binary16 midpoint and its float32 neighbours exercise ties-to-even
    h = np.arange(0, 0x7BFF, 7, dtype=np.uint16).view(np.float16).astype(np.float64)
    h_next = np.nextafter(h.astype(np.float16), np.float16(np.inf)).astype(np.float64)
    mid = ((h + h_next) / 2).astype(np.float32)
    vals += [mid, np.nextafter(mid, np.float32(0)), np.nextafter(mid, np.float32(1e9))]
    vals += [np.array([0.0, -0.0, 65504, 65519.99, 65520, 1e6, 2 ** -24, 2 ** -25,
                       2 ** -25 * 1.0000001, 2 ** -14, 6.1e-5], np.float32)]
    x = np.concatenate(vals).astype(np.float32)
    x = np.concatenate([x, -x])
    with np.errstate(over="ignore"):
        ref = x.astype(np.float16).view(np.uint16)
    got = np.array([O.float_to_half(float(v)) for v in x], dtype=np.uint16)
    assert np.array_equal(got, ref)


def test_clz32_definition():
    for v in [0, 1, 2, 3, 7, 8, 127, 128, 2 ** 31, 2 ** 32 - 1] + list(range(0, 300)):
        assert O.clz32(v) == 32 - int(v).bit_length()


# --------------------------------------------------------------------------
# LZS (Eq. 2) -- exhaustive over all int8 codes, against Appendix A's H(m)
# --------------------------------------------------------------------------

def _bitlen_H(m: int) -> int:
    """Appendix A: H(0) = 0, H(m) = floor(log2 m) + 1."""
    return 0 if m == 0 else int(np.floor(np.log2(m))) + 1


def test_lzs_exhaustive_all_int8_codes():
    codes = np.arange(-127, 128, dtype=np.int8)
    flags, c = O.lzs_encode(codes, 1)
    v = O.lzs_decode(c, flags, 1)
    hist = {}
    for q, f, ci, vi in zip(codes.astype(int), flags.astype(int), c.astype(int), v.astype(int)):
        mag = abs(q)
        H = _bitlen_H(mag)
        # Appendix A: the lower H(m) - 3 magnitude bits are discarded when H >= 4
        assert f == max(H - 3, 0)
        assert f in (0, 1, 2, 3, 4)                       # Eq. 2 range
        assert abs(ci) <= 7                                # 3 magnitude bits + sign
        assert ci == int(np.sign(q)) * (mag >> f)
        assert vi == int(np.sign(q)) * ((mag >> f) << f)
        if mag < 8:
            assert vi == q                                 # bottom 3 bits preserved
        hist[f] = hist.get(f, 0) + (1 if q >= 0 else 0)
    # magnitudes 0..127: FLAG histogram fixed by H(m)
    assert hist == {0: 8, 1: 8, 2: 16, 3: 32, 4: 64}
    mags = sorted(set(abs(int(x)) for x in v))
    assert mags == list(range(8)) + [8, 10, 12, 14, 16, 20, 24, 28, 32, 40, 48, 56, 64, 80, 96, 112]


def test_lzs_rejects_code_minus_128():
    with pytest.raises(ValueError):
        O.lzs_flag(np.array([-128], np.int8))
    with pytest.raises(ValueError):
        O.lzs_encode(np.array([3, -128], np.int8), 2)


def test_lzs_all_pairs_minimal_shift():
    """G_s = 2 over all 255^2 code pairs: FLAG is the smallest right shift
    that leaves every magnitude of the subgroup within 3 bits (the shared
    representation starts at the top-most active bit)."""
    a = np.repeat(np.arange(-127, 128), 255).astype(np.int8)
    b = np.tile(np.arange(-127, 128), 255).astype(np.int8)
    q = np.stack([a, b], axis=1).ravel()
    flags, c = O.lzs_encode(q, 2)
    mag = np.abs(q.astype(np.int32)).reshape(-1, 2)
    f_min = np.zeros(mag.shape[0], np.int32)
    for f in range(5, -1, -1):
        fits = ((mag >> f) <= 7).all(axis=1)
        f_min = np.where(fits, f, f_min)
    assert np.array_equal(flags.astype(np.int32), f_min)
    assert np.array_equal(c.astype(np.int32).reshape(-1, 2),
                          np.sign(q.astype(np.int32)).reshape(-1, 2) * (mag >> f_min[:, None]))


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
def test_lzs_truncation_bound_and_sign(gs):
    """Appendix A: truncation toward zero, error <= 2^FLAG - 1 LSBs, no sign
    error; lossless when every magnitude of the subgroup is < 8 (Section 3)."""
    rng = np.random.default_rng(gs)
    scale = np.repeat(rng.choice([0.5, 2.0, 6.0, 30.0], 64 * 512 // gs), gs)
    q = np.clip(np.round(rng.laplace(0, 1, 64 * 512) * scale), -127, 127).astype(np.int8)
    flags, c = O.lzs_encode(q, gs)
    v = O.lzs_decode(c, flags, gs).astype(np.int32)
    qi = q.astype(np.int32)
    F = np.repeat(flags.astype(np.int32), gs)
    err = np.abs(qi) - np.abs(v)
    assert (err >= 0).all() and (err <= (1 << F) - 1).all()
    assert ((np.sign(v) == np.sign(qi)) | (v == 0)).all()
    assert (np.abs(c) <= 7).all()
    # the kept window starts at the top-most active bit: |c| >= 4 somewhere
    cmax = np.abs(c.astype(np.int32)).reshape(-1, gs).max(axis=1)
    assert (cmax[flags > 0] >= 4).all()
    small = (np.abs(qi).reshape(-1, gs).max(axis=1) < 8)
    assert small.any()
    assert np.array_equal(v.reshape(-1, gs)[small], qi.reshape(-1, gs)[small])
    assert (flags[small] == 0).all()


def test_nibble_layout_and_roundtrip():
    # hand example: two's complement nibbles, even index in the low nibble
    packed = O.pack_nibbles(np.array([1, -1, 7, -7], np.int8))
    assert list(packed) == [0xF1, 0x97]
    c = np.arange(-7, 8, dtype=np.int8)
    c = np.concatenate([c, c[::-1], [0]]).astype(np.int8)
    assert np.array_equal(O.unpack_nibbles(O.pack_nibbles(c), c.size), c)


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                rows.append(line.rstrip("\n"))
    return rows


def test_lzs_golden_worked_examples():
    for line in _read_golden("lzs_worked_examples.txt"):
        q, m, clz, flag, c, v, _ = [p.strip() for p in line.split("|", 6)]
        q = np.array([int(t) for t in q.split()], np.int8)
        assert int(np.bitwise_or.reduce(np.abs(q.astype(np.int32)))) == int(m)
        assert O.clz32(int(m)) == int(clz)
        f, cc = O.lzs_encode(q, 4)
        assert int(f[0]) == int(flag)
        assert list(cc) == [int(t) for t in c.split()]
        assert list(O.lzs_decode(cc, f, 4)) == [int(t) for t in v.split()]


def test_quantize_golden_worked_example():
    g = {}
    for line in _read_golden("quantize_worked_example.txt"):
        k, *vals = line.split()
        g[k] = vals
    x = np.zeros((1, 64), np.float16)
    x[0, :3] = [1.0, -0.5, 0.25]
    q, s, z = O.quantize(x, 64, O.SYMMETRIC)
    assert int(s.view(np.uint16)[0, 0]) == int(g["scale_bits"][0], 16)
    assert list(q[0, :4]) == [int(t) for t in g["q"]]
    assert (q[0, 4:] == 0).all() and z[0, 0] == 0
    e = O.encode(x, 64, 16, O.SYMMETRIC)
    assert list(e.flags[0]) == [int(t) for t in g["flags"]]
    assert list(O.unpack_nibbles(e.codes[0], 64)[:4]) == [int(t) for t in g["c"]]
    assert list(O.decode_values(e)[0, :4]) == [int(t) for t in g["v"]]


# --------------------------------------------------------------------------
# Stage 1 quantizer (Eq. 1) against exact rational arithmetic
# --------------------------------------------------------------------------

def _nearest_half_exact(fr: Fraction) -> int:
    """bits of the binary16 value nearest to a non-negative rational,
    ties to even, by exact comparison with its two neighbours."""
    lo = np.float16(float(fr))
    cand = {lo, np.nextafter(lo, np.float16(0)), np.nextafter(lo, np.float16(np.inf))}
    best = None
    for c in cand:
        d = abs(Fraction(float(c)) - fr)
        key = (d, int(np.array(c).view(np.uint16)) & 1)
        if best is None or key < best[0]:
            best = (key, c)
    return int(np.array(best[1]).view(np.uint16))


def test_symmetric_scale_is_correctly_rounded():
    """s16 = binary16(max|x| / 127) with a single rounding of the exact
    quotient: the binary32 intermediate never lands on a binary16 tie
    because x/127 has a period-7 binary expansion."""
    x = inputs.mixture_activations(64, 4096, seed=7)
    q, s, _ = O.quantize(x, 64, O.SYMMETRIC)
    xs = x.astype(np.float32).reshape(64, -1, 64)
    amax = np.abs(xs).max(axis=2)
    sb = s.view(np.uint16)
    for i in range(0, amax.shape[0]):
        for g in range(0, amax.shape[1], 3):
            exact = Fraction(float(amax[i, g])) / 127
            assert sb[i, g] == _nearest_half_exact(exact)


def test_symmetric_codes_against_exact_rounding():
    """x_hat = clamp(round(x/s)) with exact rational x/s: identical except
    within 2^-16 of a half-integer (binary32 reciprocal-multiply), and the
    element of largest magnitude lands on |q| = 127 whenever s is normal."""
    x = inputs.laplace_activations(16, 1152, seed=3)
    q, s, z = O.quantize(x, 64, O.SYMMETRIC)
    assert (z == 0).all()
    G = 1152 // 64
    mism = 0
    for i in range(16):
        for g in range(G):
            sv = Fraction(float(s[i, g]))
            xs = x[i, g * 64:(g + 1) * 64].astype(np.float64)
            for k in range(64):
                t = Fraction(float(xs[k])) / sv
                fl = t.numerator // t.denominator
                frac = t - fl
                exact = fl + (1 if frac > Fraction(1, 2) or (frac == Fraction(1, 2) and fl % 2) else 0)
                exact = max(-127, min(127, exact))
                if exact != int(q[i, g * 64 + k]):
                    mism += 1
                    assert abs(frac - Fraction(1, 2)) < Fraction(1, 2 ** 16)
                if abs(t) < 127:
                    assert abs(Fraction(float(xs[k])) - sv * int(q[i, g * 64 + k])) <= sv / 2 * (1 + Fraction(1, 2 ** 14))
            if float(s[i, g]) >= 2 ** -14:
                assert np.abs(q[i, g * 64:(g + 1) * 64]).max() == 127
    assert mism <= 2


def test_degenerate_groups():
    x = np.zeros((3, 128), np.float16)
    x[1, 64:] = 1e-7     # underflows: max/127 < half of the smallest subnormal
    x[2, :64] = 0.5      # all equal
    for mode in (O.SYMMETRIC, O.ASYMMETRIC):
        q, s, z = O.quantize(x, 64, mode)
        assert (s.view(np.uint16)[0] == 0).all() and (q[0] == 0).all() and (z[0] == 0).all()
        assert s.view(np.uint16)[1, 1] == 0 and (q[1, 64:] == 0).all()
    q, s, z = O.quantize(x, 64, O.SYMMETRIC)
    assert (q[2, :64] == 127).all()


def test_asymmetric_reconstruction():
    """Eq. 1 with 255 levels: x ~ s*(q - z) within half a step, except that
    the clamp to [-127, 127] clips an end level by at most one step; real zero
    is exactly representable."""
    x = inputs.silu_im2col(1, 64, 8, 8, seed=5)
    x = np.concatenate([x, np.abs(x[:4])], axis=0)  # some one-sided groups
    q, s, z = O.quantize(x, 64, O.ASYMMETRIC)
    G = x.shape[1] // 64
    for i in range(x.shape[0]):
        for g in range(G):
            sv = float(s[i, g])
            if sv == 0:
                continue
            xs = x[i, g * 64:(g + 1) * 64].astype(np.float64)
            xh = sv * (q[i, g * 64:(g + 1) * 64].astype(np.float64) - z[i, g])
            err = np.abs(xs - xh)
            clipped = np.abs(q[i, g * 64:(g + 1) * 64].astype(np.int32)) == 127
            assert (err[~clipped] <= sv / 2 * (1 + 2 ** -12)).all()
            assert (err[clipped] <= sv * 1.5 * (1 + 2 ** -12)).all()
            assert -128 <= z[i, g] <= 127


# --------------------------------------------------------------------------
# GEMM and dequantised linear
# --------------------------------------------------------------------------

def test_group_partials_match_float_matmul():
    """P_g over decoded integers equals an exact float64 matmul per group
    (all sums are integers far below 2^53)."""
    a = O.encode(inputs.laplace_activations(24, 256, seed=11), 64, 16)
    w = O.encode(inputs.gaussian_weights(40, 256, seed=12), 64, 16)
    va, vw = O.decode_values(a), O.decode_values(w)
    P = O.group_partials(va, vw, 64)
    for g in range(4):
        ref = va[:, g * 64:(g + 1) * 64].astype(np.float64) @ vw[:, g * 64:(g + 1) * 64].astype(np.float64).T
        assert np.array_equal(P[g].astype(np.float64), ref)
    rows = np.array([23, 0, 7])
    assert np.array_equal(O.group_partials(va, vw, 64, rows), P[:, rows])
    assert np.abs(P).max() <= 64 * 112 * 112


def test_group_partials_tiny_closed_form():
    va = np.full((2, 128), 3, np.int16)
    va[1, 64:] = -112
    vw = np.full((1, 128), 7, np.int16)
    P = O.group_partials(va, vw, 64)
    assert P[:, :, 0].tolist() == [[64 * 21, 64 * 21], [64 * 21, -64 * 784]]


@pytest.mark.parametrize("mode", [O.SYMMETRIC, O.ASYMMETRIC])
@pytest.mark.parametrize("gs", [8, 16, 32])
def test_linear_equals_dequantised_matmul(mode, gs):
    """y = x_hat_a @ x_hat_w^T (+bias) with x_hat = s (v - z): the
    integer-partials-then-scale route equals dequantise-then-multiply."""
    xa = inputs.laplace_activations(12, 320, seed=21)
    xw = inputs.gaussian_weights(20, 320, seed=22)
    bias = inputs.gaussian_weights(1, 20, seed=23)[0]
    a, w = O.encode(xa, 64, gs, mode), O.encode(xw, 64, gs, mode)
    ref = O.dequantize(a) @ O.dequantize(w).T + bias.astype(np.float64)
    y = O.linear(a, w, bias)
    assert np.allclose(y, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())
    rows = np.array([5, 11])
    assert np.array_equal(O.linear(a, w, bias, rows), y[rows])
    # quantization noise only: near the unquantised product (a dropped scale
    # or a transposed operand gives a relative error near or above 1)
    exact = xa.astype(np.float64) @ xw.astype(np.float64).T + bias.astype(np.float64)
    rel = np.linalg.norm(y - exact) / np.linalg.norm(exact)
    assert rel < 0.5


def test_encoder_sidecars_consistent():
    x = inputs.laplace_activations(5, 256, seed=31)
    e = O.encode(x, 64, 16, O.ASYMMETRIC)
    v = O.decode_values(e).astype(np.int64)
    assert np.array_equal(v.reshape(5, 4, 64).sum(axis=2), e.gsum)
    q, s, z = O.quantize(x, 64, O.ASYMMETRIC)
    assert np.array_equal(s.view(np.uint16), e.scales.view(np.uint16))
    assert np.array_equal(z, e.zeros)
    f, c = O.lzs_encode(q.ravel(), 16)
    assert np.array_equal(f, e.flags.ravel())
    assert np.array_equal(O.pack_nibbles(c), e.codes.ravel())


# --------------------------------------------------------------------------
# Appendix A error theory and Section 4.2 entropy on generated distributions
# --------------------------------------------------------------------------

def _dists():
    rng = np.random.default_rng(99)
    return {
        "laplace": rng.laplace(0, 0.05, (8, 4096)),
        "gaussian": rng.normal(0, 0.05, (8, 4096)),
        "mixture": inputs.mixture_activations(8, 4096, seed=98).astype(np.float64),
    }


@pytest.mark.parametrize("name", ["laplace", "gaussian", "mixture"])
def test_appendix_a_error_bound(name):
    """Per-tensor symmetric int8 (one group per row) followed by LZS with
    G_s = 1: the mean truncation error is at most s8 * sum_k P_k (2^(k-3)-1)
    (Appendix A), E_total <= E_q^8 + E_LZS, and when P(|J| >= 8) < 1/2 the
    total error stays below naive 4-bit's s4/2 = 8 s8."""
    x = _dists()[name].astype(np.float16)
    R, K = x.shape
    q, s, _ = O.quantize(x, K, O.SYMMETRIC)
    flags, c = O.lzs_encode(q.ravel(), 1)
    v = O.lzs_decode(c, flags, 1).reshape(R, K).astype(np.float64)
    xf = x.astype(np.float64)
    for i in range(R):
        s8 = float(s[i, 0])
        m = np.abs(q[i].astype(np.int64))
        H = np.array([_bitlen_H(int(t)) for t in m])
        Pk = np.array([(H == k).mean() for k in range(8)])
        bound = sum(Pk[k] * (2 ** (k - 3) - 1) for k in range(4, 8))
        e_lzs = np.abs(q[i].astype(np.float64) - v[i]).mean()
        assert e_lzs <= bound + 1e-12
        e_q8 = np.abs(xf[i] - s8 * q[i]).mean()
        e_tot = np.abs(xf[i] - s8 * v[i]).mean()
        assert e_tot <= e_q8 + s8 * e_lzs + 1e-12
        if (m >= 8).mean() < 0.5:
            assert e_tot < 8 * s8


def _naive_int4_same_range(x, s8):
    """Naive signed 4-bit midtread quantizer covering the same range as the
    8-bit one, s4 = 16 s8 (Appendix A), i.e. the paper's INT4 baseline."""
    s4 = 16.0 * s8
    q4 = np.clip(np.round(x / s4), -7, 7)
    return q4.astype(np.int8), q4 * s4


def _entropy(codes):
    p = np.bincount((codes.astype(np.int32) & 15).ravel(), minlength=16) / codes.size
    p = p[p > 0]
    return -(p * np.log2(p)).sum()


@pytest.mark.parametrize("name", ["mixture", "laplace_outliers"])
@pytest.mark.parametrize("gs", [1, 16, 32])
def test_theorem1_and_entropy_vs_naive_int4(name, gs):
    """Theorem 1 / Section 4.2 in the setting the paper states them for: a
    static per-tensor activation range (Appendix C, LDM setting), here one
    quantization group per 4096-wide row, on outlier-heavy data where
    P(|J| >= 8) < 1/2.  QuaRTZ's mean absolute error is below naive INT4's
    and its 4-bit codes have higher entropy."""
    if name == "mixture":
        x = inputs.mixture_activations(8, 4096, seed=98)
    else:
        x = inputs.laplace_activations(8, 4096, seed=97)
    R, K = x.shape
    q, s, _ = O.quantize(x, K, O.SYMMETRIC)
    assert (np.abs(q.astype(np.int32)) >= 8).mean() < 0.5      # theorem's condition
    flags, c = O.lzs_encode(q.ravel(), gs)
    v = O.lzs_decode(c, flags, gs).reshape(R, K).astype(np.float64)
    s8 = np.repeat(s.astype(np.float64), K, axis=1)
    xf = x.astype(np.float64)
    q4, xh4 = _naive_int4_same_range(xf, s8)
    assert np.abs(xf - s8 * v).mean() < np.abs(xf - xh4).mean()
    assert _entropy(c) > _entropy(q4)


@pytest.mark.parametrize("name", ["laplace", "gaussian", "mixture"])
def test_elementwise_lzs_beats_naive_int4(name):
    """With G_s = 1 every element keeps its own top 3 magnitude bits; the
    error stays below naive INT4 of the same range on every distribution."""
    x = _dists()[name].astype(np.float16)
    R, K = x.shape
    q, s, _ = O.quantize(x, K, O.SYMMETRIC)
    flags, c = O.lzs_encode(q.ravel(), 1)
    v = O.lzs_decode(c, flags, 1).reshape(R, K).astype(np.float64)
    s8 = np.repeat(s.astype(np.float64), K, axis=1)
    xf = x.astype(np.float64)
    _, xh4 = _naive_int4_same_range(xf, s8)
    assert np.abs(xf - s8 * v).mean() < np.abs(xf - xh4).mean()


def test_quantize_ties_and_zero_point_golden():
    g = {}
    for line in _read_golden("quantize_ties_and_zero_point.txt"):
        k, *vals = line.split()
        g[k] = vals
    x = np.zeros((1, 64), np.float16)
    t = [float(v) for v in g["ties_x_times_1024"]]
    x[0, :len(t)] = np.array(t) * 2.0 ** -10
    q, s, z = O.quantize(x, 64, O.SYMMETRIC)
    assert int(s.view(np.uint16)[0, 0]) == int(g["ties_scale_bits"][0], 16)
    assert list(q[0, :len(t)]) == [int(v) for v in g["ties_q"]]
    x = np.zeros((1, 64), np.float16)
    t = [float(v) for v in g["asym_x"]]
    x[0, :len(t)] = t
    q, s, z = O.quantize(x, 64, O.ASYMMETRIC)
    assert int(s.view(np.uint16)[0, 0]) == int(g["asym_scale_bits"][0], 16)
    assert int(z[0, 0]) == int(g["asym_zero"][0])
    assert list(q[0, :len(t)]) == [int(v) for v in g["asym_q"]]
    assert (q[0, len(t):] == int(g["asym_zero"][0])).all()


# --- static per-tensor quantization (Appendix C, latent-diffusion setting) ---

def test_static_scale_equals_own_per_tensor_scale():
    """With the tensor's own per-tensor scale, static encoding equals dynamic
    encoding of the whole tensor as one quantization group (flattened to a
    single row): the dynamic route computes the scale from the data, the
    static route is handed it."""
    x = inputs.mixture_activations(8, 512, seed=91)
    s16 = np.float16(np.float32(np.abs(x.astype(np.float32)).max()) / np.float32(127))
    for gs in (8, 16, 32, 64):
        st = O.encode_static(x, s16, 512, gs)
        dyn = O.encode(x.reshape(1, -1), x.size, gs)
        assert np.array_equal(st.codes.reshape(-1), dyn.codes.reshape(-1))
        assert np.array_equal(st.flags.reshape(-1), dyn.flags.reshape(-1))
        assert np.all(st.scales.view(np.uint16) == dyn.scales.view(np.uint16)[0, 0])


def test_static_scale_saturates_and_rounds():
    """Closed form: q = clamp(round-half-even(x * r), -127, 127), r = RN(1/s),
    checked on values chosen exactly in units of s = 2^-4 (r exact)."""
    s16 = np.float16(2.0 ** -4)
    units = np.array([0, 1, -1, 2.5, -2.5, 3.5, 126.5, 127, 127.5, 200, -200, -300, 1000, -1e4])
    x = (units * 2.0 ** -4).astype(np.float16)
    q = O.quantize_static(x.reshape(1, -1), s16).ravel()
    expect = np.clip(np.round(units), -127, 127)      # numpy rounds half to even
    assert np.array_equal(q, expect.astype(np.int8))
    assert np.array_equal(O.quantize_static(x.reshape(1, -1), np.float16(0)).ravel(), np.zeros_like(q))


def test_static_scale_codes_follow_lzs_of_saturated_values():
    """Every saturated element becomes code +-7 with FLAG 4 (decoded +-112)."""
    x = np.full((1, 64), 50.0, np.float16)
    x[0, 1::2] = -50.0
    e = O.encode_static(x, np.float16(0.01), 64, 16)
    v = O.decode_values(e)
    assert np.all(np.abs(v) == 112) and np.all(e.flags == 4)


# --- LLM variant (Section 5): 16-bit codes compressed straight to 4 bits ---

def test_lzs16_exhaustive_all_16bit_codes():
    """Every code in [-32767, 32767] at G_s = 1: FLAG = max(H(m) - 3, 0) with
    Appendix A's bit length H, now ranging over 0..12, and FLAG is also the
    smallest right shift that leaves the magnitude within 3 bits."""
    q = np.arange(-32767, 32768, dtype=np.int16)
    flags, c = O.lzs_encode16(q, 1)
    qi = q.astype(np.int64)
    mag = np.abs(qi)
    H = np.array([int(m).bit_length() for m in mag])
    f = flags.astype(np.int64)
    assert np.array_equal(f, np.maximum(H - 3, 0))
    f_min = np.full(mag.size, -1)
    for t in range(15, -1, -1):
        f_min = np.where((mag >> t) <= 7, t, f_min)
    assert np.array_equal(f, f_min)
    assert f.max() == 12 and (np.abs(c) <= 7).all()
    assert np.array_equal(c.astype(np.int64), np.sign(qi) * (mag >> f))
    v = O.lzs_decode(c, flags, 1).astype(np.int64)
    assert np.abs(v).max() == 7 << 12 == 28672
    assert ((mag - np.abs(v)) < (1 << f)).all() and ((mag - np.abs(v)) >= 0).all()
    # FLAG histogram over magnitudes 0..32767 is fixed by H: 2^(F+2) codes per FLAG >= 1
    hist = np.bincount(f[qi >= 0], minlength=13)
    assert hist[0] == 8 and all(hist[F] == 1 << (F + 2) for F in range(1, 13))
    # the 8-bit codes are a subset: same FLAG and value on [-127, 127]
    f8, c8 = O.lzs_encode(np.arange(-127, 128, dtype=np.int8), 1)
    mid = slice(32767 - 127, 32767 + 128)
    assert np.array_equal(f8, flags[mid]) and np.array_equal(c8, c[mid])
    with pytest.raises(ValueError):
        O.lzs_encode16(np.array([5, -32768], np.int16), 2)


def test_quantize16_closed_form_on_exact_units():
    """Closed form of the 16-bit symmetric quantizer where every quantity is
    exact: max|x| = 4 gives s = binary16(4 / 32767) = 2^-13 (the quotient is
    2^-13 (1 + 1/32767), far below half a binary16 step), r = 2^13, and each
    x = u 2^-13 maps to clamp(round-half-even(u), -32767, 32767).  The value
    4.0 itself lands on 32768 and must saturate to 32767 (not wrap)."""
    units = np.array([0, 1, -1, 0.5, 1.5, 2.5, -2.5, 3.5, 513.5, 1000.5, 1001.5, 1543, 12344,
                      -12344, 20000, 32752, -32752, 32768, -32768])
    x = np.zeros((1, 64), np.float16)
    x[0, :units.size] = (units * 2.0 ** -13).astype(np.float16)
    exact = x[0, :units.size].astype(np.float64) * 2.0 ** 13
    assert np.array_equal(exact, units)    # binary16 holds every unit exactly
    q, s = O.quantize16(x, 64)
    assert s.view(np.uint16)[0, 0] == np.float16(2.0 ** -13).view(np.uint16)
    expect = np.clip(np.round(exact), -32767, 32767)   # numpy: half to even
    assert np.array_equal(q[0, :units.size].astype(np.int64), expect.astype(np.int64))
    assert q[0, list(units).index(32768)] == 32767 and q[0, list(units).index(-32768)] == -32767
    assert (q[0, units.size:] == 0).all()


def test_quantize16_against_exact_rounding():
    """16-bit codes against exact rational rounding of x / s: equal except
    within 2^-12 of a half-integer (binary32 reciprocal-multiply at 16-bit
    magnitudes), |x - s q| <= s / 2 for unsaturated elements, and the largest
    element of a group lands on 32767 up to the relative rounding error of
    the binary16 scale."""
    x = inputs.laplace_activations(4, 512, seed=13)
    q, s = O.quantize16(x, 64)
    mism = 0
    for i in range(4):
        for g in range(8):
            sv = Fraction(float(s[i, g]))
            xs = x[i, g * 64:(g + 1) * 64].astype(np.float64)
            for k in range(64):
                t = Fraction(float(xs[k])) / sv
                fl = t.numerator // t.denominator
                frac = t - fl
                ex = fl + (1 if frac > Fraction(1, 2) or (frac == Fraction(1, 2) and fl % 2) else 0)
                ex = max(-32767, min(32767, ex))
                if ex != int(q[i, g * 64 + k]):
                    mism += 1
                    assert abs(frac - Fraction(1, 2)) < Fraction(1, 2 ** 12)
                if abs(t) < 32767:
                    assert abs(Fraction(float(xs[k])) - sv * int(q[i, g * 64 + k])) <= sv / 2 * (1 + Fraction(1, 2 ** 10))
            # the binary16 scale is off max|x| / 32767 by at most half its own
            # spacing (2^-24 absolute once it is subnormal, i.e. max|x| < 2)
            rel = float(np.spacing(s[i, g])) / 2 / float(s[i, g])
            top = np.abs(q[i, g * 64:(g + 1) * 64].astype(np.int64)).max()
            assert 32767 * (1 - rel) / (1 + rel) - 1 <= top <= 32767
    assert mism <= 4


def test_encode16_truncation_bound_and_linear_exact():
    """LLM-variant encoding (G_s = 8): every decoded value is the 16-bit code
    truncated toward zero by its subgroup's FLAG (error < 2^FLAG steps, no
    sign error), and the W4A4 linear of two such operands equals the binary64
    product of the dequantised operands.  All-saturated rows make each
    64-wide group sum 64 x 28672^2 (> 2^31): an int32 accumulator would wrap."""
    xa = inputs.mixture_activations(6, 256, seed=17)
    xw = inputs.gaussian_weights(10, 256, seed=18)
    xa[0, :] = 8.0
    xw[0, :] = -2.0
    a = O.encode16(xa, 64, 8)
    w = O.encode16(xw, 64, 8)
    assert a.flags.max() == 12
    q, _ = O.quantize16(xa, 64)
    v = O.decode_values(a).astype(np.int64)
    qi = q.astype(np.int64)
    F = np.repeat(a.flags.astype(np.int64), 8, axis=1)
    err = np.abs(qi) - np.abs(v)
    assert (err >= 0).all() and (err < (1 << F)).all()
    assert ((np.sign(v) == np.sign(qi)) | (v == 0)).all()
    y = O.linear(a, w)
    ref = O.dequantize(a) @ O.dequantize(w).T
    assert np.allclose(y, ref, rtol=1e-12, atol=1e-12 * np.abs(ref).max())
    P = O.group_partials(O.decode_values(a), O.decode_values(w), 64)
    assert P[0, 0, 0] == -64 * 28672 * 28672 and abs(P[0, 0, 0]) > 2 ** 31


# --- attention decode step (Appendix D, Table 6) ----------------------------

def _attn_inputs(BH, L_max, d, gs, seed):
    q = O.encode(inputs.laplace_activations(BH, d, seed=seed, outlier_frac=0.01, outlier_scale=20.0), 64, gs)
    k = O.encode(inputs.laplace_activations(BH * L_max, d, seed=seed + 1, outlier_frac=0.01,
                                            outlier_scale=20.0), 64, gs)
    v = O.encode(inputs.mixture_activations(BH * L_max, d, seed=seed + 2), 64, gs)
    return q, k, v


@pytest.mark.parametrize("gs", [8, 16, 32])
def test_attention_equals_dense_softmax_of_dequantised(gs):
    """A different route: dequantise q, K, V (binary64), then dense
    softmax(q K^T scale) V with SciPy's softmax, per head over the first L
    cache rows of that head.  Catches a wrong cache row, a dropped scale, a
    transposed operand or a softmax over the wrong axis."""
    from scipy.special import softmax
    BH, L_max, L, d = 5, 40, 33, 128
    q, k, v = _attn_inputs(BH, L_max, d, gs, 300 + gs)
    scale = d ** -0.5
    o, oabs = O.attention_decode(q, k, v, L_max, L, scale, with_abs=True)
    qh, kh, vh = O.dequantize(q), O.dequantize(k), O.dequantize(v)
    for bh in range(BH):
        kk = kh[bh * L_max:bh * L_max + L]
        vv = vh[bh * L_max:bh * L_max + L]
        p = softmax(scale * (kk @ qh[bh]))
        ref = p @ vv
        assert np.allclose(o[bh], ref, rtol=1e-12, atol=1e-14)
        assert np.allclose(oabs[bh], p @ np.abs(vv), rtol=1e-12, atol=1e-14)


def test_attention_special_cases():
    """L = 1 returns that token's dequantised value exactly; a zero query
    gives equal weights (the mean of the V rows); every output lies in the
    hull of the V rows; rows beyond L never matter; a key aligned with the
    query and 60 nats ahead takes all the weight."""
    BH, L_max, d = 3, 20, 128
    q, k, v = _attn_inputs(BH, L_max, d, 16, 400)
    vh = O.dequantize(v)
    o1 = O.attention_decode(q, k, v, L_max, 1, 0.1)
    assert np.array_equal(o1, vh[0::L_max][:BH])
    qz = O.encode(np.zeros((BH, d), np.float16), 64, 16)
    L = 13
    oz = O.attention_decode(qz, k, v, L_max, L, 0.1)
    for bh in range(BH):
        rows = vh[bh * L_max:bh * L_max + L]
        assert np.allclose(oz[bh], rows.mean(axis=0), rtol=1e-12, atol=1e-15)
    o = O.attention_decode(q, k, v, L_max, L, 0.3)
    for bh in range(BH):
        rows = vh[bh * L_max:bh * L_max + L]
        assert (o[bh] >= rows.min(axis=0) - 1e-12).all() and (o[bh] <= rows.max(axis=0) + 1e-12).all()
    # rows beyond L ignored
    k2, v2 = _attn_inputs(BH, L_max, d, 16, 500)[1:]
    for dst, src in ((k, k2), (v, v2)):
        for bh in range(BH):
            sl = slice(bh * L_max + L, (bh + 1) * L_max)
            dst.codes[sl], dst.flags[sl], dst.scales[sl] = src.codes[sl], src.flags[sl], src.scales[sl]
    assert np.array_equal(O.attention_decode(q, k, v, L_max, L, 0.3), o)
    # a dominant key: q = k_t* = ones vs all other keys 0; after Eq. 1 and
    # LZS both decode to 112 s with s = fp16(1/127), so the gap is
    # 128 * scale * (112 s)^2 = 46.7 nats and the rest weighs < L e^-46
    xq = np.ones((1, d), np.float16)
    xk = np.zeros((L_max, d), np.float16)
    xk[7] = 1.0
    qd, kd = O.encode(xq, 64, 16), O.encode(xk, 64, 16)
    vd = O.encode(inputs.mixture_activations(L_max, d, seed=600), 64, 16)
    od = O.attention_decode(qd, kd, vd, L_max, L_max, 60.0 / 128)
    vmax = np.abs(O.dequantize(vd)).max()
    assert np.allclose(od[0], O.dequantize(vd)[7], rtol=0, atol=L_max * np.exp(-46) * vmax)
    assert not np.array_equal(od[0], O.dequantize(vd)[7])
