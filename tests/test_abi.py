"""C-ABI checks that need no GPU: the library builds and loads, exports every
symbol include/quartz.h declares, and rejects bad arguments on the host
before anything is launched."""
import ctypes as C
import os
import re

import pytest

from paper_2509_26436_gb300 import _native as N
from paper_2509_26436_gb300 import build as B

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "quartz.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return N.load()


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(quartz_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for required in ("quartz_quantize", "quartz_encode_weights", "quartz_linear",
                     "quartz_dequantize", "quartz_linear_workspace_size", "quartz_device_status"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    for name in _declared():
        assert hasattr(lib, name), name
    assert set(_declared()) == set(N.SIGNATURES)


def test_status_strings_and_version(lib):
    assert lib.quartz_status_string(0) == b"QUARTZ_OK"
    assert lib.quartz_status_string(5) == b"QUARTZ_ERR_TIMEOUT"
    assert lib.quartz_status_string(99) == b"QUARTZ_ERR_UNKNOWN"
    assert lib.quartz_version() >> 16 == 1


def _enc(rows, K, gs=16, mode=0, ptr=0x1000):
    return N.QuartzEncoded(ptr, ptr, ptr, ptr, ptr, rows, K, N.QuartzParams(64, gs, mode))


def test_encoded_sizes(lib):
    out = (C.c_size_t * 5)()
    p = N.QuartzParams(64, 16, 0)
    assert lib.quartz_encoded_sizes(10, 128, C.byref(p), out) == 0
    assert list(out) == [10 * 64, 10 * 8, 10 * 2 * 2, 10 * 2, 10 * 2 * 4]
    p = N.QuartzParams(64, 12, 0)
    assert lib.quartz_encoded_sizes(10, 128, C.byref(p), out) == N.QUARTZ_ERR_INVALID_ARG
    p = N.QuartzParams(64, 16, 0, 4)             # FLAGs two per byte
    assert lib.quartz_encoded_sizes(10, 128, C.byref(p), out) == 0
    assert out[1] == 10 * 8 // 2
    p = N.QuartzParams(64, 64, 0, 4)             # an odd number of subgroups in all
    assert lib.quartz_encoded_sizes(3, 64, C.byref(p), out) == 0
    assert out[1] == 2
    p = N.QuartzParams(64, 16, 0, 5)
    assert lib.quartz_encoded_sizes(10, 128, C.byref(p), out) == N.QUARTZ_ERR_INVALID_ARG


def test_host_validation_rejects_before_launch(lib):
    """Every case here fails in host-side validation; no CUDA call is made."""
    q = lib.quartz_quantize
    e = _enc(4, 100)                                   # K not a multiple of 64
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG
    e = _enc(4, 128, gs=12)                            # G_s not in {8,16,32,64}
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG
    e = N.QuartzEncoded(0x1000, 0x1000, 0x1000, 0, 0, 4, 256, N.QuartzParams(128, 16, 0))
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_UNSUPPORTED   # group_q neither 64 nor K
    e = N.QuartzEncoded(0x1000, 0x1000, 0x1000, 0, 0, 4, 192, N.QuartzParams(96, 16, 0))
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_UNSUPPORTED   # group_q not a multiple of 64
    e = N.QuartzEncoded(0x1000, 0x1000, 0x1000, 0x1000, 0x1000, 4, 256, N.QuartzParams(256, 16, 1))
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_UNSUPPORTED   # per-row scales are symmetric only
    e = _enc(4, 128, mode=7)
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG
    e = _enc(4, 128)
    assert q(0x1001, C.byref(e), None) == N.QUARTZ_ERR_ALIGNMENT
    assert q(None, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG
    e = _enc(4, 128, ptr=0x1008)
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_ALIGNMENT
    e = N.QuartzEncoded(0x1000, 0x1000, 0x1000, 0, 0, 4, 128, N.QuartzParams(64, 16, 1))
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG  # asym needs zeros+gsum
    e = _enc(-1, 128)
    assert q(0x1000, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG
    assert lib.quartz_dequantize(C.byref(_enc(4, 128)), None, None) == N.QUARTZ_ERR_INVALID_ARG


def test_quantize_static_validation(lib):
    qs = lib.quartz_quantize_static
    e = _enc(4, 128)
    assert qs(0x1000, 0x7C00, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG   # +inf scale
    assert qs(0x1000, 0xBC00, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG   # -1.0
    assert qs(0x1000, 0x7E00, C.byref(e), None) == N.QUARTZ_ERR_INVALID_ARG   # NaN
    assert qs(0x1001, 0x3C00, C.byref(e), None) == N.QUARTZ_ERR_ALIGNMENT
    assert qs(0x1000, 0x3C00, C.byref(_enc(4, 128, mode=1)), None) == N.QUARTZ_ERR_UNSUPPORTED
    assert qs(None, 0x3C00, C.byref(_enc(0, 128)), None) == N.QUARTZ_OK         # empty


def test_linear_validation(lib):
    L = lib.quartz_linear_ex
    a, w = _enc(16, 128), _enc(24, 128)
    ok = dict(bias=None, y=0x2000, t=0, part=None, pg=0, algo=0, ws=0x3000, wsb=1 << 30)

    def call(a, w, **kw):
        d = dict(ok, **kw)
        o = N.QuartzLinearOpts(d["part"], d["pg"], d["algo"], None, None)
        return L(C.byref(a), C.byref(w), d["bias"], d["y"], d["t"], d["ws"], d["wsb"], C.byref(o),
                 None)

    assert call(a, _enc(24, 192)) == N.QUARTZ_ERR_INVALID_ARG           # K mismatch
    assert call(a, _enc(24, 128, gs=32)) == N.QUARTZ_ERR_INVALID_ARG    # G_s mismatch
    assert call(a, _enc(20, 128)) == N.QUARTZ_ERR_INVALID_ARG           # N % 8 != 0
    assert call(a, w, t=3) == N.QUARTZ_ERR_INVALID_ARG                  # output type
    assert call(a, w, algo=9) == N.QUARTZ_ERR_INVALID_ARG
    assert call(a, w, part=0x4000, pg=2) == N.QUARTZ_ERR_INVALID_ARG    # group out of range
    assert call(a, w, y=0x2004) == N.QUARTZ_ERR_ALIGNMENT
    assert call(a, w, bias=0x2002) == N.QUARTZ_ERR_ALIGNMENT
    assert call(a, w, wsb=16) == N.QUARTZ_ERR_WORKSPACE
    assert call(a, w, ws=None) == N.QUARTZ_ERR_WORKSPACE
    assert call(a, w, y=None) == N.QUARTZ_ERR_INVALID_ARG
    p = N.QuartzParams(64, 16, 0)
    # at least both operands expanded to one byte per element
    assert lib.quartz_linear_workspace_size(16, 24, 128, C.byref(p)) > 16 * 128 + 24 * 128
    assert lib.quartz_linear_workspace_size(16, 20, 128, C.byref(p)) == 0
    assert lib.quartz_selftest_timeout(10, None) == N.QUARTZ_ERR_INVALID_ARG


def test_linear_launch_count(lib):
    """Preparation + GEMM, plus the combine kernel only where a device splits
    the last wave (never for one tile, with partials, asymmetric or on the
    SIMT / shift GEMMs); 0 for invalid sizes or M = 0."""
    cnt = lib.quartz_linear_launch_count
    p = N.QuartzParams(64, 16, 0)
    pa = N.QuartzParams(64, 16, 1)
    for algo in (N.ALGO_TCGEN05, N.ALGO_SIMT, N.ALGO_SHIFT):
        assert cnt(16, 24, 128, C.byref(p), algo, 0) == 2        # one tile: no split
        assert cnt(18432, 9216, 3072, C.byref(pa), algo, 0) == 2  # asymmetric: no split
        assert cnt(18432, 9216, 3072, C.byref(p), algo, 1) == 2   # with partials: no split
    assert cnt(18432, 9216, 3072, C.byref(p), N.ALGO_TCGEN05, 0) in (2, 3)
    assert cnt(0, 24, 128, C.byref(p), 0, 0) == 0
    assert cnt(16, 20, 128, C.byref(p), 0, 0) == 0     # N % 8 != 0
    assert cnt(16, 24, 100, C.byref(p), 0, 0) == 0     # K not a multiple of group_q
    assert cnt(16, 24, 128, C.byref(p), 9, 0) == 0     # algorithm


def test_code_bits_validation(lib):
    """16-bit stage-1 codes (Section 5 LLM variant): symmetric groups of 64;
    no SIMT GEMM and no int32 partials for them."""
    out = (C.c_size_t * 5)()
    for bits, rc in ((0, 0), (8, 0), (16, 0), (12, N.QUARTZ_ERR_INVALID_ARG), (4, N.QUARTZ_ERR_INVALID_ARG)):
        p = N.QuartzParams(64, 8, 0, 8, bits)
        assert lib.quartz_encoded_sizes(10, 128, C.byref(p), out) == rc
    p = N.QuartzParams(64, 8, 0, 4, 16)          # FLAGs 0..12 still fit in 4 bits
    assert lib.quartz_encoded_sizes(10, 128, C.byref(p), out) == 0 and out[1] == 10 * 16 // 2
    q = lib.quartz_quantize

    def enc(rows, K, gq=64, mode=0, bits=16):
        return N.QuartzEncoded(0x1000, 0x1000, 0x1000, 0x1000, 0x1000, rows, K, N.QuartzParams(gq, 8, mode, 8, bits))

    assert q(0x1000, C.byref(enc(4, 128, mode=1)), None) == N.QUARTZ_ERR_UNSUPPORTED   # asymmetric
    assert q(0x1000, C.byref(enc(4, 128, gq=128)), None) == N.QUARTZ_ERR_UNSUPPORTED   # per-row scales
    assert lib.quartz_quantize_static(0x1000, 0x3C00, C.byref(enc(4, 128)), None) == N.QUARTZ_ERR_UNSUPPORTED
    L = lib.quartz_linear_ex

    def lin(a, w, algo, part=None):
        o = N.QuartzLinearOpts(part, 0, algo, None, None)
        return L(C.byref(a), C.byref(w), None, 0x2000, 0, 0x3000, 1 << 30, C.byref(o), None)

    a, w = enc(16, 128), enc(24, 128)
    assert lin(a, w, N.ALGO_SIMT) == N.QUARTZ_ERR_UNSUPPORTED
    assert lin(a, w, N.ALGO_SHIFT, part=0x4000) == N.QUARTZ_ERR_UNSUPPORTED
    assert lin(a, w, N.ALGO_TCGEN05, part=0x4000) == N.QUARTZ_ERR_UNSUPPORTED
    assert lin(a, enc(24, 128, bits=8), N.ALGO_SHIFT) == N.QUARTZ_ERR_INVALID_ARG  # mixed widths
    # the fused path takes 16-bit codes; an a_out of the other code width is rejected
    assert lib.quartz_linear_f16(0x1000, 16, C.byref(w), None, 0x2000, 0, C.byref(enc(16, 128, bits=8)),
                                 0x3000, 1 << 30, None) == N.QUARTZ_ERR_INVALID_ARG
    assert lib.quartz_linear_f16(0x1000, 16, C.byref(enc(24, 128, mode=1)), None, 0x2000, 0, None,
                                 0x3000, 1 << 30, None) == N.QUARTZ_ERR_UNSUPPORTED


def test_attention_validation(lib):
    """Host checks of the attention decode step and the cache append."""
    def enc(rows, K=128, gs=16, mode=0, gq=64, bits=8):
        return N.QuartzEncoded(0x1000, 0x1000, 0x1000, 0x1000, 0x1000, rows, K, N.QuartzParams(gq, gs, mode, 8, bits))

    assert lib.quartz_attention_workspace_size(4, 1000) > 0
    assert lib.quartz_attention_workspace_size(0, 1000) == 0
    assert lib.quartz_attention_workspace_size(4, 0) == 0
    A = lib.quartz_attention_decode

    def att(q, k, v, L_max=50, L=40, o=0x2000, t=0, ws=0x3000, wsb=1 << 20, scale=0.1):
        return A(C.byref(q), C.byref(k), C.byref(v), L_max, L, scale, o, t, ws, wsb, None)

    q, k, v = enc(4), enc(200), enc(200)
    assert att(enc(4, K=256), enc(200, K=256), enc(200, K=256)) == N.QUARTZ_ERR_INVALID_ARG  # d != 128
    assert att(q, enc(200, gs=32), v) == N.QUARTZ_ERR_INVALID_ARG          # G_s mismatch
    assert att(q, enc(199), v) == N.QUARTZ_ERR_INVALID_ARG                 # rows != BH * L_max
    assert att(q, k, v, L=51) == N.QUARTZ_ERR_INVALID_ARG                  # L > L_max
    assert att(q, k, v, L=0) == N.QUARTZ_ERR_INVALID_ARG
    assert att(q, k, v, t=3) == N.QUARTZ_ERR_INVALID_ARG
    assert att(q, k, v, scale=float("nan")) == N.QUARTZ_ERR_INVALID_ARG
    assert att(q, k, v, o=0x2004) == N.QUARTZ_ERR_ALIGNMENT
    assert att(q, k, v, wsb=16) == N.QUARTZ_ERR_WORKSPACE
    assert att(enc(4, mode=1), enc(200, mode=1), enc(200, mode=1)) == N.QUARTZ_ERR_UNSUPPORTED
    assert att(enc(4, bits=16), enc(200, bits=16), enc(200, bits=16)) == N.QUARTZ_ERR_UNSUPPORTED
    K = lib.quartz_kv_append
    assert K(0x1000, 4, 3, C.byref(enc(200)), 50, 48, None) == N.QUARTZ_ERR_INVALID_ARG   # t0 + T > L_max
    assert K(0x1000, 4, 3, C.byref(enc(199)), 50, 0, None) == N.QUARTZ_ERR_INVALID_ARG    # rows
    assert K(0x1000, 4, 3, C.byref(enc(200, K=64)), 50, 0, None) == N.QUARTZ_ERR_UNSUPPORTED
    assert K(0x1008, 4, 3, C.byref(enc(200)), 50, 0, None) == N.QUARTZ_ERR_ALIGNMENT
    assert K(None, 4, 0, C.byref(enc(200)), 50, 0, None) == N.QUARTZ_OK                   # T == 0


def test_prepared_weights_validation(lib):
    p = N.QuartzParams(64, 16, 0)
    assert lib.quartz_prepared_weights_size(24, 128, C.byref(p)) >= 24 * 128
    assert lib.quartz_prepared_weights_size(20, 128, C.byref(p)) == 0          # N % 8
    assert lib.quartz_prepared_weights_size(24, 100, C.byref(p)) == 0          # K % 64
    P = lib.quartz_prepare_weights
    w = _enc(24, 128)
    need = lib.quartz_prepared_weights_size(24, 128, C.byref(p))
    assert P(C.byref(w), 0x4000, need - 1, None) == N.QUARTZ_ERR_WORKSPACE
    assert P(C.byref(w), None, need, None) == N.QUARTZ_ERR_WORKSPACE
    assert P(C.byref(w), 0x4008, need, None) == N.QUARTZ_ERR_ALIGNMENT
    assert P(C.byref(_enc(20, 128)), 0x4000, need, None) == N.QUARTZ_ERR_INVALID_ARG
    o = N.QuartzLinearOpts(None, 0, 0, None, None, 0x5008)                   # misaligned prepared weights
    assert lib.quartz_linear_ex(C.byref(_enc(16, 128)), C.byref(w), None, 0x2000, 0, 0x3000, 1 << 30,
                                C.byref(o), None) == N.QUARTZ_ERR_ALIGNMENT


def test_linear_f16_validation(lib):
    """Host checks of the fused activation path: nothing is launched on error."""
    L = lib.quartz_linear_f16
    w = _enc(24, 128)
    ok = dict(x=0x1000, M=16, bias=None, y=0x2000, t=0, aout=None, ws=0x3000, wsb=1 << 30)

    def call(w, **kw):
        d = dict(ok, **kw)
        return L(d["x"], d["M"], C.byref(w), d["bias"], d["y"], d["t"], d["aout"], d["ws"], d["wsb"], None)

    assert call(_enc(24, 128, mode=1)) == N.QUARTZ_ERR_UNSUPPORTED      # asymmetric not fused
    assert call(_enc(20, 128)) == N.QUARTZ_ERR_INVALID_ARG             # N % 8 != 0
    assert call(w, M=-1) == N.QUARTZ_ERR_INVALID_ARG
    assert call(w, t=3) == N.QUARTZ_ERR_INVALID_ARG
    assert call(w, x=0x1008) == N.QUARTZ_ERR_ALIGNMENT
    assert call(w, x=None) == N.QUARTZ_ERR_INVALID_ARG
    assert call(w, wsb=16) == N.QUARTZ_ERR_WORKSPACE
    assert call(w, aout=C.byref(_enc(8, 128))) == N.QUARTZ_ERR_INVALID_ARG       # rows != M
    assert call(w, aout=C.byref(_enc(16, 128, gs=32))) == N.QUARTZ_ERR_INVALID_ARG
    assert call(w, M=0, x=None, y=None) == N.QUARTZ_OK                   # empty: no-op


def test_missing_library_fails_loudly(tmp_path):
    saved = N._lib
    try:
        N._lib = None
        with pytest.raises(RuntimeError, match="no CPU or fallback"):
            N.load(str(tmp_path / "libquartz.so"))
    finally:
        N._lib = saved


def test_probe_validation(lib):
    """The pipe-rate probes reject bad sizes on the host (nothing launched)."""
    assert lib.quartz_probe_fp32_pipe(0, 10, 0x1000, None) == N.QUARTZ_ERR_INVALID_ARG
    assert lib.quartz_probe_fp32_pipe(4, 0, 0x1000, None) == N.QUARTZ_ERR_INVALID_ARG
    assert lib.quartz_probe_fp32_pipe(4, 10, None, None) == N.QUARTZ_ERR_INVALID_ARG
    assert lib.quartz_probe_mma_f8(0, 10, None) == N.QUARTZ_ERR_INVALID_ARG
    assert lib.quartz_probe_mma_f8(4, 0, None) == N.QUARTZ_ERR_INVALID_ARG
    assert lib.quartz_probe_mma_f8(1 << 17, 10, None) == N.QUARTZ_ERR_INVALID_ARG
