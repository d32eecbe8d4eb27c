"""GPU parity of the attention decode step (Appendix D, Table 6) and the
cache append against the CPU oracle.

* Cache append: codes, FLAGs and scale bits bit-exact against the oracle's
  encoder of the same rows; rows outside the appended range untouched.
* Attention: o against the oracle's binary64 result.  Tolerance from the
  kernel's arithmetic: the integer group sums are exact; each score takes
  at most 6 binary32 roundings relative to S = max_t sum_k |q_k k_k| scale,
  so in the log2 domain (|score - max| <= 2 S log2 e) its error is below
  8 x 3 S log2(e) 2^-24, plus 2 ulp of exp2f: every weight p_t is off by a
  relative eps_p = ln 2 x that + 2^-22.  The value sum and the softmax
  denominator add at most (L/8 + 2 L/128 + 80) binary32 roundings each
  (per-thread sums of L/8 terms, one rescale per 128-token tile, the 8-slot
  and split reductions).  So |o - o_ref| <= (2 eps_p + 2 (L/8 + 2L/128 + 80)
  2^-24) sum_t p_t |v_t| + the output rounding (2^-11 |o| for fp16).
"""
import numpy as np
import pytest

import oracle as O
from paper_2509_26436_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

REL = {"float16": 2.0 ** -11, "bfloat16": 2.0 ** -8, "float32": 0.0}


@pytest.fixture(scope="module")
def Q():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2509_26436_gb300 as Q
    return Q


def _gpu_enc(Q, x, gs, flag_bits=8):
    return Q.quantize(torch.from_numpy(x).cuda(), group_s=gs, flag_bits=flag_bits)


def _check(o_gpu, q, k, v, L_max, L, scale, dtype_name):
    ref, oabs = O.attention_decode(q, k, v, L_max, L, scale, with_abs=True)
    qh, kh = np.abs(O.dequantize(q)), np.abs(O.dequantize(k))
    BH = q.rows
    S = np.array([(kh[b * L_max:b * L_max + L] @ qh[b]).max() * abs(scale) for b in range(BH)])
    eps = 2.0 ** -24
    eps_p = np.log(2) * 8 * 3 * S * np.log2(np.e) * eps + 2.0 ** -22
    tol = (2 * eps_p[:, None] + 2 * (L / 8 + 2 * L / 128 + 80) * eps) * oabs + REL[dtype_name] * np.abs(ref) + 1e-30
    err = np.abs(o_gpu.astype(np.float64) - ref)
    bad = err > tol
    assert not bad.any(), (f"{bad.sum()} of {bad.size} outside tolerance; worst "
                           f"{(err / tol).max():.3g}x")
    return (err / tol).max()


def _case(Q, BH, L_max, L, gs, seed, out="float32", flag_bits=8, scale=128 ** -0.5):
    xq, xk, xv = inputs.attention_inputs(BH, L_max, seed)
    q, k, v = (_gpu_enc(Q, x, gs, flag_bits) for x in (xq, xk, xv))
    o = Q.attention_decode(q, k, v, L_max, L, scale, out_dtype=getattr(torch, out))
    assert Q.device_status() == 0
    eq, ek, ev = O.encode(xq, 64, gs), O.encode(xk, 64, gs), O.encode(xv, 64, gs)
    return _check(o.float().cpu().numpy(), eq, ek, ev, L_max, L, scale, out)


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("BH,L_max,L", [(1, 1, 1), (3, 130, 1), (5, 200, 127), (4, 300, 128), (7, 300, 129),
                                        (2, 1500, 1499), (6, 4096, 4096)])
def test_attention_decode_ragged(Q, gs, BH, L_max, L):
    _case(Q, BH, L_max, L, gs, seed=7000 + BH + L)


@pytest.mark.parametrize("out", ["float16", "bfloat16", "float32"])
@pytest.mark.parametrize("flag_bits", [8, 4])
def test_attention_decode_dtypes_and_packed_flags(Q, out, flag_bits):
    _case(Q, 9, 700, 650, 16, seed=7100, out=out, flag_bits=flag_bits)


def test_attention_single_token_is_exact(Q):
    """L = 1: the weight is exactly 1 and o is the dequantised value row."""
    xq, xk, xv = inputs.attention_inputs(12, 3, 7200)
    q, k, v = (_gpu_enc(Q, x, 8) for x in (xq, xk, xv))
    o = Q.attention_decode(q, k, v, 3, 1, 0.3, out_dtype=torch.float32)
    ref = O.attention_decode(O.encode(xq, 64, 8), O.encode(xk, 64, 8), O.encode(xv, 64, 8), 3, 1, 0.3)
    assert np.array_equal(o.cpu().numpy().astype(np.float64), ref)


def test_attention_large_scores(Q):
    """Scores of hundreds of nats (large scale): softmax concentrates on a
    few keys; the running maximum keeps every exponent finite."""
    _case(Q, 4, 1000, 1000, 16, seed=7300, scale=4.0)


@pytest.mark.parametrize("heads", inputs.ATTN_HEADS)
def test_attention_table6_sizes_sampled(Q, heads):
    """The benchmark's workload (batch 16, heads x 128, 4096 cached tokens,
    G_s 8 / 16 / 32) in its launch configuration; a sample of heads compared
    with the oracle."""
    BH, L = inputs.ATTN_BATCH * heads, inputs.ATTN_CONTEXT
    xq, xk, xv = inputs.attention_inputs(BH, L, seed=7400 + heads)
    heads_s = np.array([0, 1, BH // 2, BH - 1])
    rows = (heads_s[:, None] * L + np.arange(L)[None, :]).ravel()
    for gs in (8, 16, 32):
        q, k, v = (_gpu_enc(Q, x, gs) for x in (xq, xk, xv))
        o = Q.attention_decode(q, k, v, L, L, 128 ** -0.5)
        assert Q.device_status() == 0
        eq, ek, ev = O.encode(xq[heads_s], 64, gs), O.encode(xk[rows], 64, gs), O.encode(xv[rows], 64, gs)
        _check(o[torch.from_numpy(heads_s).cuda()].float().cpu().numpy(), eq, ek, ev, L, L, 128 ** -0.5,
               "float16")
        del q, k, v


@pytest.mark.parametrize("gs", [8, 16, 32, 64])
@pytest.mark.parametrize("flag_bits", [8, 4])
def test_kv_append_bit_exact(Q, gs, flag_bits):
    """Append T tokens per head at t0 into a cache whose other rows hold an
    earlier encoding; compare every cache row with the oracle."""
    BH, L_max, t0, T = 6, 40, 13, 9
    _, xk, _ = inputs.attention_inputs(BH, L_max, 7500 + gs)
    xnew = inputs.attention_inputs(BH, T, 7600 + gs)[1].reshape(BH, T, 128)
    cache = _gpu_enc(Q, xk, gs, flag_bits)
    Q.kv_append(torch.from_numpy(xnew).cuda(), cache, L_max, t0)
    torch.cuda.synchronize()
    assert Q.device_status() == 0
    xk2 = xk.reshape(BH, L_max, 128).copy()
    xk2[:, t0:t0 + T] = xnew
    ref = O.encode(xk2.reshape(BH * L_max, 128), 64, gs)
    assert np.array_equal(cache.codes.cpu().numpy(), ref.codes)
    assert np.array_equal(cache.scales.cpu().numpy().view(np.uint16), ref.scales.view(np.uint16))
    flags = ref.flags.reshape(-1)
    if flag_bits == 4:
        flags = flags[0::2] | (flags[1::2] << 4)
    assert np.array_equal(cache.flags.cpu().numpy().reshape(-1), flags)


def test_decode_loop_append_then_attend(Q):
    """A short decode loop: append one token per head, attend over the
    grown cache; each step against the oracle."""
    BH, L_max, gs = 8, 64, 16
    xq, xk, xv = inputs.attention_inputs(BH, L_max, 7700)
    k = Q.empty_encoded(BH * L_max, 128, Q.Params(64, gs), "cuda")
    v = Q.empty_encoded(BH * L_max, 128, Q.Params(64, gs), "cuda")
    xk3, xv3 = xk.reshape(BH, L_max, 128), xv.reshape(BH, L_max, 128)
    Q.kv_append(torch.from_numpy(np.ascontiguousarray(xk3[:, :50])).cuda(), k, L_max, 0)
    Q.kv_append(torch.from_numpy(np.ascontiguousarray(xv3[:, :50])).cuda(), v, L_max, 0)
    q = _gpu_enc(Q, xq, gs)
    eq = O.encode(xq, 64, gs)
    for L in range(51, 55):
        Q.kv_append(torch.from_numpy(np.ascontiguousarray(xk3[:, L - 1:L])).cuda(), k, L_max, L - 1)
        Q.kv_append(torch.from_numpy(np.ascontiguousarray(xv3[:, L - 1:L])).cuda(), v, L_max, L - 1)
        o = Q.attention_decode(q, k, v, L_max, L, 128 ** -0.5, out_dtype=torch.float32)
        assert Q.device_status() == 0
        kk = np.zeros_like(xk3)
        vv = np.zeros_like(xv3)
        kk[:, :L], vv[:, :L] = xk3[:, :L], xv3[:, :L]
        ek = O.encode(kk.reshape(-1, 128), 64, gs)
        ev = O.encode(vv.reshape(-1, 128), 64, gs)
        _check(o.cpu().numpy(), eq, ek, ev, L_max, L, 128 ** -0.5, "float32")
