"""QuaRTZ CPU oracle (test infrastructure only).

NumPy front end to the plain-C oracle in ``quartz_oracle.c``.  Only the test
suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline and
reference legs may import this package; the product path never does.  It
imports nothing from the CUDA package.

Every function follows a passage of arXiv 2509.26436:
  quantize        Section 3, Eq. 1 (per-group 8-bit min-max)
  lzs_encode      Section 3, Eq. 2 (FLAG = max(29 - clz(m), 0), shift)
  lzs_decode      Section 3 (the equal shift of a group is undone by FLAG)
  encode          Eq. 1 then Eq. 2 then nibble packing (Section 4.4 format)
  quantize16      Section 5 LLM variant: Eq. 1 with 16-bit codes
  lzs_encode16    Eq. 2 on 16-bit codes (FLAG 0..12)
  group_partials  Section 4.4 (integer MMA per 64-wide group)
  linear          Section 4.4 + Appendix C (16-bit group scales)
  attention_decode  Appendix D, Table 6: attention of one query per head over
                  an encoded key / value cache (reading in quartz_oracle.c)
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "quartz_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

SYMMETRIC = 0
ASYMMETRIC = 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2 -ffp-contract=off); returns the path."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11", "-fPIC",
               "-shared", "-o", tmp, _SRC, "-lm"]
        subprocess.check_call(cmd)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = C.CDLL(build())
            P = C.c_void_p
            i64, i32 = C.c_int64, C.c_int
            lib.oracle_half_to_float.argtypes = [C.c_uint16]
            lib.oracle_half_to_float.restype = C.c_float
            lib.oracle_float_to_half_rn.argtypes = [C.c_float]
            lib.oracle_float_to_half_rn.restype = C.c_uint16
            lib.oracle_clz32.argtypes = [C.c_uint32]
            lib.oracle_clz32.restype = i32
            lib.oracle_lzs_flag.argtypes = [P, i32]
            lib.oracle_quantize.argtypes = [P, i64, i64, i32, i32, P, P, P]
            lib.oracle_lzs_encode.argtypes = [P, i64, i32, P, P]
            lib.oracle_lzs_decode.argtypes = [P, P, i64, i32, P]
            lib.oracle_pack_nibbles.argtypes = [P, i64, P]
            lib.oracle_pack_nibbles.restype = None
            lib.oracle_unpack_nibbles.argtypes = [P, i64, P]
            lib.oracle_unpack_nibbles.restype = None
            lib.oracle_encode.argtypes = [P, i64, i64, i32, i32, i32, P, P, P, P, P]
            lib.oracle_quantize_static.argtypes = [P, i64, C.c_uint16, P]
            lib.oracle_quantize16.argtypes = [P, i64, i64, i32, P, P]
            lib.oracle_lzs_encode16.argtypes = [P, i64, i32, P, P]
            lib.oracle_encode16.argtypes = [P, i64, i64, i32, i32, P, P, P]
            lib.oracle_encode_static.argtypes = [P, i64, i64, C.c_uint16, i32, i32, P, P, P]
            lib.oracle_attention_decode.argtypes = [P, P, P, P, P, P, P, P, P, i64, i64, i64, i64, i32,
                                                    i32, C.c_double, P, P]
            lib.oracle_decode_codes.argtypes = [P, P, i64, i64, i32, P]
            lib.oracle_dequantize.argtypes = [P, P, P, P, i64, i64, i32, i32, P]
            lib.oracle_group_partials.argtypes = [P, P, i64, i64, i64, i32, P, i64, P]
            lib.oracle_linear.argtypes = [P, P, P, P, P, P, P, P, i64, i64, i64, i32, i32,
                                          P, P, i64, P, P, P]
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _check(rc):
    if rc != 0:
        raise ValueError(f"oracle error {rc}")


def _as_u16(x):
    """fp16 array (or its uint16 bit view) -> contiguous uint16 bits."""
    x = np.ascontiguousarray(x)
    return x.view(np.uint16) if x.dtype == np.float16 else x.astype(np.uint16, copy=False)


# --- IEEE binary16 ---------------------------------------------------------

def half_to_float(bits: int) -> float:
    return _load().oracle_half_to_float(bits)


def float_to_half(x: float) -> int:
    return _load().oracle_float_to_half_rn(x)


def clz32(v: int) -> int:
    return _load().oracle_clz32(v)


# --- stage 1 (Eq. 1) -------------------------------------------------------

def quantize(x16: np.ndarray, group_q: int = 64, mode: int = SYMMETRIC):
    """Eq. 1 per group: returns (q int8 [R,K], scales fp16 [R,K/gq], zeros int8 [R,K/gq])."""
    xb = _as_u16(x16)
    R, K = xb.shape
    q = np.empty((R, K), np.int8)
    s = np.empty((R, K // group_q), np.uint16)
    z = np.empty((R, K // group_q), np.int8)
    _check(_load().oracle_quantize(_ptr(xb), R, K, group_q, mode, _ptr(q), _ptr(s), _ptr(z)))
    return q, s.view(np.float16), z


# --- stage 2 (Eq. 2) -------------------------------------------------------

def lzs_flag(q_sub: np.ndarray) -> int:
    """FLAG of one subgroup; raises for the never-produced code -128."""
    q_sub = np.ascontiguousarray(q_sub, dtype=np.int8)
    rc = _load().oracle_lzs_flag(_ptr(q_sub), q_sub.size)
    if rc < 0:
        raise ValueError("code -128 has no 4-bit LZS form")
    return rc


def lzs_encode(q: np.ndarray, group_s: int):
    """int8 codes (flat) -> (flags uint8 [n/gs], c int8 [n] in [-7,7])."""
    q = np.ascontiguousarray(q, dtype=np.int8).ravel()
    f = np.empty(q.size // group_s, np.uint8)
    c = np.empty(q.size, np.int8)
    rc = _load().oracle_lzs_encode(_ptr(q), q.size, group_s, _ptr(f), _ptr(c))
    if rc == -2:
        raise ValueError("code -128 has no 4-bit LZS form")
    _check(rc)
    return f, c


def lzs_decode(c: np.ndarray, flags: np.ndarray, group_s: int) -> np.ndarray:
    c = np.ascontiguousarray(c, dtype=np.int8).ravel()
    flags = np.ascontiguousarray(flags, dtype=np.uint8).ravel()
    v = np.empty(c.size, np.int16)
    _check(_load().oracle_lzs_decode(_ptr(c), _ptr(flags), c.size, group_s, _ptr(v)))
    return v


def pack_nibbles(c: np.ndarray) -> np.ndarray:
    c = np.ascontiguousarray(c, dtype=np.int8).ravel()
    out = np.empty((c.size + 1) // 2, np.uint8)
    _load().oracle_pack_nibbles(_ptr(c), c.size, _ptr(out))
    return out


def unpack_nibbles(p: np.ndarray, n: int) -> np.ndarray:
    p = np.ascontiguousarray(p, dtype=np.uint8).ravel()
    out = np.empty(n, np.int8)
    _load().oracle_unpack_nibbles(_ptr(p), n, _ptr(out))
    return out


# --- whole encoder ---------------------------------------------------------

class Encoded:
    """Oracle-side encoded tensor (the Section 4.4 storage format)."""

    def __init__(self, codes, flags, scales, zeros, gsum, group_q, group_s, mode):
        self.codes, self.flags, self.scales = codes, flags, scales
        self.zeros, self.gsum = zeros, gsum
        self.group_q, self.group_s, self.mode = group_q, group_s, mode

    @property
    def rows(self):
        return self.codes.shape[0]

    @property
    def K(self):
        return self.codes.shape[1] * 2


def encode(x16: np.ndarray, group_q: int = 64, group_s: int = 16, mode: int = SYMMETRIC) -> Encoded:
    xb = _as_u16(x16)
    R, K = xb.shape
    G = K // group_q
    codes = np.empty((R, K // 2), np.uint8)
    flags = np.empty((R, K // group_s), np.uint8)
    scales = np.empty((R, G), np.uint16)
    zeros = np.empty((R, G), np.int8)
    gsum = np.empty((R, G), np.int32)
    _check(_load().oracle_encode(_ptr(xb), R, K, group_q, group_s, mode, _ptr(codes),
                                 _ptr(flags), _ptr(scales), _ptr(zeros), _ptr(gsum)))
    return Encoded(codes, flags, scales.view(np.float16), zeros, gsum, group_q, group_s, mode)


def quantize_static(x16: np.ndarray, s16) -> np.ndarray:
    """Static per-tensor Eq. 1 with a given fp16 scale: q int8, same shape."""
    xb = _as_u16(x16)
    q = np.empty(xb.shape, np.int8)
    _check(_load().oracle_quantize_static(_ptr(xb), xb.size, int(np.float16(s16).view(np.uint16)), _ptr(q)))
    return q


def encode_static(x16: np.ndarray, s16, group_q: int = 64, group_s: int = 16) -> Encoded:
    """Encoder with a static (calibrated) scale for every group (symmetric)."""
    xb = _as_u16(x16)
    R, K = xb.shape
    G = K // group_q
    codes = np.empty((R, K // 2), np.uint8)
    flags = np.empty((R, K // group_s), np.uint8)
    scales = np.empty((R, G), np.uint16)
    _check(_load().oracle_encode_static(_ptr(xb), R, K, int(np.float16(s16).view(np.uint16)), group_q,
                                        group_s, _ptr(codes), _ptr(flags), _ptr(scales)))
    return Encoded(codes, flags, scales.view(np.float16), np.zeros((R, G), np.int8),
                   np.zeros((R, G), np.int32), group_q, group_s, SYMMETRIC)


def quantize16(x16: np.ndarray, group_q: int = 64):
    """LLM variant stage 1: 16-bit codes q int16 [R, K] and fp16 scales [R, K/gq]."""
    xb = _as_u16(x16)
    R, K = xb.shape
    q = np.empty((R, K), np.int16)
    s = np.empty((R, K // group_q), np.uint16)
    _check(_load().oracle_quantize16(_ptr(xb), R, K, group_q, _ptr(q), _ptr(s)))
    return q, s.view(np.float16)


def lzs_encode16(q: np.ndarray, group_s: int):
    """Eq. 2 on 16-bit codes: (flags uint8 0..12, c int8 in [-7, 7])."""
    q = np.ascontiguousarray(q, dtype=np.int16).ravel()
    flags = np.empty(q.size // group_s, np.uint8)
    c = np.empty(q.size, np.int8)
    rc = _load().oracle_lzs_encode16(_ptr(q), q.size, group_s, _ptr(flags), _ptr(c))
    if rc == -2:
        raise ValueError("code -32768 has no 4-bit LZS form")
    _check(rc)
    return flags, c


def encode16(x16: np.ndarray, group_q: int = 64, group_s: int = 8) -> Encoded:
    """LLM-variant encoder (16-bit codes, FLAGs 0..12), symmetric."""
    xb = _as_u16(x16)
    R, K = xb.shape
    G = K // group_q
    codes = np.empty((R, K // 2), np.uint8)
    flags = np.empty((R, K // group_s), np.uint8)
    scales = np.empty((R, G), np.uint16)
    _check(_load().oracle_encode16(_ptr(xb), R, K, group_q, group_s, _ptr(codes), _ptr(flags), _ptr(scales)))
    return Encoded(codes, flags, scales.view(np.float16), np.zeros((R, G), np.int8),
                   np.zeros((R, G), np.int32), group_q, group_s, SYMMETRIC)


def decode_values(e: Encoded) -> np.ndarray:
    """Decoded LZS integers v [R, K] (int16)."""
    v = np.empty((e.rows, e.K), np.int16)
    _check(_load().oracle_decode_codes(_ptr(e.codes), _ptr(e.flags), e.rows, e.K, e.group_s,
                                       _ptr(v)))
    return v


def dequantize(e: Encoded) -> np.ndarray:
    """x_hat = s * (v - z), binary64 [R, K]."""
    out = np.empty((e.rows, e.K), np.float64)
    z = e.zeros if e.mode == ASYMMETRIC else None
    _check(_load().oracle_dequantize(_ptr(e.codes), _ptr(e.flags), _ptr(_as_u16(e.scales)),
                                     _ptr(z), e.rows, e.K, e.group_q, e.group_s, _ptr(out)))
    return out


# --- GEMM (Section 4.4) ----------------------------------------------------

def group_partials(va: np.ndarray, vw: np.ndarray, group_q: int = 64, rows=None) -> np.ndarray:
    """P [G, n_rows, N] int64 of the decoded integer operands."""
    va = np.ascontiguousarray(va, dtype=np.int16)
    vw = np.ascontiguousarray(vw, dtype=np.int16)
    M, K = va.shape
    N = vw.shape[0]
    sel = None if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    nr = M if sel is None else sel.size
    P = np.empty((K // group_q, nr, N), np.int64)
    _check(_load().oracle_group_partials(_ptr(va), _ptr(vw), M, N, K, group_q, _ptr(sel),
                                         0 if sel is None else sel.size, _ptr(P)))
    return P


def linear(a: Encoded, w: Encoded, bias16=None, rows=None, with_abs: bool = False):
    """y [n_rows, N] binary64 of the W4A4 linear (selected rows of A); with
    `with_abs` also sum_g |s_a s_w D_g| + |bias| of each output."""
    if a.K != w.K or a.group_q != w.group_q or a.group_s != w.group_s or a.mode != w.mode:
        raise ValueError("operands must share K, group sizes and mode")
    sel = None if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    nr = a.rows if sel is None else sel.size
    y = np.empty((nr, w.rows), np.float64)
    yabs = np.empty((nr, w.rows), np.float64) if with_abs else None
    scratch = np.empty((w.rows, w.K), np.int16)
    az = a.zeros if a.mode == ASYMMETRIC else None
    wz = w.zeros if w.mode == ASYMMETRIC else None
    b = None if bias16 is None else _as_u16(bias16)
    _check(_load().oracle_linear(_ptr(a.codes), _ptr(a.flags), _ptr(_as_u16(a.scales)), _ptr(az),
                                 _ptr(w.codes), _ptr(w.flags), _ptr(_as_u16(w.scales)), _ptr(wz),
                                 a.rows, w.rows, a.K, a.group_q, a.group_s, _ptr(b), _ptr(sel),
                                 0 if sel is None else sel.size, _ptr(scratch), _ptr(y),
                                 _ptr(yabs)))
    return (y, yabs) if with_abs else y


# --- attention (Appendix D, Table 6) ---------------------------------------

def attention_decode(q: Encoded, k: Encoded, v: Encoded, L_max: int, L: int, scale: float,
                     with_abs: bool = False):
    """o [BH, d] binary64: one query per (batch x head) row of `q` against the
    first L tokens of that head's rows (bh * L_max + t) of the caches."""
    if not (q.K == k.K == v.K and q.group_q == k.group_q == v.group_q and
            q.group_s == k.group_s == v.group_s and q.mode == k.mode == v.mode == SYMMETRIC):
        raise ValueError("q, k, v must share d, group sizes and the symmetric mode")
    BH, d = q.rows, q.K
    if k.rows != BH * L_max or v.rows != BH * L_max:
        raise ValueError("caches must hold BH * L_max rows")
    o = np.empty((BH, d), np.float64)
    oabs = np.empty((BH, d), np.float64) if with_abs else None
    _check(_load().oracle_attention_decode(
        _ptr(q.codes), _ptr(q.flags), _ptr(_as_u16(q.scales)), _ptr(k.codes), _ptr(k.flags),
        _ptr(_as_u16(k.scales)), _ptr(v.codes), _ptr(v.flags), _ptr(_as_u16(v.scales)), BH, L_max, L, d,
        q.group_q, q.group_s, float(scale), _ptr(o), _ptr(oabs)))
    return (o, oabs) if with_abs else o
