"""ctypes declarations of the C ABI in include/quartz.h (libquartz.so).

Loading fails loudly when the library has not been built: there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libquartz.so")

QUARTZ_OK = 0
QUARTZ_ERR_INVALID_ARG = 1
QUARTZ_ERR_ALIGNMENT = 2
QUARTZ_ERR_UNSUPPORTED = 3
QUARTZ_ERR_CUDA = 4
QUARTZ_ERR_TIMEOUT = 5
QUARTZ_ERR_WORKSPACE = 6

SYMMETRIC = 0
ASYMMETRIC = 1

OUT_F16 = 0
OUT_BF16 = 1
OUT_F32 = 2

ALGO_TCGEN05 = 0
ALGO_SIMT = 1
ALGO_SHIFT = 2

# every symbol the header declares, with (restype, argtypes)
_P = C.c_void_p
_I32 = C.c_int32
_I64 = C.c_int64
_SZ = C.c_size_t


class QuartzParams(C.Structure):
    _fields_ = [("group_q", C.c_int32), ("group_s", C.c_int32), ("mode", C.c_int32),
                ("flag_bits", C.c_int32), ("code_bits", C.c_int32)]


class QuartzEncoded(C.Structure):
    _fields_ = [("codes", _P), ("flags", _P), ("scales", _P), ("zeros", _P), ("gsum", _P),
                ("rows", C.c_int64), ("K", C.c_int64), ("p", QuartzParams)]


class QuartzLinearOpts(C.Structure):
    _fields_ = [("partials", _P), ("partials_group", C.c_int32), ("algo", C.c_int32),
                ("gemm_event_begin", _P), ("gemm_event_end", _P), ("w_prepared", _P)]


SIGNATURES = {
    "quartz_status_string": (C.c_char_p, [_I32]),
    "quartz_version": (_I32, []),
    "quartz_encoded_sizes": (_I32, [_I64, _I64, C.POINTER(QuartzParams), C.POINTER(_SZ)]),
    "quartz_quantize": (_I32, [_P, C.POINTER(QuartzEncoded), _P]),
    "quartz_quantize_static": (_I32, [_P, C.c_uint16, C.POINTER(QuartzEncoded), _P]),
    "quartz_encode_weights": (_I32, [_P, C.POINTER(QuartzEncoded), _P]),
    "quartz_dequantize": (_I32, [C.POINTER(QuartzEncoded), _P, _P]),
    "quartz_linear_workspace_size": (_SZ, [_I64, _I64, _I64, C.POINTER(QuartzParams)]),
    "quartz_linear_launch_count": (_I32, [_I64, _I64, _I64, C.POINTER(QuartzParams), _I32, _I32]),
    "quartz_linear": (_I32, [C.POINTER(QuartzEncoded), C.POINTER(QuartzEncoded), _P, _P, _I32,
                             _P, _SZ, _P]),
    "quartz_linear_ex": (_I32, [C.POINTER(QuartzEncoded), C.POINTER(QuartzEncoded), _P, _P, _I32,
                                _P, _SZ, C.POINTER(QuartzLinearOpts), _P]),
    "quartz_linear_noalloc": (_I32, [C.POINTER(QuartzEncoded), C.POINTER(QuartzEncoded), _P, _P,
                                     _I32, _P]),
    "quartz_linear_f16": (_I32, [_P, _I64, C.POINTER(QuartzEncoded), _P, _P, _I32,
                                 C.POINTER(QuartzEncoded), _P, _SZ, _P]),
    "quartz_linear_f16_ex": (_I32, [_P, _I64, C.POINTER(QuartzEncoded), _P, _P, _P, _I32,
                                    C.POINTER(QuartzEncoded), _P, _SZ, _P]),
    "quartz_prepared_weights_size": (_SZ, [_I64, _I64, C.POINTER(QuartzParams)]),
    "quartz_prepare_weights": (_I32, [C.POINTER(QuartzEncoded), _P, _SZ, _P]),
    "quartz_attention_workspace_size": (_SZ, [_I64, _I64]),
    "quartz_kv_append": (_I32, [_P, _I64, _I64, C.POINTER(QuartzEncoded), _I64, _I64, _P]),
    "quartz_attention_decode": (_I32, [C.POINTER(QuartzEncoded), C.POINTER(QuartzEncoded),
                                       C.POINTER(QuartzEncoded), _I64, _I64, C.c_float, _P, _I32, _P, _SZ,
                                       _P]),
    "quartz_device_status": (_I32, [_P]),
    "quartz_selftest_timeout": (_I32, [_I64, _P]),
    "quartz_probe_fp32_pipe": (_I32, [_I32, _I64, _P, _P]),
    "quartz_probe_mma_f8": (_I32, [_I32, _I64, _P]),
}

_lock = threading.Lock()
_lib = None


def load(path: str = LIB_PATH):
    """Load libquartz.so and declare every entry point; raises if missing."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(path):
                raise RuntimeError(
                    f"{path} is missing: build it with `python -m paper_2509_26436_gb300.build` "
                    "(there is no CPU or fallback implementation)")
            lib = C.CDLL(path)
            for name, (res, args) in SIGNATURES.items():
                fn = getattr(lib, name)
                fn.restype = res
                fn.argtypes = args
            _lib = lib
    return _lib


class QuartzError(RuntimeError):
    def __init__(self, status: int, what: str):
        name = load().quartz_status_string(status).decode()
        super().__init__(f"{what}: {name} ({status})")
        self.status = status


def check(status: int, what: str) -> None:
    if status != QUARTZ_OK:
        raise QuartzError(status, what)
