"""quartz_linear_noalloc: the linear layer for callers that cannot allocate
device memory (a plugin whose host framework owns all device memory, or a
latency-critical path that must not risk a synchronising cudaMalloc).

It runs through the C ABI with its library-owned scratch array and must match
quartz_linear (caller-provided workspace) within the tolerance the linear
parity tests use, on two calls in a row with different inputs, so the
scratch contents one call leaves behind cannot leak into the next.  This file
is collected last so a failure here never hides the rest of the suite.
"""
import ctypes as C

import numpy as np
import pytest

from paper_2509_26436_gb300 import inputs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def Q():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2509_26436_gb300 as Q
    return Q


def _noalloc(Q, a, w, bias, y):
    lib = Q._native.load()
    ac, wc = a.c(), w.c()
    rc = lib.quartz_linear_noalloc(C.byref(ac), C.byref(wc), None if bias is None else bias.data_ptr(),
                                   y.data_ptr(), Q.OUT_F32, torch.cuda.current_stream().cuda_stream)
    return rc


# (200, 264, 640): ragged M and N tiles, 10 groups.  (1100, 4400, 640): on a
# 152-SM GB300, 9 x 18 = 162 tiles, so the last 10 are cut into 4 parts each
# whose partial tiles sit in the scratch array and are added by the combine
# kernel.
NOALLOC_SHAPES = [(200, 264, 640), (1100, 4400, 640)]
SCRATCH_BYTES = 32 << 20   # QUARTZ_NOALLOC_SCRATCH_BYTES in quartz.h


@pytest.mark.parametrize("M,N,K", NOALLOC_SHAPES)
def test_noalloc_matches_workspace_entry_point(Q, M, N, K):
    assert Q.linear_workspace_size(M, N, K) <= SCRATCH_BYTES
    w16 = inputs.gaussian_weights(N, K, seed=71)
    bias = torch.from_numpy(inputs.gaussian_weights(1, N, seed=72)[0]).cuda()
    w = Q.encode_weights(torch.from_numpy(w16).cuda(), group_s=16)
    for call, seed in enumerate((73, 74)):
        x = torch.from_numpy(inputs.laplace_activations(M, K, seed=seed)).cuda()
        a = Q.quantize(x, group_s=16)
        ref = Q.linear(a, w, bias, out_dtype=torch.float32)
        y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        assert _noalloc(Q, a, w, bias, y) == 0, f"call {call}"
        assert Q.device_status() == 0
        got, exp = y.cpu().numpy().astype(np.float64), ref.cpu().numpy().astype(np.float64)
        # same tolerance as the linear parity tests (fp32 output): relative
        # 1e-5 plus a cancellation term; both calls run the same kernels, so
        # the results are in fact identical
        tol = 1e-5 * np.abs(exp) + (K // 64 + 4) * 2.0 ** -24 * np.abs(exp).max() + 2.0 ** -24
        assert (np.abs(got - exp) <= tol).all(), f"call {call}"
        assert np.array_equal(got, exp), f"call {call}: same kernels, different result"


def test_noalloc_rejects_oversized_problem(Q):
    lib = Q._native.load()
    # a workspace of more than 2 x 8192 x 4096 bytes (both operands expanded to one
    # byte per element), far above the 32 MiB scratch array
    p = Q._native.QuartzParams(64, 16, 0)
    a = Q._native.QuartzEncoded(0x1000, 0x1000, 0x1000, 0, 0, 8192, 4096, p)
    w = Q._native.QuartzEncoded(0x1000, 0x1000, 0x1000, 0, 0, 8192, 4096, p)
    rc = lib.quartz_linear_noalloc(C.byref(a), C.byref(w), None, 0x2000, 0, None)
    assert rc == Q._native.QUARTZ_ERR_WORKSPACE
