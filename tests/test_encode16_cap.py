"""Host-side check of the arithmetic behind the 16-bit-code encoder's
branch-free 32767 cap (Section 5 LLM variant, Eq. 1 with 32767 levels,
Eq. 2 with FLAGs up to 12).

The encoder takes each code's magnitude as rne(|x| r) >> FLAG from the
1.5 * 2^23 rounding sum without capping rne(|x| r) first, then saturates
every packed magnitude byte b with (b & 7) | 7 * (bit 3 of b).  That equals
min(rne(|x| r), 32767) >> FLAG as long as (a) an uncapped magnitude above
32767 only occurs in a subgroup whose FLAG is 12, and (b) b never exceeds 15.
Both depend on how far the fp16 scale RN(amax / 32767) can round down, so
they are checked here for every positive finite fp16 group maximum, with the
binary32 steps of the definition (s = fp16(amax / 32767), r = RN(1 / s),
x r rounded once, round half to even), over the 400 fp16 values at and
below each maximum (the only ones whose product can pass 32767).
"""
import numpy as np


def _fp32_steps(amax16):
    amax = amax16.astype(np.float32)
    s = (amax / np.float32(32767)).astype(np.float32).astype(np.float16).astype(np.float32)
    ok = s > 0
    r = np.where(ok, (np.float32(1) / np.where(ok, s, np.float32(1))).astype(np.float32), np.float32(0))
    return r.astype(np.float32), ok


def _flag(qmax):
    """Eq. 2 with 16-bit codes: max(bit_length(m) - 3, 0)."""
    bl = np.zeros_like(qmax)
    nz = qmax > 0
    bl[nz] = np.floor(np.log2(qmax[nz])).astype(np.int64) + 1
    return np.maximum(bl - 3, 0)


def test_branch_free_cap_every_fp16_maximum():
    top = np.arange(1, 0x7C00, dtype=np.uint16).view(np.float16)
    r, ok = _fp32_steps(top)
    qmax = np.minimum(np.rint((top.astype(np.float32) * r).astype(np.float32).astype(np.float64)), 32767)
    F = _flag(qmax.astype(np.int64))
    capped_elements, largest = 0, 0
    for d in range(400):
        idx = np.arange(len(top)) - d
        valid = (idx >= 0) & ok
        x = top[np.clip(idx, 0, None)].astype(np.float32)
        q = np.rint((x * r).astype(np.float32).astype(np.float64)).astype(np.int64)
        over = (q > 32767) & valid
        capped_elements += int(over.sum())
        largest = max(largest, int(q[valid].max()))
        # (a) a magnitude past the cap sits where the (capped) subgroup maximum has FLAG 12
        assert (F[over] == 12).all()
        b = (q >> F) & 0xFF
        # (b) the shifted magnitude byte stays below 16
        assert (b[valid] <= 15).all()
        got = (b & 7) | (((b >> 3) & 1) * 7)
        want = np.minimum(q, 32767) >> F
        assert np.array_equal(got[valid], want[valid])
    # the cap is exercised, and the rounding-down of the smallest subnormal
    # scales pushes rne(|x| r) well past 32768
    assert capped_elements > 100000
    assert 40000 < largest < 49152


def test_byte_saturation_is_per_byte():
    """The packed form: four magnitude bytes at once, no carry between bytes."""
    rng = np.random.default_rng(5)
    b = rng.integers(0, 16, size=(10000, 4)).astype(np.uint32)
    word = b[:, 0] | (b[:, 1] << 8) | (b[:, 2] << 16) | (b[:, 3] << 24)
    sat = (word & np.uint32(0x07070707)) | (((word >> np.uint32(3)) & np.uint32(0x01010101)) * np.uint32(7))
    got = np.stack([(sat >> np.uint32(8 * k)) & np.uint32(0xFF) for k in range(4)], axis=1)
    assert np.array_equal(got, np.minimum(b, 7))
