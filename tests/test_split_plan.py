"""Index plan of the tcgen05 GEMM's split last wave, checked on the CPU.

The persistent GEMM runs P = min(T, SMs) CTAs over T tiles of 128 x 256
outputs, each a sequence of G 64-wide K groups (Section 4.4, Appendix C).
When the tiles left after whole waves would leave CTAs idle, the host cuts
them along K (linear.cu: tail_split; with at most half as many tiles as
SMs every tile is cut into equal parts and the grid has tiles x parts CTAs;
with more than half, every tile's groups are spread in one range per SM)
and every CTA role walks the same work list (work_items / work_item);
tail_combine_kernel adds the parts of a cut tile and returns at once for a
tail tile that one CTA ran whole.

This file restates those three pieces of integer arithmetic in Python and
checks, over a grid of tile counts, SM counts and group counts, that
  * every (tile, group) pair is computed by exactly one CTA;
  * a tile is either whole (part -1, all G groups on one CTA) or cut into
    parts numbered 0 .. split-1 (equal parts) or 0 .. r-1 for the r CTA
    ranges it meets (range forms: r <= 2 after a wave of whole tiles, r <= 3
    with fewer tiles than SMs), whose group ranges are contiguous, ordered
    by part and cover [0, G);
  * every part's partial-tile slot index is inside the workspace that the
    host sizes (tail_tiles x split slots);
  * the combine kernel's test for "this tail tile was cut" agrees with the
    work list, so no cut tile is left unstored and no whole tile is
    overwritten;
  * the cut shortens the busiest CTA's group count as the host intends.
A regression in any of the formulas (an off-by-one in a range bound, a
wrong part number) fails one of these.
"""
import itertools

import pytest

MAX_TAIL_SPLIT = 4
MIN_STREAM_SAVING = 32


def grid_size(T, sms, tail, split, ls):
    """CTAs of the launch: one per tile up to the SM count, tiles x split
    when every tile is cut into equal parts (fewer tiles than SMs), one per
    SM when group ranges are spread over the SMs."""
    if split > 1 and ls == 0 and tail == T:
        return tail * split
    if ls > 0:
        return sms
    return min(T, sms)


def tail_split(T, sms, G):
    """(tail_tiles, split, ls) as the host chooses them (symmetric mode)."""
    P = min(T, sms)
    W, R = divmod(T, P)
    if W >= 1 and 2 * R > P:
        Ts = P + R
        U = Ts * G
        if G * (P - R) < MIN_STREAM_SAVING * P or U >= 1 << 30:
            return 0, 1, 0
        return Ts, 2, (U + P - 1) // P
    if T < sms:
        if 2 * T > sms:
            # more than half the SMs hold a tile: one contiguous range of the
            # tiles' group iterations per SM (a tile in up to 3 parts)
            U = T * G
            if G * (sms - T) < MIN_STREAM_SAVING * sms or U >= 1 << 30:
                return 0, 1, 0
            return T, 3, (U + sms - 1) // sms
        S = min(sms // T, MAX_TAIL_SPLIT, G // 2)
        return (T, S, 0) if S >= 2 else (0, 1, 0)
    if W < 1 or R == 0:
        return 0, 1, 0
    S = min(P // R, MAX_TAIL_SPLIT, G // 2)
    if S < 2:
        return 0, 1, 0
    return R, S, 0


def work_items(c, P, T, G, tail, split, ls):
    full = T - tail if split > 1 else T
    if split <= 1:
        return (T - c + P - 1) // P
    if ls > 0:
        nf = full // P
        U = tail * G
        b, e = c * ls, min(c * ls + ls, U)
        if b >= e:
            return nf
        return nf + (e - 1) // G - b // G + 1
    return full // P + (1 if c < tail * split else 0)


def work_item(c, P, T, G, tail, split, ls, k):
    """(tile, g0, g1, part, tail_index); part -1 is a whole tile."""
    full = T - tail if split > 1 else T
    if ls > 0 and k >= full // P:
        U = tail * G
        b, e = c * ls, min(c * ls + ls, U)
        t = b // G + (k - full // P)
        t0 = t * G
        g0, g1 = max(b - t0, 0), min(e - t0, G)
        if g0 == 0 and g1 == G:
            return full + t, 0, G, -1, 0
        return full + t, g0, g1, c - t0 // ls, t
    if split <= 1 or k < full // P:
        return c + k * P, 0, G, -1, 0
    ti = c // split
    part = c - ti * split
    return full + ti, part * G // split, (part + 1) * G // split, part, ti


def range_parts(tail_index, G, ls):
    """Parts of tail tile `tail_index` when group ranges of ls are spread
    over the SMs: the ranges its G group iterations meet."""
    return ((tail_index + 1) * G - 1) // ls - (tail_index * G) // ls + 1


def combine_skips(tail_index, G, ls):
    """tail_combine_kernel returns at once for this tail tile (range forms)."""
    return ls > 0 and range_parts(tail_index, G, ls) == 1


def check_plan(T, sms, G):
    tail, split, ls = tail_split(T, sms, G)
    P = grid_size(T, sms, tail, split, ls)
    assert P <= sms
    cover = {}
    busiest = 0
    for c in range(P):
        n = work_items(c, P, T, G, tail, split, ls)
        groups = 0
        for k in range(n):
            tile, g0, g1, part, ti = work_item(c, P, T, G, tail, split, ls, k)
            assert 0 <= tile < T
            assert 0 <= g0 < g1 <= G, (T, sms, G, c, k)
            groups += g1 - g0
            if part >= 0:
                assert split > 1
                assert 0 <= ti < tail and 0 <= part < split
                assert tile == T - tail + ti
            cover.setdefault(tile, []).append((g0, g1, part))
        busiest = max(busiest, groups)
    assert sorted(cover) == list(range(T)), "a tile is missing or computed twice"
    for tile, pieces in cover.items():
        pieces.sort()
        assert pieces[0][0] == 0 and pieces[-1][1] == G
        for (a0, a1, _), (b0, b1, _) in zip(pieces, pieces[1:]):
            assert a1 == b0, f"tile {tile}: groups not covered exactly once: {pieces}"
        parts = [p for _, _, p in pieces]
        if len(pieces) == 1:
            assert parts == [-1], f"tile {tile} run whole must be stored whole"
        else:
            assert -1 not in parts
            if ls > 0:
                ti = tile - (T - tail)
                assert parts == list(range(range_parts(ti, G, ls))), f"tile {tile}: range parts {parts}"
                assert len(parts) <= split, f"tile {tile}: {len(parts)} parts, {split} slots"
            else:
                assert parts == list(range(split)), f"tile {tile}: parts {parts}"
        if split > 1 and tile >= T - tail:
            ti = tile - (T - tail)
            assert combine_skips(ti, G, ls) == (len(pieces) == 1), f"combine test wrong for tail tile {ti}"
    # the plan's critical path (group iterations of the busiest CTA)
    W = T // min(T, sms)
    if split > 1 and ls == 0 and tail == T:
        assert busiest == -(-G // split)
    elif split > 1 and ls > 0 and T < sms:
        assert busiest <= ls and busiest <= G - MIN_STREAM_SAVING
    elif split > 1 and ls > 0:
        assert busiest <= (W - 1) * G + ls
        assert busiest <= (W + 1) * G - MIN_STREAM_SAVING
    elif split > 1:
        assert busiest == W * G + -(-G // split) or busiest == W * G + G // split + (G % split > 0)
        assert busiest < (W + 1) * G
    else:
        assert busiest == -(-T // P) * G
    return tail, split, ls


SMS = [1, 2, 3, 7, 16, 148, 152]
TILES = [1, 2, 5, 151, 152, 153, 160, 200, 228, 229, 230, 300, 303, 304, 305, 381, 405, 456, 500, 1000]
GROUPS = [1, 2, 3, 4, 5, 9, 18, 48, 64, 66, 68, 96, 172, 192]


@pytest.mark.parametrize("sms", SMS)
def test_split_plan_covers_every_group_once(sms):
    seen = set()
    for T, G in itertools.product(TILES, GROUPS):
        seen.add(check_plan(T, sms, G)[1:] != (1, 0))
    if sms >= 16:
        assert seen == {True, False}   # the grid exercises split and unsplit plans


def test_split_plan_forms_reached_at_152_sms():
    """The shapes the GPU parity tests use take the form the tests claim."""
    def plan(M, N, K):
        T = -(-M // 128) * -(-N // 256)
        return tail_split(T, 152, K // 64)

    # one-wave form: 4, 3, 2, 2 parts
    assert plan(1100, 4400, 640)[1] == 4
    assert plan(1614, 3816, 640)[1] == 3
    assert plan(1472, 4408, 256)[1] == 2
    assert plan(449, 9904, 320)[1] == 2
    # two-wave form after whole tiles (W = 2): 9 x 45 = 405 and 12 x 32 = 384 tiles
    for shape in ((1100, 11400, 6144), (1500, 8000, 4352)):
        tail, split, ls = plan(*shape)
        assert split == 2 and ls > 0 and tail < -(-shape[0] // 128) * -(-shape[1] // 256)
    # two-wave form over all tiles (W = 1): LLaMA-2-7B down projection at 2048 tokens
    tail, split, ls = plan(2048, 4096, 11008)
    assert split == 2 and ls > 0 and tail == 256
    # a last wave more than half full whose cut would save too little stays whole
    assert plan(2048, 4096, 4096)[1] == 1
    # fewer tiles than SMs: 256 x 1152 x 1152 (2 x 5 tiles, 18 groups) in 4 parts
    # each; one tile of 10 groups in 4; one tile of a single group stays whole
    assert plan(256, 1152, 1152) == (10, 4, 0)
    assert plan(128, 256, 640) == (1, 4, 0)
    assert plan(128, 256, 64)[1] == 1
    # more than half the SMs hold a tile: one range per SM, tiles in up to 3
    # parts (SDXL 3x3 conv on 1280 channels at 32x32: 16 x 5 = 80 tiles, 180 groups)
    assert plan(2048, 1280, 11520) == (80, 3, 95)
    assert plan(1200, 2296, 6400) == (90, 3, 60)
    assert plan(1200, 2296, 640)[1] == 1   # saving too small


def test_split_plan_exhaustive_small():
    """Every tile count up to 5 waves and every group count up to 80 on a
    small and an odd SM count."""
    for sms in (5, 13):
        for T in range(1, 5 * sms + 1):
            for G in range(1, 81):
                check_plan(T, sms, G)
