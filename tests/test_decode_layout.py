"""The shared-memory addressing of the persistent decode grid's fragment loads, checked on the CPU
(a model of the kernel's index arithmetic in `decode.cu`, decode_stream; no GPU).

A TMA box of 64 bf16 columns x R rows with the 128-byte swizzle stores row y's 16-byte chunk k
at byte y * 128 + 16 * (k ^ (y % 8)). A consumer lane (g, c) = (lane // 4, lane % 4) loads, for
the 32-column step st of a box, 8 consecutive K elements of weight rows rho(g) and rho(g) + 8
(the A fragments of two m16n8k16 MMAs) and of token g (its B fragment), with K permuted alike in
both operands. rho(g) = (g >> 1) | ((g & 1) << 2) is the MMA-row -> tile-row map; the epilogue
applies the same map to the accumulator rows.

Checked: every lane reads exactly the element the fragment layout assigns it, every weight row
and K element of a step is read once, and the A loads of each 8-lane phase of a 16-byte shared
load hit 8 distinct bank groups. The staged B loads (T > 2) hit each of 4 bank groups twice per
phase: a 2-way conflict the B layout still carries (rows t and t + 1 swizzle into the same
half of the bank window).
"""
import itertools

KBLK_ROWS = 32        # weight rows of a box (32-row tiles)


def rho8(g):
    return (g >> 1) | ((g & 1) << 2)


def swizzled_offset(row, chunk):
    """Byte offset of (row, 16-byte chunk) inside a 128-byte-swizzled box."""
    return row * 128 + 16 * (chunk ^ (row % 8))


def unswizzle(offset):
    row, pos = divmod(offset, 128)
    return row, (pos // 16) ^ (row % 8)


def a_address(lane, st, gq, half):
    """decode_stream: lane_off = rho(g) 128 + ((c ^ rho(g)) << 4); at = (base + (st >> 1) kBlk) ^
    ((st & 1) << 6); row group gq reads at + 16 gq 128 (MMA row g) and at + (16 gq + 8) 128 (row g + 8).
    Box-relative (the stage base is 1024-byte aligned)."""
    g, c = lane >> 2, lane & 3
    arow = rho8(g)
    lane_off = arow * 128 + ((c ^ arow) << 4)
    at = lane_off ^ ((st & 1) << 6)
    return (st >> 1), at + (16 * gq + 8 * half) * 128


def b_address(lane, st, T, token_map=lambda g: g, clamp=True):
    """Staged B: boff = t 128 + ((c ^ (t & 7)) << 4), read at (st >> 1) bblk + (boff ^ ((st & 1) << 6)),
    for the token t = token_map(g) of lane (g, c), clamped to T - 1 as the kernel does."""
    g, c = lane >> 2, lane & 3
    t = min(token_map(g), T - 1) if clamp else token_map(g)
    boff = t * 128 + ((c ^ (t & 7)) << 4)
    return (st >> 1), boff ^ ((st & 1) << 6)


def test_a_fragments_land_on_their_elements_and_cover_the_step():
    for st in range(4):
        seen = set()
        for lane, gq, half in itertools.product(range(32), range(2), range(2)):
            box, off = a_address(lane, st, gq, half)
            assert box == st >> 1
            row, chunk = unswizzle(off)
            g, c = lane >> 2, lane & 3
            assert row == 16 * gq + 8 * half + rho8(g)            # weight row of MMA row g (+ 8)
            assert chunk == 4 * (st & 1) + c                      # K elements 8 chunk .. + 7 of the box
            seen.add((row, chunk))
        assert seen == {(y, 4 * (st & 1) + k) for y in range(KBLK_ROWS) for k in range(4)}


def test_b_fragments_land_on_their_elements():
    for T, st in itertools.product((3, 5, 8), range(4)):
        for lane in range(32):
            box, off = b_address(lane, st, T)
            row, chunk = unswizzle(off)
            g, c = lane >> 2, lane & 3
            assert row == min(g, T - 1) and chunk == 4 * (st & 1) + c and box == st >> 1


def _worst_phase_conflict(addresses):
    """Max over the four 8-lane phases of a 16-byte load: lanes per bank group (distinct addresses)."""
    worst = 1
    for p in range(4):
        groups = {}
        for off in {addresses[lane] for lane in range(8 * p, 8 * p + 8)}:
            groups[(off // 16) % 8] = groups.get((off // 16) % 8, 0) + 1
        worst = max(worst, max(groups.values()))
    return worst


def test_a_loads_are_bank_conflict_free_and_rho_is_why():
    for st, gq, half in itertools.product(range(4), range(2), range(2)):
        addrs = [a_address(lane, st, gq, half)[1] for lane in range(32)]
        assert _worst_phase_conflict(addrs) == 1
    # without the row map (MMA row g reading tile row g) the same loads conflict 2-way
    plain = [(lane >> 2) * 128 + (((lane & 3) ^ (lane >> 2)) << 4) for lane in range(32)]
    assert _worst_phase_conflict(plain) == 2


def test_staged_b_loads_conflict_two_way_at_most():
    for T, st in itertools.product((3, 5, 8), range(4)):
        addrs = [b_address(lane, st, T)[1] for lane in range(32)]
        assert _worst_phase_conflict(addrs) <= 2
    assert _worst_phase_conflict([b_address(lane, 0, 8)[1] for lane in range(32)]) == 2


def test_reading_token_rho_removes_the_b_conflict():
    """Lane g reading token rho(g) (accumulator columns then un-permuted in the epilogue) puts the
    phase's two tokens in opposite halves of the bank window, as rho does for the weight rows --
    provided the read is not clamped to T - 1: with T <= 4 the clamped tokens fall back into one
    half. A staged box holds round8(T) rows, zero-filled by the TMA beyond T, so the clamp is not
    needed there (results for tokens >= T are never stored)."""
    for T, st in itertools.product((3, 5, 8), range(4)):
        addrs = [b_address(lane, st, T, rho8, clamp=False)[1] for lane in range(32)]
        assert _worst_phase_conflict(addrs) == 1
        for lane in range(32):
            row, chunk = unswizzle(addrs[lane])
            assert row == rho8(lane >> 2) < 8 and chunk == 4 * (st & 1) + (lane & 3)
    assert _worst_phase_conflict([b_address(lane, 0, 3, rho8)[1] for lane in range(32)]) == 2


def row_pitch(kc):
    """decode.cu row_pitch: a row's bytes, plus 64 when they are a multiple of 128."""
    return kc * 2 + (64 if (kc * 2) % 128 == 0 else 0)


def test_padded_rows_are_conflict_free():
    """decode_rows' weight rows (lane (g, c) reads row 16 gq + g [+ 8] at step * 64 + 16 c) and
    decode_stream's resident B rows (token t = g, same column offset) use row_pitch: rows g and
    g + 1 start 64 bytes apart in the bank window, so each phase covers all 8 bank groups."""
    for kc in range(32, 2048 + 1, 32):
        pitch = row_pitch(kc)
        assert pitch % 128 == 64 and pitch >= 2 * kc
        for step in range(kc // 32):
            for gq, half in itertools.product(range(4), range(2)):
                addrs = [(16 * gq + 8 * half + (lane >> 2)) * pitch + step * 64 + 16 * (lane & 3) for lane in range(32)]
                assert _worst_phase_conflict(addrs) == 1
            for T in (1, 2):                      # resident B at T <= 2 (tokens clamped to T - 1)
                addrs = [min(lane >> 2, T - 1) * pitch + step * 64 + 16 * (lane & 3) for lane in range(32)]
                assert _worst_phase_conflict(addrs) == 1
