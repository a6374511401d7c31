"""Pins for oracle.layout (format v1 of the packed cache): every code bit has its own
position (a bijection onto the row's bits), pack/unpack round-trips for every b and every
even r edge case, the row size is 16*r*b bytes, hand-derived positions from the format
text, zero tail tokens, and 256-byte aligned head regions."""
import numpy as np
import pytest

from oracle import layout as lo

RS = [2, 4, 6, 14, 16, 18, 30, 32, 34, 62, 64, 100, 126, 128]


@pytest.mark.parametrize("side", [0, 1])
@pytest.mark.parametrize("b", range(1, 9))
def test_positions_are_a_bijection(side, b):
    for r in (2, 18, 128):
        pos = lo.bit_positions(side, r, b).ravel()
        assert pos.size == 128 * r * b == 8 * lo.row_bytes(r, b)
        assert np.array_equal(np.sort(pos), np.arange(pos.size))


@pytest.mark.parametrize("side", [0, 1])
@pytest.mark.parametrize("b", range(1, 9))
def test_roundtrip(side, b):
    g = np.random.default_rng(b * 10 + side)
    for r in RS:
        codes = g.integers(0, 1 << b, size=(128, r))
        row = lo.pack_row(codes, side, b)
        assert row.dtype == np.uint8 and row.size == 16 * r * b
        assert np.array_equal(lo.unpack_row(row, side, r, b), codes)


def test_hand_positions_k():
    # K row, b = 4, r = 6: token 17 -> tau 1, tt 1 -> piece 1, rho 2; channel 3 -> strip 1, h 1.
    # strip 1 starts at byte 32*4*1 = 128, piece 1 at +16 bytes = 144 -> bit 1152;
    # code bits x = rho*b + k = 8..11 -> word 0, bits 16 + 8..11.
    pos = lo.bit_positions(0, 6, 4)
    assert list(pos[17, 3]) == [1152 + 24, 1152 + 25, 1152 + 26, 1152 + 27]
    # K row, b = 3, token 15 (tau 0, tt 15 -> piece 7, rho 1), channel 0 (strip 0, h 0):
    # piece 7 at byte 4*3*7 = 84 -> bit 672; x = 3..5 -> word 0 bits 3..5.
    assert list(lo.bit_positions(0, 2, 3)[15, 0]) == [675, 676, 677]
    # b = 3, rho 5 straddles 16-bit halves: x = 15, 16, 17 -> word 0 bit 15, word 1 bits 0, 1.
    # token 34 -> tau 2, tt 2 -> piece 2, rho 4 (x = 12..14); token 42 -> tt 10 -> piece 2,
    # rho 5.  channel 1 -> h 1 (+16).
    base = 8 * (4 * 3 * 2)
    assert list(lo.bit_positions(0, 2, 3)[42, 1]) == [base + 16 + 15, base + 32 + 16 + 0, base + 32 + 16 + 1]


def test_hand_positions_v():
    # V row, b = 2, r = 4: token 5 (tau 0, tt 5 -> j = 2, u = 0, h = 1), channel 3
    # (strip 1, c = 1) -> piece 4*1 + 2 = 6, rho 0.  strip 1 at byte 64, piece 6 at +48
    # -> bit 896; x = 0, 1 -> bits 16 + 0, 16 + 1.
    assert list(lo.bit_positions(1, 4, 2)[5, 3]) == [896 + 16, 896 + 17]
    # token 24 (tau 1, tt 8 -> j 0, u 1, h 0), channel 0 -> piece 0, rho 3 -> x = 6, 7.
    assert list(lo.bit_positions(1, 4, 2)[24, 0]) == [6, 7]


def test_pieces_hold_one_lane_fragment():
    """K piece p of strip s holds exactly tokens {16*tau + p, 16*tau + p + 8}; V piece
    4c + j holds channel 2s + c at tokens {16*tau + 2j + {0, 1, 8, 9}}."""
    r, b = 4, 2
    for side in (0, 1):
        pos = lo.bit_positions(side, r, b)
        for t in range(128):
            for i in range(r):
                byte = pos[t, i, 0] // 8
                s, p = byte // (32 * b), (byte % (32 * b)) // (4 * b)
                assert s == i // 2
                tt = t % 16
                if side == 0:
                    assert p == tt % 8
                else:
                    assert p == 4 * (i % 2) + (tt // 2) % 4


def test_tail_is_zero_and_tokens_roundtrip():
    g = np.random.default_rng(5)
    for T in (1, 127, 128, 129, 255, 256, 257):
        for side in (0, 1):
            codes = g.integers(0, 8, size=(T, 6))
            rows = lo.pack_tokens(codes, side, 3)
            assert rows.shape == (-(-T // 128), 16 * 6 * 3)
            full = lo.unpack_tokens(rows, side, 6, 3, rows.shape[0] * 128)
            assert np.array_equal(full[:T], codes)
            assert np.all(full[T:] == 0)


def test_regions():
    r = np.array([128, 0, 2, 18])
    b = np.array([1, 3, 1, 3])
    offs, total = lo.plan_regions(r, b, n_slots=3)
    assert list(offs) == [0, 6144, 6144, 6144 + 256]
    assert total == 6144 + 256 + 3 * 16 * 18 * 3 // 256 * 256 + (256 if (3 * 16 * 18 * 3) % 256 else 0)
    assert all(o % 256 == 0 for o in offs)
