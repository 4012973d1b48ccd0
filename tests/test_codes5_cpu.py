"""Pins of the oracle's strict 5-bit storage (Sec. 4: 4 shift bits and a sign bit; for shifts in [-14, 0] a
ternary sign times 15 shifts plus the zero weight is 31 states, which fit 5 bits).  Checked against what the
format and the arithmetic fix, not against the oracle itself: every one of the 31 states by brute force, a
hand-written blob, the exact size of 5 bits per weight, and results of Eq. 3 that do not change when the codes
go through the format."""
import numpy as np
import pytest

import synth_inputs as si
from oracle import deepshift_oracle as O


def _all_states():
    states = [(0, p) for p in range(-15, 1)]
    states += [(s, p) for s in (-1, 1) for p in range(-14, 1)]
    return states


def test_every_state_has_a_distinct_code_and_reads_back():
    codes = {}
    for s, p in _all_states():
        c = O.code5(s, p)
        assert 0 <= c < 32
        if s != 0:
            assert c not in codes.values()
            codes[(s, p)] = c
            assert O.decode5(c) == (s, p)
        else:
            assert c == 0 and O.decode5(0) == (0, 0)
    # 30 nonzero states and the zero weight: 31 of the 32 codes; 31 itself is never written
    assert sorted(codes.values()) == list(range(1, 31))
    assert O.decode5(31) is None


@pytest.mark.parametrize("s,p", [(1, -15), (-1, -15), (2, 0), (1, 1), (0, -16)])
def test_states_outside_the_format_are_refused(s, p):
    with pytest.raises(ValueError):
        O.code5(s, p)


def test_hand_written_blob():
    """One column, three weights: (+1, p=0) -> code 1 = 0b00001, (-1, p=-14) -> code 30 = 0b11110, a zero
    weight -> 0.  Bit plane b holds bit b of each code at the weight's position in its 32-weight chunk."""
    s = np.array([[1, -1, 0]], dtype=np.int8)
    p = np.array([[0, -14, -7]], dtype=np.int8)
    blob = O.pack_codes5(s, p)
    assert blob.size == 512  # 256-byte header + one 20-byte record, rounded to 256 bytes
    assert blob[0:4].view(np.uint32)[0] == 0x31575344 and blob[4:8].view(np.uint32)[0] == 2
    assert list(blob[8:32].view(np.int64)) == [1, 3, 1]
    planes = blob[256:276].view(np.uint32)
    assert list(planes) == [0b001, 0b010, 0b010, 0b010, 0b010]
    assert not blob[276:].any()


@pytest.mark.parametrize("n_out,k_red", [(7, 64), (3, 100), (1, 1), (33, 32)])
def test_five_bits_per_weight(n_out, k_red):
    L = O.codes5_layout(n_out, k_red)
    chunks = (k_red + 31) // 32
    assert L["n_chunks"] == chunks
    assert L["total"] >= 256 + n_out * chunks * 32 * 5 // 8
    assert L["total"] - 256 < n_out * chunks * 32 * 5 // 8 + 256
    if k_red % 32 == 0:
        # exactly 5 bits for each of the n_out * k_red weights in the planes
        assert n_out * chunks * 20 * 8 == 5 * n_out * k_red


def test_round_trip_of_random_codes():
    s = si.sign_codes(11, (9, 75))
    p = np.maximum(si.shift_codes_uniform(11, (9, 75)), -14).astype(np.int8)
    s2, p2 = O.unpack_codes5(O.pack_codes5(s, p), 9, 75)
    assert np.array_equal(s2, s)
    assert np.array_equal(p2, np.where(s == 0, 0, p))


def test_eq3_results_do_not_change_through_the_format():
    """The p of a zero weight is not stored; no term depends on it (s = 0 makes the term zero)."""
    x, s, p, b = si.fc_layer(12, 6, 70, 9, -(1 << 20), 1 << 20)
    p = np.maximum(p, -14).astype(np.int8)
    s2, p2 = O.unpack_codes5(O.pack_codes5(s, p), 9, 70)
    assert np.array_equal(O.linear_shift(x, s2, p2, b), O.linear_shift(x, s, p, b))


def test_corrupt_code_is_refused_on_read():
    blob = O.pack_codes5(np.array([[1]], np.int8), np.array([[0]], np.int8))
    blob[256:276] = 0xFF  # every plane bit set: code 31 at every position
    with pytest.raises(ValueError):
        O.unpack_codes5(blob, 1, 1)
