"""Pins of the CPU oracle against what the paper and mathematics fix.

No test here compares the oracle with a retyped copy of itself.  Each pin
reaches the expected value another way: hand-derived values (golden
fixtures), exact rational arithmetic, two's-complement bit strings, float64
library routines on inputs where the shift is exact, closed forms and
invariants.  A plausible mistake in the oracle (a dropped term, a wrong sign,
shift direction or rounding, a transposed operand, a misplaced tap, a missing
bias or clamp) fails at least one of them.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth_inputs as si
from oracle import deepshift_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                rows.append(line.split())
    return rows


def _golden_layer(case):
    d = {}
    for row in _read_golden("layer_cases.txt"):
        if row[0] == case:
            d[row[1]] = [int(v) for v in row[2:]]
    return d


# --------------------------------------------------------------------------
# Single term: Eq. 1 and Eq. 2
# --------------------------------------------------------------------------

def test_term_golden_cases():
    rows = _read_golden("term_cases.txt")
    assert len(rows) >= 20
    for x, p, s, want in rows:
        assert O.term(int(x), int(s), int(p)) == int(want), (x, p, s)


EDGE_X = [-(1 << 31), -(1 << 31) + 1, -(1 << 16) - 1, -(1 << 16), -(1 << 15) - 1, -(1 << 15),
          -(1 << 15) + 1, -3, -2, -1, 0, 1, 2, 3, (1 << 15) - 1, 1 << 15, (1 << 15) + 1,
          (1 << 20) - 1, (1 << 31) - 2, (1 << 31) - 1]


def _twos_complement_shift(x: int, k: int) -> int:
    """Arithmetic right shift done on the 32-bit two's-complement bit string."""
    bits = format(x & 0xFFFFFFFF, "032b")
    shifted = bits[0] * k + bits[:32 - k]          # replicate the sign bit
    v = int(shifted, 2)
    return v - (1 << 32) if shifted[0] == "1" else v


def test_term_exhaustive_codes_vs_rational_floor_and_bit_strings():
    """All 33 code states x edge activations: Eq. 1 as exact rational floor and as a bit-string shift."""
    for p in range(-15, 1):
        for s in (-1, 0, 1):
            for x in EDGE_X:
                want_rational = s * math.floor(Fraction(x, 2 ** (-p)))
                want_bits = s * _twos_complement_shift(x, -p)
                got = O.term(x, s, p)
                assert got == want_rational == want_bits, (x, s, p)


def test_term_rejects_out_of_range_codes():
    with pytest.raises(ValueError):
        O.shift(5, 1)
    with pytest.raises(ValueError):
        O.flip(5, 2)
    x = np.zeros((1, 2), np.int32)
    with pytest.raises(ValueError):
        O.linear_shift(x, np.array([[1, 2]]), np.array([[0, 0]]))
    with pytest.raises(ValueError):
        O.linear_shift(x, np.array([[1, 1]]), np.array([[0, -16]]))


# --------------------------------------------------------------------------
# LinearShift (Eq. 3)
# --------------------------------------------------------------------------

def test_linear_golden_cases():
    for case in ("fc1", "sat1", "sat_bias"):
        g = _golden_layer(case)
        x = np.array([g["x"]], np.int64)
        K = x.shape[1]
        N = len(g["b"])
        s = np.array(g["s"], np.int64).reshape(N, K)
        p = np.array(g["p"], np.int64).reshape(N, K)
        b = np.array(g["b"], np.int64)
        assert O.linear_shift(x, s, p, b).ravel().tolist() == g["y"]
        assert O.linear_shift(x, s, p, b, relu=True).ravel().tolist() == g["y_relu"]


def test_linear_brute_force_tiny():
    """Every output of random tiny layers equals the sum of rational-floor terms."""
    rng = np.random.default_rng(7)
    for _ in range(25):
        M, K, N = rng.integers(1, 5, size=3)
        x = rng.choice(EDGE_X, size=(M, K)).astype(np.int64)
        s = rng.integers(-1, 2, size=(N, K))
        p = rng.integers(-15, 1, size=(N, K))
        b = rng.integers(-(1 << 31), 1 << 31, size=N)
        acc = O.linear_shift_acc(x, s, p, b)
        for m in range(M):
            for n in range(N):
                want = int(b[n]) + sum(int(s[n, k]) * math.floor(Fraction(int(x[m, k]), 2 ** int(-p[n, k])))
                                       for k in range(K))
                assert acc[m, n] == want
                assert O.linear_shift_at(x, s, p, b, m, n) == want


def test_linear_exact_float64_when_x_multiple_of_2_15():
    """x = 2^15 u makes every shift exact, so acc - b equals the float64 matmul with W = s 2^p."""
    rng = np.random.default_rng(11)
    M, K, N = 13, 77, 9
    u = rng.integers(-(1 << 16), 1 << 16, size=(M, K))
    x = u * (1 << 15)
    s = rng.integers(-1, 2, size=(N, K))
    p = rng.integers(-15, 1, size=(N, K))
    b = rng.integers(-(1 << 16), 1 << 16, size=N)
    W = s.astype(np.float64) * np.ldexp(1.0, p)
    want = torch.from_numpy(x.astype(np.float64)) @ torch.from_numpy(W).T
    got = O.linear_shift_acc(x, s, p, b) - b[None, :]
    assert np.array_equal(got.astype(np.float64), want.numpy())


def test_linear_ternary_p0_is_int_matmul():
    rng = np.random.default_rng(12)
    x = rng.integers(-(1 << 20), 1 << 20, size=(6, 50))
    s = rng.integers(-1, 2, size=(7, 50))
    p = np.zeros_like(s)
    assert np.array_equal(O.linear_shift_acc(x, s, p), np.matmul(x, s.T))


def test_linear_negation_invariance():
    """s -> -s negates acc - b exactly; x -> -x does not (floor), which is documented here."""
    x, s, p, b = si.fc_layer(3, 8, 40, 6, -(1 << 20), 1 << 20)
    b = b.astype(np.int64)
    a = O.linear_shift_acc(x, s, p, b) - b
    a_neg = O.linear_shift_acc(x, -s, p, b) - b
    assert np.array_equal(a_neg, -a)
    a_xneg = O.linear_shift_acc(-x.astype(np.int64), s, p, b) - b
    assert not np.array_equal(a_xneg, -a)


def test_linear_split_k_additive():
    x, s, p, b = si.fc_layer(4, 5, 70, 3, -(1 << 20), 1 << 20)
    full = O.linear_shift_acc(x, s, p)
    part = O.linear_shift_acc(x[:, :33], s[:, :33], p[:, :33]) + O.linear_shift_acc(x[:, 33:], s[:, 33:], p[:, 33:])
    assert np.array_equal(full, part)


def test_linear_trivial_weights():
    x, s, p, b = si.fc_layer(5, 4, 30, 5, -(1 << 31), 1 << 31)
    # all-zero signs: y = sat(b)
    assert np.array_equal(O.linear_shift(x, np.zeros_like(s), p, b), np.broadcast_to(b, (4, 5)))
    # one-hot code at k0 with shift q: y = x[:, k0] >> q
    for q in (0, 1, 7, 15):
        s1 = np.zeros_like(s)
        s1[:, 3] = 1
        p1 = np.full_like(p, -q)
        want = np.floor_divide(x[:, 3].astype(np.int64), 1 << q)
        got = O.linear_shift(x, s1, p1)
        assert np.array_equal(got, np.repeat(want[:, None], 5, axis=1))


def test_linear_saturation_boundaries():
    # exact sum lands on INT32_MAX, INT32_MAX + 1, INT32_MIN, INT32_MIN - 1
    x = np.array([[(1 << 30), (1 << 30) - 1, 1]], np.int64)
    s = np.array([[1, 1, 0], [1, 1, 1], [-1, -1, -1], [-1, -1, -1]])
    p = np.zeros_like(s)
    b = np.array([0, 0, 0, -1])
    y = O.linear_shift(x, s, p, b)
    assert y.ravel().tolist() == [(1 << 31) - 1, (1 << 31) - 1, -(1 << 31), -(1 << 31)]
    acc = O.linear_shift_acc(x, s, p, b).ravel().tolist()
    assert acc == [(1 << 31) - 1, 1 << 31, -(1 << 31), -(1 << 31) - 1]


def test_accumulation_bound_holds_and_is_tight():
    rng = np.random.default_rng(21)
    for _ in range(30):
        M, K, N = 4, int(rng.integers(1, 60)), 3
        amax_bits = int(rng.integers(1, 32))
        x = rng.integers(-(1 << amax_bits), 1 << amax_bits, size=(M, K))
        x = np.clip(x, -(1 << 31), (1 << 31) - 1)
        s = rng.integers(-1, 2, size=(N, K))
        p = rng.integers(-15, 1, size=(N, K))
        b = rng.integers(-(1 << 20), 1 << 20, size=N)
        A, nnz = O.column_constants(s, p)
        amax = O.absmax(x)
        acc = O.linear_shift_acc(x, s, p, b)
        for n in range(N):
            bound = ((amax * int(A[n]) + (1 << 15) - 1) >> 15) + int(nnz[n]) + abs(int(b[n]))
            assert np.abs(acc[:, n]).max() <= bound
    # worst case attains ceil(amax / 2^k) per term
    amax = (1 << 20) + 5
    ks = np.arange(16)
    x = np.full((1, 16), -amax)
    s = -np.ones((1, 16), np.int64)
    p = -ks[None, :]
    acc = int(O.linear_shift_acc(x, s, p)[0, 0])
    assert acc == sum(-(-amax // (1 << int(k))) for k in ks)
    A, nnz = O.column_constants(s, p)
    assert acc <= ((amax * int(A[0]) + (1 << 15) - 1) >> 15) + int(nnz[0])
    # -INT32_MIN with s = -1 does not fit int32: the bound must refuse it
    assert not O.int32_accumulation_is_exact(1 << 31, 1 << 15, 1, 0)
    assert O.int32_accumulation_is_exact((1 << 31) - 2, 1 << 15, 1, 0)


def test_accumulation_bound_is_sound_at_the_int32_edge():
    """Near the int32 edge the bound admits no column whose worst-case sum overflows (reading R-acc).

    The worst case of a column with s = -1 and p = 0, -1, ..., -15 is x = -amax on every term: each term is then
    ceil(amax / 2^k), and a positive bias adds b.  That sum is written out here with Python ints.  For amax swept
    across the point where it passes INT32_MAX, the bound may answer True only when the sum fits, and it does
    answer True a little below the edge, so it is not vacuous.
    """
    ks = range(16)
    s = -np.ones((1, 16), np.int64)
    p = -np.arange(16)[None, :]
    A, nnz = O.column_constants(s, p)
    for babs in (0, 1, 2, 3, 12345, (1 << 20) + 3):   # several positions of the edge
        def worst(amax):
            return sum(-(-amax // (1 << k)) for k in ks) + babs
        lo, hi = 0, 1 << 31             # the largest amax whose worst case fits: worst(lo) <= INT32_MAX < worst(hi)
        while hi - lo > 1:
            mid = (lo + hi) // 2
            lo, hi = (mid, hi) if worst(mid) <= O.INT32_MAX else (lo, mid)
        answers = {amax: O.int32_accumulation_is_exact(amax, int(A[0]), int(nnz[0]), babs)
                   for amax in range(lo - 64, lo + 64)}
        for amax, ok in answers.items():
            assert not ok or worst(amax) <= O.INT32_MAX, (amax, babs)
        assert answers[lo - 64]


def test_column_constants_closed_forms():
    K = 37
    s = np.ones((3, K), np.int64)
    p = np.stack([np.zeros(K), np.full(K, -15), np.full(K, -3)]).astype(np.int64)
    A, nnz = O.column_constants(s, p)
    assert A.tolist() == [K << 15, K, K << 12]
    assert nnz.tolist() == [K, K, K]
    s[1, ::2] = 0
    A, nnz = O.column_constants(s, p)
    assert A[1] == K // 2 and nnz[1] == K // 2


# --------------------------------------------------------------------------
# ConvShift (Eq. 3, convolution form)
# --------------------------------------------------------------------------

def test_conv_golden_cases():
    x = np.arange(1, 10, dtype=np.int64).reshape(1, 1, 3, 3)
    s = np.zeros((1, 1, 3, 3), np.int64)
    s[0, 0, 0, 2] = 1
    p = np.zeros_like(s)
    y = O.conv2d_shift(x, s, p, None, (1, 1), (1, 1))
    assert y.ravel().tolist() == _golden_layer("conv_xcorr")["y"]
    g = _golden_layer("conv_half")
    y = O.conv2d_shift(x, np.ones_like(s), -np.ones_like(s), None, (1, 1), (1, 1))[0, 0]
    for key, (i, j) in {"y00": (0, 0), "y01": (0, 1), "y10": (1, 0), "y11": (1, 1), "y22": (2, 2)}.items():
        assert y[i, j] == g[key][0]
    # 1x1 stride 2: subsampling
    x = np.arange(16, dtype=np.int64).reshape(1, 1, 4, 4)
    y = O.conv2d_shift(x, np.ones((1, 1, 1, 1)), np.zeros((1, 1, 1, 1)), None, (2, 2), (0, 0))
    assert y.ravel().tolist() == [0, 2, 8, 10]


@pytest.mark.parametrize("geom", [(2, 3, 7, 6, 4, 3, 3, 1, 1, 1, 1), (1, 2, 9, 9, 3, 3, 3, 2, 2, 1, 1),
                                  (2, 3, 11, 10, 2, 7, 7, 2, 2, 3, 3), (1, 4, 6, 5, 3, 1, 1, 2, 2, 0, 0),
                                  (1, 2, 5, 7, 2, 3, 1, 1, 2, 0, 2)])
def test_conv_exact_float64_when_x_multiple_of_2_15(geom):
    """x = 2^15 u: acc - b equals torch's float64 conv2d with W = s 2^p (cross-correlation)."""
    N, C, H, W, K, R, S, sh, sw, ph, pw = geom
    rng = np.random.default_rng(sum(geom))
    x = rng.integers(-(1 << 16), 1 << 16, size=(N, C, H, W)) * (1 << 15)
    s = rng.integers(-1, 2, size=(K, C, R, S))
    p = rng.integers(-15, 1, size=(K, C, R, S))
    b = rng.integers(-(1 << 16), 1 << 16, size=K)
    Wt = torch.from_numpy(s.astype(np.float64) * np.ldexp(1.0, p))
    want = F.conv2d(torch.from_numpy(x.astype(np.float64)), Wt, stride=(sh, sw), padding=(ph, pw))
    got = O.conv2d_shift_acc(x, s, p, b, (sh, sw), (ph, pw)) - b[None, :, None, None]
    assert got.shape == tuple(want.shape)
    assert np.array_equal(got.astype(np.float64), want.numpy())


def _im2col(x, R, S, stride, pad):
    """Explicit patch gather: rows = (n, oh, ow), columns = (c, r, q), zero outside the image."""
    N, C, H, W = x.shape
    OH = (H + 2 * pad[0] - R) // stride[0] + 1
    OW = (W + 2 * pad[1] - S) // stride[1] + 1
    cols = np.zeros((N * OH * OW, C * R * S), dtype=np.int64)
    for n in range(N):
        for oh in range(OH):
            for ow in range(OW):
                row = (n * OH + oh) * OW + ow
                for c in range(C):
                    for r in range(R):
                        for q in range(S):
                            ih = oh * stride[0] - pad[0] + r
                            iw = ow * stride[1] - pad[1] + q
                            if 0 <= ih < H and 0 <= iw < W:
                                cols[row, (c * R + r) * S + q] = x[n, c, ih, iw]
    return cols, OH, OW


@pytest.mark.parametrize("geom", [(2, 3, 6, 5, 4, 3, 3, 1, 1, 1, 1), (1, 2, 9, 8, 3, 7, 7, 2, 2, 3, 3),
                                  (1, 3, 7, 7, 2, 3, 3, 2, 2, 1, 1)])
def test_conv_equals_im2col_plus_linear(geom):
    N, C, H, W, K, R, S, sh, sw, ph, pw = geom
    x, s, p, b = si.conv_layer(sum(geom), N, C, H, W, K, R, S, -(1 << 20), 1 << 20)
    cols, OH, OW = _im2col(x.astype(np.int64), R, S, (sh, sw), (ph, pw))
    lin = O.linear_shift_acc(cols, s.reshape(K, -1), p.reshape(K, -1), b)
    lin = lin.reshape(N, OH, OW, K).transpose(0, 3, 1, 2)
    assert np.array_equal(O.conv2d_shift_acc(x, s, p, b, (sh, sw), (ph, pw)), lin)


def test_conv_identity_and_sampled_elements():
    x, s, p, b = si.conv_layer(9, 2, 4, 6, 6, 4, 1, 1, -(1 << 31), 1 << 31)
    eye_s = np.eye(4, dtype=np.int64).reshape(4, 4, 1, 1)
    y = O.conv2d_shift(x, eye_s, np.zeros_like(eye_s), None)
    assert np.array_equal(y, x)
    x, s, p, b = si.conv_layer(10, 2, 3, 7, 6, 5, 3, 3)
    acc = O.conv2d_shift_acc(x, s, p, b, (2, 1), (1, 0))
    for (n, k, oh, ow) in [(0, 0, 0, 0), (1, 4, 3, 3), (0, 2, 1, 2), (1, 1, 3, 0)]:
        assert acc[n, k, oh, ow] == O.conv2d_shift_at(x, s, p, b, (2, 1), (1, 0), n, k, oh, ow)


def test_conv_negation_invariance():
    x, s, p, b = si.conv_layer(13, 1, 3, 6, 6, 4, 3, 3, -(1 << 20), 1 << 20)
    bb = b.astype(np.int64)[None, :, None, None]
    a = O.conv2d_shift_acc(x, s, p, b, (1, 1), (1, 1)) - bb
    assert np.array_equal(O.conv2d_shift_acc(x, -s, p, b, (1, 1), (1, 1)) - bb, -a)


# --------------------------------------------------------------------------
# Chain operators
# --------------------------------------------------------------------------

def test_maxpool_golden_and_library():
    x = np.array([[[[-1, -2], [-3, -4]]]], np.int32)
    assert O.maxpool2d(x, 3, 2, 1).ravel().tolist() == _golden_layer("maxpool_neg")["y"]
    rng = np.random.default_rng(3)
    x = rng.integers(-(1 << 31), 1 << 31, size=(2, 3, 11, 10)).astype(np.int32)
    want = F.max_pool2d(torch.from_numpy(x.astype(np.float64)), 3, 2, 1).numpy()
    assert np.array_equal(O.maxpool2d(x, 3, 2, 1).astype(np.float64), want)
    want2 = F.max_pool2d(torch.from_numpy(x.astype(np.float64)), 2, 2, 0).numpy()
    assert np.array_equal(O.maxpool2d(x, 2, 2, 0).astype(np.float64), want2)


def test_avgpool_floor_golden_and_library():
    g = _golden_layer("avgpool_floor")
    for key in ("a", "b"):
        x = np.array(g[key], np.int32).reshape(1, 1, 2, 2)
        assert O.avgpool_floor(x, 2, 2).ravel().tolist() == g[key + "_y"]
    rng = np.random.default_rng(4)
    x = rng.integers(-(1 << 31), 1 << 31, size=(2, 5, 7, 7)).astype(np.int32)
    mean = F.avg_pool2d(torch.from_numpy(x.astype(np.float64)), 7).numpy()
    assert np.array_equal(O.avgpool_floor(x, 7, 7).astype(np.float64), np.floor(mean))


def test_add_relu_golden():
    g = _golden_layer("add_relu")
    assert O.add_relu(np.array(g["a"], np.int32), np.array(g["b"], np.int32)).tolist() == g["y"]


# --------------------------------------------------------------------------
# Float variant
# --------------------------------------------------------------------------

def test_float_variant_exact_on_small_integers_and_near_library():
    rng = np.random.default_rng(5)
    M, K, N = 9, 64, 7
    xi = rng.integers(-100, 100, size=(M, K))
    s = rng.integers(-1, 2, size=(N, K))
    p = rng.integers(-15, 1, size=(N, K))
    got = O.linear_shift_float(xi.astype(np.float64), s, p)
    for m in range(M):
        for n in range(N):
            want = sum(Fraction(int(s[n, k]) * int(xi[m, k])) * Fraction(1, 2 ** int(-p[n, k])) for k in range(K))
            assert Fraction(got[m, n]) == want
    x = si.bits_to_f64(si.bf16_bits(rng.uniform(-(1 << 20), 1 << 20, size=(M, K))))
    b = rng.uniform(-1, 1, size=N)
    W = s.astype(np.float64) * np.ldexp(1.0, p)
    lib = x @ W.T + b
    got = O.linear_shift_float(x, s, p, b)
    scale = O.linear_shift_float_absterms(x, s, p) + np.abs(b)
    assert np.all(np.abs(got - lib) <= 1e-13 * scale)


# --------------------------------------------------------------------------
# Packed blob (storage format of the codes)
# --------------------------------------------------------------------------

def test_pack_golden_tiny_blob():
    g = {r[0]: [int(v) for v in r[1:]] for r in _read_golden("pack_tiny.txt")}
    s = np.array(g["s"]).reshape(2, 3)
    p = np.array(g["p"]).reshape(2, 3)
    blob = O.pack_planes6(s, p)
    L = O.blob_layout(2, 3)
    nib = np.frombuffer(blob[L["nib"]:L["bits"]].tobytes(), np.uint32).reshape(1, 2, 4)
    bits = np.frombuffer(blob[L["bits"]:L["col_a"]].tobytes(), np.uint32).reshape(1, 2, 2)
    assert nib[0, 0].tolist() == g["nib0"] and nib[0, 1].tolist() == g["nib1"]
    assert bits[0, 0].tolist() == g["bits0"] and bits[0, 1].tolist() == g["bits1"]
    colA = np.frombuffer(blob[L["col_a"]:L["nnz"]].tobytes(), np.uint64)
    nnz = np.frombuffer(blob[L["nnz"]:L["nnz"] + 8].tobytes(), np.uint32)
    assert colA.tolist() == g["colA"] and nnz.tolist() == g["nnz"]
    hdr = blob[:48]
    assert int(np.frombuffer(hdr[0:4].tobytes(), np.uint32)[0]) == 0x31575344
    assert np.frombuffer(hdr[8:32].tobytes(), np.int64).tolist() == [2, 3, 1]
    assert int(np.frombuffer(hdr[36:40].tobytes(), np.uint32)[0]) == 3
    assert int(np.frombuffer(hdr[40:48].tobytes(), np.uint64)[0]) == 32769


def test_pack_round_trip_and_sizes():
    for n_out, k_red in [(1, 1), (3, 31), (5, 32), (4, 33), (2, 100)]:
        s = si.sign_codes(n_out * 1000 + k_red, (n_out, k_red))
        p = si.shift_codes_uniform(n_out * 1000 + k_red, (n_out, k_red))
        blob = O.pack_planes6(s, p)
        L = O.blob_layout(n_out, k_red)
        assert blob.size == L["total"] and L["total"] % 256 == 0
        assert L["bits"] - L["nib"] == ((k_red + 31) // 32) * n_out * 16
        s2, p2 = O.unpack_planes6(blob, n_out, k_red)
        assert np.array_equal(s2, s)
        # a zero code's shift is still stored
        assert np.array_equal(p2, p)


def test_expand_layout_closed_form():
    """Expanded layout: word c of row (cb, k) is -p of column 32 cb + c, word 32 + c its sign."""
    s = np.array([[1, -1, 0], [0, 1, -1]])
    p = np.array([[0, -15, -3], [-1, -2, -4]])
    e = O.expand_codes(s, p)
    assert e.shape == (1, 3, 64)
    assert e[0, :, 0].tolist() == [0, 15, 3] and e[0, :, 1].tolist() == [1, 2, 4]
    assert e[0, :, 32].tolist() == [1, -1, 0] and e[0, :, 33].tolist() == [0, 1, -1]
    assert not e[0, :, 2:32].any() and not e[0, :, 34:].any()
    s2 = np.ones((40, 2), np.int64)
    e2 = O.expand_codes(s2, np.zeros_like(s2))
    assert e2.shape == (2, 2, 64) and e2[1, :, 32:40].all() and not e2[1, :, 40:].any()


# --------------------------------------------------------------------------
# Chained forward: the ResNet composition against float64 library routines
# --------------------------------------------------------------------------

def _one_hot_params(shapes, seed):
    """p = 0 and exactly one non-zero sign per output channel: every term is exact, activations stay bounded."""
    rng = np.random.default_rng(seed)
    params = []
    for shp in shapes:
        K = shp[0]
        fan = int(np.prod(shp[1:]))
        s = np.zeros((K, fan), np.int64)
        s[np.arange(K), rng.integers(0, fan, K)] = rng.choice([-1, 1], K)
        params.append((s.reshape(shp), np.zeros(shp, np.int64), rng.integers(-(1 << 10), 1 << 10, K)))
    return params


def _torch_resnet(x, params, kind, blocks):
    """float64 torch restatement (library conv2d / pools / linear) of the same ResNet topology."""
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    it = iter(params)

    def conv(v, prm, stride, pad):
        s, p, b = prm
        return F.conv2d(v, t(s * np.ldexp(1.0, p)), t(b), stride=stride, padding=pad)

    v = F.relu(conv(t(x), next(it), 2, 3))
    v = F.max_pool2d(v, 3, 2, 1)
    for stage, nb in enumerate(blocks):
        planes = 64 * 2 ** stage
        out_c = planes if kind == "basic" else 4 * planes
        for bi in range(nb):
            stride = 2 if (stage > 0 and bi == 0) else 1
            need_ds = stride != 1 or v.shape[1] != out_c
            if kind == "basic":
                c1, c2 = next(it), next(it)
                ds = next(it) if need_ds else None
                m = conv(F.relu(conv(v, c1, stride, 1)), c2, 1, 1)
            else:
                c1, c2, c3 = next(it), next(it), next(it)
                ds = next(it) if need_ds else None
                m = conv(F.relu(conv(F.relu(conv(v, c1, 1, 0)), c2, stride, 1)), c3, 1, 0)
            sc = conv(v, ds, stride, 0) if ds is not None else v
            v = F.relu(m + sc)
    v = torch.floor(F.avg_pool2d(v, v.shape[2]))
    s, p, b = next(it)
    return F.linear(v.reshape(v.shape[0], -1), t(s.reshape(s.shape[0], -1) * np.ldexp(1.0, p.reshape(p.shape[0], -1))),
                    t(b))


@pytest.mark.parametrize("arch,kind,blocks", [("resnet18", "basic", [2, 2, 2, 2]),
                                              ("resnet50", "bottleneck", [3, 4, 6, 3])])
def test_resnet_chain_matches_float64_library_case(arch, kind, blocks):
    from oracle import networks as ON
    from paper_1905_13298_gb300 import networks as PN   # layer shapes only (no library call)
    _, shapes = PN.resnet_program(arch, 32, 32)
    params = _one_hot_params(shapes, 3)
    x = si.image_batch(5, 2, 3, 32, 32)
    got = ON.resnet_forward(x, params, arch)
    want = _torch_resnet(x, params, kind, blocks).numpy()
    assert np.abs(want).max() < 2 ** 31
    assert np.array_equal(got.astype(np.float64), want)


def _torch_vgg16(x, params):
    """float64 torch restatement (library conv2d / max_pool2d / linear) of VGG16 (configuration D)."""
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    it = iter(params)
    v = t(x)
    for c in (64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M", 512, 512, 512, "M"):
        if c == "M":
            v = F.max_pool2d(v, 2, 2)
        else:
            s, p, b = next(it)
            v = F.relu(F.conv2d(v, t(s * np.ldexp(1.0, p)), t(b), stride=1, padding=1))
    v = v.reshape(v.shape[0], -1)
    for i in range(3):
        s, p, b = next(it)
        w = s.reshape(s.shape[0], -1) * np.ldexp(1.0, p.reshape(p.shape[0], -1))
        v = F.linear(v, t(w), t(b))
        if i < 2:
            v = F.relu(v)
    return v


def test_vgg16_chain_matches_float64_library_case():
    """VGG16 (32 x 32 input, so the first FC has 512 inputs): one-hot codes with p = 0 make every
    term exact, so the oracle's chain equals the float64 library composition exactly."""
    from oracle import networks as ON
    from paper_1905_13298_gb300 import networks as PN   # layer shapes only (no library call)
    _, shapes = PN.vgg16_program(32, 32)
    params = _one_hot_params(shapes, 4)
    x = si.image_batch(6, 2, 3, 32, 32)
    got = ON.vgg16_forward(x, params)
    want = _torch_vgg16(x, params).numpy()
    assert np.abs(want).max() < 2 ** 31
    assert np.array_equal(got.astype(np.float64), want)


def test_bf16_weight_bits_decode_to_s_times_power_of_two():
    """bf16 patterns of the float variant's weights decode (via float32 bit casts) to s * 2^p exactly."""
    s = np.array([[1, -1, 0, 1], [-1, 1, 1, 0]])
    p = np.array([[0, -15, -3, -7], [-1, -2, 0, -15]])
    bits = O.weights_bf16_bits(s, p)
    assert bits[0, 0] == 0x3F80 and bits[0, 1] == 0xB800 and bits[0, 2] == 0 and bits[1, 2] == 0x3F80
    vals = si.bits_to_f64(bits)
    assert np.array_equal(vals, s * np.ldexp(1.0, p))


# ---------------------------------------------------------------------------
# DeepShift-Q quantizer (Eq. 4-6) and Q16.16 input rounding (Sec. 4)
# ---------------------------------------------------------------------------
def _exact_round_log2(a: float) -> int:
    """round(log2 a) for a float a > 0 from exact rationals: the n with
    2^(2n-1) <= a^2 < 2^(2n+1) (the bound 2^(n+1/2) is irrational, so no ties)."""
    from fractions import Fraction
    q = Fraction(a) ** 2
    n = 0
    while q >= Fraction(2) ** (2 * n + 1):
        n += 1
    while q < Fraction(2) ** (2 * n - 1):
        n -= 1
    return n


def test_quantize_weights_powers_of_two_are_fixed_points():
    """W = +-2^k quantizes to s = +-1, p = k inside [-15, 0] and to the clip bound outside it."""
    ks = np.arange(-20, 4)
    for sign in (1.0, -1.0):
        w = (sign * np.ldexp(1.0, ks)).astype(np.float32)
        s, p = O.quantize_weights(w)
        assert (s == int(sign)).all()
        assert np.array_equal(p, np.clip(ks, -15, 0))


def test_quantize_weights_against_exact_rationals():
    """Random float32 weights, and the float32 neighbours of every rounding bound 2^(n+1/2):
    p equals the clipped exact round(log2|W|), s the sign."""
    w = si.float_weights(31, (4000,), -19, 2)
    bounds = []
    for n in range(-18, 3):
        c = np.float32(2.0 ** (n + 0.5))
        bounds += [c, np.nextafter(c, np.float32(0)), np.nextafter(c, np.float32(10))]
    w = np.concatenate([w, np.array(bounds, np.float32), -np.array(bounds, np.float32)])
    for p_min in (-15, -14):
        s, p = O.quantize_weights(w, p_min)
        for wi, si_, pi in zip(w.tolist(), s.tolist(), p.tolist()):
            assert si_ == (1 if wi > 0 else -1)
            assert pi == min(max(_exact_round_log2(abs(wi)), p_min), 0), (wi, pi)


def test_quantize_weights_matches_log2_library_away_from_bounds():
    """np.round(np.log2(|W|)), a different route, agrees wherever log2|W| is not within 1e-6 of a half-integer."""
    w = si.float_weights(32, (200000,), -17, 1)
    lg = np.log2(np.abs(w.astype(np.float64)))
    far = np.abs(lg - np.floor(lg) - 0.5) > 1e-6
    s, p = O.quantize_weights(w)
    assert np.array_equal(p[far], np.clip(np.round(lg[far]), -15, 0).astype(np.int8))
    assert np.array_equal(s, np.sign(w).astype(np.int8))


def test_quantize_weights_special_values():
    w = np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 1e-45, -1e-40, 3.0, -1.0e30], np.float32)
    s, p = O.quantize_weights(w)
    assert s.tolist() == [0, 0, 0, 1, -1, 1, -1, 1, -1]
    assert p.tolist() == [-15, -15, -15, 0, 0, -15, -15, 0, 0]
    s, p = O.quantize_weights(w, -14)
    assert p.tolist() == [-14, -14, -14, 0, 0, -14, -14, 0, 0]
    with pytest.raises(ValueError):
        O.quantize_weights(w, -16)


def test_quantize_weights_then_flip_reproduces_powers_of_two():
    """Eq. 6: flip(2^p, s) of the codes is the nearest power of two in log scale, clipped."""
    w = si.float_weights(33, (5000,), -14, -1)
    s, p = O.quantize_weights(w)
    wq = s.astype(np.float64) * np.ldexp(1.0, p.astype(np.int64))
    ratio = np.abs(w.astype(np.float64)) / np.abs(wq)
    assert (ratio >= 2 ** -0.5).all() and (ratio < 2 ** 0.5).all()


def test_quantize_activations_ties_saturation_and_specials():
    half = 1.0 / 65536
    x = np.array([0.5 * half, 1.5 * half, 2.5 * half, -0.5 * half, -1.5 * half, -2.5 * half,
                  32767.0, 32768.0, -32768.0, -32768.5, 1e30, -1e30, np.nan, np.inf, -np.inf], np.float32)
    q = O.quantize_activations(x)
    assert q.tolist() == [0, 2, 2, 0, -2, -2, 32767 << 16, 2 ** 31 - 1, -(2 ** 31), -(2 ** 31),
                          2 ** 31 - 1, -(2 ** 31), 0, 2 ** 31 - 1, -(2 ** 31)]


def test_quantize_activations_against_exact_rationals_and_torch_round():
    """Exact rational round-half-even on random values (including ties), and torch.round (also half to
    even) as a library route for values inside the range."""
    from fractions import Fraction
    x = si.float_activations(34, (3000,), -20, 14)
    q = O.quantize_activations(x)
    for xi, qi in zip(x.tolist(), q.tolist()):
        v = Fraction(xi) * 65536
        fl = v.numerator // v.denominator
        d = v - fl
        r = fl + (1 if d > Fraction(1, 2) or (d == Fraction(1, 2) and fl % 2 == 1) else 0)
        assert qi == max(min(r, 2 ** 31 - 1), -(2 ** 31)), xi
    t = torch.round(torch.from_numpy(x.astype(np.float64)) * 65536).to(torch.int64).numpy()
    assert np.array_equal(q.astype(np.int64), t)


# ---------------------------------------------------------------------------
# Input gradient (Eq. 7 and its footnote)
# ---------------------------------------------------------------------------
BWD_GEOMS = [  # N, C, H, W, K, R, S, stride, pad
    (2, 3, 7, 6, 4, 3, 3, 1, 1), (2, 3, 7, 6, 4, 3, 3, 2, 1), (1, 2, 9, 9, 3, 7, 7, 2, 3),
    (2, 5, 6, 5, 3, 1, 1, 2, 0), (1, 4, 5, 5, 2, 3, 3, 1, 0), (1, 2, 8, 7, 3, 5, 3, 2, 2),
]


@pytest.mark.parametrize("geom", BWD_GEOMS)
def test_conv_backward_x_equals_float64_autograd_on_exact_inputs(geom):
    """dy a multiple of 2^15 makes every shift exact, so dC/dX is torch's float64 autograd of conv2d with
    W = s * 2^p (a library route through the transposed convolution)."""
    N, C, H, W, K, R, S, st, pd = geom
    s = si.sign_codes(sum(geom), (K, C, R, S))
    p = si.shift_codes_uniform(sum(geom), (K, C, R, S))
    OH, OW = O.conv_out_size(H, R, st, pd), O.conv_out_size(W, S, st, pd)
    dy = si.uniform_int(sum(geom) + 1, si.STREAM_X, (N, K, OH, OW), -4096, 4096) * (1 << 15)
    got = O.conv2d_shift_backward_x_acc(dy, s, p, (H, W), (st, st), (pd, pd))
    wt = torch.tensor(s * np.ldexp(1.0, p.astype(np.int64)), dtype=torch.float64)
    x = torch.zeros((N, C, H, W), dtype=torch.float64, requires_grad=True)
    F.conv2d(x, wt, stride=st, padding=pd).backward(torch.tensor(dy, dtype=torch.float64))
    assert np.array_equal(got, x.grad.numpy().astype(np.int64))


def test_linear_backward_x_equals_float64_matmul_on_exact_inputs():
    M, K, N = 7, 19, 11
    s = si.sign_codes(3, (N, K))
    p = si.shift_codes_uniform(3, (N, K))
    dy = si.uniform_int(4, si.STREAM_X, (M, N), -4096, 4096) * (1 << 15)
    wt = torch.tensor(s * np.ldexp(1.0, p.astype(np.int64)), dtype=torch.float64)
    want = (torch.tensor(dy, dtype=torch.float64) @ wt).numpy().astype(np.int64)
    assert np.array_equal(O.linear_shift_backward_x_acc(dy, s, p), want)


@pytest.mark.parametrize("geom", BWD_GEOMS[:4])
def test_conv_backward_x_brute_force_gather_with_floor(geom):
    """Non-exact gradients (floor matters): each input position gathers, with Python ints, every
    (output, tap) pair that read it in the forward pass."""
    N, C, H, W, K, R, S, st, pd = geom
    s = si.sign_codes(sum(geom) + 2, (K, C, R, S))
    p = si.shift_codes_uniform(sum(geom) + 2, (K, C, R, S))
    OH, OW = O.conv_out_size(H, R, st, pd), O.conv_out_size(W, S, st, pd)
    dy = si.activations(sum(geom) + 3, (N, K, OH, OW), -(1 << 20), 1 << 20)
    got = O.conv2d_shift_backward_x(dy, s, p, (H, W), (st, st), (pd, pd))
    for n in range(N):
        for c in range(C):
            for i in range(H):
                for j in range(W):
                    acc = 0
                    for k in range(K):
                        for r in range(R):
                            for q in range(S):
                                u, v = i + pd - r, j + pd - q
                                if u % st or v % st:
                                    continue
                                oh, ow = u // st, v // st
                                if 0 <= oh < OH and 0 <= ow < OW:
                                    acc += int(s[k, c, r, q]) * (int(dy[n, k, oh, ow]) // (1 << -int(p[k, c, r, q])))
                    assert got[n, c, i, j] == max(min(acc, 2 ** 31 - 1), -(2 ** 31))


@pytest.mark.parametrize("geom", [g for g in BWD_GEOMS if g[7] == 1])
def test_conv_backward_x_stride1_is_forward_conv_with_rot180_codes(geom):
    """For stride 1 the input gradient is the forward ConvShift of dy with the rot180 / transposed codes
    (Eq. 7 footnote) and padding R - 1 - pad."""
    N, C, H, W, K, R, S, st, pd = geom
    s = si.sign_codes(sum(geom) + 4, (K, C, R, S))
    p = si.shift_codes_uniform(sum(geom) + 4, (K, C, R, S))
    OH, OW = O.conv_out_size(H, R, 1, pd), O.conv_out_size(W, S, 1, pd)
    dy = si.activations(sum(geom) + 5, (N, K, OH, OW), -(1 << 24), 1 << 24)
    sb, pb = O.backward_codes(s, p)
    assert sb.shape == (C, K, R, S) and sb[0, 0, 0, 0] == s[0, 0, R - 1, S - 1]
    want = O.conv2d_shift_backward_x(dy, s, p, (H, W), (1, 1), (pd, pd))
    assert np.array_equal(O.conv2d_shift(dy, sb, pb, None, (1, 1), (R - 1 - pd, S - 1 - pd)), want)


def test_linear_backward_x_is_forward_with_transposed_codes():
    s = si.sign_codes(6, (13, 29))
    p = si.shift_codes_uniform(6, (13, 29))
    dy = si.activations(7, (5, 13), -(1 << 30), 1 << 30)
    sb, pb = O.backward_codes(s, p)
    assert np.array_equal(O.linear_shift(dy, sb[:, :, 0, 0], pb[:, :, 0, 0]), O.linear_shift_backward_x(dy, s, p))


@pytest.mark.parametrize("geom", BWD_GEOMS)
def test_conv_backward_x_phase_decomposition(geom):
    """The input gradient equals, phase by phase, a stride-1 correlation of dy with the phase's rot180
    sub-kernel (backward_phase_codes) and padding Th - 1 - c, placed at rows sh i' + rho (the algorithm of
    the GPU path for strided layers), restated here with Python ints."""
    N, C, H, W, K, R, S, st, pd = geom
    s = si.sign_codes(sum(geom) + 8, (K, C, R, S))
    p = si.shift_codes_uniform(sum(geom) + 8, (K, C, R, S))
    OH, OW = O.conv_out_size(H, R, st, pd), O.conv_out_size(W, S, st, pd)
    dy = si.activations(sum(geom) + 9, (N, K, OH, OW), -(1 << 20), 1 << 20)
    want = O.conv2d_shift_backward_x_acc(dy, s, p, (H, W), (st, st), (pd, pd))
    phases = O.backward_phase_codes(s, p, (st, st))
    got = np.zeros_like(want)
    for rh in range(min(st, H)):
        for rw in range(min(st, W)):
            a, b = (rh + pd) % st, (rw + pd) % st
            if phases[(a, b)] is None:
                continue
            sp, pp = phases[(a, b)]
            th, tw = sp.shape[2], sp.shape[3]
            ph, pw = th - 1 - (rh + pd - a) // st, tw - 1 - (rw + pd - b) // st
            for i in range((H - rh + st - 1) // st):
                for j in range((W - rw + st - 1) // st):
                    for n in range(N):
                        for c in range(C):
                            acc = 0
                            for k in range(K):
                                for t in range(th):
                                    for u in range(tw):
                                        ih, iw = i - ph + t, j - pw + u
                                        if 0 <= ih < OH and 0 <= iw < OW:
                                            acc += int(sp[c, k, t, u]) * (int(dy[n, k, ih, iw]) >> -int(pp[c, k, t, u]))
                            got[n, c, st * i + rh, st * j + rw] = acc
    assert np.array_equal(got, want)
    if st == 1:
        sb, pb = O.backward_codes(s, p)
        assert np.array_equal(phases[(0, 0)][0], sb) and np.array_equal(phases[(0, 0)][1], pb)
