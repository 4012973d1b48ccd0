"""GPU parity of the float variant (bf16 x, tcgen05 tensor cores, fp32 accumulation).

The integer operators are bit-exact; this one rounds its fp32 sums in an
order of the hardware's choosing, so it is held to
|y - y_exact| <= 1e-5 * (sum_k |x W| + |bias|) per output, y_exact from the
float64 oracle.
"""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu
TOL = 1e-5


def _case(seed, M, K, N, lo=-(1 << 20), hi=1 << 20):
    rng = np.random.default_rng(seed)
    bits = si.bf16_bits(rng.uniform(lo, hi, size=(M, K)))
    s = si.sign_codes(seed, (N, K))
    p = si.shift_codes_uniform(seed, (N, K))
    b = (si.bias(seed, N).astype(np.float64) / 65536.0).astype(np.float32)
    return bits, s, p, b


def _run(ds, bits, s, p, b, relu=False):
    x = torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)
    w = ds.pack_shift_weights(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    ds.expand_shift_weights_bf16(w)
    y = ds.linear_shift_bf16(x, w, torch.from_numpy(b).cuda(), relu=relu)
    torch.cuda.synchronize()
    assert ds.ds_bf16_fault_flag() == 0
    return y.cpu().numpy().astype(np.float64), w


def _check(y, bits, s, p, b, relu=False, rows=None):
    xf = si.bits_to_f64(bits if rows is None else bits[rows])
    want = O.linear_shift_float(xf, s, p, b.astype(np.float64))
    scale = O.linear_shift_float_absterms(xf, s, p) + np.abs(b.astype(np.float64))[None, :]
    if relu:
        want = np.maximum(want, 0)
    got = y if rows is None else y[rows]
    err = np.abs(got - want)
    assert np.all(err <= TOL * scale + 1e-30), float((err / np.maximum(scale, 1e-30)).max())


def test_bf16_weight_layout_bitexact(dslib):
    s = si.sign_codes(3, (70, 100))
    p = si.shift_codes_uniform(3, (70, 100))
    w = dslib.pack_shift_weights(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    dslib.expand_shift_weights_bf16(w)
    got = w.bf16.cpu().numpy().view(np.uint16)[:70 * 104].reshape(70, 104)
    assert np.array_equal(got[:, :100], O.weights_bf16_bits(s, p))
    assert not got[:, 100:].any()


@pytest.mark.parametrize("M,K,N", [(128, 64, 256), (128, 256, 256), (200, 136, 300), (1, 8, 1), (300, 520, 260)])
def test_bf16_small_shapes(dslib, M, K, N):
    bits, s, p, b = _case(M * 7 + K + N, M, K, N)
    y, _ = _run(dslib, bits, s, p, b)
    _check(y, bits, s, p, b)


@pytest.mark.parametrize("M,K,N", [(2560, 72, 2560), (1000, 40, 5000)])
def test_bf16_more_tiles_than_sms(dslib, M, K, N):
    """More 128 x 256 output tiles (200, 160) than SMs, ragged edges: every output checked."""
    bits, s, p, b = _case(M + 3 * K + N, M, K, N)
    y, _ = _run(dslib, bits, s, p, b, relu=True)
    _check(y, bits, s, p, b, relu=True)


def test_bf16_relu_and_exact_small_integers(dslib):
    """Small-integer activations with few terms: the fp32 sum is exact, so the result is bit-exact."""
    M, K, N = 130, 64, 257
    rng = np.random.default_rng(1)
    bits = si.bf16_bits(rng.integers(-100, 100, size=(M, K)).astype(np.float64))
    s = si.sign_codes(9, (N, K))
    p = np.zeros((N, K), np.int8)
    b = np.zeros(N, np.float32)
    y, _ = _run(dslib, bits, s, p, b, relu=True)
    want = np.maximum(O.linear_shift_float(si.bits_to_f64(bits), s, p), 0)
    assert np.array_equal(y, want)


@pytest.mark.parametrize("M,K,N", [(1, 8, 1), (300, 520, 260)])
def test_bf16_zero_codes_give_the_bias(dslib, M, K, N):
    """Every sign zero decodes to W = +0, so every product and the fp32 sum are exact zeros: y equals the
    bias exactly (and ReLU of it)."""
    bits, s, p, b = _case(M * 5 + K + N, M, K, N)
    for relu in (False, True):
        y, _ = _run(dslib, bits, np.zeros_like(s), p, b, relu=relu)
        want = np.broadcast_to(b.astype(np.float64), (M, N))
        assert np.array_equal(y, np.maximum(want, 0) if relu else want)


def test_bf16_config4_float_sampled(dslib):
    """The float variant of the large FC shape, 8192 x 4096 x 4096, on sampled rows."""
    M, K, N = 8192, 4096, 4096
    bits, s, p, b = _case(si.SEED_BASE + 44, M, K, N)
    y, _ = _run(dslib, bits, s, p, b)
    rows = np.array([0, 1, 127, 128, 4095, 8191])
    _check(y, bits, s, p, b, rows=rows)


def test_bounded_wait_expiry_is_reported_and_recovered(dslib):
    """Failure detection without a fault: with the wait limit cut to one cycle every launch's first bounded wait
    runs out, so the launch stops issuing, lets its issued copies and MMAs finish, frees its tensor memory and sets
    the fault flag.  The flag reads 1 (and reading clears it); with the default limit restored the next call is
    correct and reads 0."""
    ds = dslib
    bits, s, p, b = _case(77, 256, 512, 512)
    x = torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)
    w = ds.pack_shift_weights(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    ds.expand_shift_weights_bf16(w)
    bd = torch.from_numpy(b).cuda()
    assert ds.ds_bf16_fault_flag() == 0
    try:
        ds.ds_bf16_set_wait_limit(1)
        ds.linear_shift_bf16(x, w, bd)
        torch.cuda.synchronize()
    finally:
        ds.ds_bf16_set_wait_limit(0)
    assert ds.ds_bf16_fault_flag() == 1
    assert ds.ds_bf16_fault_flag() == 0  # read and cleared
    y = ds.linear_shift_bf16(x, w, bd)
    torch.cuda.synchronize()
    assert ds.ds_bf16_fault_flag() == 0
    _check(y.cpu().numpy().astype(np.float64), bits, s, p, b)
