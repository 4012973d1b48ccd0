"""GPU parity of the float -> code quantizer (DeepShift-Q, Eq. 4-6) and the float -> Q16.16 rounding
(Sec. 4) against the CPU oracle (bit-exact)."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu

SPECIALS = np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 1e-45, -1e-40, 2.0 ** -126, 1.0, -1.0, 0.5, 2.0 ** -15,
                     2.0 ** -16, 1.5, 3.0, 1e30, -1e30] +
                    [np.float32(2.0 ** (n + 0.5)) for n in range(-17, 2)] +
                    [np.nextafter(np.float32(2.0 ** (n + 0.5)), np.float32(0)) for n in range(-17, 2)], np.float32)


def _weights(seed, n):
    w = si.float_weights(seed, (n,), -20, 2)
    w[: min(n, SPECIALS.size)] = SPECIALS[: min(n, SPECIALS.size)]
    return w


@pytest.mark.parametrize("n", [1, 3, 4, 5, 37, 1000, 4099, (1 << 20) + 3])
@pytest.mark.parametrize("p_min", [-15, -14, -8])
def test_quantize_weights_bitexact(dslib, n, p_min):
    w = _weights(n + 7 * p_min, n)
    s, p = dslib.quantize_shift_weights(torch.from_numpy(w).cuda(), p_min)
    ws, wp = O.quantize_weights(w, p_min)
    assert np.array_equal(s.cpu().numpy(), ws)
    assert np.array_equal(p.cpu().numpy(), wp)


@pytest.mark.parametrize("offset", [1, 2, 3])
def test_quantize_weights_unaligned_views(dslib, offset):
    """Views that start off a 16-byte boundary take the scalar path."""
    w = _weights(11, 2051)
    wd = torch.from_numpy(w).cuda()[offset:]
    s = torch.empty(wd.numel() + 1, dtype=torch.int8, device="cuda")[1:]
    p = torch.empty(wd.numel() + 3, dtype=torch.int8, device="cuda")[3:]
    dslib.ds_quantize_shift_weights(wd, wd.numel(), -15, s, p)
    ws, wp = O.quantize_weights(w[offset:])
    assert np.array_equal(s.cpu().numpy(), ws)
    assert np.array_equal(p.cpu().numpy(), wp)


def test_quantize_weights_vgg16_fc1_full_size(dslib):
    """The 4096 x 25088 weight matrix of VGG16's first FC layer (103 M weights), every code checked."""
    w = si.float_weights(12, (4096, 25088), -18, 1)
    s, p = dslib.quantize_shift_weights(torch.from_numpy(w).cuda())
    ws, wp = O.quantize_weights(w)
    assert np.array_equal(s.cpu().numpy(), ws)
    assert np.array_equal(p.cpu().numpy(), wp)


@pytest.mark.parametrize("n", [1, 2, 4, 7, 1000, 4101, (1 << 20) + 1])
def test_quantize_q16_bitexact(dslib, n):
    x = si.float_activations(100 + n, (n,), -20, 17)
    sp = np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 32768.0, -32768.0, -32768.5, 0.5 / 65536, 1.5 / 65536,
                   -2.5 / 65536, 1e-45], np.float32)
    x[: min(n, sp.size)] = sp[: min(n, sp.size)]
    q = dslib.quantize_q16(torch.from_numpy(x).cuda())
    assert np.array_equal(q.cpu().numpy(), O.quantize_activations(x))


def test_quantize_q16_unaligned_view(dslib):
    x = si.float_activations(5, (1031,), -20, 17)
    xd = torch.from_numpy(x).cuda()[1:]
    q = torch.empty(xd.numel() + 1, dtype=torch.int32, device="cuda")[1:]
    dslib.ds_quantize_q16(xd, xd.numel(), q)
    assert np.array_equal(q.cpu().numpy(), O.quantize_activations(x[1:]))


def test_float_layer_end_to_end(dslib):
    """Float weights, input and bias -> codes and Q16.16 on the GPU -> pack -> LinearShift: equals the
    oracle's LinearShift of the oracle's conversions."""
    M, K, N = 48, 300, 70
    w = si.float_weights(21, (N, K), -12, -2)
    x = si.float_activations(22, (M, K), -6, 6)
    b = si.float_activations(23, (N,), -8, 2)
    s, p = dslib.quantize_shift_weights(torch.from_numpy(w).cuda())
    xq = dslib.quantize_q16(torch.from_numpy(x).cuda())
    bq = dslib.quantize_q16(torch.from_numpy(b).cuda())
    packed = dslib.pack_shift_weights(s, p)
    y = dslib.linear_shift(xq, packed, bq, relu=True).cpu().numpy()
    ws, wp = O.quantize_weights(w)
    want = O.linear_shift(O.quantize_activations(x), ws, wp, O.quantize_activations(b), relu=True)
    assert np.array_equal(y, want)
