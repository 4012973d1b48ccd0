"""GPU parity of the input gradient (Eq. 7 and its footnote) of LinearShift and ConvShift, and of the
input-gradient code packing, against the CPU oracle (bit-exact)."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


@pytest.mark.parametrize("dims,stride", [((1, 1, 1, 1), 1), ((5, 3, 3, 3), 1), ((64, 33, 1, 1), 1),
                                         ((7, 40, 7, 7), 2), ((3, 70, 3, 2), 2), ((6, 9, 1, 1), 2),
                                         ((4, 5, 5, 3), 3)])
def test_pack_backward_phase_blobs_bitexact(dslib, dims, stride):
    K, C, R, S = dims
    s = si.sign_codes(sum(dims), dims)
    p = si.shift_codes_uniform(sum(dims), dims)
    w = dslib.pack_shift_weights_backward(_dev(s), _dev(p), (stride, stride))
    blob = w.blob.cpu().numpy()
    for (a, b), codes in O.backward_phase_codes(s, p, (stride, stride)).items():
        d = w.desc[a * stride + b]
        assert d.n_out == C
        if codes is None:
            assert d.k_red == 0 and not d.packed
            continue
        sp, pp = codes
        assert d.k_red == sp[0].size
        want = O.pack_planes6(sp.reshape(C, -1), pp.reshape(C, -1))
        off = d.packed - w.blob.data_ptr()
        assert np.array_equal(blob[off:off + want.size], want)


FC_SHAPES = [(1, 1, 1), (3, 7, 5), (64, 784, 512), (33, 130, 65), (200, 64, 1000)]


@pytest.mark.parametrize("M,K,N", FC_SHAPES)
@pytest.mark.parametrize("flags", [0, 16])
@pytest.mark.parametrize("expand", [False, True])
def test_linear_backward_x_bitexact(dslib, M, K, N, flags, expand):
    s = si.sign_codes(M + K + N, (N, K))
    p = si.shift_codes_uniform(M + K + N, (N, K))
    dy = si.activations(M * 7 + N, (M, N), -(1 << 22), 1 << 22)
    w = dslib.pack_shift_weights_backward(_dev(s), _dev(p), expand=expand)
    dx = torch.empty((M, K), dtype=torch.int32, device="cuda")
    amax = torch.zeros(2, dtype=torch.int32, device="cuda")
    dslib.ds_linear_shift_backward_x(_dev(dy), w.desc[0], dx, M, K, N, flags | dslib.DS_AMAX_OUT, amax)
    want = O.linear_shift_backward_x(dy, s, p)
    assert np.array_equal(dx.cpu().numpy(), want)
    assert amax.cpu().numpy().view(np.uint32)[1] == O.absmax(want)


def test_linear_backward_x_saturates(dslib):
    M, K, N = 9, 40, 300
    s = si.sign_codes(1, (N, K))
    p = np.zeros((N, K), np.int8)
    dy = si.activations(2, (M, N), -(1 << 31), 1 << 31)
    w = dslib.pack_shift_weights_backward(_dev(s), _dev(p))
    dx = torch.empty((M, K), dtype=torch.int32, device="cuda")
    amax = torch.zeros(2, dtype=torch.int32, device="cuda")
    dslib.ds_linear_shift_backward_x(_dev(dy), w.desc[0], dx, M, K, N, 0, amax)
    want = O.linear_shift_backward_x(dy, s, p)
    assert (np.abs(O.linear_shift_backward_x_acc(dy, s, p)) > O.INT32_MAX).any()
    assert np.array_equal(dx.cpu().numpy(), want)


def _degenerate_cases(seed, code_shape, dy_shape, bwd):
    """(s, p, dy, want) for the degenerate codes: every sign zero (dX = 0), and s = -1, p = 0 on dY = INT32_MIN,
    where every term is 2^31 (outside int32): dX saturates wherever a term reaches it."""
    zero = (np.zeros(code_shape, np.int8), si.shift_codes_uniform(seed, code_shape),
            si.activations(seed + 1, dy_shape, -(1 << 31), 1 << 31))
    edge = (-np.ones(code_shape, np.int8), np.zeros(code_shape, np.int8), np.full(dy_shape, -(1 << 31), np.int32))
    out = []
    for s, p, dy in (zero, edge):
        out.append((s, p, dy, bwd(dy, s, p)))
    assert not out[0][3].any()
    assert out[1][3].max() == O.INT32_MAX and out[1][3].min() >= 0
    return out


@pytest.mark.parametrize("M,K,N", [(1, 1, 1), (33, 130, 65), (200, 64, 1000)])
def test_linear_backward_x_degenerate_codes(dslib, M, K, N):
    for s, p, dy, want in _degenerate_cases(M + K + N, (N, K), (M, N), O.linear_shift_backward_x):
        w = dslib.pack_shift_weights_backward(_dev(s), _dev(p))
        dx = torch.empty((M, K), dtype=torch.int32, device="cuda")
        amax = torch.zeros(2, dtype=torch.int32, device="cuda")
        dslib.ds_linear_shift_backward_x(_dev(dy), w.desc[0], dx, M, K, N, dslib.DS_AMAX_OUT, amax)
        assert np.array_equal(dx.cpu().numpy(), want)
        assert amax.cpu().numpy().view(np.uint32)[1] == O.absmax(want)


# N, C, H, W, K, R, S, stride, pad
CONV_GEOMS = [
    (2, 3, 7, 6, 4, 3, 3, 1, 1),
    (2, 3, 7, 6, 4, 3, 3, 2, 1),
    (1, 3, 23, 21, 16, 7, 7, 2, 3),     # stem-shaped
    (2, 16, 9, 9, 20, 1, 1, 2, 0),      # 1x1 / 2 downsample
    (1, 8, 11, 13, 70, 3, 3, 2, 1),
    (3, 32, 8, 8, 64, 3, 3, 1, 1),
    (1, 40, 7, 7, 130, 1, 1, 1, 0),
    (1, 5, 6, 6, 3, 1, 1, 1, 1),        # pad > R - 1: the gather path even at stride 1
    (2, 4, 10, 9, 6, 5, 3, 2, 2),       # non-square kernel
    (1, 6, 11, 10, 5, 5, 5, 3, 2),      # stride 3
    (2, 7, 9, 9, 4, 3, 3, 2, 0),        # stride 2, no padding: (9 - 3) / 2 whole steps, every row is reached
    (2, 7, 10, 10, 4, 3, 3, 2, 0),      # stride 2, no padding: the last input row and column get no gradient
]


@pytest.mark.parametrize("geom", CONV_GEOMS)
@pytest.mark.parametrize("flags", [0, 16, 32])  # default / forced 64-bit / forced gather path
@pytest.mark.parametrize("expand", [False, True])
def test_conv_backward_x_bitexact(dslib, geom, flags, expand):
    N, C, H, W, K, R, S, st, pd = geom
    s = si.sign_codes(sum(geom) * 3, (K, C, R, S))
    p = si.shift_codes_uniform(sum(geom) * 3, (K, C, R, S))
    OH, OW = O.conv_out_size(H, R, st, pd), O.conv_out_size(W, S, st, pd)
    dy = si.activations(sum(geom) + flags, (N, K, OH, OW), -(1 << 22), 1 << 22)
    w = dslib.pack_shift_weights_backward(_dev(s), _dev(p), (st, st), expand=expand)
    dx = torch.empty((N, C, H, W), dtype=torch.int32, device="cuda")
    amax = torch.zeros(2, dtype=torch.int32, device="cuda")
    dslib.ds_conv2d_shift_backward_x(_dev(dy), w.desc, dx, N, C, H, W, K, R, S, st, st, pd, pd,
                                     flags | dslib.DS_AMAX_OUT, amax)
    want = O.conv2d_shift_backward_x(dy, s, p, (H, W), (st, st), (pd, pd))
    assert np.array_equal(dx.cpu().numpy(), want)
    assert amax.cpu().numpy().view(np.uint32)[1] == O.absmax(want)


@pytest.mark.parametrize("geom", [CONV_GEOMS[0], CONV_GEOMS[1], CONV_GEOMS[2], CONV_GEOMS[-2], CONV_GEOMS[-1]])
@pytest.mark.parametrize("flags", [0, 32])  # default / forced gather path
def test_conv_backward_x_degenerate_codes(dslib, geom, flags):
    """Zero codes give dX = 0 everywhere; s = -1, p = 0 on dY = INT32_MIN saturates every position a tap
    reaches and leaves 0 where none does (stride 2 without padding: the last row and column)."""
    N, C, H, W, K, R, S, st, pd = geom
    OH, OW = O.conv_out_size(H, R, st, pd), O.conv_out_size(W, S, st, pd)
    bwd = lambda dy, s, p: O.conv2d_shift_backward_x(dy, s, p, (H, W), (st, st), (pd, pd))
    for s, p, dy, want in _degenerate_cases(sum(geom) + flags, (K, C, R, S), (N, K, OH, OW), bwd):
        w = dslib.pack_shift_weights_backward(_dev(s), _dev(p), (st, st))
        dx = torch.empty((N, C, H, W), dtype=torch.int32, device="cuda")
        amax = torch.zeros(2, dtype=torch.int32, device="cuda")
        dslib.ds_conv2d_shift_backward_x(_dev(dy), w.desc, dx, N, C, H, W, K, R, S, st, st, pd, pd,
                                         flags | dslib.DS_AMAX_OUT, amax)
        assert np.array_equal(dx.cpu().numpy(), want)
        assert amax.cpu().numpy().view(np.uint32)[1] == O.absmax(want)


@pytest.mark.parametrize("geom", [(2, 64, 56, 56, 64, 3, 3, 1, 1), (2, 64, 56, 56, 128, 1, 1, 2, 0),
                                  (2, 64, 56, 56, 128, 3, 3, 2, 1), (2, 3, 224, 224, 64, 7, 7, 2, 3)])
def test_conv_backward_x_resnet_layers(dslib, geom):
    """ResNet18 layer shapes (conv2_x, the 1x1/2 and 3x3/2 transitions, the 7x7/2 stem whose 3-column gradient
    runs the narrow kernel), 2 images, every output."""
    N, C, H, W, K, R, S, st, pd = geom
    s = si.sign_codes(sum(geom), (K, C, R, S))
    p = si.shift_codes_geometric(sum(geom), (K, C, R, S), -6)
    OH, OW = O.conv_out_size(H, R, st, pd), O.conv_out_size(W, S, st, pd)
    dy = si.activations(sum(geom) + 1, (N, K, OH, OW), -(1 << 20), 1 << 20)
    w = dslib.pack_shift_weights_backward(_dev(s), _dev(p), (st, st), expand=True)
    dx = torch.empty((N, C, H, W), dtype=torch.int32, device="cuda")
    amax = torch.zeros(2, dtype=torch.int32, device="cuda")
    dslib.ds_conv2d_shift_backward_x(_dev(dy), w.desc, dx, N, C, H, W, K, R, S, st, st, pd, pd, 0, amax)
    assert np.array_equal(dx.cpu().numpy(), O.conv2d_shift_backward_x(dy, s, p, (H, W), (st, st), (pd, pd)))
