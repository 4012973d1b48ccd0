"""GPU parity of the weight-specialised ConvShift (codes compiled into the kernel at run time) against the CPU
oracle and the generic ConvShift kernels, bit-exact.  Each specialisation compiles a kernel with NVRTC (seconds),
so the cases are few and small, plus VGG16's first layer (C = 3, 64 channels, 3x3) at four images."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _run(ds, h, x, b, res, N, C, H, W, K, OH, OW, flags):
    y = torch.full((N, K, OH, OW), 7, dtype=torch.int32, device="cuda")
    amax_io = torch.zeros(2, dtype=torch.int32, device="cuda")
    ds.ds_conv2d_shift_specialized(h, _dev(x), _dev(b) if b is not None else None,
                                   _dev(res) if res is not None else None, y, N, H, W, flags | ds.DS_AMAX_OUT,
                                   amax_io)
    torch.cuda.synchronize()
    return y.cpu().numpy(), amax_io.cpu().numpy().view(np.uint32)


# N, C, H, W, K, R (= S), stride, pad
GEOMS = [
    (2, 3, 17, 19, 8, 3, 1, 1),      # VGG-like 3x3/1, ragged width and height
    (1, 3, 30, 28, 16, 5, 2, 2),     # 5x5/2
    (2, 4, 9, 23, 5, 1, 1, 0),       # 1x1, a ragged channel group
    (1, 2, 13, 11, 12, 7, 2, 3),     # 7x7/2 stem-like, small
]


@pytest.mark.parametrize("geom", GEOMS)
def test_specialized_matches_oracle_and_generic(dslib, geom):
    ds = dslib
    N, C, H, W, K, R, st, pd = geom
    x, s, p, b = si.conv_layer(sum(geom) * 41, N, C, H, W, K, R, R, -(1 << 20), 1 << 20, -4)
    OH = (H + 2 * pd - R) // st + 1
    OW = (W + 2 * pd - R) // st + 1
    res = si.activations(sum(geom), (N, K, OH, OW), -(1 << 30), 1 << 30)
    h = ds.ds_specialize_conv2d_shift(s, p, K, C, R, R, st, pd)
    try:
        acc = O.conv2d_shift(x, s, p, b, (st, st), (pd, pd))
        # the 32-bit path (the bound holds for these inputs), with and without the fused epilogue
        got, amax = _run(ds, h, x, b, None, N, C, H, W, K, OH, OW, 0)
        assert np.array_equal(got, acc)
        assert amax[1] == O.absmax(acc)
        want = O.add_relu(acc, res)
        got, _ = _run(ds, h, x, b, res, N, C, H, W, K, OH, OW, ds.DS_RELU | ds.DS_RESIDUAL)
        assert np.array_equal(got, want)
        # the 64-bit path, forced
        got, _ = _run(ds, h, x, b, None, N, C, H, W, K, OH, OW, ds.DS_FORCE_INT64 | ds.DS_RELU)
        assert np.array_equal(got, np.maximum(acc, 0))
        # the generic kernels on the same layer
        w = ds.pack_shift_weights(_dev(s), _dev(p))
        gen = ds.conv2d_shift(_dev(x), w, (R, R), _dev(b), (st, st), (pd, pd),
                              amax_io=torch.zeros(2, dtype=torch.int32, device="cuda"))
        assert np.array_equal(gen.cpu().numpy(), acc)
    finally:
        ds.ds_specialized_destroy(h)


def test_specialized_saturating_inputs_take_the_64bit_path(dslib):
    """Full-range inputs with many p = 0 weights: the bound fails, the CTA sums in 64 bits and saturates."""
    ds = dslib
    N, C, H, W, K, R = 1, 3, 12, 15, 8, 3
    x, s, p, b = si.conv_layer(902, N, C, H, W, K, R, R, -(1 << 31), 1 << 31, -1)
    acc = O.conv2d_shift_acc(x, s, p, b, (1, 1), (1, 1))
    assert (np.abs(acc) > O.INT32_MAX).any()
    h = ds.ds_specialize_conv2d_shift(s, p, K, C, R, R, 1, 1)
    try:
        got, _ = _run(ds, h, x, b, None, N, C, H, W, K, H, W, 0)
        assert np.array_equal(got, O.conv2d_shift(x, s, p, b, (1, 1), (1, 1)))
    finally:
        ds.ds_specialized_destroy(h)


def test_specialized_zero_codes_give_the_bias(dslib):
    """Every weight zero: the generated kernel has no terms at all, and every output is its bias."""
    ds = dslib
    N, C, H, W, K, R = 2, 3, 10, 9, 6, 3
    x, s, p, b = si.conv_layer(903, N, C, H, W, K, R, R)
    h = ds.ds_specialize_conv2d_shift(np.zeros_like(s), p, K, C, R, R, 1, 1)
    try:
        got, _ = _run(ds, h, x, b, None, N, C, H, W, K, H, W, 0)
        assert np.array_equal(got, np.broadcast_to(b[None, :, None, None], got.shape))
    finally:
        ds.ds_specialized_destroy(h)


def test_specialized_vgg16_first_layer(dslib):
    """VGG16's first conv (3 -> 64, 3x3/1/1) at 224 x 224, the layer specialisation is meant for: every output of
    four images against the oracle."""
    ds = dslib
    x, s, p, b = si.conv_layer(904, 4, 3, 224, 224, 64, 3, 3, -(1 << 17), 1 << 17, si.layer_centre(3, 3, 3))
    h = ds.ds_specialize_conv2d_shift(s, p, 64, 3, 3, 3, 1, 1)
    try:
        got, _ = _run(ds, h, x, b, None, 4, 3, 224, 224, 64, 224, 224, ds.DS_RELU)
        assert np.array_equal(got, O.conv2d_shift(x, s, p, b, (1, 1), (1, 1), relu=True))
    finally:
        ds.ds_specialized_destroy(h)


def test_specialized_many_images_walk_tiles(dslib):
    """Many small images (three row tiles each, the last one ragged) with a residual and no ReLU: a grid of
    thousands of CTAs, the residual join saturating, max|y| over the joined outputs."""
    ds = dslib
    N, C, H, W, K, R = 640, 2, 40, 22, 8, 3
    x, s, p, b = si.conv_layer(905, N, C, H, W, K, R, R, -(1 << 20), 1 << 20, -3)
    res = si.activations(906, (N, K, H, W), -(1 << 30), 1 << 30)
    h = ds.ds_specialize_conv2d_shift(s, p, K, C, R, R, 1, 1)
    try:
        got, amax = _run(ds, h, x, b, res, N, C, H, W, K, H, W, ds.DS_RESIDUAL)
        # the residual join without ReLU: one saturation of the layer's output plus the residual
        want = O.sat32(O.conv2d_shift(x, s, p, b, (1, 1), (1, 1)).astype(np.int64) + res.astype(np.int64))
        assert amax[1] == O.absmax(want)
        assert np.array_equal(got, want)
    finally:
        ds.ds_specialized_destroy(h)
