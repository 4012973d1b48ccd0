"""GPU parity of ConvShift against the CPU oracle (bit-exact)."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _run(ds, x, s, p, b, stride, pad, relu=False, residual=None, flags=0, expand=False):
    w = ds.pack_shift_weights(_dev(s), _dev(p), expand=expand)
    amax_io = torch.zeros(2, dtype=torch.int32, device="cuda")
    y = ds.conv2d_shift(_dev(x), w, s.shape[2:], _dev(b) if b is not None else None, stride, pad, relu=relu,
                        residual=_dev(residual) if residual is not None else None, amax_io=amax_io,
                        flags=flags | ds.DS_AMAX_OUT)
    torch.cuda.synchronize()
    return y.cpu().numpy(), amax_io.cpu().numpy().view(np.uint32)


# N, C, H, W, K, R, S, stride, pad
GEOMS = [
    (2, 3, 7, 6, 4, 3, 3, 1, 1),
    (1, 3, 23, 21, 64, 7, 7, 2, 3),     # ResNet stem shape, small image
    (2, 16, 9, 9, 20, 1, 1, 2, 0),      # 1x1 / 2 downsample
    (1, 8, 11, 13, 70, 3, 3, 2, 1),     # 3x3 / 2
    (3, 32, 8, 8, 64, 3, 3, 1, 1),
    (1, 64, 14, 14, 64, 3, 3, 1, 1),
    (2, 5, 5, 5, 3, 5, 5, 1, 0),        # kernel covers the image
    (1, 1, 1, 1, 1, 1, 1, 1, 0),
    (1, 40, 7, 7, 130, 1, 1, 1, 0),
    (2, 48, 8, 8, 72, 1, 1, 1, 0),      # 1x1, OH*OW % 4 == 0: 16-byte epilogue, ragged channel tile
    (1, 20, 16, 16, 36, 1, 1, 2, 0),    # 1x1 / 2, 16-byte epilogue, channels not a multiple of 16
    # stride 2: halo slots start one column early; 8-byte pieces need an even width and an odd padding
    (2, 6, 10, 10, 12, 3, 3, 2, 0),     # even padding: 4-byte copies, 8-pixel groups
    (1, 4, 20, 20, 8, 3, 3, 2, 1),      # 8-byte pieces, 8-pixel groups (OW = 10)
    (2, 5, 28, 30, 9, 7, 7, 2, 3),      # 7x7/2 with 8-byte pieces, OW = 15
    (1, 3, 17, 14, 5, 3, 3, 2, 2),      # padding 2: 4-byte copies
]


@pytest.mark.parametrize("geom", GEOMS)
@pytest.mark.parametrize("flags", [0, 16, 32, 48])  # direct / forced 64-bit / implicit GEMM / both
@pytest.mark.parametrize("expand", [False, True])
def test_conv_bitexact(dslib, geom, flags, expand):
    N, C, H, W, K, R, S, st, pd = geom
    x, s, p, b = si.conv_layer(sum(geom) * 31 + flags, N, C, H, W, K, R, S, -(1 << 20), 1 << 20)
    want = O.conv2d_shift(x, s, p, b, (st, st), (pd, pd))
    got, amax = _run(dslib, x, s, p, b, (st, st), (pd, pd), flags=flags, expand=expand)
    assert np.array_equal(got, want)
    assert amax[1] == O.absmax(want)


@pytest.mark.parametrize("geom", [GEOMS[0], GEOMS[2], GEOMS[4], GEOMS[9], GEOMS[10]])
@pytest.mark.parametrize("flags", [0, 16, 32])
def test_conv_relu_residual(dslib, geom, flags):
    N, C, H, W, K, R, S, st, pd = geom
    x, s, p, b = si.conv_layer(sum(geom) + 5, N, C, H, W, K, R, S, -(1 << 24), 1 << 24)
    OH = (H + 2 * pd - R) // st + 1
    OW = (W + 2 * pd - S) // st + 1
    res = si.activations(99, (N, K, OH, OW), -(1 << 31), 1 << 31)
    want = O.add_relu(O.conv2d_shift(x, s, p, b, (st, st), (pd, pd)), res)
    got, _ = _run(dslib, x, s, p, b, (st, st), (pd, pd), relu=True, residual=res, flags=flags)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("flags", [0, 32])
def test_conv_saturating_inputs(dslib, flags):
    x, s, p, b = si.conv_layer(123, 1, 16, 8, 8, 32, 3, 3, -(1 << 31), 1 << 31, centre=-1)
    want = O.conv2d_shift(x, s, p, b, (1, 1), (1, 1), relu=True)
    assert (np.abs(O.conv2d_shift_acc(x, s, p, b, (1, 1), (1, 1))) > O.INT32_MAX).any()
    got, _ = _run(dslib, x, s, p, b, (1, 1), (1, 1), relu=True, flags=flags)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("geom", [GEOMS[0], GEOMS[1], GEOMS[2]])
@pytest.mark.parametrize("flags", [0, 32])
@pytest.mark.parametrize("expand", [False, True])
def test_conv_degenerate_codes(dslib, geom, flags, expand):
    """The degenerate cases of the method on the conv kernels: every sign zero gives y = sat32(b) at every
    position (padding included); s = -1, p = 0 on x = INT32_MIN makes every in-image term 2^31, outside
    int32, so the 64-bit path is taken (every window here holds at least four such terms: all outputs
    saturate)."""
    N, C, H, W, K, R, S, st, pd = geom
    x, s, p, b = si.conv_layer(sum(geom) * 13 + flags, N, C, H, W, K, R, S, -(1 << 31), 1 << 31)
    OH = (H + 2 * pd - R) // st + 1
    OW = (W + 2 * pd - S) // st + 1
    got, amax = _run(dslib, x, np.zeros_like(s), p, b, (st, st), (pd, pd), flags=flags, expand=expand)
    assert np.array_equal(got, np.broadcast_to(b[None, :, None, None], (N, K, OH, OW)))
    assert amax[1] == O.absmax(b)
    xm = np.full(x.shape, -(1 << 31), np.int32)
    sm = -np.ones(s.shape, np.int8)
    pm = np.zeros(s.shape, np.int8)
    want = O.conv2d_shift(xm, sm, pm, b, (st, st), (pd, pd))
    assert (want == O.INT32_MAX).all()
    got, amax = _run(dslib, xm, sm, pm, b, (st, st), (pd, pd), flags=flags, expand=expand)
    assert np.array_equal(got, want)
    assert amax[1] == O.absmax(want)


# Standalone calls whose grid does not fill the SMs at the batch the layer sweeps time them: the reduction is
# split over the CTAs of a thread-block cluster (1x1: pointwise kernel; 3x3/2: direct kernel)
SPLIT_GEOMS = [
    (32, 256, 14, 14, 512, 1, 1, 2, 0),   # ResNet18 downsample 1x1/2, batch 32
    (32, 128, 28, 28, 256, 1, 1, 2, 0),   # ResNet18 downsample 1x1/2, batch 32
    (8, 2048, 7, 7, 512, 1, 1, 1, 0),     # ResNet50 bottleneck reduce on 7 x 7
    (32, 256, 14, 14, 512, 3, 3, 2, 1),   # ResNet18 conv5_1 3x3/2, batch 32
]


@pytest.mark.parametrize("geom", SPLIT_GEOMS)
@pytest.mark.parametrize("flags,residual", [(0, False), (16, False), (0, True)])
def test_conv_standalone_cluster_split(dslib, geom, flags, residual):
    """Every output of the under-filled layers, with the expanded codes the sweeps use: the 32-bit path, the
    forced 64-bit path, and the residual join with ReLU."""
    N, C, H, W, K, R, S, st, pd = geom
    x, s, p, b = si.conv_layer(sum(geom) * 17 + flags, N, C, H, W, K, R, S, 0, 1 << 20, si.layer_centre(C, R, S))
    OH = (H + 2 * pd - R) // st + 1
    OW = (W + 2 * pd - S) // st + 1
    res = si.activations(77, (N, K, OH, OW), -(1 << 31), 1 << 31) if residual else None
    acc = O.conv2d_shift(x, s, p, b, (st, st), (pd, pd))
    want = O.add_relu(acc, res) if residual else np.maximum(acc, 0)
    got, amax = _run(dslib, x, s, p, b, (st, st), (pd, pd), relu=True, residual=res, flags=flags, expand=True)
    assert np.array_equal(got, want)
    assert amax[1] == O.absmax(want)


# ResNet18 / ResNet50 / VGG16 layer shapes at a small batch, both kernels
NET_GEOMS = [
    (1, 3, 224, 224, 64, 7, 7, 2, 3),    # stem 7x7/2
    (2, 64, 56, 56, 64, 3, 3, 1, 1),     # conv2_x
    (2, 64, 56, 56, 128, 3, 3, 2, 1),    # conv3_1 3x3/2
    (2, 64, 56, 56, 128, 1, 1, 2, 0),    # downsample 1x1/2
    (2, 128, 28, 28, 128, 3, 3, 1, 1),
    (2, 256, 14, 14, 256, 3, 3, 1, 1),
    (2, 512, 7, 7, 512, 3, 3, 1, 1),
    (2, 64, 56, 56, 256, 1, 1, 1, 0),    # bottleneck expand
    (1, 3, 32, 32, 64, 3, 3, 1, 1),      # VGG first conv (small image)
]


@pytest.mark.parametrize("geom", NET_GEOMS)
def test_conv_network_layer_shapes(dslib, geom):
    N, C, H, W, K, R, S, st, pd = geom
    x, s, p, b = si.conv_layer(sum(geom) * 7, N, C, H, W, K, R, S, 0, 1 << 20)
    want = O.conv2d_shift(x, s, p, b, (st, st), (pd, pd), relu=True)
    for flags, expand in ((0, False), (0, True), (32, False), (16, True)):
        got, _ = _run(dslib, x, s, p, b, (st, st), (pd, pd), relu=True, flags=flags, expand=expand)
        assert np.array_equal(got, want), (flags, expand)


@pytest.mark.parametrize("expand", [False, True])
def test_conv_config2_two_images_full(dslib, expand):
    """The ResNet18 conv2_x layer (64 -> 64, 56 x 56, 3x3/1/1) on two images, every output."""
    x, s, p, b = si.config2(N=2)
    want = O.conv2d_shift(x, s, p, b, (1, 1), (1, 1))
    got, _ = _run(dslib, x, s, p, b, (1, 1), (1, 1), expand=expand)
    assert np.array_equal(got, want)


_CONFIG2_ORACLE = {}


def _config2_oracle(x, s, p, b):
    """The oracle on the whole N = 32 batch (about 15 s), computed once per session."""
    if "y" not in _CONFIG2_ORACLE:
        _CONFIG2_ORACLE["y"] = O.conv2d_shift(x, s, p, b, (1, 1), (1, 1))
    return _CONFIG2_ORACLE["y"]


@pytest.mark.parametrize("expand", [False, True])
def test_conv_config2_full_batch_every_output(dslib, expand):
    """The full N = 32 launch as the benchmark times it (the expanded layout; the packed blob too): every one
    of the 6.4 M outputs against the oracle."""
    x, s, p, b = si.config2()
    got, _ = _run(dslib, x, s, p, b, (1, 1), (1, 1), expand=expand)
    assert np.array_equal(got, _config2_oracle(x, s, p, b))
