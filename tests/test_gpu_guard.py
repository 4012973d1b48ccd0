"""Guard bands around every buffer a call touches: evidence on the GPU that no kernel reads or writes outside its
arguments (compute-sanitizer is not available on this machine).

Each buffer sits inside a larger allocation whose margins (16 KB on each side) hold a canary.  Output margins must
be unchanged after the call, so nothing wrote past an output.  Input margins hold large values (0x40000000 in the
activations, codes that are not valid codes in the weight blobs), so a read past an input would change the
results; every result is compared bit for bit with the CPU oracle.  The paths covered are those of the other
parity tests: direct, pointwise, cluster-split and implicit-GEMM convolutions, both FC kernels, both code layouts,
the 64-bit accumulators, the input gradient, the chained forward with its workspace, the pools, the conversion
kernels, the bf16 tensor-core kernel and the run-time compiled conv."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu

G = 16384  # margin in bytes on each side of a buffer
X_CANARY = 0x40000000
Y_CANARY = 0x5A5A5A5A


class Guarded:
    """A flat device buffer of n elements with G bytes of canary on each side."""

    def __init__(self, n, dtype, canary, data=None):
        esz = torch.tensor([], dtype=dtype).element_size()
        self.g = G // esz
        self.n = n
        self.canary = canary
        self.full = torch.full((n + 2 * self.g,), canary, dtype=dtype, device="cuda")
        self.view = self.full[self.g:self.g + n]
        if data is not None:
            self.view.copy_(torch.from_numpy(np.ascontiguousarray(data).reshape(-1)).to("cuda"))

    def margins_intact(self):
        torch.cuda.synchronize()
        c = torch.tensor(self.canary, dtype=self.full.dtype, device="cuda")
        return bool((self.full[:self.g] == c).all()) and bool((self.full[self.g + self.n:] == c).all())

    def numpy(self, shape):
        return self.view.cpu().numpy().reshape(shape)


def _weights(ds, s, p, expand):
    """Packs codes into a guarded blob (and expands them into a guarded buffer); returns the descriptor and the
    guarded buffers.  The blob margins hold 0xFF bytes: as codes, every nonzero weight with a large shift."""
    n_out, k_red = s.shape[0], int(np.prod(s.shape[1:]))
    nb = ds.ds_packed_weight_bytes(n_out, k_red)
    blob = Guarded(nb, torch.uint8, 0xFF)
    sd = torch.from_numpy(np.ascontiguousarray(s.reshape(n_out, k_red))).cuda()
    pd = torch.from_numpy(np.ascontiguousarray(p.reshape(n_out, k_red))).cuda()
    desc = ds.ds_pack_shift_weights(sd, pd, n_out, k_red, blob.view, nb)
    assert blob.margins_intact()
    bufs = [blob]
    if expand:
        eb = ds.ds_expanded_weight_bytes(n_out, k_red)
        exp = Guarded(eb // 4, torch.int32, 0x7F7F7F7F)
        ds.ds_expand_shift_weights(desc, exp.view, eb)
        assert exp.margins_intact()
        bufs.append(exp)
    return desc, bufs


# N, C, H, W, K, R, stride, pad, flags
CONVS = [
    (2, 5, 13, 17, 9, 3, 1, 1, 0),          # direct 3x3/1, ragged
    (2, 6, 15, 14, 10, 3, 2, 1, 0),         # direct 3x3/2
    (1, 3, 30, 30, 8, 7, 2, 3, 0),          # 7x7/2 stem
    (2, 16, 9, 11, 24, 1, 1, 0, 0),         # pointwise 1x1/1
    (2, 16, 14, 14, 32, 1, 2, 0, 0),        # pointwise 1x1/2
    (1, 64, 7, 7, 64, 3, 1, 1, 0),          # under-filled grid: cluster split
    (1, 256, 7, 7, 128, 1, 1, 0, 0),        # under-filled 1x1: cluster split
    (2, 5, 13, 17, 9, 3, 1, 1, 32),         # implicit GEMM (DS_CONV_IM2COL)
    (2, 5, 11, 12, 7, 5, 2, 2, 32),         # implicit GEMM, 5x5/2
    (2, 5, 13, 17, 9, 3, 1, 1, 16),         # forced 64-bit accumulators
]


@pytest.mark.parametrize("expand", [True, False])
@pytest.mark.parametrize("geom", CONVS)
def test_conv_stays_inside_its_buffers(dslib, geom, expand):
    ds = dslib
    N, C, H, W, K, R, st, pd, flags = geom
    x, s, p, b = si.conv_layer(sum(geom) + 3, N, C, H, W, K, R, R, -(1 << 20), 1 << 20, -5)
    OH, OW = (H + 2 * pd - R) // st + 1, (W + 2 * pd - R) // st + 1
    res = si.activations(sum(geom) + 4, (N, K, OH, OW), -(1 << 30), 1 << 30)
    desc, wbufs = _weights(ds, s, p, expand)
    xg = Guarded(x.size, torch.int32, X_CANARY, x)
    bg = Guarded(K, torch.int32, X_CANARY, b)
    rg = Guarded(res.size, torch.int32, X_CANARY, res)
    yg = Guarded(N * K * OH * OW, torch.int32, Y_CANARY)
    ag = Guarded(2, torch.int32, Y_CANARY, np.zeros(2, np.int32))
    ds.ds_conv2d_shift(xg.view, desc, bg.view, rg.view, yg.view, N, C, H, W, K, R, R, st, st, pd, pd,
                       flags | ds.DS_RESIDUAL | ds.DS_RELU | ds.DS_AMAX_OUT, ag.view)
    for g in [xg, bg, rg, yg, ag] + wbufs:
        assert g.margins_intact()
    want = O.add_relu(O.conv2d_shift(x, s, p, b, (st, st), (pd, pd)), res)
    assert np.array_equal(yg.numpy(want.shape), want)
    assert ag.numpy(2).view(np.uint32)[1] == O.absmax(want)


# M, K, N, flags
FCS = [(5, 300, 70, 0), (64, 784, 512, 0), (700, 200, 130, 0), (37, 333, 65, 16), (300, 129, 67, 16)]


@pytest.mark.parametrize("expand", [True, False])
@pytest.mark.parametrize("shape", FCS)
def test_linear_stays_inside_its_buffers(dslib, shape, expand):
    ds = dslib
    M, K, N, flags = shape
    x, s, p, b = si.fc_layer(sum(shape), M, K, N, -(1 << 24), 1 << 24)
    desc, wbufs = _weights(ds, s, p, expand)
    xg = Guarded(x.size, torch.int32, X_CANARY, x)
    bg = Guarded(N, torch.int32, X_CANARY, b)
    yg = Guarded(M * N, torch.int32, Y_CANARY)
    ag = Guarded(2, torch.int32, Y_CANARY, np.zeros(2, np.int32))
    ds.ds_linear_shift(xg.view, desc, bg.view, yg.view, M, K, N, flags | ds.DS_AMAX_OUT, ag.view)
    for g in [xg, bg, yg, ag] + wbufs:
        assert g.margins_intact()
    want = O.linear_shift(x, s, p, b)
    assert np.array_equal(yg.numpy(want.shape), want)


@pytest.mark.parametrize("geom", [(2, 6, 11, 12, 8, 3, 2, 1), (2, 20, 11, 12, 8, 3, 2, 1), (1, 3, 23, 21, 16, 7, 2, 3)])
def test_conv_input_gradient_stays_inside_its_buffers(dslib, geom):
    """Stride 2: the tap phases with their own descriptors into one guarded blob; 6 and 3 gradient columns run
    the narrow kernel, 20 the implicit GEMMs of all phases in one launch."""
    ds = dslib
    N, C, H, W, K, R, st, pd = geom
    _, s, p, _ = si.conv_layer(77, N, C, H, W, K, R, R)
    OH, OW = (H + 2 * pd - R) // st + 1, (W + 2 * pd - R) // st + 1
    dy = si.activations(78, (N, K, OH, OW), -(1 << 20), 1 << 20)
    nb = ds.ds_packed_weight_bytes_backward(K, C, R, R, st, st)
    blob = Guarded(nb, torch.uint8, 0xFF)
    descs = ds.ds_pack_shift_weights_backward(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda(), K, C, R, R,
                                              st, st, blob.view, nb)
    dyg = Guarded(dy.size, torch.int32, X_CANARY, dy)
    dxg = Guarded(N * C * H * W, torch.int32, Y_CANARY)
    ds.ds_conv2d_shift_backward_x(dyg.view, descs, dxg.view, N, C, H, W, K, R, R, st, st, pd, pd)
    for g in (blob, dyg, dxg):
        assert g.margins_intact()
    want = O.conv2d_shift_backward_x(dy, s, p, (H, W), (st, st), (pd, pd))
    assert np.array_equal(dxg.numpy(want.shape), want)


def test_linear_input_gradient_stays_inside_its_buffers(dslib):
    ds = dslib
    M, K, N = 33, 150, 70
    _, s, p, _ = si.fc_layer(79, M, K, N, 0, 1)
    dy = si.activations(80, (M, N), -(1 << 20), 1 << 20)
    nb = ds.ds_packed_weight_bytes_backward(N, K, 1, 1)
    blob = Guarded(nb, torch.uint8, 0xFF)
    descs = ds.ds_pack_shift_weights_backward(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda(), N, K, 1, 1,
                                              1, 1, blob.view, nb)
    dyg = Guarded(dy.size, torch.int32, X_CANARY, dy)
    dxg = Guarded(M * K, torch.int32, Y_CANARY)
    ds.ds_linear_shift_backward_x(dyg.view, descs[0], dxg.view, M, K, N)
    for g in (blob, dyg, dxg):
        assert g.margins_intact()
    want = O.linear_shift_backward_x(dy, s, p)
    assert np.array_equal(dxg.numpy(want.shape), want)


def test_chained_forward_stays_inside_its_workspace(dslib):
    """ResNet18 at 64 x 64, two images: every layer's slot, the split scratch and the max|x| words live in one
    guarded workspace; the pools, the split finalize and the FC run between them."""
    ds = dslib
    from oracle import networks as ON
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet18", 64, 64)
    params = si.network_params(prog[1], 101)
    x = si.image_batch(11, 2, 3, 64, 64)
    net = PN.ShiftNetwork(prog[0], params, batch=2)
    nbytes = net.workspace.numel()
    wsg = Guarded(nbytes, torch.uint8, 0xA5)
    xg = Guarded(x.size, torch.int32, X_CANARY, x)
    yg = Guarded(2 * 1000, torch.int32, Y_CANARY)
    ds.ds_shift_forward(net.layers, len(net.specs), xg.view, yg.view, wsg.view, nbytes, 2)
    for g in (wsg, xg, yg):
        assert g.margins_intact()
    assert np.array_equal(yg.numpy((2, 1000)), ON.resnet_forward(x, params, "resnet18"))


def test_conversion_kernels_stay_inside_their_buffers(dslib):
    ds = dslib
    n = 10007
    rng = np.random.default_rng(5)
    wf = (rng.standard_normal(n) * 0.05).astype(np.float32)
    wg = Guarded(n, torch.float32, float("nan"), wf)
    sg = Guarded(n, torch.int8, 0x55)
    pg = Guarded(n, torch.int8, 0x55)
    ds.ds_quantize_shift_weights(wg.view, n, -15, sg.view, pg.view)
    torch.cuda.synchronize()
    assert sg.margins_intact() and pg.margins_intact()
    s_want, p_want = O.quantize_weights(wf, -15)
    assert np.array_equal(sg.numpy(n), s_want) and np.array_equal(pg.numpy(n), p_want)
    xf = (rng.standard_normal(n) * 100).astype(np.float32)
    xg = Guarded(n, torch.float32, float("nan"), xf)
    qg = Guarded(n, torch.int32, Y_CANARY)
    ds.ds_quantize_q16(xg.view, n, qg.view)
    assert qg.margins_intact()
    assert np.array_equal(qg.numpy(n), O.quantize_activations(xf))


def test_bf16_kernel_stays_inside_its_buffers(dslib):
    """The TMA loads of the tensor-core kernel read tiles clipped to the tensor maps' extents; its margins hold
    large bf16 values, so a read past x would show in the results."""
    ds = dslib
    M, K, N = 130, 200, 72
    rng = np.random.default_rng(81)
    bits = si.bf16_bits(rng.uniform(-(1 << 20), 1 << 20, size=(M, K)))
    s = si.sign_codes(81, (N, K))
    p = si.shift_codes_uniform(81, (N, K))
    bf = (si.bias(81, N).astype(np.float64) / 65536.0).astype(np.float32)
    desc, wbufs = _weights(ds, s, p, False)
    wb = ds.ds_bf16_weight_bytes(N, K)
    w16 = Guarded(wb, torch.uint8, 0x7F)
    ds.ds_expand_shift_weights_bf16(desc, w16.view, wb)
    xg = Guarded(M * K, torch.int16, 0x7F00, bits.view(np.int16))
    bg = Guarded(N, torch.float32, float("inf"), bf)
    yg = Guarded(M * N, torch.float32, 12345.0)
    ds.ds_linear_shift_bf16(xg.view, desc, bg.view, yg.view, M, K, N)
    for g in [w16, xg, bg, yg] + wbufs:
        assert g.margins_intact()
    assert ds.ds_bf16_fault_flag() == 0
    got = yg.numpy((M, N)).astype(np.float64)
    xf = si.bits_to_f64(bits)
    want = O.linear_shift_float(xf, s, p, bf.astype(np.float64))
    scale = O.linear_shift_float_absterms(xf, s, p) + np.abs(bf.astype(np.float64))[None, :]
    assert np.all(np.abs(got - want) <= 1e-5 * scale + 1e-30)


def test_specialized_conv_stays_inside_its_buffers(dslib):
    """The run-time compiled kernel: 16-byte-aligned row staging with zero fill, ragged tiles, residual."""
    ds = dslib
    N, C, H, W, K, R = 2, 3, 19, 23, 8, 3
    x, s, p, b = si.conv_layer(83, N, C, H, W, K, R, R, -(1 << 20), 1 << 20, -3)
    res = si.activations(84, (N, K, H, W), -(1 << 30), 1 << 30)
    h = ds.ds_specialize_conv2d_shift(s, p, K, C, R, R, 1, 1)
    try:
        xg = Guarded(x.size, torch.int32, X_CANARY, x)
        bg = Guarded(K, torch.int32, X_CANARY, b)
        rg = Guarded(res.size, torch.int32, X_CANARY, res)
        yg = Guarded(N * K * H * W, torch.int32, Y_CANARY)
        ag = Guarded(2, torch.int32, Y_CANARY, np.zeros(2, np.int32))
        ds.ds_conv2d_shift_specialized(h, xg.view, bg.view, rg.view, yg.view, N, H, W,
                                       ds.DS_RESIDUAL | ds.DS_RELU | ds.DS_AMAX_OUT, ag.view)
        for g in (xg, bg, rg, yg, ag):
            assert g.margins_intact()
        want = O.add_relu(O.conv2d_shift(x, s, p, b, (1, 1), (1, 1)), res)
        assert np.array_equal(yg.numpy(want.shape), want)
    finally:
        ds.ds_specialized_destroy(h)
