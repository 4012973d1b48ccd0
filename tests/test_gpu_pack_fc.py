"""GPU parity of weight packing and LinearShift against the CPU oracle (bit-exact)."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _pack(ds, s, p, expand=False):
    return ds.pack_shift_weights(_dev(s.astype(np.int8)), _dev(p.astype(np.int8)), expand=expand)


@pytest.mark.parametrize("n_out,k_red", [(1, 1), (3, 31), (64, 576), (65, 33), (512, 784), (130, 100),
                                         (3, 100000), (1024, 1152), (9, 4129), (7, 48), (5, 528)])
def test_pack_blob_bitexact(dslib, n_out, k_red):
    seed = n_out * 7919 + k_red
    s = si.sign_codes(seed, (n_out, k_red))
    p = si.shift_codes_uniform(seed, (n_out, k_red))
    w = _pack(dslib, s, p)
    torch.cuda.synchronize()
    want = O.pack_planes6(s, p)
    got = w.blob.cpu().numpy()
    assert got.size == want.size
    assert np.array_equal(got, want)
    A, nnz = O.column_constants(s, p)
    assert w.desc.a_max == int(A.max()) and w.desc.nnz_max == int(nnz.max())


@pytest.mark.parametrize("n_out,k_red", [(1, 1), (33, 31), (64, 576), (70, 100)])
def test_expand_bitexact(dslib, n_out, k_red):
    seed = n_out * 31 + k_red
    s = si.sign_codes(seed, (n_out, k_red))
    p = si.shift_codes_uniform(seed, (n_out, k_red))
    w = dslib.pack_shift_weights(_dev(s), _dev(p), expand=True)
    torch.cuda.synchronize()
    want = O.expand_codes(s, p)
    got = w.expanded.cpu().numpy().reshape(want.shape)
    assert np.array_equal(got, want)
    assert w.desc.expanded == w.expanded.data_ptr()


def test_pack_rejects_bad_codes(dslib):
    s = np.ones((4, 10), np.int8)
    p = np.zeros((4, 10), np.int8)
    s[2, 3] = 2
    with pytest.raises(dslib.DsError) as e:
        _pack(dslib, s, p)
    assert e.value.status == dslib.DS_ERR_CODE_RANGE
    s[2, 3] = 1
    p[1, 1] = 1
    with pytest.raises(dslib.DsError):
        _pack(dslib, s, p)
    p[1, 1] = -16
    with pytest.raises(dslib.DsError):
        _pack(dslib, s, p)


@pytest.mark.parametrize("k_red", [10, 48, 100, 512])
def test_pack_counts_every_bad_code(dslib, k_red):
    """The out-of-range codes are counted exactly by every packing kernel (scalar, 4 and 16 codes per lane: k_red
    10, 100 / 48, 512), including positions in a chunk's second half and a tail chunk."""
    s = si.sign_codes(k_red, (5, k_red))
    p = si.shift_codes_uniform(k_red, (5, k_red))
    bad = [(0, 0, 2, 0), (1, k_red - 1, 1, 1), (3, k_red // 2, -2, -3), (4, k_red - 2, 0, -16), (2, 5, -1, 5)]
    for n, k, sv, pv in bad:
        s[n, k], p[n, k] = sv, pv
    with pytest.raises(dslib.DsError) as e:
        _pack(dslib, s, p)
    assert e.value.status == dslib.DS_ERR_CODE_RANGE
    assert str(e.value).split(": ", 1)[1].startswith(f"{len(bad)} codes"), str(e.value)


def _run_fc(ds, x, s, p, b, flags=0, amax=True, expand=False):
    w = _pack(ds, s, p, expand)
    xd = _dev(x.astype(np.int32))
    bd = _dev(b.astype(np.int32)) if b is not None else None
    amax_io = torch.zeros(2, dtype=torch.int32, device="cuda") if amax else None
    y = ds.linear_shift(xd, w, bd, amax_io=amax_io, flags=flags)
    torch.cuda.synchronize()
    return y.cpu().numpy(), (amax_io.cpu().numpy().view(np.uint32) if amax else None)


# Small and medium batches take the cluster kernel (the reduction split over up
# to 16 CTAs); (1024, 40, 3712) fills the SMs with 128 x 64 tiles and takes
# the plain shift GEMM.  K covers < 32, non-multiples of 4 and of 32, and long
# reductions with several chunks per CTA of a cluster.
FC_SHAPES = [(1, 1, 1), (3, 5, 7), (64, 784, 512), (129, 33, 65), (130, 100, 130), (257, 64, 64),
             (5, 1000, 3), (200, 4, 70), (31, 129, 1), (2, 8195, 96), (64, 4100, 200), (9, 2000, 130),
             (1024, 40, 3712)]


@pytest.mark.parametrize("M,K,N", FC_SHAPES)
@pytest.mark.parametrize("flags", [0, 1, 16, 17])
@pytest.mark.parametrize("expand", [False, True])
def test_linear_shift_bitexact(dslib, M, K, N, flags, expand):
    x, s, p, b = si.fc_layer(M * 1000 + K * 10 + N, M, K, N, -(1 << 20), 1 << 20)
    want = O.linear_shift(x, s, p, b, relu=bool(flags & 1))
    got, amax = _run_fc(dslib, x, s, p, b, flags | dslib.DS_AMAX_OUT, expand=expand)
    assert np.array_equal(got, want)
    assert amax[0] == O.absmax(x)
    assert amax[1] == O.absmax(want)


# one shape per FC kernel: cluster (small M) and shift GEMM (M = 1024, N = 3712)
@pytest.mark.parametrize("M,K,N", [(1, 1, 1), (9, 700, 130), (1024, 40, 3712)])
@pytest.mark.parametrize("expand", [False, True])
def test_linear_shift_degenerate_codes(dslib, M, K, N, expand):
    """The degenerate cases of the method: every sign zero gives y = sat32(b) (nnz = 0 and A = 0 in every
    column); s = -1, p = 0 on x = INT32_MIN makes every term 2^31, the one term value outside int32, so the
    accumulator bound must refuse the 32-bit path wherever the exact sums leave int32."""
    x, s, p, b = si.fc_layer(M + 7 * K + N, M, K, N, -(1 << 31), 1 << 31)
    got, amax = _run_fc(dslib, x, np.zeros_like(s), p, b, dslib.DS_AMAX_OUT, expand=expand)
    assert np.array_equal(got, np.broadcast_to(b, (M, N)))
    assert amax[1] == O.absmax(b)
    xm = np.full((M, K), -(1 << 31), np.int32)
    sm = -np.ones((N, K), np.int8)
    pm = np.zeros((N, K), np.int8)
    want = O.linear_shift(xm, sm, pm, b)
    assert K == 1 or (O.linear_shift_acc(xm, sm, pm, b) > O.INT32_MAX).all()
    got, amax = _run_fc(dslib, xm, sm, pm, b, dslib.DS_AMAX_OUT, expand=expand)
    assert np.array_equal(got, want)
    assert amax[0] == 1 << 31 and amax[1] == O.absmax(want)


def test_linear_shift_config1_bitexact(dslib):
    x, s, p, b = si.config1()
    want = O.linear_shift(x, s, p, b)
    got, _ = _run_fc(dslib, x, s, p, b)
    assert np.array_equal(got, want)


def test_linear_shift_no_bias_no_amax(dslib):
    x, s, p, b = si.fc_layer(77, 40, 70, 90, -(1 << 31), 1 << 31)
    got, _ = _run_fc(dslib, x, s, p, None, 0, amax=False)
    assert np.array_equal(got, O.linear_shift(x, s, p, None))


@pytest.mark.parametrize("M,K,N", [(70, 300, 66), (128, 64, 64), (3, 5000, 40)])
def test_linear_shift_saturating_inputs(dslib, M, K, N):
    """Full-range int32 activations: the 64-bit path must take over and saturate exactly."""
    x, s, p, b = si.fc_layer(M + K + N, M, K, N, -(1 << 31), 1 << 31)
    p = np.where(np.arange(K)[None, :] % 3 == 0, 0, p).astype(np.int8)  # many unit weights
    want = O.linear_shift(x, s, p, b, relu=True)
    assert (np.abs(O.linear_shift_acc(x, s, p, b)) > O.INT32_MAX).any()
    got, _ = _run_fc(dslib, x, s, p, b, dslib.DS_RELU)
    assert np.array_equal(got, want)


def test_linear_shift_amax_in_is_used(dslib):
    """A caller-provided amax that proves int32 safety gives the same exact result."""
    x, s, p, b = si.fc_layer(5, 96, 96, 96, -(1 << 20), 1 << 20)
    w = _pack(dslib, s, p)
    amax_io = torch.tensor([O.absmax(x), 0], dtype=torch.int64).to(torch.int32).cuda()
    y = dslib.linear_shift(_dev(x), w, _dev(b), amax_io=amax_io, flags=dslib.DS_AMAX_IN)
    assert np.array_equal(y.cpu().numpy(), O.linear_shift(x, s, p, b))


@pytest.mark.parametrize("expand", [False, True])
def test_linear_shift_config4_sampled(dslib, expand):
    """Full-size 8192 x 4096 x 4096 launch (the expanded layout is the one the benchmark times); sampled
    outputs checked one by one, and 24 whole rows (tile edges, the last row, random rows) against the
    vectorised oracle."""
    x, s, p, b = si.config4_int()
    w = _pack(dslib, s, p, expand=expand)
    amax_io = torch.zeros(2, dtype=torch.int32, device="cuda")
    y = dslib.linear_shift(_dev(x), w, _dev(b), amax_io=amax_io).cpu().numpy()
    rng = np.random.default_rng(0)
    rows = np.concatenate([[0, 8191], rng.integers(0, 8192, 30)])
    cols = np.concatenate([[0, 4095], rng.integers(0, 4096, 30)])
    for m, n in zip(rows, cols):
        want = O.linear_shift_at(x, s, p, b, int(m), int(n))
        assert y[m, n] == max(min(want, O.INT32_MAX), O.INT32_MIN)
    whole = [0, 127, 128, 4095, 4096, 4097, 8064, 8191] + [int(v) for v in rng.integers(0, 8192, 16)]
    for m in whole:
        assert np.array_equal(y[m:m + 1], O.linear_shift(x[m:m + 1], s, p, b)), m
