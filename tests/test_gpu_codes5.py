"""GPU parity of the strict 5-bit code storage against the oracle, byte for byte: ds_pack_shift_weights5 writes
the oracle's blob (header, planes, zero tail), ds_unpack_shift_weights5 reads back the oracle's codes, codes
outside the 31 states are refused on both sides, and a layer run from the read-back codes gives the results of
the original codes."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _codes(seed, n_out, k_red):
    s = si.sign_codes(seed, (n_out, k_red))
    p = np.maximum(si.shift_codes_uniform(seed, (n_out, k_red)), -14).astype(np.int8)
    p[s == 0] = si.shift_codes_uniform(seed + 1, (n_out, k_red))[s == 0]  # zero weights may carry p = -15
    return s, p


@pytest.mark.parametrize("n_out,k_red", [(1, 3), (7, 64), (33, 32), (5, 100), (70, 1025), (512, 784)])
def test_pack5_blob_and_round_trip(dslib, n_out, k_red):
    ds = dslib
    s, p = _codes(n_out * 1000 + k_red, n_out, k_red)
    blob = ds.pack_shift_weights5(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    torch.cuda.synchronize()
    want = O.pack_codes5(s, p)
    assert np.array_equal(blob.cpu().numpy(), want)
    s2, p2 = ds.unpack_shift_weights5(blob, n_out, k_red)
    ws, wp = O.unpack_codes5(want, n_out, k_red)
    assert np.array_equal(s2.cpu().numpy(), ws) and np.array_equal(p2.cpu().numpy(), wp)
    assert np.array_equal(ws, s) and np.array_equal(wp, np.where(s == 0, 0, p))


def test_every_state_through_the_gpu(dslib):
    """All 46 (s, p) pairs that have a 5-bit code (zero weights with any p in [-15, 0]) in one column."""
    ds = dslib
    pairs = [(0, q) for q in range(-15, 1)] + [(sv, q) for sv in (-1, 1) for q in range(-14, 1)]
    s = np.array([[a for a, _ in pairs]], np.int8)
    p = np.array([[b for _, b in pairs]], np.int8)
    blob = ds.pack_shift_weights5(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    assert np.array_equal(blob.cpu().numpy(), O.pack_codes5(s, p))
    s2, p2 = ds.unpack_shift_weights5(blob, 1, len(pairs))
    assert [(int(a), int(b)) for a, b in zip(s2.cpu().numpy()[0], p2.cpu().numpy()[0])] == \
        [O.decode5(O.code5(a, b)) for a, b in pairs]


@pytest.mark.parametrize("bad", [(1, -15), (-1, -15), (2, 0), (1, 1)])
def test_codes_without_a_5bit_state_are_refused(dslib, bad):
    ds = dslib
    s, p = _codes(3, 4, 40)
    s[2, 17], p[2, 17] = bad
    with pytest.raises(ds.DsError) as e:
        ds.pack_shift_weights5(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    assert e.value.status == ds.DS_ERR_CODE_RANGE


def test_unpack_refuses_a_corrupt_or_foreign_blob(dslib):
    ds = dslib
    s, p = _codes(4, 3, 50)
    blob = ds.pack_shift_weights5(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    with pytest.raises(ds.DsError) as e:  # other dims
        ds.unpack_shift_weights5(blob, 3, 49)
    assert e.value.status == ds.DS_ERR_SHAPE
    planes = blob.clone()
    planes[256:276] = 0xFF  # code 31 everywhere in the first record
    with pytest.raises(ds.DsError) as e:
        ds.unpack_shift_weights5(planes, 3, 50)
    assert e.value.status == ds.DS_ERR_CODE_RANGE
    six = ds.pack_shift_weights(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    with pytest.raises(ds.DsError) as e:  # a 6-bit blob is not a 5-bit one
        ds.unpack_shift_weights5(six.blob, 3, 50)
    assert e.value.status == ds.DS_ERR_INVALID_ARG


def test_layer_from_read_back_codes(dslib):
    """Store, read back, pack to the 6-bit blob and run: the FC results equal those of the original codes."""
    ds = dslib
    M, K, N = 40, 300, 70
    x, s, p, b = si.fc_layer(5, M, K, N, -(1 << 20), 1 << 20)
    p = np.maximum(p, -14).astype(np.int8)
    blob = ds.pack_shift_weights5(torch.from_numpy(s).cuda(), torch.from_numpy(p).cuda())
    s2, p2 = ds.unpack_shift_weights5(blob, N, K)
    w = ds.pack_shift_weights(s2, p2, expand=True)
    y = ds.linear_shift(torch.from_numpy(x).cuda(), w, torch.from_numpy(b).cuda())
    assert np.array_equal(y.cpu().numpy(), O.linear_shift(x, s, p, b))
