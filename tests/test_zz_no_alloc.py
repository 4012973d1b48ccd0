"""The allocation-free LinearShift entry point.

ds_linear_shift_static_scratch serves callers that cannot allocate device
memory (a plugin handed only its buffers, a host callback, a real-time path):
its two scratch words live in a static device array of the library.  These
checks call it through the C ABI on three calls in a row and compare every
output with ds_linear_shift (caller-allocated scratch) and with the CPU
oracle.

The calls alternate small and full-range activations (small, full range,
small), so each call runs after one whose max|x| differs from its own.  What
they check is output parity after any history of the shared array.  They do
not observe the array itself: the pre-pass folds max|x| in with a max, so a
leftover value can only be larger than the true one, which selects the 64-bit
path, and that path is exact too.  A leftover value therefore cannot change
an output.

This file is collected last so that a run that stops at the first failure
has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _reference(ds, x, w, b, M, K, N, flags):
    y = torch.empty((M, N), dtype=torch.int32, device="cuda")
    amax_io = torch.zeros(2, dtype=torch.int32, device="cuda")
    ds.ds_linear_shift(x, w.desc, b, y, M, K, N, flags, amax_io)
    return y


def test_static_scratch_matches_allocating_entry_point(dslib):
    ds = dslib
    L = ds.lib()
    stream = torch.cuda.current_stream().cuda_stream
    M, K, N = 150, 300, 70
    # small activations (32-bit path), full-range ones (64-bit path), small again
    cases = [(0, si.fc_layer(42, M, K, N, -(1 << 20), 1 << 20)),
             (ds.DS_RELU, si.fc_layer(41, M, K, N, -(1 << 31), 1 << 31)),
             (ds.DS_RELU, si.fc_layer(43, M, K, N, -(1 << 18), 1 << 18))]
    for flags, (x, s, p, b) in cases:
        w = ds.pack_shift_weights(_dev(s), _dev(p))
        xd, bd = _dev(x), _dev(b)
        want = _reference(ds, xd, w, bd, M, K, N, flags)
        y = torch.full((M, N), 7, dtype=torch.int32, device="cuda")
        st = L.ds_linear_shift_static_scratch(xd.data_ptr(), ctypes.byref(w.desc), bd.data_ptr(), y.data_ptr(),
                                              M, K, N, flags, stream)
        assert st == ds.DS_OK, ds.ds_last_error()
        torch.cuda.synchronize()
        # integer path: the tolerance of every parity test here is bit-exact
        assert torch.equal(y, want)
        assert np.array_equal(y.cpu().numpy(), O.linear_shift(x, s, p, b, relu=bool(flags & ds.DS_RELU)))


def test_static_scratch_rejects_amax_flags(dslib):
    ds = dslib
    x = torch.zeros((4, 4), dtype=torch.int32, device="cuda")
    y = torch.zeros((4, 4), dtype=torch.int32, device="cuda")
    w = ds.pack_shift_weights(torch.ones((4, 4), dtype=torch.int8, device="cuda"),
                              torch.zeros((4, 4), dtype=torch.int8, device="cuda"))
    with pytest.raises(ds.DsError) as e:
        ds.ds_linear_shift_static_scratch(x, w.desc, None, y, 4, 4, 4, ds.DS_AMAX_OUT)
    assert e.value.status == ds.DS_ERR_INVALID_ARG
