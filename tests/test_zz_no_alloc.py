"""The allocation-free LinearShift entry point.

ds_linear_shift_static_scratch serves callers that cannot allocate device
memory (a plugin handed only its buffers, a host callback, a real-time path):
its two scratch words live in a static device array of the library.  These
checks call it through the C ABI and compare it with ds_linear_shift, which
takes caller-allocated scratch, on two calls in a row.  The second call uses
inputs with a different max|x| so that a stale value left in the shared array
by the first call would show up.  This file is collected last so that a run
that stops at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth_inputs as si

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
    # call 1: full-range activations (64-bit path); call 2: small activations (32-bit path)
    cases = [si.fc_layer(41, M, K, N, -(1 << 31), 1 << 31), si.fc_layer(42, M, K, N, -(1 << 20), 1 << 20)]
    for flags, (x, s, p, b) in zip((ds.DS_RELU, 0), cases):
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


def test_static_scratch_rejects_amax_flags(dslib):
    ds = dslib
    x = torch.zeros((4, 4), dtype=torch.int32, device="cuda")
    y = torch.zeros((4, 4), dtype=torch.int32, device="cuda")
    w = ds.pack_shift_weights(torch.ones((4, 4), dtype=torch.int8, device="cuda"),
                              torch.zeros((4, 4), dtype=torch.int8, device="cuda"))
    with pytest.raises(ds.DsError) as e:
        ds.ds_linear_shift_static_scratch(x, w.desc, None, y, 4, 4, 4, ds.DS_AMAX_OUT)
    assert e.value.status == ds.DS_ERR_INVALID_ARG
