"""GPU parity of the chained forward's integer pools (one-layer programs through ds_shift_forward) against the
oracle's pools, bit-exact: the paired 3x3 / 2 max-pool of the ResNet stems (W a multiple of 4), the generic
max-pool (other widths, 2x2 / 2 of VGG) and the whole-plane and windowed floor average pools, on values that
include INT32_MIN, INT32_MAX and negative sums."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _run_pool(op, x, R, stride, pad):
    import paper_1905_13298_gb300 as ds
    from paper_1905_13298_gb300.networks import LayerSpec, ShiftNetwork
    N, C, H, W = x.shape
    spec = LayerSpec(op=op, inp=0, aux=-1, out=1, C=C, H=H, W=W, R=R, S=R, stride=stride, pad=pad)
    net = ShiftNetwork([spec], [], batch=N)
    y = net.forward(torch.from_numpy(np.ascontiguousarray(x)).cuda())
    torch.cuda.synchronize()
    return y.cpu().numpy()


def _inputs(seed, shape):
    x = si.activations(seed, shape, -(1 << 31), 1 << 31)
    flat = x.reshape(-1)
    flat[::97] = np.iinfo(np.int32).min
    flat[5::89] = np.iinfo(np.int32).max
    return x


@pytest.mark.parametrize("shape", [(3, 5, 112, 112), (2, 3, 13, 20), (1, 4, 4, 4), (2, 3, 12, 18), (1, 2, 9, 7)])
def test_maxpool_3x3_stride2(dslib, shape):
    import paper_1905_13298_gb300 as ds
    x = _inputs(sum(shape), shape)
    got = _run_pool(ds.DS_OP_MAXPOOL, x, 3, 2, 1)
    assert np.array_equal(got, O.maxpool2d(x, 3, 2, 1))


def test_maxpool_2x2_stride2(dslib):
    import paper_1905_13298_gb300 as ds
    x = _inputs(71, (2, 6, 14, 14))
    assert np.array_equal(_run_pool(ds.DS_OP_MAXPOOL, x, 2, 2, 0), O.maxpool2d(x, 2, 2, 0))


@pytest.mark.parametrize("shape", [(4, 512, 7, 7), (3, 7, 1, 1), (2, 9, 6, 6), (1, 40, 11, 11)])
def test_avgpool_whole_plane(dslib, shape):
    """The global pool: negative sums floor toward minus infinity, sums beyond int32 are exact."""
    import paper_1905_13298_gb300 as ds
    x = _inputs(sum(shape) + 1, shape)
    k = shape[2]
    assert shape[2] == shape[3]
    assert np.array_equal(_run_pool(ds.DS_OP_AVGPOOL, x, k, 1, 0), O.avgpool_floor(x, k, 1))


def test_avgpool_windowed(dslib):
    import paper_1905_13298_gb300 as ds
    x = _inputs(72, (2, 3, 10, 10))
    assert np.array_equal(_run_pool(ds.DS_OP_AVGPOOL, x, 2, 2, 0), O.avgpool_floor(x, 2, 2))
