"""Two host threads drive the library at once, each on its own stream (the
launchers' one-time attribute calls and cluster-capacity caches are shared
process state): results stay bit-exact with the oracle."""
import threading

import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import deepshift_oracle as O

pytestmark = pytest.mark.gpu


def _work(ds, seed, out, errors):
    try:
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            dev = torch.device("cuda")
            # a small-batch FC (cluster kernel) and a standalone conv with a cluster split
            x, s, p, b = si.fc_layer(seed, 9, 700, 130, -(1 << 20), 1 << 20)
            w = ds.pack_shift_weights(torch.from_numpy(s).to(dev), torch.from_numpy(p).to(dev), expand=True)
            y = ds.linear_shift(torch.from_numpy(x).to(dev), w, torch.from_numpy(b).to(dev),
                                amax_io=torch.zeros(2, dtype=torch.int32, device=dev),
                                flags=ds.DS_AMAX_OUT, stream=stream.cuda_stream)
            xc, sc, pc, bc = si.conv_layer(seed + 1, 1, 64, 14, 14, 64, 3, 3, 0, 1 << 20)
            wc = ds.pack_shift_weights(torch.from_numpy(sc).to(dev), torch.from_numpy(pc).to(dev), expand=True)
            yc = ds.conv2d_shift(torch.from_numpy(xc).to(dev), wc, (3, 3), torch.from_numpy(bc).to(dev),
                                 (1, 1), (1, 1), stream=stream.cuda_stream)
        stream.synchronize()
        out[seed] = (y.cpu().numpy(), O.linear_shift(x, s, p, b), yc.cpu().numpy(),
                     O.conv2d_shift(xc, sc, pc, bc, (1, 1), (1, 1)))
    except Exception as e:  # reported by the main thread
        errors.append(e)


def test_two_host_threads(dslib):
    out, errors = {}, []
    threads = [threading.Thread(target=_work, args=(dslib, seed, out, errors)) for seed in (11, 23)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    for seed, (y, want, yc, wantc) in out.items():
        assert np.array_equal(y, want), seed
        assert np.array_equal(yc, wantc), seed
