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


def _forward_work(seed, out, errors):
    try:
        from paper_1905_13298_gb300 import networks as PN
        prog = PN.resnet_program("resnet18", 64, 64)
        params = si.network_params(prog[1], 103)
        x = si.image_batch(seed, 2, 3, 64, 64)
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            net = PN.ShiftNetwork(prog[0], params, batch=2)
            xd = torch.from_numpy(x).cuda()
            for _ in range(3):  # each thread's shortcut layers run on that thread's own side stream
                y = net.forward(xd, stream=stream.cuda_stream)
        stream.synchronize()
        out[seed] = (y.cpu().numpy().reshape(2, -1), x, params)
    except Exception as e:  # reported by the main thread
        errors.append(e)


def test_chained_forwards_on_four_host_threads(dslib):
    """Four threads run the ResNet18 forward at once, each on its own stream (and its own side stream for the
    shortcut layers): every result equals the oracle."""
    from oracle import networks as ON
    out, errors = {}, []
    threads = [threading.Thread(target=_forward_work, args=(seed, out, errors)) for seed in (31, 32, 33, 34)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    for seed, (y, x, params) in out.items():
        assert np.array_equal(y, ON.resnet_forward(x, params, "resnet18")), seed
