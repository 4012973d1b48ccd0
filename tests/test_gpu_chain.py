"""GPU parity of the chained forward (ds_shift_forward) against the CPU oracle (bit-exact)."""
import numpy as np
import pytest
import torch

import synth_inputs as si
from oracle import networks as ON

pytestmark = pytest.mark.gpu


def _run(program, params, x, expand=True):
    from paper_1905_13298_gb300.networks import ShiftNetwork
    specs, _ = program
    net = ShiftNetwork(specs, params, batch=x.shape[0], expand=expand)
    y = net.forward(torch.from_numpy(x).cuda())
    torch.cuda.synchronize()
    return y.cpu().numpy().reshape(x.shape[0], -1)


@pytest.mark.parametrize("expand", [True, False])
def test_resnet18_small_images(dslib, expand):
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet18", 64, 64)
    params = si.network_params(prog[1], 100)
    x = si.image_batch(7, 2, 3, 64, 64)
    assert np.array_equal(_run(prog, params, x, expand), ON.resnet_forward(x, params, "resnet18"))


def test_resnet50_small_image(dslib):
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet50", 64, 64)
    params = si.network_params(prog[1], 200)
    x = si.image_batch(8, 1, 3, 64, 64)
    assert np.array_equal(_run(prog, params, x), ON.resnet_forward(x, params, "resnet50"))


def test_vgg16_small_images(dslib):
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.vgg16_program(32, 32)
    params = si.network_params(prog[1], 300)
    x = si.image_batch(9, 2, 3, 32, 32)
    assert np.array_equal(_run(prog, params, x), ON.vgg16_forward(x, params))


def test_resnet18_stress_codes_saturate_exactly(dslib):
    """Codes centred at -6 in every layer (the stress law): activations saturate; results stay exact."""
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet18", 32, 32)
    params = []
    for i, shp in enumerate(prog[1]):
        params.append((si.sign_codes(400 + i, shp), si.shift_codes_geometric(400 + i, shp, -6), si.bias(400 + i, shp[0])))
    x = si.image_batch(10, 2, 3, 32, 32)
    want = ON.resnet_forward(x, params, "resnet18")
    assert (np.abs(want) == 2 ** 31 - 1).any() or (want == -(2 ** 31)).any()
    assert np.array_equal(_run(prog, params, x), want)


def test_resnet18_zero_codes(dslib):
    """Every sign zero (nnz = 0 and A = 0 in every column of every layer): each layer's output is its bias after
    the epilogue, carried through pools, residual joins and the max|x| hand-off between layers."""
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet18", 32, 32)
    params = [(np.zeros_like(s), p, b) for s, p, b in si.network_params(prog[1], 500)]
    x = si.image_batch(11, 2, 3, 32, 32)
    want = ON.resnet_forward(x, params, "resnet18")
    assert np.array_equal(want, np.broadcast_to(params[-1][2], want.shape))   # the FC sees only its bias
    assert np.array_equal(_run(prog, params, x), want)


def test_resnet18_full_size_batch1(dslib):
    """The ResNet18-architecture forward at 224 x 224, batch 1: every output."""
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet18")
    params = si.network_params(prog[1], si.SEED_BASE + 3)
    x = si.image_batch(si.SEED_BASE + 3, 1)
    assert np.array_equal(_run(prog, params, x), ON.resnet_forward(x, params, "resnet18"))


@pytest.mark.parametrize("batch", [1, 3])
def test_resnet18_small_batches_split_reduction(dslib, batch):
    """Small batches: tiles span image boundaries and small layers split their reduction (int64 partials)."""
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet18", 64, 64)
    params = si.network_params(prog[1], 500 + batch)
    x = si.image_batch(11 + batch, batch, 3, 64, 64)
    assert np.array_equal(_run(prog, params, x), ON.resnet_forward(x, params, "resnet18"))


def test_resnet18_stress_codes_small_batch(dslib):
    """Saturating codes at batch 1: the split reduction takes the 64-bit path and saturates exactly."""
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program("resnet18", 32, 32)
    params = []
    for i, shp in enumerate(prog[1]):
        params.append((si.sign_codes(600 + i, shp), si.shift_codes_geometric(600 + i, shp, -6), si.bias(600 + i, shp[0])))
    x = si.image_batch(12, 1, 3, 32, 32)
    assert np.array_equal(_run(prog, params, x), ON.resnet_forward(x, params, "resnet18"))


def _pointwise_pair_program(C, H, W, K1):
    """x [C,H,W] -> 1x1 conv K1 + ReLU -> 1x1 conv C, + x, ReLU (a bottleneck-style pair of 1x1 layers)."""
    from paper_1905_13298_gb300 import networks as PN
    b = PN._Builder(C, H, W)
    a = b.conv(0, K1, 1, 1, 0, relu=True)
    b.conv(a, C, 1, 1, 0, relu=True, residual=0, out=1)
    return (b.specs, b.shapes)


def _pointwise_pair_oracle(x, params):
    from oracle import deepshift_oracle as O
    (s1, p1, b1), (s2, p2, b2) = params
    a = O.conv2d_shift(x, s1, p1, b1, (1, 1), (0, 0), relu=True)
    return O.add_relu(O.conv2d_shift(a, s2, p2, b2, (1, 1), (0, 0)), x)


@pytest.mark.parametrize("batch,hw", [(1, 7), (2, 5)])
@pytest.mark.parametrize("stress", [False, True])
def test_pointwise_split_reduction(dslib, batch, hw, stress):
    """1x1 layers with 512 / 256 input channels on tiny maps: the chained forward splits their reduction
    over CTAs (int64 partials, then the finalize epilogue with residual and ReLU).  Pixel tiles span
    image boundaries (49 and 25 pixels per image).  Stress codes force the 64-bit path and saturation."""
    prog = _pointwise_pair_program(512, hw, hw, 256)
    if stress:
        params = [(si.sign_codes(700 + i, shp), si.shift_codes_geometric(700 + i, shp, -1), si.bias(700 + i, shp[0]))
                  for i, shp in enumerate(prog[1])]
    else:
        params = si.network_params(prog[1], 710 + batch)
    x = si.activations(720 + batch, (batch, 512, hw, hw), -(1 << 24), 1 << 24)
    want = _pointwise_pair_oracle(x, params).reshape(batch, -1)
    if stress:
        assert (np.abs(want) == 2 ** 31 - 1).any()
    assert np.array_equal(_run(prog, params, x), want)


def test_split_scratch_large_then_small_layers(dslib):
    """A split layer whose int64 scratch exceeds the 2 MB zero prefix (zeroed before its launch) followed by
    split layers that rely on the prefix being left zero (3x3 64 -> 128 on 28x28 at batch 4, then a 3x3/2 and
    a 1x1 on 14x14), twice in a row."""
    from paper_1905_13298_gb300 import networks as PN
    from oracle import deepshift_oracle as O
    b = PN._Builder(64, 28, 28)
    a1 = b.conv(0, 128, 3, 1, 1, relu=True)
    a2 = b.conv(a1, 128, 3, 2, 1, relu=True)
    b.conv(a2, 256, 1, 1, 0, relu=True, out=1)
    prog = (b.specs, b.shapes)
    params = si.network_params(prog[1], 820)
    x = si.activations(821, (4, 64, 28, 28), 0, 1 << 20)
    (s1, p1, b1), (s2, p2, b2), (s3, p3, b3) = params
    h = O.conv2d_shift(x, s1, p1, b1, (1, 1), (1, 1), relu=True)
    h = O.conv2d_shift(h, s2, p2, b2, (2, 2), (1, 1), relu=True)
    want = O.conv2d_shift(h, s3, p3, b3, (1, 1), (0, 0), relu=True).reshape(4, -1)
    from paper_1905_13298_gb300.networks import ShiftNetwork
    net = ShiftNetwork(prog[0], params, batch=4, expand=True)
    xd = torch.from_numpy(x).cuda()
    for _ in range(2):
        y = net.forward(xd)
        torch.cuda.synchronize()
        assert np.array_equal(y.cpu().numpy().reshape(4, -1), want)


def _stored_logits():
    """Oracle logits of the full-size forwards (tests/golden/network_outputs_224.txt, written by
    tests/golden/make_network_outputs.py with oracle/networks.py): (arch, batch, image) -> (digests, logits)."""
    import os
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "network_outputs_224.txt")
    out = {}
    with open(path) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            v = line.split()
            out[(v[0], int(v[1]), int(v[2]))] = ((v[3], v[4]), np.array([int(t) for t in v[5:]], dtype=np.int64))
    return out


def _digests(x, params):
    import hashlib
    hx = hashlib.sha256(np.ascontiguousarray(x).tobytes()).hexdigest()[:16]
    h = hashlib.sha256()
    for s, p, b in params:
        for a in (s, p, b):
            h.update(np.ascontiguousarray(a).tobytes())
    return hx, h.hexdigest()[:16]


@pytest.mark.parametrize("arch,batch", [("resnet18", 32), ("resnet50", 64), ("vgg16", 64)])
def test_full_size_chain_first_and_last_image(dslib, arch, batch):
    """The benchmarked chained forwards at full size (224 x 224; ResNet18 at batch 32, ResNet50 and VGG16 at
    batch 64), run as the benchmark runs them (one ds_shift_forward over the whole batch, expanded codes): the
    first and the last image's 1000 logits equal the oracle's, element by element."""
    from paper_1905_13298_gb300 import networks as PN
    prog = PN.resnet_program(arch) if arch != "vgg16" else PN.vgg16_program()
    params = si.network_params(prog[1], si.SEED_BASE + 3)
    x = si.image_batch(si.SEED_BASE + 3, batch)
    stored = _stored_logits()
    y = _run(prog, params, x)
    for image in (0, batch - 1):
        digests, want = stored[(arch, batch, image)]
        assert _digests(x[image:image + 1], params) == digests, "stale fixture: regenerate the stored logits"
        assert np.array_equal(y[image], want), image


def test_forward_replays_from_a_cuda_graph(dslib):
    """The chained forward captured in a CUDA graph (after one eager call) and replayed on new inputs copied into
    the captured input buffer: every replay equals the oracle, as the eager call does."""
    from paper_1905_13298_gb300 import networks as PN
    from oracle import networks as ON
    prog = PN.resnet_program("resnet18", 64, 64)
    params = si.network_params(prog[1], 102)
    net = PN.ShiftNetwork(prog[0], params, batch=2)
    xs = [si.image_batch(20 + i, 2, 3, 64, 64) for i in range(3)]
    xd = torch.from_numpy(xs[0]).cuda()
    y = torch.empty(net.out_shape, dtype=torch.int32, device="cuda")
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        net.forward(xd, y, stream.cuda_stream)  # eager first: one-time attribute and occupancy queries
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream, capture_error_mode="relaxed"):
            net.forward(xd, y, stream.cuda_stream)
    torch.cuda.synchronize()
    for x in xs:
        xd.copy_(torch.from_numpy(x))
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(y.cpu().numpy().reshape(2, -1), ON.resnet_forward(x, params, "resnet18"))
