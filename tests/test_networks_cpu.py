"""The ResNet18 / ResNet50 / VGG16 layer programs against their architectures.

The term count of a forward (one shift-op per weight-activation product, the
multiply-accumulate count of the float network) is rebuilt here layer by layer
from the architecture tables, independently of the program builder: ResNet18
and ResNet50 (He et al., basic and bottleneck blocks, 224 x 224 input) and
VGG16 (configuration D of Simonyan and Zisserman).  A missing block, a wrong
stride or a transposed channel count changes the totals.
"""
import paper_1905_13298_gb300 as ds
from paper_1905_13298_gb300 import networks as PN


def _conv(cout, cin, k, oh):
    return cout * oh * oh * cin * k * k


def _resnet18_per_image():
    t = _conv(64, 3, 7, 112)                       # stem 7x7/2
    t += 4 * _conv(64, 64, 3, 56)                  # stage 1: two basic blocks
    for c, hw in ((128, 28), (256, 14), (512, 7)):
        t += _conv(c, c // 2, 3, hw)               # first 3x3, stride 2
        t += 3 * _conv(c, c, 3, hw)                # the other three 3x3
        t += _conv(c, c // 2, 1, hw)               # 1x1/2 shortcut
    return t + 512 * 1000                          # FC


def _resnet50_per_image():
    t = _conv(64, 3, 7, 112)
    cin = 64
    for planes, nb, hw_in, hw in ((64, 3, 56, 56), (128, 4, 56, 28), (256, 6, 28, 14), (512, 3, 14, 7)):
        for i in range(nb):
            t += _conv(planes, cin, 1, hw_in if i == 0 else hw)  # 1x1 reduce (before the stride)
            t += _conv(planes, planes, 3, hw)                     # 3x3 (stride 2 in the first block of stages 2-4)
            t += _conv(4 * planes, planes, 1, hw)                 # 1x1 expand
            if i == 0:
                t += _conv(4 * planes, cin, 1, hw)                # projection shortcut
            cin = 4 * planes
    return t + 2048 * 1000


def _vgg16_per_image():
    t, cin, hw = 0, 3, 224
    for block in ((64, 64), (128, 128), (256, 256, 256), (512, 512, 512), (512, 512, 512)):
        for c in block:
            t += _conv(c, cin, 3, hw)
            cin = c
        hw //= 2
    return t + 25088 * 4096 + 4096 * 4096 + 4096 * 1000


def _counts(specs):
    return (sum(1 for s in specs if s.op == ds.DS_OP_CONV), sum(1 for s in specs if s.op == ds.DS_OP_FC))


def test_resnet18_terms_and_layers():
    specs, _ = PN.resnet_program("resnet18")
    assert _resnet18_per_image() == 1_814_073_344
    assert PN.shift_terms(specs, 1) == _resnet18_per_image()
    assert PN.shift_terms(specs, 32) == 32 * _resnet18_per_image()
    assert _counts(specs) == (20, 1)


def test_resnet50_terms_and_layers():
    specs, _ = PN.resnet_program("resnet50")
    assert PN.shift_terms(specs, 64) == 64 * _resnet50_per_image()
    assert _counts(specs) == (53, 1)


def test_vgg16_terms_and_layers():
    specs, _ = PN.vgg16_program()
    assert _vgg16_per_image() == 15_470_264_320
    assert PN.shift_terms(specs, 64) == 64 * _vgg16_per_image()
    assert _counts(specs) == (13, 3)


def test_programs_and_oracle_agree_on_layer_shapes():
    """The layer programs the library runs and the oracle's architectures (which write the stored full-size
    logits) list the same shift layers, in the same parameter order, at every image size the tests use."""
    from oracle import networks as ON
    for arch in ("resnet18", "resnet50"):
        for hw in ((224, 224), (64, 64), (32, 32)):
            assert [tuple(s) for s in PN.resnet_program(arch, *hw)[1]] == ON.layer_shapes(arch, *hw)
    for hw in ((224, 224), (32, 32)):
        assert [tuple(s) for s in PN.vgg16_program(*hw)[1]] == ON.layer_shapes("vgg16", *hw)
