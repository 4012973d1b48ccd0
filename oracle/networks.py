"""CPU oracle of chained DeepShift forwards.  TEST INFRASTRUCTURE ONLY.

Every conv and FC layer of the network is a shift layer (Eq. 3 with the
Sec. 4 fixed point; DeepShift converts all layers, including the first and the
last), composed with the integer pools of ``deepshift_oracle``.  BatchNorm is
omitted (reading R-bn: it is not a shift op and the codes are synthetic).
The architectures follow the standard definitions that the paper evaluates:

* ResNet18 / ResNet50 (He et al.): 7x7/2 stem conv + ReLU, 3x3/2 max-pool
  (pad 1), four stages of basic (18) or bottleneck (50) blocks, floor
  average pool over the final 7x7 map, FC to 1000.  A block computes
  ReLU(sat32(main + shortcut)); the shortcut is the identity or a 1x1 conv
  with the block's stride (no ReLU); in bottleneck blocks the stride sits on
  the 3x3 conv.
* VGG16 (Simonyan and Zisserman): thirteen 3x3/1/1 convs + ReLU with 2x2/2
  max-pools, then FC 25088 -> 4096 -> 4096 (ReLU) -> 1000.

Parameter order (``params`` is a list of (s, p, b) per shift layer):
ResNet: stem; then per block conv1, conv2 (, conv3 for bottleneck) and the
downsample conv if the block has one; then the FC.  VGG16: the 13 convs,
then the 3 FCs.

Pins: the chain is built only from pinned parts (conv, FC, pools, residual
join), and the whole chain of each network equals a float64 composition of
library routines (torch conv2d, max_pool2d, avg_pool2d + floor, linear) on a
special case where every term is exact: one non-zero code per output channel
with p = 0 (tests/test_oracle_pins.py, *_chain_matches_float64_library_case,
ResNet18, ResNet50 and VGG16 on 32 x 32 images).  A wrong stride, padding,
pool, shortcut, ReLU placement or layer order changes that result.
"""
from __future__ import annotations

import numpy as np

from . import deepshift_oracle as O

RESNET_STAGES = {"resnet18": ("basic", [2, 2, 2, 2]), "resnet50": ("bottleneck", [3, 4, 6, 3])}
VGG16_CFG = [64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M", 512, 512, 512, "M"]


def layer_shapes(arch: str, H: int = 224, W: int = 224):
    """Shapes of the shift layers of an architecture, in parameter order: (K, C, R, S) per conv and
    (n_out, k_in) per FC, as the forwards below consume them."""
    if arch == "vgg16":
        shapes, c, h, w = [], 3, H, W
        for v in VGG16_CFG:
            if v == "M":
                h, w = h // 2, w // 2
            else:
                shapes.append((v, c, 3, 3))
                c = v
        k = c * h * w
        for n in (4096, 4096, 1000):
            shapes.append((n, k))
            k = n
        return shapes
    kind, blocks = RESNET_STAGES[arch]
    shapes, c = [(64, 3, 7, 7)], 64
    for stage, nb in enumerate(blocks):
        for bi in range(nb):
            stride = 2 if (stage > 0 and bi == 0) else 1
            planes = 64 * (2 ** stage)
            out_c = planes if kind == "basic" else planes * 4
            if kind == "basic":
                shapes += [(planes, c, 3, 3), (planes, planes, 3, 3)]
            else:
                shapes += [(planes, c, 1, 1), (planes, planes, 3, 3), (out_c, planes, 1, 1)]
            if stride != 1 or c != out_c:
                shapes.append((out_c, c, 1, 1))
            c = out_c
    shapes.append((1000, c))
    return shapes


def _conv(x, prm, stride, pad, relu, residual=None):
    """One ConvShift layer of a chain (Eq. 3, convolutional form; readings R-conv, R-acc), then either the
    residual join ReLU(sat32(y + residual)) or the optional ReLU."""
    s, p, b = prm
    y = O.conv2d_shift(x, s, p, b, (stride, stride), (pad, pad), relu=False)
    if residual is not None:
        return O.add_relu(y, residual)
    return np.maximum(y, 0).astype(np.int32) if relu else y


def resnet_forward(x, params, arch: str = "resnet18"):
    """Forward of an all-shift ResNet; x int32 [N, 3, 224, 224]; returns int32 [N, 1000].

    Every conv and FC is a shift layer (Eq. 3 with Sec. 4's fixed point); pools follow reading R-pool, and
    BatchNorm is omitted (reading R-bn)."""
    kind, blocks = RESNET_STAGES[arch]
    it = iter(params)
    x = _conv(x, next(it), 2, 3, relu=True)
    x = O.maxpool2d(x, 3, 2, 1)
    for stage, nb in enumerate(blocks):
        for bi in range(nb):
            stride = 2 if (stage > 0 and bi == 0) else 1
            planes = 64 * (2 ** stage)
            out_c = planes if kind == "basic" else planes * 4
            need_ds = stride != 1 or x.shape[1] != out_c
            if kind == "basic":
                c1, c2 = next(it), next(it)
                ds = next(it) if need_ds else None
                t = _conv(x, c1, stride, 1, relu=True)
                sc = _conv(x, ds, stride, 0, relu=False) if ds is not None else x
                x = _conv(t, c2, 1, 1, relu=True, residual=sc)
            else:
                c1, c2, c3 = next(it), next(it), next(it)
                ds = next(it) if need_ds else None
                t = _conv(x, c1, 1, 0, relu=True)
                t = _conv(t, c2, stride, 1, relu=True)
                sc = _conv(x, ds, stride, 0, relu=False) if ds is not None else x
                x = _conv(t, c3, 1, 0, relu=True, residual=sc)
    k = x.shape[2]
    x = O.avgpool_floor(x, k, k)
    s, p, b = next(it)
    y = O.linear_shift(x.reshape(x.shape[0], -1), s.reshape(s.shape[0], -1), p.reshape(p.shape[0], -1), b)
    if next(it, None) is not None:
        raise ValueError("unused parameters")
    return y


def vgg16_forward(x, params):
    """Forward of an all-shift VGG16; x int32 [N, 3, H, W] (224 x 224 in the workloads); returns int32 [N, 1000].

    Every conv and FC is a shift layer (Eq. 3 with Sec. 4's fixed point); max-pools follow reading R-pool."""
    it = iter(params)
    for v in VGG16_CFG:
        if v == "M":
            x = O.maxpool2d(x, 2, 2, 0)
        else:
            x = _conv(x, next(it), 1, 1, relu=True)
    x = x.reshape(x.shape[0], -1)
    for i in range(3):
        s, p, b = next(it)
        x = O.linear_shift(x, s.reshape(s.shape[0], -1), p.reshape(p.shape[0], -1), b, relu=(i < 2))
    if next(it, None) is not None:
        raise ValueError("unused parameters")
    return x
