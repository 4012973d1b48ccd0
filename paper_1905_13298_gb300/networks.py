"""Layer programs of all-shift ResNet18 / ResNet50 / VGG16 for ds_shift_forward.

A program is a list of LayerSpec (one ds_layer each) plus the shapes of its
shift layers' codes in parameter order (ResNet: stem; per block conv1, conv2
(, conv3), downsample if any; FC.  VGG16: 13 convs, 3 FCs).  BatchNorm is
omitted: it is not a shift operation and the codes are synthetic.
"""
from __future__ import annotations

import ctypes
import math
from dataclasses import dataclass

import numpy as np

from . import (DS_OP_AVGPOOL, DS_OP_CONV, DS_OP_FC, DS_OP_MAXPOOL, DS_RELU, DS_RESIDUAL, _need, _on_one_gpu,
               ds_last_error, ds_layer, ds_shift_forward, ds_shift_forward_workspace_bytes, pack_shift_weights)


@dataclass
class LayerSpec:
    op: int
    inp: int
    aux: int
    out: int
    C: int
    H: int
    W: int
    K: int = 0
    R: int = 1
    S: int = 1
    stride: int = 1
    pad: int = 0
    flags: int = 0
    param: int = -1  # index into the parameter list, -1 for pools


class _Builder:
    def __init__(self, C, H, W):
        self.specs, self.shapes = [], []
        self.free = []
        self.next_slot = 2
        self.shape = {0: (C, H, W)}

    def slot(self):
        if self.free:
            return self.free.pop()
        s = self.next_slot
        self.next_slot += 1
        return s

    def release(self, s):
        if s >= 2 and s not in self.free:
            self.free.append(s)

    def conv(self, inp, K, R, stride, pad, relu=True, residual=None, param=None, out=None):
        C, H, W = self.shape[inp]
        out = self.slot() if out is None else out
        idx = len(self.shapes) if param is None else param
        if param is None:
            self.shapes.append((K, C, R, R))
        flags = (DS_RELU if relu else 0) | (DS_RESIDUAL if residual is not None else 0)
        self.specs.append(LayerSpec(DS_OP_CONV, inp, -1 if residual is None else residual, out, C, H, W, K, R, R,
                                    stride, pad, flags, idx))
        self.shape[out] = (K, (H + 2 * pad - R) // stride + 1, (W + 2 * pad - R) // stride + 1)
        return out

    def reserve_param(self, shape):
        self.shapes.append(shape)
        return len(self.shapes) - 1

    def fc(self, inp, K, relu, out=None):
        C, H, W = self.shape[inp]
        out = self.slot() if out is None else out
        self.shapes.append((K, C * H * W))
        self.specs.append(LayerSpec(DS_OP_FC, inp, -1, out, C, H, W, K, 1, 1, 1, 0, DS_RELU if relu else 0,
                                    len(self.shapes) - 1))
        self.shape[out] = (K, 1, 1)
        return out

    def pool(self, op, inp, R, stride, pad):
        C, H, W = self.shape[inp]
        out = self.slot()
        self.specs.append(LayerSpec(op, inp, -1, out, C, H, W, 0, R, R, stride, pad, 0, -1))
        self.shape[out] = (C, (H + 2 * pad - R) // stride + 1, (W + 2 * pad - R) // stride + 1)
        return out


def resnet_program(arch: str = "resnet18", H: int = 224, W: int = 224):
    kind, blocks = {"resnet18": ("basic", [2, 2, 2, 2]), "resnet50": ("bottleneck", [3, 4, 6, 3])}[arch]
    b = _Builder(3, H, W)
    x = b.conv(0, 64, 7, 2, 3)
    y = b.pool(DS_OP_MAXPOOL, x, 3, 2, 1)
    b.release(x)
    x = y
    for stage, nb in enumerate(blocks):
        planes = 64 * 2 ** stage
        out_c = planes if kind == "basic" else 4 * planes
        for bi in range(nb):
            stride = 2 if (stage > 0 and bi == 0) else 1
            need_ds = stride != 1 or b.shape[x][0] != out_c
            if kind == "basic":
                p1 = b.reserve_param((planes, b.shape[x][0], 3, 3))
                p2 = b.reserve_param((planes, planes, 3, 3))
                pds = b.reserve_param((out_c, b.shape[x][0], 1, 1)) if need_ds else None
                t = b.conv(x, planes, 3, stride, 1, param=p1)
                sc = b.conv(x, out_c, 1, stride, 0, relu=False, param=pds) if need_ds else x
                o = b.conv(t, planes, 3, 1, 1, residual=sc, param=p2)
                b.release(t)
            else:
                p1 = b.reserve_param((planes, b.shape[x][0], 1, 1))
                p2 = b.reserve_param((planes, planes, 3, 3))
                p3 = b.reserve_param((out_c, planes, 1, 1))
                pds = b.reserve_param((out_c, b.shape[x][0], 1, 1)) if need_ds else None
                t1 = b.conv(x, planes, 1, 1, 0, param=p1)
                t2 = b.conv(t1, planes, 3, stride, 1, param=p2)
                # the shortcut before t1's slot is freed: it then writes no slot the main branch still
                # reads, so the executor can run it beside the main branch
                sc = b.conv(x, out_c, 1, stride, 0, relu=False, param=pds) if need_ds else x
                b.release(t1)
                o = b.conv(t2, out_c, 1, 1, 0, residual=sc, param=p3)
                b.release(t2)
            if need_ds:
                b.release(sc)
            b.release(x)
            x = o
    k = b.shape[x][1]
    y = b.pool(DS_OP_AVGPOOL, x, k, k, 0)
    b.fc(y, 1000, relu=False, out=1)
    return b.specs, b.shapes


def vgg16_program(H: int = 224, W: int = 224):
    cfg = [64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M", 512, 512, 512, "M"]
    b = _Builder(3, H, W)
    x = 0
    for v in cfg:
        if v == "M":
            y = b.pool(DS_OP_MAXPOOL, x, 2, 2, 0)
        else:
            y = b.conv(x, v, 3, 1, 1)
        b.release(x)
        x = y
    x1 = b.fc(x, 4096, relu=True)
    b.release(x)
    x2 = b.fc(x1, 4096, relu=True)
    b.release(x1)
    b.fc(x2, 1000, relu=False, out=1)
    return b.specs, b.shapes


def shift_terms(specs, batch: int) -> int:
    """Shift-op terms (one shift + one add each) of one forward at this batch."""
    total = 0
    for s in specs:
        if s.op == DS_OP_CONV:
            oh = (s.H + 2 * s.pad - s.R) // s.stride + 1
            ow = (s.W + 2 * s.pad - s.S) // s.stride + 1
            total += batch * s.K * oh * ow * s.C * s.R * s.S
        elif s.op == DS_OP_FC:
            total += batch * s.K * s.C * s.H * s.W
    return total


def output_shape(sp):
    """(channels, height, width) a layer writes per image."""
    if sp.op == DS_OP_FC:
        return (sp.K, 1, 1)
    OH = (sp.H + 2 * sp.pad - sp.R) // sp.stride + 1
    OW = (sp.W + 2 * sp.pad - sp.S) // sp.stride + 1
    return (sp.K if sp.op == DS_OP_CONV else sp.C, OH, OW)


class ShiftNetwork:
    """A packed all-shift network bound to device memory, run with ds_shift_forward."""

    def __init__(self, specs, params, batch: int, device="cuda", expand: bool = True):
        import torch
        self.specs = specs
        self.batch = batch
        self.weights = []
        self.biases = []
        for i, (s, p, bias) in enumerate(params):
            b = np.asarray(bias)
            if b.shape != (np.shape(s)[0],) or not np.issubdtype(b.dtype, np.integer):
                raise ValueError(f"bias {i} must be {np.shape(s)[0]} integers (one per output channel)")
            if b.size and (b.min() < -(1 << 31) or b.max() >= (1 << 31)):
                raise ValueError(f"bias {i} does not fit int32")
            w = pack_shift_weights(torch.from_numpy(s).to(device), torch.from_numpy(p).to(device), expand=expand)
            self.weights.append(w)
            self.biases.append(torch.from_numpy(np.ascontiguousarray(b, dtype=np.int32)).to(device))
        self.layers = (ds_layer * len(specs))()
        for i, sp in enumerate(specs):
            L = self.layers[i]
            L.op, L.in_, L.aux, L.out = sp.op, sp.inp, sp.aux, sp.out
            L.C, L.H, L.W, L.K, L.R, L.S = sp.C, sp.H, sp.W, sp.K, sp.R, sp.S
            L.stride, L.pad, L.flags = sp.stride, sp.pad, sp.flags
            if sp.param >= 0:
                L.w = ctypes.pointer(self.weights[sp.param].desc)
                L.bias = self.biases[sp.param].data_ptr()
        nbytes = ds_shift_forward_workspace_bytes(self.layers, len(specs), batch)
        if nbytes == 0:
            raise ValueError(f"the layer program was refused: {ds_last_error()}")
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.in_shape = (batch, specs[0].C, specs[0].H, specs[0].W)
        self.out_shape = (batch,) + output_shape([sp for sp in specs if sp.out == 1][-1])

    def forward(self, x, y=None, stream=None):
        """Runs the program on int32 x of shape (batch, C, H, W) (the first layer's input) into y (new, or
        a contiguous int32 tensor of at least out_shape's size) on the workspace's device."""
        import torch
        _need(x, "x", torch.int32, self.in_shape)
        if y is not None and (y.dtype != torch.int32 or not y.is_contiguous() or y.numel() < math.prod(self.out_shape)):
            raise ValueError(f"y must be a contiguous int32 tensor of at least {math.prod(self.out_shape)} elements")
        _on_one_gpu(workspace=self.workspace, x=x, y=y)
        if y is None:
            y = torch.empty(self.out_shape, dtype=torch.int32, device=x.device)
        ds_shift_forward(self.layers, len(self.specs), x, y, self.workspace, self.workspace.numel(), self.batch,
                         stream)
        return y
