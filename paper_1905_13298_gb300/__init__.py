"""DeepShift shift operators on GB300: thin Python binding of libdeepshift.so.

The functions named ``ds_*`` mirror the C ABI of ``include/deepshift.h`` one
to one (argument marshalling only: every step runs in the library's CUDA
kernels).  PyTorch supplies device memory and the current CUDA stream.  There
is no CPU fallback: importing works without a GPU, but every compute call
needs the built library and a CUDA device, and fails loudly otherwise.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libdeepshift.so")

# status codes (deepshift.h)
DS_OK = 0
DS_ERR_INVALID_ARG = 1
DS_ERR_SHAPE = 2
DS_ERR_CODE_RANGE = 3
DS_ERR_ALIGNMENT = 4
DS_ERR_BUFFER_TOO_SMALL = 5
DS_ERR_UNSUPPORTED = 6
DS_ERR_CUDA = 7
STATUS_NAMES = {0: "DS_OK", 1: "DS_ERR_INVALID_ARG", 2: "DS_ERR_SHAPE", 3: "DS_ERR_CODE_RANGE",
                4: "DS_ERR_ALIGNMENT", 5: "DS_ERR_BUFFER_TOO_SMALL", 6: "DS_ERR_UNSUPPORTED",
                7: "DS_ERR_CUDA"}

# flags
DS_RELU = 1
DS_AMAX_IN = 2
DS_AMAX_OUT = 4
DS_RESIDUAL = 8
DS_FORCE_INT64 = 16
DS_CONV_IM2COL = 32

DS_OP_CONV = 1
DS_OP_FC = 2
DS_OP_MAXPOOL = 3
DS_OP_AVGPOOL = 4

DS_WEIGHTS_MAGIC = 0x31575344
DS_FORMAT_PLANES6 = 1
DS_FORMAT_CODES5 = 2


class DsError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class ds_weights(ctypes.Structure):
    _fields_ = [("magic", ctypes.c_uint32), ("format", ctypes.c_uint32),
                ("n_out", ctypes.c_int64), ("k_red", ctypes.c_int64), ("n_chunks", ctypes.c_int64),
                ("packed", ctypes.c_void_p), ("packed_bytes", ctypes.c_size_t),
                ("a_max", ctypes.c_uint64), ("nnz_max", ctypes.c_uint32), ("reserved", ctypes.c_uint32),
                ("expanded", ctypes.c_void_p), ("expanded_bytes", ctypes.c_size_t),
                ("weights_bf16", ctypes.c_void_p), ("weights_bf16_bytes", ctypes.c_size_t)]


class ds_layer(ctypes.Structure):
    _fields_ = [("op", ctypes.c_int32), ("in_", ctypes.c_int32), ("aux", ctypes.c_int32), ("out", ctypes.c_int32),
                ("C", ctypes.c_int32), ("H", ctypes.c_int32), ("W", ctypes.c_int32), ("K", ctypes.c_int32),
                ("R", ctypes.c_int32), ("S", ctypes.c_int32), ("stride", ctypes.c_int32), ("pad", ctypes.c_int32),
                ("flags", ctypes.c_uint32), ("w", ctypes.POINTER(ds_weights)), ("bias", ctypes.c_void_p)]


_lib = None

_SIGNATURES = {
    "ds_last_error": (ctypes.c_char_p, []),
    "ds_version": (ctypes.c_int, []),
    "ds_abi_struct_size": (ctypes.c_size_t, [ctypes.c_int]),
    "ds_packed_weight_bytes": (ctypes.c_size_t, [ctypes.c_int64, ctypes.c_int64]),
    "ds_pack_shift_weights": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64,
                                             ctypes.c_void_p, ctypes.c_size_t, ctypes.POINTER(ds_weights),
                                             ctypes.c_void_p]),
    "ds_linear_shift": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ds_weights), ctypes.c_void_p,
                                       ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                       ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p]),
    "ds_conv2d_shift": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ds_weights), ctypes.c_void_p,
                                       ctypes.c_void_p, ctypes.c_void_p] + [ctypes.c_int] * 11 +
                        [ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p]),
    "ds_linear_shift_static_scratch": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ds_weights),
                                                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                                      ctypes.c_int64, ctypes.c_int64, ctypes.c_uint32,
                                                      ctypes.c_void_p]),
    "ds_packed5_weight_bytes": (ctypes.c_size_t, [ctypes.c_int64, ctypes.c_int64]),
    "ds_pack_shift_weights5": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64,
                                              ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]),
    "ds_unpack_shift_weights5": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int64, ctypes.c_int64,
                                                ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "ds_expanded_weight_bytes": (ctypes.c_size_t, [ctypes.c_int64, ctypes.c_int64]),
    "ds_expand_shift_weights": (ctypes.c_int, [ctypes.POINTER(ds_weights), ctypes.c_void_p, ctypes.c_size_t,
                                               ctypes.c_void_p]),
    "ds_shift_forward_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(ds_layer), ctypes.c_int, ctypes.c_int]),
    "ds_shift_forward": (ctypes.c_int, [ctypes.POINTER(ds_layer), ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p,
                                        ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_void_p]),
    "ds_bf16_weight_bytes": (ctypes.c_size_t, [ctypes.c_int64, ctypes.c_int64]),
    "ds_expand_shift_weights_bf16": (ctypes.c_int, [ctypes.POINTER(ds_weights), ctypes.c_void_p, ctypes.c_size_t,
                                                    ctypes.c_void_p]),
    "ds_linear_shift_bf16": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ds_weights), ctypes.c_void_p,
                                            ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                            ctypes.c_uint32, ctypes.c_void_p]),
    "ds_bf16_fault_flag": (ctypes.c_int, []),
    "ds_bf16_set_wait_limit": (None, [ctypes.c_longlong]),
    "ds_specialize_conv2d_shift": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p] + [ctypes.c_int] * 6 +
                                   [ctypes.POINTER(ctypes.c_void_p)]),
    "ds_conv2d_shift_specialized": (ctypes.c_int, [ctypes.c_void_p] * 5 + [ctypes.c_int] * 3 +
                                    [ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p]),
    "ds_specialized_destroy": (None, [ctypes.c_void_p]),
    "ds_absmax": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]),
    "ds_quantize_shift_weights": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_void_p,
                                                 ctypes.c_void_p, ctypes.c_void_p]),
    "ds_quantize_q16": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]),
    "ds_packed_weight_bytes_backward": (ctypes.c_size_t, [ctypes.c_int] * 6),
    "ds_pack_shift_weights_backward": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p] + [ctypes.c_int] * 6 +
                                       [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_void_p]),
    "ds_linear_shift_backward_x": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                                  ctypes.c_int64, ctypes.c_int64, ctypes.c_uint32, ctypes.c_void_p,
                                                  ctypes.c_void_p]),
    "ds_conv2d_shift_backward_x": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p] +
                                   [ctypes.c_int] * 11 + [ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p]),
}


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built (there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with paper_1905_13298_gb300.build.build_library()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        for which, st in ((0, ds_weights), (1, ds_layer)):
            if L.ds_abi_struct_size(which) != ctypes.sizeof(st):
                raise ImportError(f"{st.__name__} layout differs between the binding and {LIB_PATH}")
        _lib = L
    return _lib


def ds_last_error() -> str:
    return lib().ds_last_error().decode()


def _check(status: int) -> None:
    if status != DS_OK:
        raise DsError(status, ds_last_error())


def _ptr(t) -> int | None:
    """Device (or host) address of a tensor, None for None; ints pass through."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _need(t, name: str, dtypes, shape=None, min_numel: int = 0) -> None:
    """Checks a tensor argument of the tensor-level helpers (None passes).  The C ABI sees only an
    address, so a tensor of another dtype, a strided view or a wrong shape would be read as something
    it is not: each is refused here instead."""
    if t is None:
        return
    dtypes = dtypes if isinstance(dtypes, tuple) else (dtypes,)
    if t.dtype not in dtypes:
        raise ValueError(f"{name} must be {' or '.join(str(d) for d in dtypes)}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    if t.numel() < min_numel:
        raise ValueError(f"{name} needs at least {min_numel} elements")


def _on_one_gpu(**tensors) -> None:
    """Every tensor given (None passes) is CUDA memory on the first one's device."""
    device = None
    for name, t in tensors.items():
        if t is None:
            continue
        if t.device.type != "cuda":
            raise ValueError(f"{name} must be a CUDA tensor")
        device = device or t.device
        if t.device != device:
            raise ValueError(f"{name} is on {t.device}, the input on {device}")


def _need_amax(amax_io) -> None:
    import torch
    _need(amax_io, "amax_io", (torch.int32, torch.uint32), min_numel=2)


def _stream(stream) -> int | None:
    if stream is not None:
        return stream if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


# ---------------------------------------------------------------------------
# One-to-one wrappers of the C ABI
# ---------------------------------------------------------------------------

def ds_packed_weight_bytes(n_out: int, k_red: int) -> int:
    return int(lib().ds_packed_weight_bytes(n_out, k_red))


def ds_pack_shift_weights(s, p, n_out: int, k_red: int, packed, packed_bytes: int, stream=None) -> ds_weights:
    desc = ds_weights()
    _check(lib().ds_pack_shift_weights(_ptr(s), _ptr(p), n_out, k_red, _ptr(packed), packed_bytes,
                                       ctypes.byref(desc), _stream(stream)))
    return desc


def ds_packed5_weight_bytes(n_out: int, k_red: int) -> int:
    return int(lib().ds_packed5_weight_bytes(n_out, k_red))


def ds_pack_shift_weights5(s, p, n_out: int, k_red: int, packed5, packed5_bytes: int, stream=None) -> None:
    _check(lib().ds_pack_shift_weights5(_ptr(s), _ptr(p), n_out, k_red, _ptr(packed5), packed5_bytes,
                                        _stream(stream)))


def ds_unpack_shift_weights5(packed5, packed5_bytes: int, n_out: int, k_red: int, s, p, stream=None) -> None:
    _check(lib().ds_unpack_shift_weights5(_ptr(packed5), packed5_bytes, n_out, k_red, _ptr(s), _ptr(p),
                                          _stream(stream)))


def ds_expanded_weight_bytes(n_out: int, k_red: int) -> int:
    return int(lib().ds_expanded_weight_bytes(n_out, k_red))


def ds_expand_shift_weights(w: ds_weights, expanded, expanded_bytes: int, stream=None) -> None:
    _check(lib().ds_expand_shift_weights(ctypes.byref(w), _ptr(expanded), expanded_bytes, _stream(stream)))


def ds_linear_shift(x, w: ds_weights, bias, y, M: int, K: int, N: int, flags: int = 0, amax_io=None,
                    stream=None) -> None:
    _check(lib().ds_linear_shift(_ptr(x), ctypes.byref(w), _ptr(bias), _ptr(y), M, K, N, flags,
                                 _ptr(amax_io), _stream(stream)))


def ds_conv2d_shift(x, w: ds_weights, bias, residual, y, N, C, H, W, K, R, S, stride_h, stride_w,
                    pad_h, pad_w, flags: int = 0, amax_io=None, stream=None) -> None:
    _check(lib().ds_conv2d_shift(_ptr(x), ctypes.byref(w), _ptr(bias), _ptr(residual), _ptr(y), N, C, H,
                                 W, K, R, S, stride_h, stride_w, pad_h, pad_w, flags, _ptr(amax_io),
                                 _stream(stream)))


def ds_linear_shift_static_scratch(x, w: ds_weights, bias, y, M: int, K: int, N: int, flags: int = 0,
                                   stream=None) -> None:
    """ds_linear_shift with its scratch in the library's static device array (no allocation)."""
    _check(lib().ds_linear_shift_static_scratch(_ptr(x), ctypes.byref(w), _ptr(bias), _ptr(y), M, K, N, flags,
                                                _stream(stream)))


def ds_shift_forward_workspace_bytes(layers, n: int, batch: int) -> int:
    return int(lib().ds_shift_forward_workspace_bytes(layers, n, batch))


def ds_shift_forward(layers, n: int, x, y, ws, ws_bytes: int, batch: int, stream=None) -> None:
    _check(lib().ds_shift_forward(layers, n, _ptr(x), _ptr(y), _ptr(ws), ws_bytes, batch, _stream(stream)))


def ds_bf16_weight_bytes(n_out: int, k_red: int) -> int:
    return int(lib().ds_bf16_weight_bytes(n_out, k_red))


def ds_expand_shift_weights_bf16(w: ds_weights, buf, nbytes: int, stream=None) -> None:
    _check(lib().ds_expand_shift_weights_bf16(ctypes.byref(w), _ptr(buf), nbytes, _stream(stream)))


def ds_linear_shift_bf16(x, w: ds_weights, bias, y, M: int, K: int, N: int, flags: int = 0, stream=None) -> None:
    _check(lib().ds_linear_shift_bf16(_ptr(x), ctypes.byref(w), _ptr(bias), _ptr(y), M, K, N, flags, _stream(stream)))


def ds_bf16_fault_flag() -> int:
    return int(lib().ds_bf16_fault_flag())


def ds_bf16_set_wait_limit(cycles: int) -> None:
    lib().ds_bf16_set_wait_limit(cycles)


def ds_specialize_conv2d_shift(s, p, K: int, C: int, R: int, S: int, stride: int, pad: int) -> int:
    """s, p: HOST int8 arrays [K][C][R][S] (numpy, C-contiguous).  Returns the handle (an address)."""
    import numpy as np
    s = np.ascontiguousarray(s, dtype=np.int8)
    p = np.ascontiguousarray(p, dtype=np.int8)
    if s.size != K * C * R * S or p.size != K * C * R * S:
        raise DsError(DS_ERR_SHAPE, "codes must hold K*C*R*S values")
    out = ctypes.c_void_p()
    _check(lib().ds_specialize_conv2d_shift(s.ctypes.data, p.ctypes.data, K, C, R, S, stride, pad,
                                            ctypes.byref(out)))
    return int(out.value)


def ds_conv2d_shift_specialized(h: int, x, bias, residual, y, N: int, H: int, W: int, flags: int = 0,
                                amax_io=None, stream=None) -> None:
    _check(lib().ds_conv2d_shift_specialized(h, _ptr(x), _ptr(bias), _ptr(residual), _ptr(y), N, H, W, flags,
                                             _ptr(amax_io), _stream(stream)))


def ds_specialized_destroy(h: int) -> None:
    lib().ds_specialized_destroy(h)


def ds_absmax(x, n: int, amax, stream=None) -> None:
    _check(lib().ds_absmax(_ptr(x), n, _ptr(amax), _stream(stream)))


def ds_packed_weight_bytes_backward(K: int, C: int, R: int, S: int, stride_h: int = 1, stride_w: int = 1) -> int:
    return int(lib().ds_packed_weight_bytes_backward(K, C, R, S, stride_h, stride_w))


def ds_pack_shift_weights_backward(s, p, K: int, C: int, R: int, S: int, stride_h: int, stride_w: int, packed,
                                   packed_bytes: int, stream=None):
    """Returns a ctypes array of stride_h * stride_w descriptors (one per tap phase)."""
    descs = (ds_weights * (stride_h * stride_w))()
    _check(lib().ds_pack_shift_weights_backward(_ptr(s), _ptr(p), K, C, R, S, stride_h, stride_w, _ptr(packed),
                                                packed_bytes, descs, _stream(stream)))
    return descs


def ds_linear_shift_backward_x(dy, w: ds_weights, dx, M: int, K: int, N: int, flags: int = 0, amax_io=None,
                               stream=None) -> None:
    _check(lib().ds_linear_shift_backward_x(_ptr(dy), ctypes.byref(w), _ptr(dx), M, K, N, flags, _ptr(amax_io),
                                            _stream(stream)))


def ds_conv2d_shift_backward_x(dy, w, dx, N, C, H, W, K, R, S, stride_h, stride_w, pad_h, pad_w,
                               flags: int = 0, amax_io=None, stream=None) -> None:
    """w: the ctypes descriptor array of ds_pack_shift_weights_backward (or one descriptor for stride 1)."""
    ref = w if isinstance(w, ctypes.Array) else ctypes.byref(w)
    _check(lib().ds_conv2d_shift_backward_x(_ptr(dy), ref, _ptr(dx), N, C, H, W, K, R, S, stride_h,
                                            stride_w, pad_h, pad_w, flags, _ptr(amax_io), _stream(stream)))


def ds_quantize_shift_weights(w, n: int, p_min: int, s, p, stream=None) -> None:
    _check(lib().ds_quantize_shift_weights(_ptr(w), n, p_min, _ptr(s), _ptr(p), _stream(stream)))


def ds_quantize_q16(x, n: int, q, stream=None) -> None:
    _check(lib().ds_quantize_q16(_ptr(x), n, _ptr(q), _stream(stream)))


# ---------------------------------------------------------------------------
# Tensor-level helpers (allocate outputs with torch, then call the ABI)
# ---------------------------------------------------------------------------

class PackedShiftWeights:
    """A packed blob (device uint8 tensor) plus its ds_weights descriptor and,
    optionally, the expanded execution layout (device int32 tensor)."""

    def __init__(self, blob, desc: ds_weights):
        self.blob = blob
        self.desc = desc
        self.expanded = None
        self.bf16 = None

    @property
    def n_out(self) -> int:
        return int(self.desc.n_out)

    @property
    def k_red(self) -> int:
        return int(self.desc.k_red)


def expand_shift_weights(w: PackedShiftWeights, stream=None) -> PackedShiftWeights:
    """Adds the expanded execution layout to packed weights (8 bytes per weight)."""
    import torch
    nbytes = ds_expanded_weight_bytes(w.n_out, w.k_red)
    buf = torch.empty(nbytes // 4, dtype=torch.int32, device=w.blob.device)
    ds_expand_shift_weights(w.desc, buf, nbytes, stream)
    w.expanded = buf
    return w


def expand_shift_weights_bf16(w: PackedShiftWeights, stream=None) -> PackedShiftWeights:
    """Adds the bf16 weight layout W = s * 2^p used by the float variant."""
    import torch
    nbytes = ds_bf16_weight_bytes(w.n_out, w.k_red)
    buf = torch.empty(nbytes, dtype=torch.uint8, device=w.blob.device)
    ds_expand_shift_weights_bf16(w.desc, buf, nbytes, stream)
    w.bf16 = buf
    return w


def linear_shift_bf16(x, w: PackedShiftWeights, bias=None, relu: bool = False, out=None, stream=None):
    """Float LinearShift: fp32 y = bias + x @ W^T (ReLU) for bf16 x [M, K] on the tensor cores."""
    import torch
    _need(x, "x", torch.bfloat16)
    if x.dim() != 2:
        raise ValueError("x must be [M, K]")
    M, K = x.shape
    N = w.n_out
    _need(bias, "bias", torch.float32, (N,))
    _need(out, "out", torch.float32, (M, N))
    _on_one_gpu(x=x, bias=bias, out=out)
    y = out if out is not None else torch.empty((M, N), dtype=torch.float32, device=x.device)
    ds_linear_shift_bf16(x, w.desc, bias, y, M, K, N, DS_RELU if relu else 0, stream)
    return y


class PackedBackwardWeights:
    """The input-gradient codes of one layer: a device blob holding one packed matrix per tap phase,
    the ctypes array of their descriptors, and optionally each phase's expanded layout."""

    def __init__(self, blob, descs, stride):
        self.blob = blob
        self.desc = descs  # pass to ds_conv2d_shift_backward_x; descs[0] to ds_linear_shift_backward_x
        self.stride = stride
        self.expanded = []

    def expand(self, stream=None):
        import torch
        for d in self.desc:
            if d.k_red == 0:
                continue
            nbytes = ds_expanded_weight_bytes(d.n_out, d.k_red)
            buf = torch.empty(nbytes // 4, dtype=torch.int32, device=self.blob.device)
            ds_expand_shift_weights(d, buf, nbytes, stream)
            self.expanded.append(buf)
        return self


def pack_shift_weights_backward(s, p, stride=(1, 1), stream=None, expand: bool = False) -> PackedBackwardWeights:
    """Packs the input-gradient codes (Eq. 7 footnote: rot180, channels swapped, split into the tap phases
    of a strided layer) of forward int8 codes [K, C, R, S] or [N, K] (device)."""
    import torch
    if s.device.type != "cuda" or p.device.type != "cuda":
        raise ValueError("codes must be CUDA tensors")
    dims = tuple(s.shape) + (1,) * (4 - s.dim())
    K, C, R, S = dims
    sh, sw = stride
    s4 = s.reshape(dims).to(torch.int8).contiguous()
    p4 = p.reshape(dims).to(torch.int8).contiguous()
    nbytes = ds_packed_weight_bytes_backward(K, C, R, S, sh, sw)
    if nbytes == 0:
        raise DsError(DS_ERR_SHAPE, "invalid code matrix shape")
    blob = torch.empty(nbytes, dtype=torch.uint8, device=s.device)
    descs = ds_pack_shift_weights_backward(s4, p4, K, C, R, S, sh, sw, blob, nbytes, stream)
    w = PackedBackwardWeights(blob, descs, (sh, sw))
    if expand:
        w.expand(stream)
    return w


def quantize_shift_weights(w, p_min: int = -15, stream=None):
    """DeepShift-Q codes (Eq. 4-6) of a float32 CUDA weight tensor: int8 tensors s, p of w's shape."""
    import torch
    if w.device.type != "cuda" or w.dtype != torch.float32:
        raise ValueError("w must be a float32 CUDA tensor")
    w = w.contiguous()
    s = torch.empty(w.shape, dtype=torch.int8, device=w.device)
    p = torch.empty(w.shape, dtype=torch.int8, device=w.device)
    ds_quantize_shift_weights(w, w.numel(), p_min, s, p, stream)
    return s, p


def quantize_q16(x, out=None, stream=None):
    """Q16.16 int32 tensor of a float32 CUDA tensor (Sec. 4: ties to even, saturating, NaN -> 0)."""
    import torch
    if x.device.type != "cuda" or x.dtype != torch.float32:
        raise ValueError("x must be a float32 CUDA tensor")
    x = x.contiguous()
    q = out if out is not None else torch.empty(x.shape, dtype=torch.int32, device=x.device)
    ds_quantize_q16(x, x.numel(), q, stream)
    return q


def pack_shift_weights5(s, p, stream=None):
    """Stores int8 codes [n_out, ...] (every shift of a nonzero weight in [-14, 0]) in a new 5-bit blob (device
    uint8 tensor)."""
    import torch
    _need(s, "s", torch.int8)
    _need(p, "p", torch.int8, tuple(s.shape))
    _on_one_gpu(s=s, p=p)
    n_out, k_red = s.shape[0], s[0].numel()
    nbytes = ds_packed5_weight_bytes(n_out, k_red)
    blob = torch.empty(nbytes, dtype=torch.uint8, device=s.device)
    ds_pack_shift_weights5(s, p, n_out, k_red, blob, nbytes, stream)
    return blob


def unpack_shift_weights5(blob, n_out: int, k_red: int, stream=None):
    """Reads a 5-bit blob back into int8 codes (s, p) of shape [n_out, k_red] (p = 0 where s = 0)."""
    import torch
    _need(blob, "blob", torch.uint8)
    s = torch.empty((n_out, k_red), dtype=torch.int8, device=blob.device)
    p = torch.empty((n_out, k_red), dtype=torch.int8, device=blob.device)
    ds_unpack_shift_weights5(blob, blob.numel(), n_out, k_red, s, p, stream)
    return s, p


def pack_shift_weights(s, p, stream=None, expand: bool = False) -> PackedShiftWeights:
    """Packs int8 sign/shift code tensors [n_out, ...] (device) into a new blob;
    with expand=True also builds the expanded execution layout."""
    import torch
    if s.device.type != "cuda" or p.device.type != "cuda":
        raise ValueError("codes must be CUDA tensors")
    n_out = s.shape[0]
    k_red = s[0].numel() if n_out else 0
    s2 = s.reshape(n_out, k_red).to(torch.int8).contiguous()
    p2 = p.reshape(n_out, k_red).to(torch.int8).contiguous()
    nbytes = ds_packed_weight_bytes(n_out, k_red)
    if nbytes == 0:
        raise DsError(DS_ERR_SHAPE, "invalid code matrix shape")
    blob = torch.empty(nbytes, dtype=torch.uint8, device=s.device)
    desc = ds_pack_shift_weights(s2, p2, n_out, k_red, blob, nbytes, stream)
    w = PackedShiftWeights(blob, desc)
    if expand:
        expand_shift_weights(w, stream)
    return w


def linear_shift(x, w: PackedShiftWeights, bias=None, relu: bool = False, amax_io=None, flags: int = 0,
                 out=None, stream=None):
    """y = sat32(bias + sum s * (x >> -p)) [ReLU] for int32 x [M, K] on the GPU."""
    import torch
    _need(x, "x", torch.int32)
    if x.dim() != 2:
        raise ValueError("x must be [M, K]")
    M, K = x.shape
    N = w.n_out
    _need(bias, "bias", torch.int32, (N,))
    _need(out, "out", torch.int32, (M, N))
    _need_amax(amax_io)
    _on_one_gpu(x=x, bias=bias, out=out, amax_io=amax_io)
    y = out if out is not None else torch.empty((M, N), dtype=torch.int32, device=x.device)
    ds_linear_shift(x, w.desc, bias, y, M, K, N, flags | (DS_RELU if relu else 0), amax_io, stream)
    return y


def conv2d_shift(x, w: PackedShiftWeights, kernel_size, bias=None, stride=(1, 1), padding=(0, 0),
                 relu: bool = False, residual=None, amax_io=None, flags: int = 0, out=None, stream=None):
    """ConvShift forward on int32 NCHW x; w packed from OIHW codes."""
    import torch
    _need(x, "x", torch.int32)
    if x.dim() != 4:
        raise ValueError("x must be [N, C, H, W]")
    N, C, H, W = x.shape
    R, S = kernel_size
    K = w.n_out
    OH = (H + 2 * padding[0] - R) // stride[0] + 1
    OW = (W + 2 * padding[1] - S) // stride[1] + 1
    _need(bias, "bias", torch.int32, (K,))
    _need(residual, "residual", torch.int32, (N, K, OH, OW))
    _need(out, "out", torch.int32, (N, K, OH, OW))
    _need_amax(amax_io)
    _on_one_gpu(x=x, bias=bias, residual=residual, out=out, amax_io=amax_io)
    y = out if out is not None else torch.empty((N, K, OH, OW), dtype=torch.int32, device=x.device)
    f = flags | (DS_RELU if relu else 0) | (DS_RESIDUAL if residual is not None else 0)
    ds_conv2d_shift(x, w.desc, bias, residual, y, N, C, H, W, K, R, S, stride[0], stride[1], padding[0],
                    padding[1], f, amax_io, stream)
    return y
