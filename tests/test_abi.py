"""Host-side checks of the C ABI: the library loads without a GPU, exports
every entry point its header declares, and rejects bad arguments before it
touches CUDA."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import deepshift_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def ds():
    from paper_1905_13298_gb300 import build
    build.build_library()
    import paper_1905_13298_gb300 as ds
    ds.lib()
    return ds


def _declared_functions():
    names = set()
    for hdr in os.listdir(os.path.join(ROOT, "include")):
        if not hdr.endswith(".h"):
            continue
        text = open(os.path.join(ROOT, "include", hdr)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        names |= set(re.findall(r"\b(ds_\w+)\s*\(", text))
    return sorted(names)


def test_every_declared_symbol_is_exported(ds):
    names = _declared_functions()
    assert "ds_linear_shift" in names and "ds_conv2d_shift" in names and "ds_pack_shift_weights" in names
    L = ds.lib()
    for n in names:
        assert hasattr(L, n), n
        assert n in ds._SIGNATURES or n.startswith("ds_"), n


def test_binding_covers_every_declared_symbol(ds):
    for n in _declared_functions():
        assert n in ds._SIGNATURES, f"{n} has no ctypes signature in the binding"


def test_packed_bytes_match_documented_layout(ds):
    for n_out, k_red in [(1, 1), (64, 576), (512, 784), (4096, 4096), (1000, 512), (3, 33)]:
        assert ds.ds_packed_weight_bytes(n_out, k_red) == O.blob_layout(n_out, k_red)["total"]
    assert ds.ds_packed_weight_bytes(0, 5) == 0
    assert ds.ds_packed_weight_bytes(5, -1) == 0


def test_struct_layouts_match_library(ds):
    L = ds.lib()
    assert L.ds_abi_struct_size(0) == ctypes.sizeof(ds.ds_weights) == 96
    assert L.ds_abi_struct_size(1) == ctypes.sizeof(ds.ds_layer)
    assert L.ds_abi_struct_size(7) == 0
    assert ds.ds_weights.packed.offset == 32


def test_validation_happens_before_cuda(ds):
    L = ds.lib()
    w = ds.ds_weights()
    # NULL pointers
    assert L.ds_linear_shift(None, ctypes.byref(w), None, None, 1, 1, 1, 0, None, None) == ds.DS_ERR_INVALID_ARG
    assert "NULL" in ds.ds_last_error()
    # bad shapes
    assert L.ds_linear_shift(16, ctypes.byref(w), None, 4096, 0, 1, 1, 0, None, None) == ds.DS_ERR_SHAPE
    assert L.ds_conv2d_shift(16, ctypes.byref(w), None, None, 4096, 1, 1, 3, 3, 1, 3, 3, 0, 1, 1, 1, 0, None,
                             None) == ds.DS_ERR_SHAPE
    # misaligned pointers
    assert L.ds_linear_shift(20, ctypes.byref(w), None, 4096, 1, 1, 1, 0, None, None) == ds.DS_ERR_ALIGNMENT
    # unfilled descriptor
    assert L.ds_linear_shift(16, ctypes.byref(w), None, 4096, 1, 1, 1, 0, None, None) == ds.DS_ERR_INVALID_ARG
    assert "ds_pack_shift_weights" in ds.ds_last_error()
    # unknown flags, residual on FC, amax flags without a buffer
    assert L.ds_linear_shift(16, ctypes.byref(w), None, 4096, 1, 1, 1, 1 << 20, None, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_linear_shift(16, ctypes.byref(w), None, 4096, 1, 1, 1, ds.DS_RESIDUAL, None, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_linear_shift(16, ctypes.byref(w), None, 4096, 1, 1, 1, ds.DS_AMAX_IN, None, None) == ds.DS_ERR_INVALID_ARG
    # pack: buffer too small, misaligned blob
    d = ds.ds_weights()
    assert L.ds_pack_shift_weights(16, 16, 4, 4, 256, 10, ctypes.byref(d), None) == ds.DS_ERR_BUFFER_TOO_SMALL
    assert L.ds_pack_shift_weights(16, 16, 4, 4, 272, 4096, ctypes.byref(d), None) == ds.DS_ERR_ALIGNMENT
    assert L.ds_pack_shift_weights(16, 16, 0, 4, 256, 4096, ctypes.byref(d), None) == ds.DS_ERR_SHAPE
    assert d.magic == 0
    # descriptor/dims mismatch
    w2 = ds.ds_weights(magic=ds.DS_WEIGHTS_MAGIC, format=ds.DS_FORMAT_PLANES6, n_out=8, k_red=8, n_chunks=1,
                       packed=256, packed_bytes=ds.ds_packed_weight_bytes(8, 8))
    assert L.ds_linear_shift(16, ctypes.byref(w2), None, 4096, 2, 9, 8, 0, None, None) == ds.DS_ERR_SHAPE
    # overlap of x and y
    assert L.ds_linear_shift(4096, ctypes.byref(w2), None, 4096, 2, 8, 8, 0, None, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_absmax(None, 4, 16, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_absmax(16, 0, 16, None) == ds.DS_ERR_SHAPE
    # input-gradient calls: bad flags (ReLU / residual / bias-like flags do not apply), shapes, buffers
    assert L.ds_linear_shift_backward_x(16, ctypes.byref(w), 4096, 1, 1, 1, ds.DS_RELU, None, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_conv2d_shift_backward_x(16, ctypes.byref(w), 4096, 1, 1, 3, 3, 1, 3, 3, 1, 1, 1, 1,
                                        ds.DS_RESIDUAL, None, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_conv2d_shift_backward_x(None, ctypes.byref(w), 4096, 1, 1, 3, 3, 1, 3, 3, 1, 1, 1, 1, 0, None,
                                        None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_conv2d_shift_backward_x(16, ctypes.byref(w), 4096, 1, 1, 3, 3, 1, 3, 3, 0, 1, 1, 1, 0, None,
                                        None) == ds.DS_ERR_SHAPE
    w4 = (ds.ds_weights * 4)()
    assert L.ds_conv2d_shift_backward_x(16, w4, 4096, 1, 1, 3, 3, 1, 3, 3, 2, 2, 1, 1, 0, None,
                                        None) == ds.DS_ERR_INVALID_ARG  # unfilled descriptors
    d4 = (ds.ds_weights * 4)()
    assert L.ds_pack_shift_weights_backward(16, 16, 4, 4, 3, 3, 1, 1, 256, 10, d4, None) == ds.DS_ERR_BUFFER_TOO_SMALL
    assert L.ds_pack_shift_weights_backward(16, 16, 4, 0, 3, 3, 1, 1, 256, 4096, d4, None) == ds.DS_ERR_SHAPE
    assert L.ds_pack_shift_weights_backward(16, 16, 4, 4, 3, 3, 0, 1, 256, 4096, d4, None) == ds.DS_ERR_SHAPE
    assert L.ds_pack_shift_weights_backward(16, 16, 4, 4, 1, 1, 1, 1, 272, 4096, d4, None) == ds.DS_ERR_ALIGNMENT
    # phase sizes: a 3x3 / 2 layer has phases of 2x2, 2x1, 1x2, 1x1 taps; a 1x1 / 2 layer one non-empty phase
    ph = [ds.ds_packed_weight_bytes(5, 4 * t) for t in (4, 2, 2, 1)]
    assert ds.ds_packed_weight_bytes_backward(4, 5, 3, 3, 2, 2) == sum((b + 255) // 256 * 256 for b in ph)
    assert ds.ds_packed_weight_bytes_backward(4, 5, 1, 1, 2, 2) == (ds.ds_packed_weight_bytes(5, 4) + 255) // 256 * 256
    assert ds.ds_packed_weight_bytes_backward(4, 5, 3, 3, 0, 2) == 0
    # quantizers: NULL pointers, p_min range, sizes, alignment
    assert L.ds_quantize_shift_weights(None, 4, -15, 16, 32, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_quantize_shift_weights(16, 4, -16, 16, 32, None) == ds.DS_ERR_INVALID_ARG
    assert "p_min" in ds.ds_last_error()
    assert L.ds_quantize_shift_weights(16, 4, 1, 16, 32, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_quantize_shift_weights(16, 0, -15, 16, 32, None) == ds.DS_ERR_SHAPE
    assert L.ds_quantize_shift_weights(18, 4, -15, 16, 32, None) == ds.DS_ERR_ALIGNMENT
    assert L.ds_quantize_q16(16, 4, None, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_quantize_q16(16, -1, 32, None) == ds.DS_ERR_SHAPE
    assert L.ds_quantize_q16(16, 4, 34, None) == ds.DS_ERR_ALIGNMENT


def _descriptor(ds, n_out, k_red):
    """A descriptor that passes the host checks for an (n_out, k_red) code matrix (its blob is never read)."""
    return ds.ds_weights(magic=ds.DS_WEIGHTS_MAGIC, format=ds.DS_FORMAT_PLANES6, n_out=n_out, k_red=k_red,
                         n_chunks=(k_red + 31) // 32, packed=256, packed_bytes=ds.ds_packed_weight_bytes(n_out, k_red))


def test_size_arithmetic_never_wraps(ds):
    """Sizes formed from caller dimensions are bounded before they can overflow 64 bits: absurd dimensions give
    a status, never a wrapped size or a check done on wrapped numbers."""
    L = ds.lib()
    # size queries: each dimension in range but the product too large gives 0, not a wrapped size
    assert ds.ds_packed_weight_bytes(1 << 20, 1 << 28) > 0            # 2^48 codes: the largest accepted
    assert ds.ds_packed_weight_bytes(1 << 20, (1 << 28) + 1) == 0
    assert ds.ds_packed_weight_bytes(1 << 31, 1 << 40) == 0
    assert ds.ds_expanded_weight_bytes(1 << 31, 1 << 36) == 0
    assert ds.ds_bf16_weight_bytes(1 << 31, 1 << 36) == 0
    assert ds.ds_expanded_weight_bytes(64, 1024) == 2 * 1024 * 64 * 4
    # a forged descriptor outside the range is refused before its layout is computed
    n_big = 65535 * 64                                                 # the widest FC layer accepted
    big = ds.ds_weights(magic=ds.DS_WEIGHTS_MAGIC, format=ds.DS_FORMAT_PLANES6, n_out=n_big, k_red=1 << 40,
                        n_chunks=1 << 35, packed=256, packed_bytes=(1 << 64) - 1)
    assert L.ds_linear_shift(16, ctypes.byref(big), None, 4096, 1, 1 << 40, n_big, 0, None,
                             None) == ds.DS_ERR_UNSUPPORTED
    assert "supported range" in ds.ds_last_error()
    # FC: M x K x 4 bytes = 2^72 would wrap to 0
    w = _descriptor(ds, 1, 1 << 30)
    assert L.ds_linear_shift(16, ctypes.byref(w), None, 1 << 48, 1 << 40, 1 << 30, 1, 0, None,
                             None) == ds.DS_ERR_UNSUPPORTED
    assert "2^62" in ds.ds_last_error()
    # conv: 2 x pad overflows int32; the padded extent is formed in 64 bits
    w1 = _descriptor(ds, 1, 9)
    for pad in ((1 << 30) + 5, (1 << 31) - 1):
        assert L.ds_conv2d_shift(16, ctypes.byref(w1), None, None, 1 << 40, 1, 1, 8, 8, 1, 3, 3, 1, 1, pad, 0, 0,
                                 None, None) == ds.DS_ERR_UNSUPPORTED
        assert "padded" in ds.ds_last_error()
        assert L.ds_conv2d_shift_backward_x(16, ctypes.byref(w1), 1 << 40, 1, 1, 8, 8, 1, 3, 3, 2, 2, pad, 0, 0,
                                            None, None) == ds.DS_ERR_UNSUPPORTED
    # conv: an image past the kernels' 32-bit per-image indexing, and a batch past 2^62 bytes
    wc = _descriptor(ds, 1, (1 << 31) - 1)
    assert L.ds_conv2d_shift(16, ctypes.byref(wc), None, None, 1 << 40, 1, (1 << 31) - 1, 2, 2, 1, 1, 1, 1, 1, 0,
                             0, 0, None, None) == ds.DS_ERR_UNSUPPORTED
    assert "image too large" in ds.ds_last_error()
    wk = _descriptor(ds, 1 << 16, 16)
    assert L.ds_conv2d_shift(16, ctypes.byref(wk), None, None, 1 << 40, (1 << 31) - 1, 16, 1 << 7, 1 << 7, 1 << 16,
                             1, 1, 1, 1, 0, 0, 0, None, None) == ds.DS_ERR_UNSUPPORTED
    assert "2^62" in ds.ds_last_error()


def test_program_size_arithmetic_never_wraps(ds):
    """The layer-program planner applies the same bounds: the padded extent, the per-image limits and the
    workspace size are checked without overflow, and the failing layer is named."""
    L = ds.lib()

    def program(pad=0, K=4, H=32, batch=2):
        w = _descriptor(ds, K, 1)
        layers = (ds.ds_layer * 2)()
        conv, pool = layers[0], layers[1]
        conv.op, conv.in_, conv.aux, conv.out = ds.DS_OP_CONV, 0, -1, 2
        conv.C, conv.H, conv.W, conv.K, conv.R, conv.S, conv.stride, conv.pad = 1, H, H, K, 1, 1, 1, pad
        conv.w = ctypes.pointer(w)
        OH = H + 2 * pad if pad < (1 << 20) else 1  # the conv is refused before the pool is looked at
        pool.op, pool.in_, pool.aux, pool.out = ds.DS_OP_MAXPOOL, 2, -1, 1
        pool.C, pool.H, pool.W, pool.K, pool.R, pool.S, pool.stride, pool.pad = K, OH, OH, 0, 1, 1, 1, 0
        return layers, batch, w

    layers, batch, _w = program()
    assert ds.ds_shift_forward_workspace_bytes(layers, 2, batch) > 2 * 4 * 32 * 32 * 4
    layers, batch, _w = program(pad=(1 << 30) + 5)
    assert ds.ds_shift_forward_workspace_bytes(layers, 2, batch) == 0
    assert ds.ds_last_error().startswith("layer 0:") and "padded" in ds.ds_last_error()
    # 2^16 channels of 2^20 outputs per image is 2^38 bytes; 2^24 images of that pass 2^62
    layers, batch, _w = program(K=1 << 16, H=1 << 10, batch=1 << 24)
    assert ds.ds_shift_forward_workspace_bytes(layers, 2, batch) == 0
    assert "2^62" in ds.ds_last_error()
    layers, batch, _w = program(K=1 << 16, H=1 << 10, batch=1 << 10)
    assert ds.ds_shift_forward_workspace_bytes(layers, 2, batch) >= (1 << 48)
    # the network input itself: non-positive or past the per-image limit
    layers, batch, _w = program(H=1 << 16)
    assert ds.ds_shift_forward_workspace_bytes(layers, 2, batch) == 0
    assert "too large" in ds.ds_last_error()


def test_tensor_helpers_refuse_mismatched_tensors(ds):
    """The tensor-level helpers check dtype, layout, shape and device before the ABI sees an address."""
    import torch
    w = ds.PackedShiftWeights(None, _descriptor(ds, 4, 8))
    x = torch.zeros((3, 8), dtype=torch.int32)
    i32 = lambda *shape: torch.zeros(shape, dtype=torch.int32)
    wc = ds.PackedShiftWeights(None, _descriptor(ds, 6, 2 * 3 * 3))
    xc = i32(1, 2, 5, 5)
    conv = lambda **kw: ds.conv2d_shift(xc if "x" not in kw else kw.pop("x"), wc, (3, 3), padding=(1, 1), **kw)
    xb = torch.zeros((3, 8), dtype=torch.bfloat16)
    cases = [
        (lambda: ds.linear_shift(x.float(), w), "int32"),
        (lambda: ds.linear_shift(i32(8, 3).t(), w), "contiguous"),
        (lambda: ds.linear_shift(x[0], w), "[M, K]"),
        (lambda: ds.linear_shift(x, w, bias=i32(5)), "shape"),
        (lambda: ds.linear_shift(x, w, bias=torch.zeros(4, dtype=torch.int64)), "int32"),
        (lambda: ds.linear_shift(x, w, out=i32(3, 5)), "shape"),
        (lambda: ds.linear_shift(x, w, amax_io=i32(1)), "at least 2"),
        (lambda: ds.linear_shift(x, w, bias=i32(4), out=i32(3, 4), amax_io=i32(2)), "CUDA"),
        (lambda: conv(x=i32(2, 5, 5)), "[N, C, H, W]"),
        (lambda: conv(bias=i32(5)), "shape"),
        (lambda: conv(residual=i32(1, 6, 4, 4)), "shape"),
        (lambda: conv(out=torch.zeros((1, 6, 5, 5), dtype=torch.float32)), "int32"),
        (lambda: conv(bias=i32(6), residual=i32(1, 6, 5, 5), out=i32(1, 6, 5, 5)), "CUDA"),
        (lambda: ds.linear_shift_bf16(xb.float(), w), "bfloat16"),
        (lambda: ds.linear_shift_bf16(xb, w, bias=i32(4)), "float32"),
        (lambda: ds.linear_shift_bf16(xb, w, bias=torch.zeros(4)), "CUDA"),
    ]
    for call, what in cases:
        with pytest.raises(ValueError, match=re.escape(what)):
            call()


def test_last_error_is_per_thread(ds):
    """ds_last_error is thread-local: threads that fail different checks each read their own message."""
    import threading
    L = ds.lib()
    w = ds.ds_weights()
    calls = {
        "NULL": lambda: L.ds_linear_shift(None, ctypes.byref(w), None, None, 1, 1, 1, 0, None, None),
        "n must be positive": lambda: L.ds_absmax(16, 0, 16, None),
        "p_min": lambda: L.ds_quantize_shift_weights(16, 4, -16, 16, 32, None),
    }
    wrong = []

    def worker(expect, call):
        for _ in range(2000):
            call()
            msg = ds.ds_last_error()
            if expect not in msg:
                wrong.append((expect, msg))
                return

    threads = [threading.Thread(target=worker, args=kv) for kv in calls.items()]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not wrong, wrong[:3]


def test_plain_c_client_builds_and_runs(tmp_path, ds):
    """The header is C99 and the library links into a plain C program (no Python, no torch): size queries and
    argument validation answer as documented without a GPU (tests/c_abi_client.c)."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lib_dir = os.path.dirname(ds.LIB_PATH)
    exe = str(tmp_path / "c_abi_client")
    cmd = [cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I", os.path.join(ROOT, "include"),
           os.path.join(ROOT, "tests", "c_abi_client.c"), "-o", exe, "-L", lib_dir, "-ldeepshift",
           f"-Wl,-rpath,{lib_dir}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    env = dict(os.environ)
    env["LD_LIBRARY_PATH"] = os.pathsep.join(p for p in ("/usr/local/cuda/lib64", env.get("LD_LIBRARY_PATH")) if p)
    r = subprocess.run([exe], capture_output=True, text=True, env=env, timeout=60)
    assert r.returncode == 0, f"check {r.returncode} failed: {r.stdout}{r.stderr}"
    assert "c abi client ok" in r.stdout


def test_no_cpu_fallback_without_library(tmp_path, monkeypatch, ds):
    """The binding refuses to run when the shared library is missing."""
    monkeypatch.setattr(ds, "_lib", None)
    monkeypatch.setattr(ds, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(ImportError):
        ds.lib()


def test_forward_program_validation_without_gpu(ds):
    """Programs are validated on the host: bad shapes and slots are rejected before anything runs."""
    from paper_1905_13298_gb300 import networks as PN
    specs, shapes = PN.resnet_program("resnet18")
    ws = [ds.ds_weights(magic=ds.DS_WEIGHTS_MAGIC, format=ds.DS_FORMAT_PLANES6, n_out=shp[0],
                        k_red=int(np.prod(shp[1:])), n_chunks=(int(np.prod(shp[1:])) + 31) // 32, packed=4096,
                        packed_bytes=ds.ds_packed_weight_bytes(shp[0], int(np.prod(shp[1:]))))
          for shp in shapes]
    layers = (ds.ds_layer * len(specs))()
    for i, sp in enumerate(specs):
        L = layers[i]
        L.op, L.in_, L.aux, L.out = sp.op, sp.inp, sp.aux, sp.out
        L.C, L.H, L.W, L.K, L.R, L.S, L.stride, L.pad, L.flags = (sp.C, sp.H, sp.W, sp.K, sp.R, sp.S, sp.stride,
                                                                  sp.pad, sp.flags)
        if sp.param >= 0:
            L.w = ctypes.pointer(ws[sp.param])
    n = len(specs)
    good = ds.ds_shift_forward_workspace_bytes(layers, n, 32)
    # the largest slot is the stem output 64 x 112 x 112 per image
    assert good >= 32 * 64 * 112 * 112 * 4
    assert ds.ds_shift_forward_workspace_bytes(layers, n, 0) == 0
    layers[3].C += 1                   # a conv whose input channels disagree with its producer
    assert ds.ds_shift_forward_workspace_bytes(layers, n, 32) == 0
    assert "input" in ds.ds_last_error()
    layers[3].C -= 1
    saved = layers[n - 1].out
    layers[n - 1].out = 7              # nobody writes the output slot
    assert ds.ds_shift_forward_workspace_bytes(layers, n, 32) == 0
    layers[n - 1].out = saved
    assert ds.ds_shift_forward_workspace_bytes(layers, n, 32) == good
    L = ds.lib()
    assert L.ds_shift_forward(layers, n, 16, 16, 256, good - 1, 32, None) == ds.DS_ERR_BUFFER_TOO_SMALL


def test_network_refuses_mismatched_inputs_and_biases(ds):
    """ShiftNetwork checks its biases before packing and its input against the program before a launch:
    an input with fewer images than the program was built for would otherwise be read past its end."""
    import torch
    from paper_1905_13298_gb300 import networks as PN
    specs, shapes = PN.resnet_program("resnet18", 32, 32)
    s = np.zeros(shapes[0], np.int8)
    for bias, what in ((np.zeros(63, np.int32), "bias 0"), (np.zeros(64, np.float32), "bias 0"),
                       (np.full(64, 1 << 31, np.int64), "int32")):
        with pytest.raises(ValueError, match=what):
            PN.ShiftNetwork(specs, [(s, s, bias)], batch=2, device="cpu")
    with pytest.raises(ValueError, match="CUDA"):   # an in-range int64 bias passes; packing wants the GPU
        PN.ShiftNetwork(specs, [(s, s, np.zeros(64, np.int64))], batch=2, device="cpu")
    net = object.__new__(PN.ShiftNetwork)
    net.specs, net.batch = specs, 2
    net.in_shape, net.out_shape = (2, 3, 32, 32), (2, 1000, 1, 1)
    net.workspace = torch.empty(256, dtype=torch.uint8)
    x = torch.zeros(net.in_shape, dtype=torch.int32)
    cases = [(lambda: net.forward(torch.zeros((1, 3, 32, 32), dtype=torch.int32)), "shape"),
             (lambda: net.forward(x.float()), "int32"),
             (lambda: net.forward(torch.zeros((2, 3, 32, 32), dtype=torch.int32).transpose(2, 3)), "contiguous"),
             (lambda: net.forward(x, torch.zeros(net.out_shape)), "y must be"),
             (lambda: net.forward(x, torch.zeros((2, 999), dtype=torch.int32)), "y must be"),
             (lambda: net.forward(x, torch.zeros(net.out_shape, dtype=torch.int32)), "CUDA")]
    for call, what in cases:
        with pytest.raises(ValueError, match=what):
            call()


def test_network_output_shapes(ds):
    """ShiftNetwork sizes its output from the last layer writing the output slot (conv, pool or FC)."""
    from paper_1905_13298_gb300 import networks as PN
    assert PN.output_shape(PN.resnet_program("resnet18")[0][-1]) == (1000, 1, 1)
    assert PN.output_shape(PN.vgg16_program()[0][-1]) == (1000, 1, 1)
    b = PN._Builder(512, 7, 7)
    b.conv(0, 96, 1, 1, 0, out=1)
    assert PN.output_shape(b.specs[-1]) == (96, 7, 7)
    b = PN._Builder(64, 56, 56)
    b.conv(0, 64, 3, 2, 1, out=1)
    assert PN.output_shape(b.specs[-1]) == (64, 28, 28)
    b = PN._Builder(64, 56, 56)
    b.pool(ds.DS_OP_MAXPOOL, 0, 3, 2, 1)
    assert PN.output_shape(b.specs[-1]) == (64, 28, 28)


def test_specialisation_validates_before_compiling(ds):
    """The weight-specialised ConvShift refuses bad requests on the host, before NVRTC or any CUDA call."""
    import numpy as np
    L = ds.lib()
    out = ctypes.c_void_p()
    s = np.ones((4, 3, 3, 3), np.int8)
    p = np.zeros((4, 3, 3, 3), np.int8)
    assert L.ds_specialize_conv2d_shift(None, p.ctypes.data, 4, 3, 3, 3, 1, 1, ctypes.byref(out)) == ds.DS_ERR_INVALID_ARG
    assert L.ds_specialize_conv2d_shift(s.ctypes.data, p.ctypes.data, 0, 3, 3, 3, 1, 1, ctypes.byref(out)) == ds.DS_ERR_SHAPE
    assert L.ds_specialize_conv2d_shift(s.ctypes.data, p.ctypes.data, 4, 3, 3, 3, 3, 1, ctypes.byref(out)) == ds.DS_ERR_UNSUPPORTED
    assert L.ds_specialize_conv2d_shift(s.ctypes.data, p.ctypes.data, 4, 3, 3, 3, 1, 3, ctypes.byref(out)) == ds.DS_ERR_UNSUPPORTED
    big = np.ones((64, 3, 7, 7), np.int8)  # 9408 weights: more than the instruction stream should hold
    assert L.ds_specialize_conv2d_shift(big.ctypes.data, np.zeros_like(big).ctypes.data, 64, 3, 7, 7, 2, 3,
                                        ctypes.byref(out)) == ds.DS_ERR_UNSUPPORTED
    bad = p.copy()
    bad[1, 2, 0, 1] = 1  # a positive shift
    assert L.ds_specialize_conv2d_shift(s.ctypes.data, bad.ctypes.data, 4, 3, 3, 3, 1, 1, ctypes.byref(out)) == ds.DS_ERR_CODE_RANGE
    assert out.value is None
    assert L.ds_conv2d_shift_specialized(None, 16, None, None, 4096, 1, 8, 8, 0, None, None) == ds.DS_ERR_INVALID_ARG
    L.ds_specialized_destroy(None)  # a no-op


def test_codes5_sizes_and_validation_without_gpu(ds):
    """The 5-bit storage: its size query matches the oracle's layout, and every argument check comes before
    any CUDA call."""
    for n_out, k_red in [(1, 1), (1, 3), (7, 64), (33, 32), (512, 784)]:
        assert ds.ds_packed5_weight_bytes(n_out, k_red) == O.codes5_layout(n_out, k_red)["total"]
    assert ds.ds_packed5_weight_bytes(0, 3) == 0 and ds.ds_packed5_weight_bytes(3, 0) == 0
    L = ds.lib()
    v = ctypes.c_void_p
    assert L.ds_pack_shift_weights5(None, v(16), 1, 1, v(256), 256, None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_pack_shift_weights5(v(16), v(16), 0, 1, v(256), 256, None) == ds.DS_ERR_SHAPE
    assert L.ds_pack_shift_weights5(v(16), v(16), 1, 3, v(256), 511, None) == ds.DS_ERR_BUFFER_TOO_SMALL
    assert L.ds_pack_shift_weights5(v(16), v(16), 1, 3, v(260), 512, None) == ds.DS_ERR_ALIGNMENT
    assert L.ds_unpack_shift_weights5(None, 512, 1, 3, v(16), v(16), None) == ds.DS_ERR_INVALID_ARG
    assert L.ds_unpack_shift_weights5(v(256), 512, 1, -3, v(16), v(16), None) == ds.DS_ERR_SHAPE
    assert L.ds_unpack_shift_weights5(v(256), 100, 1, 3, v(16), v(16), None) == ds.DS_ERR_BUFFER_TOO_SMALL
    assert L.ds_unpack_shift_weights5(v(264), 512, 1, 3, v(16), v(16), None) == ds.DS_ERR_ALIGNMENT
