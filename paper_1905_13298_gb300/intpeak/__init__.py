"""Integer issue-rate microbenchmark: the measured side of the shift kernels' ALU roofline.

`measure()` builds libds_intpeak.so (nvcc, sm_103a) next to this file, runs
each instruction mix on one full wave of CTAs, and returns thread
instructions per SM clock for each mix (from clock64 cycles, so independent
of the clock frequency) and the wall-clock rate.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "int_issue_rate.cu")
LIB = os.path.join(HERE, "libds_intpeak.so")
KINDS = {0: "SHF", 1: "IMAD", 2: "SHF+IMAD", 3: "IADD", 4: "LOP", 5: "IMAD.HI", 6: "ADD+ADD"}
# instructions per inner iteration: 64 of the mix (128 for SHF+IMAD) + 8 x-updates
INSTR_PER_ITER = {0: 72, 1: 72, 2: 136, 3: 72, 4: 72, 5: 72, 6: 136}


def build() -> str:
    if not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        subprocess.run(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-shared",
                        "-Xcompiler", "-fPIC", "-o", LIB, SRC], check=True)
    return LIB


def measure(iters: int = 4096, threads: int = 256, blocks_per_sm: int = 2):
    import torch
    L = ctypes.CDLL(build())
    props = torch.cuda.get_device_properties(0)
    sms = props.multi_processor_count
    blocks = sms * blocks_per_sm
    seed = torch.randint(1, 1 << 20, (80,), dtype=torch.int32, device="cuda")
    out = torch.empty(blocks * threads, dtype=torch.int32, device="cuda")
    cyc = torch.empty(blocks, dtype=torch.int64, device="cuda")
    res = {}
    for kind, name in KINDS.items():
        ms = ctypes.c_float()
        for _ in range(2):  # first run warms up
            rc = L.ds_probe_int_mix(kind, blocks, threads, iters, ctypes.c_void_p(seed.data_ptr()),
                                    ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(cyc.data_ptr()),
                                    ctypes.byref(ms))
            if rc != 0:
                raise RuntimeError(f"probe kind {kind} failed with CUDA error {rc}")
        cycles = float(cyc.double().max())
        instr_per_sm = blocks_per_sm * threads * iters * INSTR_PER_ITER[kind]
        res[name] = {"thread_instr_per_clk_per_sm": instr_per_sm / cycles,
                     "wall_tinstr_per_s": blocks * threads * iters * INSTR_PER_ITER[kind] / (ms.value / 1e3) / 1e12,
                     "ms": ms.value}
    return res


if __name__ == "__main__":
    import json
    print(json.dumps(measure(), indent=1))
