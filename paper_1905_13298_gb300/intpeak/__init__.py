"""Integer issue-rate microbenchmark: the measured side of the shift kernels' ALU roofline.

`measure()` builds libds_intpeak.so (nvcc, sm_103a) next to this file, runs
each instruction mix on a grid of 2 CTAs per SM, and returns thread
instructions per SM clock for each mix and the wall-clock rate.  The per-SM
rate divides the instructions of an SM's CTAs by that SM's span of clock64
(first start to last end), so it stays right when a mix's register count
lets only one CTA per SM be resident at a time.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "int_issue_rate.cu")
LIB = os.path.join(HERE, "libds_intpeak.so")
KINDS = {0: "SHF", 1: "IMAD", 2: "SHF+IMAD", 3: "IADD", 4: "LOP", 5: "IMAD.HI", 6: "ADD+ADD", 7: "SWAR16"}
# instructions per inner iteration: 64 of the mix (128 for the pairs, 192 for the SWAR triple) + 8 x-updates
INSTR_PER_ITER = {0: 72, 1: 72, 2: 136, 3: 72, 4: 72, 5: 72, 6: 136, 7: 200}
# DeepShift terms (shift + sign flip + accumulate) per inner iteration, for the mixes that form a term:
# SHF+IMAD one term per pair, IMAD.HI one per instruction, SWAR16 two (one per 16-bit lane) per triple
TERMS_PER_ITER = {2: 64, 5: 64, 7: 128}


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
    cyc = torch.empty(2 * blocks, dtype=torch.int64, device="cuda")
    smid = torch.empty(blocks, dtype=torch.int32, device="cuda")
    res = {}
    for kind, name in KINDS.items():
        ms = ctypes.c_float()
        for _ in range(2):  # first run warms up
            rc = L.ds_probe_int_mix(kind, blocks, threads, iters, ctypes.c_void_p(seed.data_ptr()),
                                    ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(cyc.data_ptr()),
                                    ctypes.c_void_p(smid.data_ptr()), ctypes.byref(ms))
            if rc != 0:
                raise RuntimeError(f"probe kind {kind} failed with CUDA error {rc}")
        c = cyc.view(blocks, 2).cpu().numpy()
        sm = smid.cpu().numpy()
        rates = []
        for s in set(sm.tolist()):
            sel = sm == s
            span = float(c[sel, 1].max() - c[sel, 0].min())
            rates.append(int(sel.sum()) * threads * iters * INSTR_PER_ITER[kind] / span)
        rate = sum(rates) / len(rates)
        if kind in TERMS_PER_ITER:
            res.setdefault("terms_per_clk_per_sm", {})[name] = rate * TERMS_PER_ITER[kind] / INSTR_PER_ITER[kind]
        res[name] = {"thread_instr_per_clk_per_sm": rate,
                     "wall_tinstr_per_s": blocks * threads * iters * INSTR_PER_ITER[kind] / (ms.value / 1e3) / 1e12,
                     "ms": ms.value}
    return res


if __name__ == "__main__":
    import json
    print(json.dumps(measure(), indent=1))
