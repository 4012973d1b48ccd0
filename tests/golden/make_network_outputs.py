"""Writes network_outputs_224.txt: CPU-oracle logits of the full-size chained forwards.

The benchmarked network workloads run whole batches at 224 x 224 (ResNet18 at
batch 32, ResNet50 and VGG16 at batch 64).  The oracle needs minutes per image
for these networks, too long to rerun inside every GPU test session, so this
script computes the first and the last image of each batch once with
``oracle/networks.py`` and stores the 1000 logits of each.  The GPU test runs
the whole batch through ds_shift_forward and compares those two images element
by element.  The images of a batch are independent (every layer is applied
per image), so the two images' logits do not depend on the batch size.

Each record also stores a SHA-256 of the image and of the layer parameters, so
a change to the input generators shows up as a stale fixture instead of a
false failure.  Inputs come from ``synth_inputs`` with the seeds the
benchmark uses; nothing here calls the CUDA path.

    python tests/golden/make_network_outputs.py        # about 2-4 minutes on 8 cores
"""
from __future__ import annotations

import hashlib
import multiprocessing as mp
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

OUT = os.path.join(HERE, "network_outputs_224.txt")
# (architecture, batch of the benchmarked workload)
CASES = [("resnet18", 32), ("resnet50", 64), ("vgg16", 64)]


def network_shapes(arch: str):
    """Layer shapes of the architecture in parameter order (oracle/networks.py's order)."""
    from oracle import networks as ON
    return ON.layer_shapes(arch)


def case_inputs(arch: str, batch: int, image: int):
    import synth_inputs as si
    params = si.network_params(network_shapes(arch), si.SEED_BASE + 3)
    x = si.image_batch(si.SEED_BASE + 3, batch)[image:image + 1]
    return x, params


def digest(x, params) -> tuple[str, str]:
    hx = hashlib.sha256(np.ascontiguousarray(x).tobytes()).hexdigest()[:16]
    h = hashlib.sha256()
    for s, p, b in params:
        for a in (s, p, b):
            h.update(np.ascontiguousarray(a).tobytes())
    return hx, h.hexdigest()[:16]


def one(job):
    arch, batch, image = job
    from oracle import networks as ON
    x, params = case_inputs(arch, batch, image)
    y = ON.vgg16_forward(x, params) if arch == "vgg16" else ON.resnet_forward(x, params, arch)
    return arch, batch, image, digest(x, params), y.reshape(-1)


def main():
    jobs = [(a, b, i) for a, b in CASES for i in (0, b - 1)]
    # the largest jobs first, so the pool's tail is short
    jobs.sort(key=lambda j: {"vgg16": 0, "resnet50": 1, "resnet18": 2}[j[0]])
    with mp.get_context("spawn").Pool(min(len(jobs), os.cpu_count() or 1)) as pool:
        res = pool.map(one, jobs)
    res.sort(key=lambda r: ([a for a, _ in CASES].index(r[0]), r[2]))
    with open(OUT, "w") as f:
        f.write("# Logits of the full-size chained forwards (224 x 224), computed by the CPU oracle\n")
        f.write("# (oracle/networks.py: every conv and FC a shift layer per Eq. 3 on the Sec. 4 fixed point).\n")
        f.write("# Written by tests/golden/make_network_outputs.py; one record per (arch, batch, image):\n")
        f.write("#   <arch> <batch> <image> <sha256(image)[:16]> <sha256(params)[:16]> <1000 int32 logits>\n")
        for arch, batch, image, (hx, hp), y in res:
            f.write(f"{arch} {batch} {image} {hx} {hp} " + " ".join(str(int(v)) for v in y) + "\n")
    print(f"wrote {OUT}")


if __name__ == "__main__":
    main()
