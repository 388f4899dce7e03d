"""Freeze the per-layer requantization shifts of the synthetic workloads.

TEST INFRASTRUCTURE: runs only the oracle (and the seeded input generator).

Recipe (the workload definition for the CIFAR-10-shaped network, the sub-byte
layers and the large-layer sweep): for each layer, the shift is the smallest
s in [0, 62] such that at most 5% of the layer's outputs exceed 2^Q - 1 before
the clip, i.e. floor(((acc + bias) * kappa + lambda) / 2^s) > 2^Q - 1 for at
most 5% of them.  It is measured on the first CAL_IMAGES images of the batch,
layer after layer (each CIFAR layer sees the oracle's output of the previous
layer after 2x2 max-pooling), and written to
paper_1908_11263_gb300/calibrated_shifts.json.

Usage:  python oracle/calibrate_shifts.py [--check]
"""
from __future__ import annotations

import argparse
import json
import os
import sys

import numpy as np

_ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if _ROOT not in sys.path:
    sys.path.insert(0, _ROOT)

import oracle  # noqa: E402
from paper_1908_11263_gb300 import inputs  # noqa: E402

OUT = os.path.join(_ROOT, "paper_1908_11263_gb300", "calibrated_shifts.json")
CLIP_FRACTION = 0.05
CAL_IMAGES = {"w3": 64, "w4": 64, "w5": 2}


def smallest_shift(acc: np.ndarray, bias, kappa, lam, bits: int) -> int:
    """Smallest s with at most CLIP_FRACTION of outputs above 2^Q-1 before the clip."""
    m = acc.shape[-1]
    a = acc.reshape(-1, m).astype(np.int64)
    t = (a + bias.astype(np.int64)) * kappa.astype(np.int64) + lam.astype(np.int64)
    top = (1 << bits) - 1
    for s in range(63):
        above = np.count_nonzero((t >> s) > top)   # numpy's >> on int64 is floor division by 2^s
        if above <= CLIP_FRACTION * t.size:
            return s
    return 62


def layer_acc(ld: inputs.LayerData, layer: inputs.ConvLayer, n: int):
    return oracle.conv_acc(ld.x[:n].astype(np.int32), ld.w.astype(np.int32),
                           (layer.stride, layer.stride), (layer.pad, layer.pad))


def calibrate() -> dict:
    table = {}
    # sub-byte benchmark layers and the large-layer sweep: inputs drawn directly
    for which, tag in ((inputs.WORKLOAD_SUBBYTE, "w4"), (inputs.WORKLOAD_SWEEP, "w5")):
        for key, layer, wl, lid in inputs.single_layer_workload(which):
            n = min(layer.n, CAL_IMAGES[tag])
            x = inputs.draw_activations(wl, lid, (layer.n, layer.h, layer.w, layer.c), layer.bits)[:n]
            layer.shift = 0  # placeholder so make_layer does not look the value up
            ld = inputs.make_layer(key, layer, wl, lid, x=x)
            table[key] = smallest_shift(layer_acc(ld, layer, n), ld.bias, ld.kappa, ld.lam, layer.bits)
    # CIFAR-shaped network: layer by layer on the oracle's own activations
    n = CAL_IMAGES["w3"]
    x = inputs.cifar_input(1024)[:n]
    for key, layer, wl, lid in inputs.cifar_layers(1024):
        layer.shift = 0
        ld = inputs.make_layer(key, layer, wl, lid, x=x)
        s = smallest_shift(layer_acc(ld, layer, n), ld.bias, ld.kappa, ld.lam, 8)
        table[key] = s
        shape = layer.shape()
        shape["n"] = n
        y = oracle.conv_hwc(x.reshape(-1), ld.w.reshape(-1).view(np.uint8), shape, ld.bias, ld.kappa, ld.lam,
                            shift=s)
        y = oracle.maxpool(y, n, layer.oh, layer.ow, layer.m, 2, 2, 8)
        x = y.reshape(n, layer.oh // 2, layer.ow // 2, layer.m)
    return table


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--check", action="store_true", help="recompute and compare with the stored table")
    args = ap.parse_args()
    table = calibrate()
    if args.check:
        with open(OUT) as f:
            stored = json.load(f)
        ok = stored == table
        print("match" if ok else f"MISMATCH stored={stored} computed={table}")
        sys.exit(0 if ok else 1)
    with open(OUT, "w") as f:
        json.dump(table, f, indent=1, sort_keys=True)
        f.write("\n")
    print(json.dumps(table, sort_keys=True))


if __name__ == "__main__":
    main()
