"""Seeded synthetic inputs for the quantized HWC convolution workloads.

This module holds no arithmetic of the method: it only draws integers.  Both the
GPU path and the oracle receive the same arrays from it; each side then packs,
convolves and compresses with its own code.

Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014; constants as published with that algorithm),
one stream per tensor.  Element i of a stream with seed s is
splitmix64_mix(s + (i + 1) * 0x9E3779B97F4A7C15), and a uniform integer in
[lo, hi] is lo + (u >> 11) mod (hi - lo + 1).

Seeds: 0x5EED0000 + 256 * workload + 16 * layer + tensor, with tensor ids
X=0, W=1, BIAS=2, KAPPA=3, LAMBDA=4.

Workload shapes follow the benchmark layer of the paper (Sec. V-A: 16x16x32
HWC input, 64 filters 3x3x32, stride 1, pad 1), the CIFAR-10 network of
Sec. V-E (3 convolutions and 1 fully-connected layer) and a sweep of larger
layers.  Value ranges: activations uniform over the unsigned Q-bit range,
weights uniform over the signed Q-bit range, bias uniform in [-2^12, 2^12],
kappa in [1, 64], lambda in [-2^15, 2^15].
"""
from __future__ import annotations

import json
import os
from dataclasses import dataclass, field

import numpy as np

_GOLDEN = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB
_MASK = (1 << 64) - 1

X, W, BIAS, KAPPA, LAMBDA = 0, 1, 2, 3, 4


def seed_for(workload: int, layer: int, tensor: int) -> int:
    return 0x5EED0000 + 256 * workload + 16 * layer + tensor


def splitmix64(seed: int, count: int) -> np.ndarray:
    """The first `count` outputs of a SplitMix64 stream, as uint64."""
    with np.errstate(over="ignore"):
        i = np.arange(1, count + 1, dtype=np.uint64)
        z = np.uint64(seed & _MASK) + i * np.uint64(_GOLDEN)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(_M1)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(_M2)
        z = z ^ (z >> np.uint64(31))
    return z


def uniform_int(seed: int, count: int, lo: int, hi: int) -> np.ndarray:
    """`count` integers uniform in [lo, hi] (int64)."""
    u = splitmix64(seed, count) >> np.uint64(11)
    return (u % np.uint64(hi - lo + 1)).astype(np.int64) + lo


@dataclass
class ConvLayer:
    """One quantized convolution layer: NHWC input, [M][KH][KW][C] filters."""
    n: int
    h: int
    w: int
    c: int
    m: int
    k: int
    stride: int = 1
    pad: int = 0
    bits: int = 8
    shift: int | None = None          # scalar shift; None = calibrated value from the table
    per_channel_shift: bool = False   # pass shifts[M] (all equal to the layer's shift)
    name: str = ""

    @property
    def oh(self):
        return (self.h + 2 * self.pad - self.k) // self.stride + 1

    @property
    def ow(self):
        return (self.w + 2 * self.pad - self.k) // self.stride + 1

    @property
    def macs(self):
        return self.n * self.oh * self.ow * self.m * self.k * self.k * self.c

    def shape(self):
        return dict(n=self.n, h=self.h, w=self.w, c=self.c, m=self.m, kh=self.k, kw=self.k,
                    sh=self.stride, sw=self.stride, ph=self.pad, pw=self.pad, bits=self.bits)

    def algorithmic_bytes(self):
        """Input + output + weights (packed sizes) + per-channel parameters, each moved once."""
        q = self.bits
        xb = self.n * self.h * self.w * self.c * q // 8
        yb = self.n * self.oh * self.ow * self.m * q // 8
        wb = self.m * self.k * self.k * self.c * q // 8
        pb = self.m * (4 + 2 + 4 + (1 if self.per_channel_shift else 0))
        return xb + yb + wb + pb


@dataclass
class LayerData:
    """Unpacked integer tensors of one layer (numpy)."""
    x: np.ndarray        # [N,H,W,C] int in [0, 2^Q-1]
    w: np.ndarray        # [M,KH,KW,C] int in [-2^(Q-1), 2^(Q-1)-1]
    bias: np.ndarray     # [M] int32
    kappa: np.ndarray    # [M] int16
    lam: np.ndarray      # [M] int32
    shift: int
    shifts: np.ndarray | None = None   # [M] uint8 or None


def draw_params(workload: int, layer: int, m: int):
    bias = uniform_int(seed_for(workload, layer, BIAS), m, -(1 << 12), 1 << 12).astype(np.int32)
    kappa = uniform_int(seed_for(workload, layer, KAPPA), m, 1, 64).astype(np.int16)
    lam = uniform_int(seed_for(workload, layer, LAMBDA), m, -(1 << 15), 1 << 15).astype(np.int32)
    return bias, kappa, lam


def draw_activations(workload: int, layer: int, shape, bits: int) -> np.ndarray:
    count = int(np.prod(shape))
    return uniform_int(seed_for(workload, layer, X), count, 0, (1 << bits) - 1).astype(np.uint8).reshape(shape)


def draw_weights(workload: int, layer: int, shape, bits: int) -> np.ndarray:
    count = int(np.prod(shape))
    lo, hi = -(1 << (bits - 1)), (1 << (bits - 1)) - 1
    return uniform_int(seed_for(workload, layer, W), count, lo, hi).astype(np.int8).reshape(shape)


_SHIFTS_FILE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "calibrated_shifts.json")


def calibrated_shifts() -> dict:
    """Per-layer shifts frozen by oracle/calibrate_shifts.py (smallest shift with <= 5% of outputs
    above 2^Q-1 before the clip, measured on the first images of the workload)."""
    if not os.path.exists(_SHIFTS_FILE):
        return {}
    with open(_SHIFTS_FILE) as f:
        return json.load(f)


def layer_shift(key: str, layer: ConvLayer) -> int:
    if layer.shift is not None:
        return layer.shift
    table = calibrated_shifts()
    if key not in table:
        raise KeyError(f"no calibrated shift for {key}; run oracle/calibrate_shifts.py")
    return int(table[key])


# ---------------------------------------------------------------- workloads

def benchmark_layer(n: int, bits: int = 8, shift: int | None = 12) -> ConvLayer:
    """Sec. V-A benchmark layer: 16x16x32 input, 64 filters 3x3x32, stride 1, pad 1."""
    return ConvLayer(n=n, h=16, w=16, c=32, m=64, k=3, stride=1, pad=1, bits=bits, shift=shift,
                     name=f"conv3x3_16x16x32_to_64_int{bits}_n{n}")


WORKLOAD_SINGLE = 1      # batch 1, INT-8, shift 12
WORKLOAD_BATCH = 2       # batch 512, INT-8, shift 12
WORKLOAD_CIFAR = 3       # CIFAR-10-shaped network, batch 1024
WORKLOAD_SUBBYTE = 4     # INT-4 / INT-2 benchmark layer, batch 512
WORKLOAD_SWEEP = 5       # larger layers, batch 64


def single_layer_workload(which: int):
    """Workloads 1, 2 and 4: (key, ConvLayer, workload id, layer id)."""
    if which == WORKLOAD_SINGLE:
        return [("w1", benchmark_layer(1), 1, 0)]
    if which == WORKLOAD_BATCH:
        return [("w2", benchmark_layer(512), 2, 0)]
    if which == WORKLOAD_SUBBYTE:
        return [("w4_int4", benchmark_layer(512, bits=4, shift=None), 4, 0),
                ("w4_int2", benchmark_layer(512, bits=2, shift=None), 4, 1)]
    if which == WORKLOAD_SWEEP:
        return [
            ("w5_56", ConvLayer(64, 56, 56, 64, 64, 3, 1, 1, 8, None, True, "conv3x3_56x56x64_to_64_n64"), 5, 0),
            ("w5_28", ConvLayer(64, 28, 28, 128, 128, 3, 1, 1, 8, None, True, "conv3x3_28x28x128_to_128_n64"), 5, 1),
            ("w5_14", ConvLayer(64, 14, 14, 256, 256, 3, 1, 1, 8, None, True, "conv3x3_14x14x256_to_256_n64"), 5, 2),
            ("w5_1x1", ConvLayer(64, 14, 14, 256, 512, 1, 1, 0, 8, None, True, "conv1x1_14x14x256_to_512_n64"), 5, 3),
        ]
    raise ValueError(which)


def cifar_layers(n: int = 1024):
    """Sec. V-E network shape: conv5x5 3->32, pool, conv5x5 32->32, pool, conv5x5 32->64, pool, FC 1024->10."""
    return [
        ("w3_conv1", ConvLayer(n, 32, 32, 3, 32, 5, 1, 2, 8, None, False, "cifar_conv1"), 3, 0),
        ("w3_conv2", ConvLayer(n, 16, 16, 32, 32, 5, 1, 2, 8, None, False, "cifar_conv2"), 3, 1),
        ("w3_conv3", ConvLayer(n, 8, 8, 32, 64, 5, 1, 2, 8, None, False, "cifar_conv3"), 3, 2),
    ]


CIFAR_FC = dict(k=1024, m=10)


def cifar_fc(workload: int = WORKLOAD_CIFAR):
    w = uniform_int(seed_for(workload, 3, W), CIFAR_FC["m"] * CIFAR_FC["k"], -128, 127).astype(np.int8)
    bias = uniform_int(seed_for(workload, 3, BIAS), CIFAR_FC["m"], -(1 << 12), 1 << 12).astype(np.int32)
    return w.reshape(CIFAR_FC["m"], CIFAR_FC["k"]), bias


def cifar_input(n: int = 1024, workload: int = WORKLOAD_CIFAR):
    return draw_activations(workload, 0, (n, 32, 32, 3), 8)


def make_layer(key: str, layer: ConvLayer, workload: int, lid: int, x: np.ndarray | None = None) -> LayerData:
    """Draw (or take) the input and draw the parameters of one layer."""
    if x is None:
        x = draw_activations(workload, lid, (layer.n, layer.h, layer.w, layer.c), layer.bits)
    wt = draw_weights(workload, lid, (layer.m, layer.k, layer.k, layer.c), layer.bits)
    bias, kappa, lam = draw_params(workload, lid, layer.m)
    shift = layer_shift(key, layer)
    shifts = np.full(layer.m, shift, np.uint8) if layer.per_channel_shift else None
    return LayerData(x=x, w=wt, bias=bias, kappa=kappa, lam=lam, shift=shift, shifts=shifts)
