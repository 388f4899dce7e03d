"""Pins for the oracle: each test checks oracle/ against something other than
itself (brute force written differently, a library special case, an algebraic
identity of the paper, an invariant, or a hand-worked value), chosen so that a
dropped term, a wrong sign or index, or a transposed operand fails one of them.
CPU only."""
import itertools
import json
import os
from fractions import Fraction
import math

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


# ------------------------------------------------------------------ helpers

def scatter_conv(x, w, stride, pad):
    """Brute force written as a scatter: every input value adds its products to
    every output it reaches.  Independent of the oracle's gather loop order."""
    n, h, wd, c = x.shape
    m, kh, kw, _ = w.shape
    oh = (h + 2 * pad[0] - kh) // stride[0] + 1
    ow = (wd + 2 * pad[1] - kw) // stride[1] + 1
    out = [[[[0] * m for _ in range(ow)] for _ in range(oh)] for _ in range(n)]
    for b in range(n):
        for iy in range(h):
            for ix in range(wd):
                for i in range(kh):
                    ty = iy + pad[0] - i
                    if ty % stride[0]:
                        continue
                    oy = ty // stride[0]
                    if not 0 <= oy < oh:
                        continue
                    for j in range(kw):
                        tx = ix + pad[1] - j
                        if tx % stride[1]:
                            continue
                        ox = tx // stride[1]
                        if not 0 <= ox < ow:
                            continue
                        for o in range(m):
                            s = 0
                            for ch in range(c):
                                s += int(x[b, iy, ix, ch]) * int(w[o, i, j, ch])
                            out[b][oy][ox][o] += s
    return np.array(out, dtype=np.int64).reshape(n, oh, ow, m)


def im2col(x, kh, kw, stride, pad):
    """Explicit im2col matrix of Sec. III-B: one row per output pixel, columns in (i, j, c) order."""
    n, h, wd, c = x.shape
    xp = np.zeros((n, h + 2 * pad[0], wd + 2 * pad[1], c), np.int64)
    xp[:, pad[0]:pad[0] + h, pad[1]:pad[1] + wd, :] = x
    oh = (h + 2 * pad[0] - kh) // stride[0] + 1
    ow = (wd + 2 * pad[1] - kw) // stride[1] + 1
    rows = []
    for b in range(n):
        for oy in range(oh):
            for ox in range(ow):
                patch = xp[b, oy * stride[0]:oy * stride[0] + kh, ox * stride[1]:ox * stride[1] + kw, :]
                rows.append(patch.reshape(-1))
    return np.array(rows), (n, oh, ow)


def rand_layer(n, h, w, c, m, k, bits=8):
    x = rng.integers(0, 1 << bits, size=(n, h, w, c))
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, k, k, c))
    return x, wt


def requant_ref(acc, bias, kappa, lam, s, bits):
    """Compression with exact rationals: floor(((acc+bias)*kappa+lam) / 2^s) clipped."""
    t = Fraction((acc + bias) * kappa + lam, 2 ** s)
    return min(max(math.floor(t), 0), (1 << bits) - 1)


# ------------------------------------------------------------------ MAC core (Eq. 2, Eq. 6)

@pytest.mark.parametrize("k,stride,pad", [(1, 1, 0), (3, 1, 1), (3, 2, 1), (5, 1, 2), (3, 1, 0), (5, 2, 2),
                                          (3, 2, 0), (1, 2, 0), (3, 1, 2)])
def test_conv_acc_matches_scatter_brute_force(k, stride, pad):
    n, h, w, c, m = 2, 5, 4, 3, 4
    if k > h + 2 * pad:
        pytest.skip("kernel larger than padded input")
    x, wt = rand_layer(n, h, w, c, m, k)
    got = oracle.conv_acc(x, wt, (stride, stride), (pad, pad))
    want = scatter_conv(x, wt, (stride, stride), (pad, pad))
    np.testing.assert_array_equal(got, want)


def test_conv_acc_rectangular_stride_pad():
    x, wt = rand_layer(1, 5, 6, 2, 3, 3)
    wt = wt[:, :, :2, :]  # 3x2 kernel
    got = oracle.conv_acc(x, wt, (2, 1), (1, 0))
    want = scatter_conv(x, wt, (2, 1), (1, 0))
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("k,stride,pad", [(3, 1, 1), (5, 1, 2), (3, 2, 1), (1, 1, 0)])
def test_conv_acc_matches_torch_conv2d_float64(k, stride, pad):
    """Library special case: exact in float64 while |acc| < 2^53."""
    torch = pytest.importorskip("torch")
    x, wt = rand_layer(2, 9, 7, 8, 5, k)
    got = oracle.conv_acc(x, wt, (stride, stride), (pad, pad))
    xt = torch.from_numpy(x.astype(np.float64)).permute(0, 3, 1, 2)
    wtt = torch.from_numpy(wt.astype(np.float64)).permute(0, 3, 1, 2)
    want = torch.nn.functional.conv2d(xt, wtt, stride=stride, padding=pad).permute(0, 2, 3, 1).numpy()
    np.testing.assert_array_equal(got, want.astype(np.int64))


def test_im2col_times_weights_equals_direct_conv():
    """Eq. 6: O(m,x,y) = dot(W(m), im2col(x,y)) with W(m) stored in im2col order."""
    x, wt = rand_layer(2, 6, 5, 4, 6, 3)
    cols, (n, oh, ow) = im2col(x, 3, 3, (1, 1), (1, 1))
    via_matmul = (cols @ wt.reshape(wt.shape[0], -1).T.astype(np.int64)).reshape(n, oh, ow, -1)
    np.testing.assert_array_equal(oracle.conv_acc(x, wt, (1, 1), (1, 1)), via_matmul)


def test_adjacent_pixels_share_weights_eq7():
    """Eq. 7: output (x+1, y) uses the same W(m) with the next im2col buffer."""
    x, wt = rand_layer(1, 6, 6, 4, 3, 3)
    acc = oracle.conv_acc(x, wt, (1, 1), (0, 0))
    cols, _ = im2col(x, 3, 3, (1, 1), (0, 0))
    cols = cols.reshape(4, 4, -1)
    for o in range(3):
        bank = wt[o].reshape(-1)
        assert acc[0, 2, 1, o] == int(np.dot(bank, cols[2, 1]))
        assert acc[0, 2, 2, o] == int(np.dot(bank, cols[2, 2]))


def test_linearity_in_weights_and_inputs():
    x1, w1 = rand_layer(1, 5, 5, 4, 3, 3)
    x2, w2 = rand_layer(1, 5, 5, 4, 3, 3)
    a = lambda x, w: oracle.conv_acc(x, w, (1, 1), (1, 1))
    np.testing.assert_array_equal(a(x1, w1 + w2), a(x1, w1) + a(x1, w2))
    np.testing.assert_array_equal(a(x1 + x2, w1), a(x1, w1) + a(x2, w1))


def test_translation_equivariance_away_from_border():
    x, wt = rand_layer(1, 8, 8, 3, 2, 3)
    shifted = np.zeros_like(x)
    shifted[:, 1:, 2:, :] = x[:, :-1, :-2, :]
    a = oracle.conv_acc(x, wt, (1, 1), (1, 1))
    b = oracle.conv_acc(shifted, wt, (1, 1), (1, 1))
    np.testing.assert_array_equal(b[:, 2:7, 3:7, :], a[:, 1:6, 1:5, :])


# ------------------------------------------------------------------ compression (Sec. III-A)

def test_floor_shift_is_floor_division():
    for t in [-9, -8, -7, -1, 0, 1, 7, 8, 9, -(1 << 40) - 3, (1 << 45) + 5, -(1 << 62)]:
        for s in [0, 1, 2, 3, 31, 32, 40, 62]:
            assert oracle.floor_shift(t, s) == math.floor(Fraction(t, 2 ** s))


def test_requant_matches_rational_definition():
    cases = itertools.product([-300000, -5, 0, 7, 123456, (1 << 31) - 5000], [-4096, 0, 4096],
                              [1, 64, -3, 32767, -32768], [-(1 << 15), 0, 1 << 15], [0, 1, 12, 31, 40, 62],
                              [8, 4, 2])
    for acc, bias, kappa, lam, s, bits in cases:
        assert oracle.requant(acc, bias, kappa, lam, s, bits) == requant_ref(acc, bias, kappa, lam, s, bits)


def test_requant_special_cases():
    # kappa = 2^s, lambda = 0, bias = 0 -> clip(acc)
    for acc in [-10, 0, 5, 200, 255, 256, 100000]:
        assert oracle.requant(acc, 0, 1 << 6, 0, 6, 8) == min(max(acc, 0), 255)
    # kappa = 1, lambda = 0, s = 0 -> saturating ReLU
    for acc in [-1, 0, 1, 14, 15, 16]:
        assert oracle.requant(acc, 0, 1, 0, 0, 4) == min(max(acc, 0), 15)
    # negative t -> 0 ; t >= 2^Q * 2^s -> 2^Q - 1
    assert oracle.requant(-1, 0, 1, 0, 0, 8) == 0
    assert oracle.requant(1 << 20, 0, 1, 0, 12, 8) == 255
    assert oracle.requant((1 << 20) - 1, 0, 1, 0, 12, 8) == 255
    assert oracle.requant((255 << 12), 0, 1, 0, 12, 8) == 255
    assert oracle.requant((255 << 12) - 1, 0, 1, 0, 12, 8) == 254
    # bias is added before kappa: (acc + bias) * kappa, not acc * kappa + bias
    assert oracle.requant(10, 5, 3, 0, 0, 8) == 45


def full_layer_ref(x, wt, bias, kappa, lam, shifts, bits, stride, pad):
    acc = scatter_conv(x, wt, stride, pad)
    out = np.empty(acc.shape, np.int64)
    for idx in np.ndindex(acc.shape):
        o = idx[-1]
        out[idx] = requant_ref(int(acc[idx]), int(bias[o]), int(kappa[o]), int(lam[o]), int(shifts[o]), bits)
    return out


@pytest.mark.parametrize("bits", [8, 4, 2])
def test_full_layer_against_independent_reference(bits):
    n, h, w, c, m, k = 2, 5, 5, 8, 8, 3
    x, wt = rand_layer(n, h, w, c, m, k, bits)
    bias = rng.integers(-50, 50, m)
    kappa = rng.integers(-5, 40, m)
    lam = rng.integers(-300, 300, m)
    shifts = rng.integers(0, 8, m)
    want = full_layer_ref(x, wt, bias, kappa, lam, shifts, bits, (1, 1), (1, 1))
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=k, kw=k, sh=1, sw=1, ph=1, pw=1, bits=bits)
    xp = oracle.pack(x.reshape(-1), bits)
    wp = oracle.pack(wt.reshape(-1), bits)
    y = oracle.conv_hwc(xp, wp, shape, bias, kappa, lam, shifts=shifts)
    got = oracle.unpack(y, want.size, bits, False).reshape(want.shape)
    np.testing.assert_array_equal(got, want)
    # spot pixels through the per-pixel entry point
    pix = [(0, 0, 0), (1, 4, 4), (1, 2, 3)]
    yp = oracle.conv_hwc_pixels(xp, wp, shape, bias, kappa, lam, pix, shifts=shifts)
    for r, (b, oy, ox) in enumerate(pix):
        np.testing.assert_array_equal(yp[r], want[b, oy, ox])


@pytest.mark.parametrize("bits", [8, 4, 2])
def test_conv_pool2_against_independent_reference(bits):
    """A conv layer and then a 2x2 stride-2 max-pool over its quantized output (Sec. IV-A): the
    independent scatter-form layer above, then the maximum of every window written as four
    explicit comparisons.  Odd output sizes check the floor rule (the last row and column drop)."""
    n, h, w, c, m, k = 2, 7, 5, 8, 8, 3
    g = np.random.default_rng(1000 + bits)  # own stream: the case does not depend on test order
    top = (1 << bits) - 1
    x = g.integers(0, top + 1, size=(n, h, w, c))
    wt = g.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, k, k, c))
    # centre the accumulators (weights average -1/2) and scale their spread onto [0, top]
    shift = {8: 13, 4: 8, 2: 5}[bits]
    bias = k * k * c * top // 4 + g.integers(-20, 21, m)
    kappa = g.integers(10, 30, m)
    lam = (top // 2) << shift
    lam = lam + g.integers(-(1 << (shift - 1)), 1 << (shift - 1), m)
    shifts = np.full(m, shift)
    t = full_layer_ref(x, wt, bias, kappa, lam, shifts, bits, (1, 1), (1, 1))  # [n, 7, 5, m]
    assert len(np.unique(t)) > min(top, 6), "layer outputs nearly constant: the pooling check would be weak"
    want = np.empty((n, 3, 2, m), np.int64)
    for b, py, px, o in np.ndindex(want.shape):
        a0, a1 = t[b, 2 * py, 2 * px, o], t[b, 2 * py, 2 * px + 1, o]
        a2, a3 = t[b, 2 * py + 1, 2 * px, o], t[b, 2 * py + 1, 2 * px + 1, o]
        best = a0
        for v in (a1, a2, a3):
            if v > best:
                best = v
        want[b, py, px, o] = best
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=k, kw=k, sh=1, sw=1, ph=1, pw=1, bits=bits)
    y = oracle.conv_hwc_pool2(oracle.pack(x.reshape(-1), bits), oracle.pack(wt.reshape(-1), bits), shape, bias,
                              kappa, lam, shifts=shifts)
    got = oracle.unpack(y, want.size, bits, False).reshape(want.shape)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("bits", [4, 2])
def test_staircase_realises_batch_norm_then_quantisation(bits):
    """Footnote to Eq. 3: the thresholds absorb the bias and batch normalisation
    y = gamma/sigma * (b + phi - mu) + beta. For gamma > 0 and the Q-bit output floor(y) clipped to
    [0, 2^Q - 1], the thresholds tau_p = ceil(mu - b + (p - beta) * sigma / gamma), p = 1 .. 2^Q - 1,
    make the staircase count of Eq. 4 equal that output for every accumulator phi. The reference
    side is exact rational arithmetic; accumulators around each threshold are included."""
    g = np.random.default_rng(100 + bits)
    top = (1 << bits) - 1
    for _ in range(25):
        gamma = Fraction(int(g.integers(1, 60)), int(g.integers(1, 60)))
        sigma = Fraction(int(g.integers(1, 60)), int(g.integers(1, 20)))
        beta = Fraction(int(g.integers(-60, 60)), 7)
        mu = Fraction(int(g.integers(-900, 900)), 3)
        b = int(g.integers(-300, 300))
        tau = [math.ceil(mu - b + (p - beta) * sigma / gamma) for p in range(1, top + 1)]
        assert tau == sorted(tau)
        phis = set(range(-3000, 3000, 37))
        for t in tau:
            phis.update((t - 1, t, t + 1))
        for phi in sorted(phis):
            y = gamma / sigma * (b + phi - mu) + beta
            want = min(max(math.floor(y), 0), top)
            assert oracle.staircase(phi, tau, bits) == want, (phi, tau)


def test_zero_weights_give_bias_only_output():
    n, h, w, c, m = 1, 4, 4, 8, 4
    x, _ = rand_layer(n, h, w, c, m, 3)
    wt = np.zeros((m, 3, 3, c), np.int64)
    bias = np.array([100, -100, 3000, 7])
    kappa = np.array([3, 2, 1, -1])
    lam = np.array([10, 0, -5, 1000])
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=3, kw=3, sh=1, sw=1, ph=1, pw=1, bits=8)
    y = oracle.conv_hwc(x.reshape(-1), wt.reshape(-1).astype(np.int8).view(np.uint8), shape, bias, kappa, lam,
                        shift=2).reshape(n, h, w, m)
    for o in range(m):
        expect = min(max(math.floor(Fraction(int(bias[o]) * int(kappa[o]) + int(lam[o]), 4)), 0), 255)
        assert np.all(y[..., o] == expect)


def test_centred_one_hot_kernel_copies_a_channel():
    n, h, w, c, m = 2, 6, 5, 8, 3
    x, _ = rand_layer(n, h, w, c, m, 3)
    wt = np.zeros((m, 3, 3, c), np.int64)
    src = [5, 0, 7]
    for o, ch in enumerate(src):
        wt[o, 1, 1, ch] = 1
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=3, kw=3, sh=1, sw=1, ph=1, pw=1, bits=8)
    y = oracle.conv_hwc(x.reshape(-1), wt.reshape(-1).astype(np.int8).view(np.uint8), shape,
                        np.zeros(m), np.ones(m), np.zeros(m), shift=0).reshape(n, h, w, m)
    for o, ch in enumerate(src):
        np.testing.assert_array_equal(y[..., o], x[..., ch])


def test_int4_layer_equals_int8_oracle_on_unpacked_values():
    """Cross bit-width: the INT-4 path is the INT-8 convolution of the unpacked values, clipped at 15."""
    n, h, w, c, m = 1, 5, 5, 8, 4
    x, wt = rand_layer(n, h, w, c, m, 3, bits=4)
    bias, kappa, lam = rng.integers(-20, 20, m), rng.integers(1, 9, m), rng.integers(-50, 50, m)
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=3, kw=3, sh=1, sw=1, ph=1, pw=1, bits=4)
    y4 = oracle.conv_hwc(oracle.pack(x.reshape(-1), 4), oracle.pack(wt.reshape(-1), 4), shape, bias, kappa, lam,
                         shift=3)
    y4 = oracle.unpack(y4, n * h * w * m, 4, False)
    shape8 = dict(shape, bits=8)
    y8 = oracle.conv_hwc(x.reshape(-1).astype(np.uint8), wt.reshape(-1).astype(np.int8).view(np.uint8), shape8,
                         bias, kappa, lam, shift=3)
    np.testing.assert_array_equal(y4, np.minimum(y8, 15))


def test_accumulator_outside_int32_is_rejected():
    c = 70000  # 255 * 127 * 70000 > 2^31
    x = np.full((1, 1, 1, c), 255, np.uint8)
    wt = np.full((1, 1, 1, c), 127, np.int8)
    shape = dict(n=1, h=1, w=1, c=c, m=1, kh=1, kw=1, sh=1, sw=1, ph=0, pw=0, bits=8)
    with pytest.raises(OverflowError):
        oracle.conv_hwc(x.reshape(-1), wt.reshape(-1).view(np.uint8), shape, np.zeros(1), np.ones(1),
                        np.zeros(1), shift=0)


# ------------------------------------------------------------------ packing (Sec. IV-A)

def test_packing_worked_bytes():
    with open(os.path.join(GOLDEN, "packing_worked_bytes.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        got = oracle.pack(np.array(case["values"]), case["bits"])
        assert list(got) == case["bytes"], case
        back = oracle.unpack(np.array(case["bytes"], np.uint8), len(case["values"]), case["bits"], case["signed"])
        assert list(back) == case["values"], case


@pytest.mark.parametrize("bits", [8, 4, 2])
@pytest.mark.parametrize("signed", [False, True])
def test_pack_unpack_round_trip_over_all_bytes(bits, signed):
    allbytes = np.arange(256, dtype=np.uint8)
    per = 8 // bits
    vals = oracle.unpack(allbytes, 256 * per, bits, signed)
    lo, hi = (-(1 << (bits - 1)), (1 << (bits - 1)) - 1) if signed else (0, (1 << bits) - 1)
    assert vals.min() >= lo and vals.max() <= hi
    np.testing.assert_array_equal(oracle.pack(vals, bits), allbytes)


# ------------------------------------------------------------------ max-pool and fully connected

def test_maxpool_matches_torch():
    torch = pytest.importorskip("torch")
    x = rng.integers(0, 256, size=(2, 8, 6, 16)).astype(np.uint8)
    y = oracle.maxpool(x.reshape(-1), 2, 8, 6, 16, 2, 2, 8).reshape(2, 4, 3, 16)
    xt = torch.from_numpy(x.astype(np.float32)).permute(0, 3, 1, 2)
    want = torch.nn.functional.max_pool2d(xt, 2, 2).permute(0, 2, 3, 1).numpy().astype(np.uint8)
    np.testing.assert_array_equal(y, want)


@pytest.mark.parametrize("bits", [4, 2])
def test_maxpool_subbyte_matches_unpacked(bits):
    x = rng.integers(0, 1 << bits, size=(1, 7, 5, 8))
    y = oracle.maxpool(oracle.pack(x.reshape(-1), bits), 1, 7, 5, 8, 3, 2, bits)
    got = oracle.unpack(y, 3 * 2 * 8, bits, False).reshape(1, 3, 2, 8)
    want = np.zeros((1, 3, 2, 8), np.int64)
    for oy in range(3):
        for ox in range(2):
            want[0, oy, ox] = x[0, 2 * oy:2 * oy + 3, 2 * ox:2 * ox + 3].reshape(-1, 8).max(axis=0)
    np.testing.assert_array_equal(got, want)


def test_linear_matches_numpy_int64():
    x = rng.integers(0, 256, size=(7, 1024)).astype(np.uint8)
    w = rng.integers(-128, 128, size=(10, 1024)).astype(np.int8)
    b = rng.integers(-4096, 4097, size=10).astype(np.int32)
    want = x.astype(np.int64) @ w.astype(np.int64).T + b
    np.testing.assert_array_equal(oracle.linear(x, w, b), want)
    np.testing.assert_array_equal(oracle.linear(x, w, None), want - b)


def test_paper_benchmark_layer_mac_count():
    """Sec. V-A layer: 16x16x32 -> 64 filters 3x3x32 is 4,718,592 MACs; an all-ones
    layer without padding makes every accumulator count its own terms."""
    with open(os.path.join(GOLDEN, "paper_benchmark_layer.json")) as f:
        g = json.load(f)
    h, w, c = g["input_hwc"]
    m, kh, kw, _ = g["filters_mkkc"]
    x = np.ones((1, h + 2, w + 2, c), np.int64)  # explicit zero-free padding ring
    wt = np.ones((m, kh, kw, c), np.int64)
    acc = oracle.conv_acc(x, wt, (1, 1), (0, 0))
    assert acc.shape == (1,) + tuple(g["output_hwc"])
    assert int(acc.sum()) == g["macs"]
    # the paper's own cycle counts give 13.07 MAC/cycle on 8 cores
    assert round(g["macs"] / g["table2_cycles_8cores"], 2) == 13.07


# ------------------------------------------------------------------ staircase compression (Eq. 4)

def eq4_staircase(acc, tau, bits):
    """Eq. 4 written out: the sum over output levels p of p times the characteristic function of
    [tau_p, tau_p+1).  Levels run 0..2^Q-1 (unsigned outputs); the lowest interval is open below
    and the highest open above."""
    bounds = [-float("inf")] + [int(t) for t in tau] + [float("inf")]
    return sum(p * (1 if bounds[p] <= acc < bounds[p + 1] else 0) for p in range(1 << bits))


@pytest.mark.parametrize("bits", [4, 2])
def test_staircase_is_eq4_on_sorted_thresholds(bits):
    rng = np.random.default_rng(40 + bits)
    for _ in range(300):
        tau = np.sort(rng.integers(-5000, 5000, size=(1 << bits) - 1))
        if rng.random() < 0.3:  # ties: empty intervals
            tau[rng.integers(0, tau.size - 1)] = tau[-1]
            tau = np.sort(tau)
        for acc in list(rng.integers(-6000, 6000, size=8)) + [int(tau[0]), int(tau[-1]), int(tau[0]) - 1]:
            assert oracle.staircase(int(acc), tau, bits) == eq4_staircase(int(acc), tau, bits)


def affine_thresholds(bias, kappa, lam, shift, bits):
    """Thresholds at which clip(floor(((acc + b) * kappa + lam) / 2^s), 0, 2^Q-1) steps up, for kappa > 0:
    the output reaches p exactly when acc >= ceil((p * 2^s - lam) / kappa) - b."""
    tau = []
    for p in range(1, 1 << bits):
        num = p * (1 << shift) - int(lam)
        t = -((-num) // int(kappa)) - int(bias)  # ceil division
        tau.append(min(max(t, -(1 << 31)), (1 << 31) - 1))
    return tau


@pytest.mark.parametrize("bits", [4, 2])
def test_thresholds_reproduce_affine_compression(bits):
    """A layer compressed by thresholds derived from (bias, kappa, lambda, shift) equals the same layer
    compressed by scaling and clipping: two formulations of Sec. III-A agree on every output."""
    rng = np.random.default_rng(50 + bits)
    n, h, w, c, m, k = 2, 6, 7, 16, 16, 3
    top = (1 << bits) - 1
    x = rng.integers(0, top + 1, size=(n, h, w, c))
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, k, k, c))
    bias = rng.integers(-300, 300, size=m).astype(np.int32)
    kappa = rng.integers(1, 60, size=m).astype(np.int16)
    lam = rng.integers(-4000, 4000, size=m).astype(np.int32)
    shift = 9
    tau = np.array([affine_thresholds(bias[o], kappa[o], lam[o], shift, bits) for o in range(m)], np.int32)
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=k, kw=k, sh=1, sw=1, ph=1, pw=1, bits=bits)
    xp, wp = oracle.pack(x.reshape(-1), bits), oracle.pack(wt.reshape(-1), bits)
    got = oracle.conv_hwc_thresholds(xp, wp, shape, tau)
    want = oracle.conv_hwc(xp, wp, shape, bias, kappa, lam, shift=shift)
    np.testing.assert_array_equal(got, want)
    assert len(np.unique(oracle.unpack(want, want.size * 8 // bits, bits, False))) > 2  # not all clipped


@pytest.mark.parametrize("bits", [4, 2])
def test_staircase_extremes(bits):
    n_tau = (1 << bits) - 1
    for acc in (-(1 << 30), -1, 0, 1, (1 << 30) - 1):
        assert oracle.staircase(acc, [(1 << 31) - 1] * n_tau, bits) == 0
        assert oracle.staircase(acc, [-(1 << 31)] * n_tau, bits) == n_tau
        assert oracle.staircase(acc, [acc] * n_tau, bits) == n_tau        # tau <= acc counts
        assert oracle.staircase(acc, [acc + 1] * n_tau, bits) == 0


# ------------------------------------------------------------------ INT-1 (Eq. 5)

def bits_pack(v01):
    """Pack 0/1 values eight per byte, element e at bit e mod 8 of byte e / 8."""
    return np.packbits(np.asarray(v01, np.uint8).reshape(-1), bitorder="little")


def test_binary_popcount_equals_pm1_dot_product():
    """popcount(W xnor X) over the in-image window equals (S + K_valid) / 2, where S is the +-1 dot
    product with zero padding and K_valid the number of in-image taps times C (torch conv2d, float64)."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(61)
    for (n, h, w, c, m, k, s, p) in [(2, 7, 9, 16, 8, 3, 1, 1), (1, 8, 8, 8, 16, 5, 2, 2), (3, 5, 6, 24, 8, 1, 1, 0),
                                     (1, 6, 6, 32, 8, 3, 2, 0)]:
        xb = rng.integers(0, 2, size=(n, h, w, c))
        wb = rng.integers(0, 2, size=(m, k, k, c))
        shape = dict(n=n, h=h, w=w, c=c, m=m, kh=k, kw=k, sh=s, sw=s, ph=p, pw=p)
        _, acc = oracle.conv_binary(bits_pack(xb), bits_pack(wb), shape, np.zeros(m, np.int32), with_acc=True)
        xt = torch.from_numpy((2.0 * xb - 1).transpose(0, 3, 1, 2)).double()
        wt = torch.from_numpy((2.0 * wb - 1).transpose(0, 3, 1, 2)).double()
        sdot = torch.nn.functional.conv2d(xt, wt, stride=s, padding=p)
        kvalid = torch.nn.functional.conv2d(torch.ones_like(xt), torch.ones_like(wt), stride=s, padding=p)
        want = ((sdot + kvalid) / 2).permute(0, 2, 3, 1).numpy().reshape(-1)
        np.testing.assert_array_equal(acc, want.astype(np.int64))


def test_binary_threshold_and_bit_order():
    rng = np.random.default_rng(62)
    n, h, w, c, m, k = 2, 5, 5, 16, 16, 3
    xb = rng.integers(0, 2, size=(n, h, w, c))
    wb = rng.integers(0, 2, size=(m, k, k, c))
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=k, kw=k, sh=1, sw=1, ph=1, pw=1)
    tau = rng.integers(40, 100, size=m).astype(np.int32)
    y, acc = oracle.conv_binary(bits_pack(xb), bits_pack(wb), shape, tau, with_acc=True)
    want = (acc.reshape(-1, m) >= tau).astype(np.uint8).reshape(-1)
    np.testing.assert_array_equal(np.unpackbits(y, bitorder="little"), want)
    # all +1 everywhere: every in-image tap matches; the corner pixel sees 4 of 9 taps
    ones = np.ones((1, 4, 4, 8), np.int64)
    shape1 = dict(n=1, h=4, w=4, c=8, m=8, kh=3, kw=3, sh=1, sw=1, ph=1, pw=1)
    _, a1 = oracle.conv_binary(bits_pack(ones), bits_pack(np.ones((8, 3, 3, 8))), shape1, np.zeros(8, np.int32),
                               with_acc=True)
    assert a1.reshape(4, 4, 8)[0, 0, 0] == 4 * 8 and a1.reshape(4, 4, 8)[1, 1, 0] == 9 * 8
    # weights the complement of the inputs: no matches at all
    _, a2 = oracle.conv_binary(bits_pack(ones), bits_pack(np.zeros((8, 3, 3, 8))), shape1, np.zeros(8, np.int32),
                               with_acc=True)
    assert np.all(a2 == 0)
