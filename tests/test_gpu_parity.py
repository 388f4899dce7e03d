"""GPU parity: the CUDA path, called through the C ABI, against the oracle,
element by element (bit-exact: every result is an integer) on the same seeded
inputs.  Small shapes span several tiles and ragged tails; the workloads run
at full size and every output byte is compared."""
import numpy as np
import pytest
import torch

import oracle
from paper_1908_11263_gb300 import inputs, qnn

from gpu_util import (conv_gpu, conv_oracle, first_mismatch, guarded_output, check_guard, to_dev, pack_gpu,
                      layer_tensors, THREADS, tc_algos, all_algos)

pytestmark = pytest.mark.gpu
ALGOS = [qnn.ALGO_TENSORCORE, qnn.ALGO_DIRECT]


@pytest.fixture(scope="module", autouse=True)
def loaded():
    qnn.load(build_if_missing=True)
    torch.cuda.set_device(0)


def rand_case(seed, n, h, w, c, m, kh, kw, bits, shift_lo=0, shift_hi=20, per_channel=True, kappa_neg=True):
    rng = np.random.default_rng(seed)
    x = rng.integers(0, 1 << bits, size=(n, h, w, c))
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, kh, kw, c))
    bias = rng.integers(-4096, 4097, size=m).astype(np.int32)
    kappa = rng.integers(-64 if kappa_neg else 1, 65, size=m).astype(np.int16)
    lam = rng.integers(-(1 << 15), (1 << 15) + 1, size=m).astype(np.int32)
    shifts = rng.integers(shift_lo, shift_hi + 1, size=m).astype(np.uint8) if per_channel else None
    shift = int(rng.integers(shift_lo, shift_hi + 1))
    return x, wt, bias, kappa, lam, shifts, shift


# (n, h, w, c, m, kh, kw, stride, pad, bits): tile multiples, ragged tails, odd widths,
# channel padding, several slabs and output-channel tiles, rectangular kernels
SHAPES = [
    (2, 16, 16, 32, 64, 3, 3, (1, 1), (1, 1), 8),
    (1, 16, 16, 32, 64, 3, 3, (1, 1), (1, 1), 4),
    (1, 16, 16, 32, 64, 3, 3, (1, 1), (1, 1), 2),
    (3, 10, 10, 16, 16, 3, 3, (1, 1), (1, 1), 8),
    (2, 14, 14, 64, 48, 3, 3, (1, 1), (1, 1), 8),
    (1, 15, 20, 24, 40, 3, 3, (1, 1), (1, 1), 8),
    (2, 9, 33, 8, 8, 1, 1, (1, 1), (0, 0), 8),
    (1, 12, 12, 3, 32, 5, 5, (1, 1), (2, 2), 8),
    (2, 8, 8, 32, 64, 5, 5, (1, 1), (2, 2), 8),
    (1, 7, 7, 128, 136, 3, 3, (1, 1), (1, 1), 8),
    (1, 6, 6, 256, 256, 3, 3, (1, 1), (1, 1), 8),
    (1, 5, 9, 32, 16, 3, 2, (1, 1), (0, 1), 8),
    (1, 11, 13, 16, 32, 2, 4, (1, 1), (1, 2), 8),
    (1, 1, 40, 16, 16, 1, 3, (1, 1), (0, 1), 8),
    (2, 13, 13, 32, 24, 3, 3, (1, 1), (0, 0), 4),
    (1, 10, 12, 48, 32, 5, 5, (1, 1), (2, 2), 4),
    (2, 9, 9, 64, 64, 3, 3, (1, 1), (1, 1), 2),
    (1, 9, 7, 8, 12, 3, 3, (1, 1), (1, 1), 2),
    (1, 16, 16, 12, 16, 3, 3, (1, 1), (1, 1), 4),
    (2, 16, 16, 32, 64, 3, 3, (2, 2), (1, 1), 8),
    (1, 17, 15, 16, 32, 3, 3, (2, 1), (1, 1), 4),
    # 16 x 8 strip tiles: a partial bottom block of rows, three and five column
    # blocks, a 5x5 window, sub-byte inputs and two channel slabs
    (2, 30, 16, 32, 64, 3, 3, (1, 1), (1, 1), 8),
    (1, 16, 24, 32, 48, 5, 5, (1, 1), (2, 2), 8),
    (1, 47, 40, 32, 32, 3, 3, (1, 1), (1, 1), 4),
    (1, 47, 40, 64, 32, 3, 3, (1, 1), (1, 1), 2),
]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(str(v) for v in s[:7]) + f"_s{s[7][0]}{s[7][1]}_p{s[8][0]}{s[8][1]}_q{s[9]}")
def test_conv_random_shapes(shape):
    n, h, w, c, m, kh, kw, stride, pad, bits = shape
    x, wt, bias, kappa, lam, shifts, shift = rand_case(hash(shape) & 0xFFFF, n, h, w, c, m, kh, kw, bits)
    want = conv_oracle(x, wt, bias, kappa, lam, shifts, shift, bits, stride, pad)
    want_scalar = conv_oracle(x, wt, None, kappa, lam, None, shift, bits, stride, pad)
    desc = qnn.conv_desc(n, h, w, c, m, kh, kw, stride, pad, bits, shift)
    tc = qnn.conv_algo(desc) == qnn.ALGO_TENSORCORE
    for algo in all_algos(n, h, w, c, m, kh, kw, stride, pad, bits):
        got = conv_gpu(x, wt, bias, kappa, lam, shifts, shift, bits, stride, pad, algo)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))
        got = conv_gpu(x, wt, None, kappa, lam, None, shift, bits, stride, pad, algo)
        assert first_mismatch(got, want_scalar) is None, (algo, "scalar shift, no bias",
                                                          first_mismatch(got, want_scalar))
    # the tensor-core kernel takes every stride-1 layer whose input rows are whole 16-byte units
    if stride == (1, 1) and (w * c * bits // 8) % 16 == 0:
        assert tc


@pytest.mark.parametrize("shift", [0, 1, 31, 40, 62])
def test_conv_shift_extremes(shift):
    x, wt, bias, kappa, lam, _, _ = rand_case(shift + 7, 1, 8, 8, 32, 32, 3, 3, 8)
    lam = lam * 1000 if shift > 30 else lam
    for algo in all_algos(1, 8, 8, 32, 32, 3, 3, (1, 1), (1, 1), 8):
        got = conv_gpu(x, wt, bias, kappa, lam.astype(np.int32), None, shift, 8, (1, 1), (1, 1), algo)
        want = conv_oracle(x, wt, bias, kappa, lam.astype(np.int32), None, shift, 8, (1, 1), (1, 1))
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))


@pytest.mark.parametrize("bits", [4, 2])
@pytest.mark.parametrize("k,c", [(3, 32), (3, 256), (1, 256)])
@pytest.mark.parametrize("pick", ["max_neg", "max_pos", "mixed"])
def test_subbyte_exact_accumulation_at_the_bounds(bits, k, c, pick):
    """Sub-byte layers with C a multiple of 32 stage e4m3 bytes and run kind::f8f6f4 MMAs. Constant
    activations at the top of the range, with weights at either end of theirs, drive every
    accumulator to its extreme (K up to 2304). With kappa=1, shift=0 and lambda = 1 - acc, every
    output reads 1 only if the accumulator is exact."""
    n, m = 1, 16
    top, lo, hi = (1 << bits) - 1, -(1 << (bits - 1)), (1 << (bits - 1)) - 1
    h, w = (4, 32) if k == 1 else (6, 6)
    x = np.full((n, h, w, c), top)
    wval = {"max_neg": lo, "max_pos": hi, "mixed": lo}[pick]
    wt = np.full((m, k, k, c), wval)
    if pick == "mixed":  # alternate the extremes along K and flip them across channels
        wt[..., 1::2] = hi
        wt[1::2] = lo + hi - wt[1::2]
    acc = (top * wt.reshape(m, -1).sum(axis=1)).astype(np.int64)
    lam = (1 - acc).astype(np.int32)
    kappa = np.ones(m, np.int16)
    assert qnn.conv_algo(qnn.conv_desc(n, h, w, c, m, k, k, 1, 0, bits, 0)) == qnn.ALGO_TENSORCORE
    want = conv_oracle(x, wt, None, kappa, lam, None, 0, bits, (1, 1), (0, 0))
    for algo in tc_algos(n, h, w, c, m, k, k, (1, 1), (0, 0), bits):
        got = conv_gpu(x, wt, None, kappa, lam, None, 0, bits, (1, 1), (0, 0), algo)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))
    per = 8 // bits
    assert np.all(oracle.unpack(want, want.size * per, bits, False) == 1)


@pytest.mark.parametrize("xval,wval", [(0, -128), (255, 127), (255, -128), (0, 127), (128, -128), (1, -1)])
@pytest.mark.parametrize("k,c", [(1, 256), (3, 128), (3, 256)])
def test_exact_accumulation_at_the_bounds(xval, wval, k, c):
    """Constant layers without padding drive every accumulator chunk to its extreme
    (K = 256, 1152, 2304); with kappa=1, shift=0 and lambda = 100 - acc every output
    reads 100 only if acc is exact."""
    n, m = 1, 16
    h, w = (4, 32) if k == 1 else (6, 6)
    x = np.full((n, h, w, c), xval)
    wt = np.full((m, k, k, c), wval)
    wt[1::2] = -wt[1::2] - (1 if wval > 0 else 0)  # mix signs across channels (stay inside int8)
    wt = np.clip(wt, -128, 127)
    acc = (xval * wt.reshape(m, -1).sum(axis=1)).astype(np.int64)
    lam = (100 - acc).astype(np.int32)
    kappa = np.ones(m, np.int16)
    assert qnn.conv_algo(qnn.conv_desc(n, h, w, c, m, k, k, 1, 0, 8, 0)) == qnn.ALGO_TENSORCORE
    for algo in all_algos(n, h, w, c, m, k, k, (1, 1), (0, 0), 8):
        got = conv_gpu(x, wt, None, kappa, lam, None, 0, 8, (1, 1), (0, 0), algo)
        assert np.all(got == 100), (algo, np.unique(got))


@pytest.mark.parametrize("bits", [8, 4, 2])
def test_exact_accumulation_random_long_k(bits):
    """K = 9 * 256 with random data: outputs compared against the oracle with kappa=1
    and per-channel lambda centring each channel's accumulators, shift 0."""
    rng = np.random.default_rng(bits)
    n, h, w, c, m = 1, 6, 6, 256, 32
    x = rng.integers(0, 1 << bits, size=(n, h, w, c))
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, 3, 3, c))
    acc = oracle.conv_acc(x, wt, (1, 1), (1, 1))
    lam = (128 - np.median(acc.reshape(-1, m), axis=0)).astype(np.int32) if bits == 8 else \
          ((1 << (bits - 1)) - np.median(acc.reshape(-1, m), axis=0)).astype(np.int32)
    kappa = np.ones(m, np.int16)
    want = conv_oracle(x, wt, None, kappa, lam, None, 0, bits, (1, 1), (1, 1))
    for algo in all_algos(n, h, w, c, m, 3, 3, (1, 1), (1, 1), bits):
        got = conv_gpu(x, wt, None, kappa, lam, None, 0, bits, (1, 1), (1, 1), algo)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))


def test_extreme_values_all_layers():
    for xval, wval in [(0, 0), (255, 127), (255, -128), (0, -128)]:
        x = np.full((2, 16, 16, 32), xval)
        wt = np.full((64, 3, 3, 32), wval)
        _, _, bias, kappa, lam, shifts, shift = rand_case(xval + wval + 1000, 2, 16, 16, 32, 64, 3, 3, 8)
        want = conv_oracle(x, wt, bias, kappa, lam, shifts, shift, 8, (1, 1), (1, 1))
        for algo in all_algos(2, 16, 16, 32, 64, 3, 3, (1, 1), (1, 1), 8):
            got = conv_gpu(x, wt, bias, kappa, lam, shifts, shift, 8, (1, 1), (1, 1), algo)
            assert first_mismatch(got, want) is None, (xval, wval, algo)


def test_empty_batch_is_a_no_op():
    x = torch.empty((0, 16, 16, 32), dtype=torch.uint8, device="cuda")
    w = torch.zeros((64, 3, 3, 32), dtype=torch.int8, device="cuda")
    k = torch.ones(64, dtype=torch.int16, device="cuda")
    lam = torch.zeros(64, dtype=torch.int32, device="cuda")
    for algo in (qnn.ALGO_TENSORCORE, qnn.ALGO_TC_WINDOW, qnn.ALGO_TC_GENERAL, qnn.ALGO_DIRECT):
        y = qnn.conv_hwc(x, w, k, lam, shift=3, bits=8, stride=1, pad=1, algo=algo)
        assert y.shape == (0, 16, 16, 64)
    qnn.device_status()


# ------------------------------------------------------------------ workloads at full size

def run_workload_layer(key, layer, wl, lid):
    ld = inputs.make_layer(key, layer, wl, lid)
    x, wt, bias, kappa, lam, shifts, shift = layer_tensors(ld)
    st, pd = (layer.stride, layer.stride), (layer.pad, layer.pad)
    want = conv_oracle(x, wt, bias, kappa, lam, shifts, shift, layer.bits, st, pd)
    algos = all_algos(layer.n, layer.h, layer.w, layer.c, layer.m, layer.k, layer.k, st, pd, layer.bits)
    assert len(algos) >= 2, (key, algos)
    for algo in algos:
        got = conv_gpu(x, wt, bias, kappa, lam, shifts, shift, layer.bits, st, pd, algo)
        assert first_mismatch(got, want) is None, (key, algo, first_mismatch(got, want))
    return want


def test_workload_single_layer_batch1():
    (key, layer, wl, lid), = inputs.single_layer_workload(inputs.WORKLOAD_SINGLE)
    assert layer.macs == 4718592
    run_workload_layer(key, layer, wl, lid)


def test_workload_single_layer_batch512():
    (key, layer, wl, lid), = inputs.single_layer_workload(inputs.WORKLOAD_BATCH)
    assert layer.macs == 2415919104
    run_workload_layer(key, layer, wl, lid)


@pytest.mark.parametrize("which", ["w4_int4", "w4_int2"])
def test_workload_subbyte(which):
    for key, layer, wl, lid in inputs.single_layer_workload(inputs.WORKLOAD_SUBBYTE):
        if key == which:
            run_workload_layer(key, layer, wl, lid)


def sample_pixels(n, oh, ow, count, seed):
    rng = np.random.default_rng(seed)
    fixed = [(0, 0, 0), (0, 0, ow - 1), (0, oh - 1, 0), (n - 1, oh - 1, ow - 1), (n - 1, oh // 2, ow // 2),
             (n // 2, 0, ow // 2), (n // 2, oh - 1, ow // 3)]
    rand = [(int(rng.integers(n)), int(rng.integers(oh)), int(rng.integers(ow))) for _ in range(count)]
    return fixed + rand


@pytest.mark.parametrize("key", ["w5_56", "w5_28", "w5_14", "w5_1x1"])
def test_workload_sweep_full(key):
    """Large layers at full batch in the benchmark's launch configuration: sampled pixels
    against the oracle's per-pixel routine first (a fast pre-check that names the first
    bad pixel), then every output byte against the oracle's whole layer, and the whole
    output against the independent CUDA-core kernel."""
    (k2, layer, wl, lid), = [t for t in inputs.single_layer_workload(inputs.WORKLOAD_SWEEP) if t[0] == key]
    ld = inputs.make_layer(k2, layer, wl, lid)
    x, wt, bias, kappa, lam, shifts, shift = layer_tensors(ld)
    st, pd = (layer.stride, layer.stride), (layer.pad, layer.pad)
    pix = sample_pixels(layer.n, layer.oh, layer.ow, 40, lid)
    want_pix = oracle.conv_hwc_pixels(x.astype(np.uint8).reshape(-1), wt.astype(np.int8).reshape(-1).view(np.uint8),
                                      layer.shape(), bias, kappa, lam, pix, shifts=shifts, shift=shift)
    want = conv_oracle(x, wt, bias, kappa, lam, shifts, shift, 8, st, pd)
    outs = {}
    for algo in all_algos(layer.n, layer.h, layer.w, layer.c, layer.m, layer.k, layer.k, st, pd, 8):
        got = conv_gpu(x, wt, bias, kappa, lam, shifts, shift, 8, st, pd, algo)
        g = got.reshape(layer.n, layer.oh, layer.ow, layer.m)
        for r, (b, oy, ox) in enumerate(pix):
            np.testing.assert_array_equal(g[b, oy, ox], want_pix[r], err_msg=f"{key} algo {algo} pixel {(b, oy, ox)}")
        assert first_mismatch(got, want) is None, (key, algo, first_mismatch(got, want))
        outs[algo] = got
    assert len(np.unique(want)) > 16, "outputs nearly constant: the comparison is weak"


def test_workload_cifar_pipeline():
    """The CIFAR-10-shaped network (Sec. V-E shape) at batch 1024: three conv layers with
    2x2 max-pooling and the fully connected layer, GPU chain vs oracle chain."""
    n = 1024
    x = inputs.cifar_input(n)
    xd = to_dev(x)
    xo = x.reshape(-1)
    for key, layer, wl, lid in inputs.cifar_layers(n):
        ld = inputs.make_layer(key, layer, wl, lid, x=np.zeros(1))
        kappa, lam, bias = to_dev(ld.kappa, torch.int16), to_dev(ld.lam, torch.int32), to_dev(ld.bias, torch.int32)
        yd = qnn.conv_hwc(xd, to_dev(ld.w), kappa, lam, bias=bias, shift=ld.shift, bits=8, stride=1, pad=layer.pad)
        xd = qnn.maxpool(yd, 2, 2, 8)
        yo = oracle.conv_hwc(xo, ld.w.reshape(-1).view(np.uint8), layer.shape(), ld.bias, ld.kappa, ld.lam,
                             shift=ld.shift, nthreads=THREADS)
        np.testing.assert_array_equal(yd.cpu().numpy().reshape(-1), yo, err_msg=key)
        xo = oracle.maxpool(yo, n, layer.oh, layer.ow, layer.m, 2, 2, 8)
        np.testing.assert_array_equal(xd.cpu().numpy().reshape(-1), xo, err_msg=key + " pool")
    wfc, bfc = inputs.cifar_fc()
    yd = qnn.linear(xd.view(n, -1), to_dev(wfc), to_dev(bfc))
    yo = oracle.linear(xo.reshape(n, -1), wfc, bfc)
    np.testing.assert_array_equal(yd.cpu().numpy(), yo)
    qnn.device_status()


# ------------------------------------------------------------------ max-pool, FC, packing

@pytest.mark.parametrize("bits,c,k,s", [(8, 32, 2, 2), (8, 64, 3, 2), (8, 24, 2, 2), (8, 5, 2, 1), (4, 32, 2, 2),
                                        (2, 16, 3, 3), (4, 6, 2, 2), (4, 64, 2, 2), (2, 64, 3, 2), (2, 128, 2, 2)])
def test_maxpool_parity(bits, c, k, s):
    rng = np.random.default_rng(c * k + bits)
    n, h, w = 3, 11, 9
    x = rng.integers(0, 1 << bits, size=(n, h, w, c))
    xp = oracle.pack(x.reshape(-1), bits) if bits < 8 else x.astype(np.uint8).reshape(-1)
    want = oracle.maxpool(xp, n, h, w, c, k, s, bits)
    xd = pack_gpu(x, bits).view(n, h, w, c * bits // 8)
    oh, ow = (h - k) // s + 1, (w - k) // s + 1
    out, buf = guarded_output((n, oh, ow, c * bits // 8))
    qnn.maxpool(xd, k, s, bits, out=out)
    check_guard(buf)
    np.testing.assert_array_equal(out.cpu().numpy().reshape(-1), want)


@pytest.mark.parametrize("n,k,m", [(1024, 1024, 10), (5, 7, 3), (33, 64, 17), (1, 4, 1), (64, 2048, 40),
                                   (8, 4096, 64)])
def test_linear_parity(n, k, m):
    rng = np.random.default_rng(n + k + m)
    x = rng.integers(0, 256, size=(n, k)).astype(np.uint8)
    w = rng.integers(-128, 128, size=(m, k)).astype(np.int8)
    b = rng.integers(-4096, 4097, size=m).astype(np.int32)
    for bias in (b, None):
        got = qnn.linear(to_dev(x), to_dev(w), None if bias is None else to_dev(bias))
        np.testing.assert_array_equal(got.cpu().numpy(), oracle.linear(x, w, bias))


@pytest.mark.parametrize("bits", [8, 4, 2])
@pytest.mark.parametrize("signed", [False, True])
def test_pack_unpack_parity(bits, signed):
    allbytes = np.arange(256, dtype=np.uint8)
    per = 8 // bits
    vals = oracle.unpack(allbytes, 256 * per, bits, signed)
    got = qnn.unpack_subbyte(to_dev(allbytes), bits, signed)
    np.testing.assert_array_equal(got.cpu().numpy().astype(np.int32) if signed or bits < 8 else
                                  got.cpu().numpy().view(np.uint8), vals)
    if bits < 8:
        rng = np.random.default_rng(bits)
        lo, hi = (-(1 << (bits - 1)), 1 << (bits - 1)) if signed else (0, 1 << bits)
        v = rng.integers(lo, hi, size=4096)
        np.testing.assert_array_equal(qnn.pack_subbyte(to_dev(v.astype(np.int8)), bits).cpu().numpy(),
                                      oracle.pack(v, bits))


def test_device_status_clean():
    qnn.device_status()
