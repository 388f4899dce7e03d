"""Fused convolution + 2x2 stride-2 max-pooling (qconv_hwc_pool2) against the oracle's two
layers in sequence (Sec. IV-A), bit for bit, plus its argument checks (without a GPU)."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_1908_11263_gb300 import build as qbuild
from paper_1908_11263_gb300 import qnn
from gpu_util import THREADS, check_guard, first_mismatch, guarded_output, pack_gpu, tc_algos, to_dev

FAKE = 0x10000  # 16-byte aligned, never dereferenced: validation fails first


def spread_case(seed, n, h, w, c, m, k, bits, per_channel_shift):
    """Seeded layer whose outputs spread over [0, 2^Q - 1]: the bias cancels the accumulators'
    mean (weights average -1/2), kappa is positive and the shift matches their spread."""
    rng = np.random.default_rng(seed)
    top = (1 << bits) - 1
    x = rng.integers(0, top + 1, size=(n, h, w, c))
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, k, k, c))
    taps = k * k * c
    centre = taps * top // 4
    spread = int(np.sqrt(taps) * ((top + 1) ** 2 - 1) / 12) + 1
    bias = (centre + rng.integers(-spread, spread + 1, size=m)).astype(np.int32)
    kappa = rng.integers(1, 400, size=m).astype(np.int16)
    shift = max(2, int(np.log2(spread * 400 / (top + 1))) + 1)
    lam = rng.integers(0, (top + 1) << (shift - 1), size=m).astype(np.int32)
    shifts = rng.integers(shift - 2, shift + 3, size=m).astype(np.uint8) if per_channel_shift else None
    return x, wt, bias, kappa, lam, shifts, shift


def packed_dev(v, bits, shape):
    per = 8 // bits
    t = pack_gpu(v.reshape(-1), bits)
    return t.view(*shape[:-1], shape[-1] // per)


def run_fused(x, wt, bias, kappa, lam, shifts, shift, bits, pad, algo=qnn.ALGO_AUTO):
    n, h, w, c = x.shape
    m, k, _, _ = wt.shape
    per = 8 // bits
    oh, ow = h + 2 * pad - k + 1, w + 2 * pad - k + 1
    out, buf = guarded_output((n, oh // 2, ow // 2, m // per))
    wd = packed_dev(wt, bits, wt.shape)
    if bits == 8:
        wd = wd.view(torch.int8)
    qnn.conv_hwc_pool2(packed_dev(x, bits, x.shape), wd, to_dev(kappa, torch.int16), to_dev(lam, torch.int32),
                       bias=to_dev(bias, torch.int32), shifts=None if shifts is None else to_dev(shifts, torch.uint8),
                       shift=shift, bits=bits, pad=pad, algo=algo, out=out)
    qnn.device_status()
    check_guard(buf)
    return out, wd


def run_oracle(x, wt, bias, kappa, lam, shifts, shift, bits, pad):
    n, h, w, c = x.shape
    m, k, _, _ = wt.shape
    shape = dict(n=n, h=h, w=w, c=c, m=m, kh=k, kw=k, sh=1, sw=1, ph=pad, pw=pad, bits=bits)
    return oracle.conv_hwc_pool2(oracle.pack(x.reshape(-1), bits), oracle.pack(wt.reshape(-1), bits), shape, bias,
                                 kappa, lam, shifts=shifts, shift=shift, nthreads=THREADS)


# (n, h, w, c, m, k, pad, bits): the CIFAR layers' shapes at small batch, partial strips at the
# right and bottom, odd output sizes (floor), 1x1 and 5x5 windows, C not a multiple of 8, two
# output-channel tiles, several channel slabs, sub-byte outputs
SHAPES = [
    (2, 32, 32, 3, 32, 5, 2, 8),
    (2, 16, 16, 32, 32, 5, 2, 8),
    (3, 8, 8, 32, 64, 5, 2, 8),
    (2, 16, 16, 32, 64, 3, 1, 8),
    (1, 30, 20, 32, 48, 5, 2, 8),
    (2, 15, 13, 16, 24, 3, 1, 8),
    (1, 12, 12, 32, 136, 3, 1, 8),
    (1, 10, 10, 128, 64, 3, 1, 8),
    (2, 9, 11, 16, 16, 1, 0, 8),
    (2, 16, 16, 32, 64, 3, 1, 4),
    (1, 13, 18, 64, 32, 3, 1, 4),
    (2, 9, 9, 64, 64, 3, 0, 2),
    (1, 14, 22, 32, 32, 3, 1, 2),
]


@pytest.mark.gpu
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s[:6])) + f"_p{s[6]}_q{s[7]}")
def test_conv_pool2_matches_oracle(shape):
    n, h, w, c, m, k, pad, bits = shape
    case = spread_case(hash(shape) & 0xFFFF, n, h, w, c, m, k, bits, per_channel_shift=(h % 2 == 0))
    want = run_oracle(*case, bits, pad)
    algos = tc_algos(n, h, w, c, m, k, k, (1, 1), (pad, pad), bits)
    assert algos
    for algo in algos:
        out, _ = run_fused(*case, bits, pad, algo)
        got = out.cpu().numpy().reshape(-1)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))
    assert len(np.unique(want)) > 4, "pooled outputs nearly constant: the check is weak"


@pytest.mark.gpu
def test_conv_pool2_equals_conv_then_qmaxpool_on_gpu():
    """The fused kernel against the library's own two launches (qconv_hwc, then qmaxpool)."""
    n, h, w, c, m, k, pad, bits = 4, 32, 32, 32, 64, 5, 2, 8
    x, wt, bias, kappa, lam, shifts, shift = spread_case(99, n, h, w, c, m, k, bits, True)
    fused, wd = run_fused(x, wt, bias, kappa, lam, shifts, shift, bits, pad)
    full = qnn.conv_hwc(packed_dev(x, bits, x.shape), wd, to_dev(kappa, torch.int16), to_dev(lam, torch.int32),
                        bias=to_dev(bias, torch.int32), shifts=to_dev(shifts, torch.uint8), shift=shift, bits=bits,
                        pad=pad)
    two_step = qnn.maxpool(full, 2, 2, bits=bits)
    torch.cuda.synchronize()
    assert torch.equal(fused, two_step)

@pytest.mark.gpu
def test_conv_pool2_cifar_chain_batch1024():
    """The CIFAR-10-shaped network of Sec. V-E at batch 1024, run as the benchmark runs it: each
    convolution with its 2x2 max-pool fused (qconv_hwc_pool2), chained on the device, then the
    fully connected layer.  Every pooled activation and every FC output is compared with the
    oracle's chain (conv_hwc then maxpool per layer, then linear)."""
    from paper_1908_11263_gb300 import inputs
    n = 1024
    x = inputs.cifar_input(n)
    xd = to_dev(x.astype(np.uint8))
    xo = x.astype(np.uint8).reshape(-1)
    for key, layer, wl, lid in inputs.cifar_layers(n):
        ld = inputs.make_layer(key, layer, wl, lid, x=np.zeros(1))
        yo = oracle.conv_hwc_pool2(xo, ld.w.reshape(-1).view(np.uint8), layer.shape(), ld.bias, ld.kappa, ld.lam,
                                   shift=ld.shift, nthreads=THREADS)
        for algo in tc_algos(n, layer.h, layer.w, layer.c, layer.m, layer.k, layer.k, (1, 1), (layer.pad, layer.pad), 8):
            yd = qnn.conv_hwc_pool2(xd, to_dev(ld.w), to_dev(ld.kappa, torch.int16), to_dev(ld.lam, torch.int32),
                                    bias=to_dev(ld.bias, torch.int32), shift=ld.shift, bits=8, pad=layer.pad,
                                    algo=algo)
            qnn.device_status()
            got = yd.cpu().numpy().reshape(-1)
            assert first_mismatch(got, yo) is None, (key, algo, first_mismatch(got, yo))
        assert len(np.unique(yo)) > 16, f"{key}: pooled outputs nearly constant, the check is weak"
        xd, xo = yd, yo
    wfc, bfc = inputs.cifar_fc()
    yd = qnn.linear(xd.view(n, -1), to_dev(wfc), to_dev(bfc))
    yo = oracle.linear(xo.reshape(n, -1), wfc, bfc)
    np.testing.assert_array_equal(yd.cpu().numpy(), yo)


@pytest.mark.gpu
def test_conv_pool2_prepared_cifar_chain_batch1024():
    """The CIFAR-10-shaped network of Sec. V-E at batch 1024 on prepared filters: each layer's
    filters prepared once (qconv_hwc_prepare), then every convolution with its 2x2 max-pool
    fused run from the prepared workspace (qconv_hwc_pool2_run), chained on the device, twice
    over the same input (the workspaces are reused), then the fully connected layer.  Every
    pooled activation and the FC outputs equal the oracle's chain."""
    from paper_1908_11263_gb300 import inputs
    n = 1024
    x = inputs.cifar_input(n)
    x0 = to_dev(x.astype(np.uint8))
    layers = inputs.cifar_layers(n)
    preps, want = [], []
    xo = x.astype(np.uint8).reshape(-1)
    for key, layer, wl, lid in layers:
        ld = inputs.make_layer(key, layer, wl, lid, x=np.zeros(1))
        preps.append(qnn.PreparedConv(to_dev(ld.w), to_dev(ld.kappa, torch.int16), to_dev(ld.lam, torch.int32),
                                      n=n, h=layer.h, wd=layer.w, bias=to_dev(ld.bias, torch.int32), shift=ld.shift,
                                      bits=8, stride=1, pad=layer.pad))
        xo = oracle.conv_hwc_pool2(xo, ld.w.reshape(-1).view(np.uint8), layer.shape(), ld.bias, ld.kappa, ld.lam,
                                   shift=ld.shift, nthreads=THREADS)
        want.append(xo)
    wfc, bfc = inputs.cifar_fc()
    want_fc = oracle.linear(want[-1].reshape(n, -1), wfc, bfc)
    for trial in range(2):
        xd = x0
        for (key, _, _, _), prep, yo in zip(layers, preps, want):
            xd = prep.pool2(xd)
            qnn.device_status()
            got = xd.cpu().numpy().reshape(-1)
            assert first_mismatch(got, yo) is None, (trial, key, first_mismatch(got, yo))
        yd = qnn.linear(xd.view(n, -1), to_dev(wfc), to_dev(bfc))
        np.testing.assert_array_equal(yd.cpu().numpy(), want_fc)


@pytest.fixture(scope="module")
def lib():
    qbuild.build()
    return qnn.load()


def test_conv_pool2_run_rejects_what_it_cannot_run(lib):
    """qconv_hwc_pool2_run: argument checks only (no CUDA call is reached)."""
    P = ctypes.c_void_p

    def status(d, ws=FAKE, nbytes=1 << 30, x=FAKE):
        return lib.qconv_hwc_pool2_run(ctypes.byref(d), P(x), P(FAKE), P(ws), ctypes.c_size_t(nbytes), None)

    ok = qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 8, 10)
    assert status(qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 2, 1, 8, 10)) == qnn.QNN_EUNSUPPORTED  # stride 2
    assert status(qnn.conv_desc(64, 14, 14, 256, 512, 1, 1, 1, 0, 8, 10)) == qnn.QNN_EUNSUPPORTED  # general kernel
    assert status(qnn.conv_desc(1, 2, 2, 32, 32, 3, 3, 1, 0, 8, 10)) == qnn.QNN_EINVAL  # 0 x 0 output
    assert status(ok, x=FAKE + 2) == qnn.QNN_EALIGN
    assert status(ok, ws=None) == qnn.QNN_EWORKSPACE
    assert status(ok, nbytes=256) == qnn.QNN_EWORKSPACE
    assert status(ok, ws=FAKE + 16) == qnn.QNN_EWORKSPACE


def test_conv_pool2_rejects_what_it_cannot_run(lib):
    """Argument checks only (no CUDA call is reached), so this runs without a GPU."""
    P = ctypes.c_void_p

    def status(d, x=FAKE, y=FAKE, ws=FAKE):
        return lib.qconv_hwc_pool2(ctypes.byref(d), P(x), P(FAKE), P(FAKE), P(FAKE), P(FAKE), None, P(y), P(ws),
                                   ctypes.c_size_t(1 << 30), None)

    ok = qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 8, 10)
    # stride 2 has no tensor-core kernel; a forced CUDA-core kernel has no fused pool
    assert status(qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 2, 1, 8, 10)) == qnn.QNN_EUNSUPPORTED
    assert status(qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 8, 10, qnn.ALGO_DIRECT)) == qnn.QNN_EUNSUPPORTED
    # a 1-pixel-wide output has no pooled pixel
    assert status(qnn.conv_desc(1, 8, 3, 32, 32, 3, 3, 1, 0, 8, 10)) == qnn.QNN_EINVAL
    assert status(ok, x=0) == qnn.QNN_EINVAL
    assert status(ok, y=FAKE + 8) == qnn.QNN_EALIGN
    # the general kernel needs its workspace; the window kernel (this layer's default) reads the
    # filters in place
    assert status(qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 8, 10, qnn.ALGO_TC_GENERAL), ws=0) == qnn.QNN_EWORKSPACE
