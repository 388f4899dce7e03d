"""Staircase (threshold) compression on the GPU (Sec. III-A, Eq. 4) against the oracle,
through both kernels, plus its rejection of INT-8 (checked without a GPU)."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_1908_11263_gb300 import build as qbuild
from paper_1908_11263_gb300 import qnn
from gpu_util import check_guard, dev, first_mismatch, guarded_output, pack_gpu, tc_algos, to_dev

FAKE = 0x10000


def run_gpu(x, w, tau, bits, stride, pad, algo):
    n, h, wd, c = x.shape
    m, kh, kw, _ = w.shape
    per = 8 // bits
    oh, ow = (h + 2 * pad - kh) // stride + 1, (wd + 2 * pad - kw) // stride + 1
    xd = pack_gpu(x, bits).view(n, h, wd, c // per)
    wd_ = pack_gpu(w, bits).view(m, kh, kw, c // per)
    out, buf = guarded_output((n, oh, ow, m // per))
    qnn.conv_hwc_thresholds(xd, wd_, to_dev(tau, torch.int32), bits=bits, stride=stride, pad=pad, algo=algo, out=out)
    qnn.device_status()
    check_guard(buf)
    return out.cpu().numpy().reshape(-1)


def run_oracle(x, w, tau, bits, stride, pad):
    n, h, wd, c = x.shape
    m, kh, kw, _ = w.shape
    shape = dict(n=n, h=h, w=wd, c=c, m=m, kh=kh, kw=kw, sh=stride, sw=stride, ph=pad, pw=pad, bits=bits)
    return oracle.conv_hwc_thresholds(oracle.pack(x.reshape(-1), bits), oracle.pack(w.reshape(-1), bits), shape, tau)


def layer(rng, n, h, w, c, m, k, bits):
    top = (1 << bits) - 1
    x = rng.integers(0, top + 1, size=(n, h, w, c))
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, k, k, c))
    return x, wt


def sorted_thresholds(rng, m, bits, taps):
    """Thresholds spread over the accumulators' range: centred on their mean (weights average -1/2)
    and about one standard deviation either side, with ties (empty intervals) in some channels."""
    top = (1 << bits) - 1
    centre = -taps * top // 4
    spread = max(8, int(np.sqrt(taps) * ((top + 1) ** 2 - 1) / 12))
    tau = np.sort(rng.integers(centre - spread, centre + spread, size=(m, top)), axis=1)
    tau[::3, 1] = tau[::3, 0]
    return tau.astype(np.int32)


@pytest.mark.gpu
@pytest.mark.parametrize("bits", [4, 2])
@pytest.mark.parametrize("shape", [(2, 16, 16, 32, 64, 3, 1, 1), (3, 9, 13, 64, 32, 3, 1, 1), (2, 12, 12, 32, 128, 5, 1, 2),
                                   (1, 11, 11, 16, 16, 3, 2, 1), (2, 8, 8, 256, 64, 1, 1, 0)])
def test_thresholds_match_oracle(bits, shape):
    n, h, w, c, m, k, stride, pad = shape
    rng = np.random.default_rng(sum(shape) + bits)
    x, wt = layer(rng, n, h, w, c, m, k, bits)
    tau = sorted_thresholds(rng, m, bits, k * k * c)
    want = run_oracle(x, wt, tau, bits, stride, pad)
    assert len(np.unique(want)) > 4
    algos = [qnn.ALGO_DIRECT] + (tc_algos(n, h, w, c, m, k, k, (1, 1), (pad, pad), bits) if stride == 1 else [])
    for algo in algos:
        got = run_gpu(x, wt, tau, bits, stride, pad, algo)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))


@pytest.mark.gpu
@pytest.mark.parametrize("bits", [4, 2])
def test_unsorted_thresholds_count(bits):
    """Any threshold values: the output counts the thresholds not above the accumulator."""
    rng = np.random.default_rng(77 + bits)
    x, wt = layer(rng, 2, 10, 16, 32, 32, 3, bits)
    top = (1 << bits) - 1
    centre = -9 * 32 * top // 4
    tau = rng.integers(centre - 200, centre + 200, size=(32, top)).astype(np.int32)
    want = run_oracle(x, wt, tau, bits, 1, 1)
    assert len(np.unique(want)) > 4
    for algo in [qnn.ALGO_DIRECT] + tc_algos(2, 10, 16, 32, 32, 3, 3, (1, 1), (1, 1), bits):
        got = run_gpu(x, wt, tau, bits, 1, 1, algo)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))


@pytest.mark.gpu
@pytest.mark.parametrize("bits", [4, 2])
def test_affine_thresholds_equal_scaling_and_clip_on_gpu(bits):
    """Thresholds derived from (bias, kappa, lambda, shift) give qconv_hwc's own output, bit for bit."""
    from test_oracle_pins import affine_thresholds
    rng = np.random.default_rng(90 + bits)
    n, h, w, c, m, k = 4, 16, 16, 32, 64, 3
    x, wt = layer(rng, n, h, w, c, m, k, bits)
    bias = rng.integers(-300, 300, size=m).astype(np.int32)
    kappa = rng.integers(1, 60, size=m).astype(np.int16)
    lam = rng.integers(-4000, 4000, size=m).astype(np.int32)
    shift = 11
    tau = np.array([affine_thresholds(bias[o], kappa[o], lam[o], shift, bits) for o in range(m)], np.int32)
    per = 8 // bits
    xd = pack_gpu(x, bits).view(n, h, w, c // per)
    wd_ = pack_gpu(wt, bits).view(m, k, k, c // per)
    ref = qnn.conv_hwc(xd, wd_, to_dev(kappa, torch.int16), to_dev(lam, torch.int32), bias=to_dev(bias, torch.int32),
                       shift=shift, bits=bits, pad=1)
    for algo in [qnn.ALGO_DIRECT] + tc_algos(n, h, w, c, m, k, k, (1, 1), (1, 1), bits):
        got = qnn.conv_hwc_thresholds(xd, wd_, to_dev(tau, torch.int32), bits=bits, pad=1, algo=algo)
        assert torch.equal(got, ref), algo


def test_thresholds_reject_int8_and_bad_arguments():
    qbuild.build()
    lib = qnn.load()
    P = ctypes.c_void_p

    def status(d, x=FAKE, w=FAKE, t=FAKE, y=FAKE):
        return lib.qconv_hwc_thresholds(ctypes.byref(d), P(x), P(w), P(t), P(y), P(FAKE), ctypes.c_size_t(1 << 30), None)

    assert status(qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 8, 0)) == qnn.QNN_EUNSUPPORTED
    d4 = qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 4, 0)
    assert status(d4, t=0) == qnn.QNN_EINVAL
    assert status(d4, t=FAKE + 2) == qnn.QNN_EALIGN
    assert status(d4, x=0) == qnn.QNN_EINVAL
