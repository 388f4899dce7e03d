"""INT-1 convolution (Sec. III-A, Eq. 5) on the GPU against the oracle, and its argument
checks (without a GPU)."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_1908_11263_gb300 import build as qbuild
from paper_1908_11263_gb300 import qnn
from gpu_util import check_guard, dev, guarded_output

FAKE = 0x10000


def bits_pack(v01):
    return np.packbits(np.asarray(v01, np.uint8).reshape(-1), bitorder="little")


@pytest.mark.gpu
@pytest.mark.parametrize("shape", [(2, 16, 16, 32, 64, 3, 1, 1), (3, 9, 13, 64, 40, 3, 1, 1), (1, 12, 12, 8, 16, 5, 2, 2),
                                   (2, 7, 9, 24, 8, 3, 1, 0), (512, 16, 16, 32, 64, 3, 1, 1), (1, 14, 14, 256, 96, 1, 1, 0),
                                   (0, 8, 8, 32, 8, 3, 1, 1)])
def test_binary_matches_oracle(shape):
    n, h, w, c, m, k, s, p = shape
    rng = np.random.default_rng(sum(shape))
    xb = rng.integers(0, 2, size=(n, h, w, c))
    wb = rng.integers(0, 2, size=(m, k, k, c))
    kk = k * k * c
    tau = rng.integers(kk // 2 - int(np.sqrt(kk)), kk // 2 + int(np.sqrt(kk)) + 1, size=m).astype(np.int32)
    oh, ow = (h + 2 * p - k) // s + 1, (w + 2 * p - k) // s + 1
    shp = dict(n=n, h=h, w=w, c=c, m=m, kh=k, kw=k, sh=s, sw=s, ph=p, pw=p)
    want = oracle.conv_binary(bits_pack(xb), bits_pack(wb), shp, tau) if n else np.zeros(0, np.uint8)
    xd = torch.from_numpy(bits_pack(xb)).to(dev()).view(n, h, w, c // 8)
    wd_ = torch.from_numpy(bits_pack(wb)).to(dev()).view(m, k, k, c // 8)
    out, buf = guarded_output((n, oh, ow, m // 8))
    qnn.conv_binary(xd, wd_, torch.from_numpy(tau).to(dev()), stride=s, pad=p, out=out)
    qnn.device_status()
    check_guard(buf)
    got = out.cpu().numpy().reshape(-1)
    np.testing.assert_array_equal(got, want)
    if n:
        ones = np.unpackbits(want, bitorder="little").mean()
        assert 0.1 < ones < 0.9  # thresholds near the middle: both output values occur


def test_binary_argument_checks():
    qbuild.build()
    lib = qnn.load()
    P = ctypes.c_void_p

    def status(d, x=FAKE, t=FAKE):
        return lib.qconv_hwc_binary(ctypes.byref(d), P(x), P(FAKE), P(t), P(FAKE), None)

    assert status(qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 8, 0)) == qnn.QNN_EUNSUPPORTED  # bits must be 1
    assert status(qnn.conv_desc(1, 8, 8, 12, 32, 3, 3, 1, 1, 1, 0)) == qnn.QNN_EUNSUPPORTED  # c % 8
    assert status(qnn.conv_desc(1, 8, 8, 32, 12, 3, 3, 1, 1, 1, 0)) == qnn.QNN_EUNSUPPORTED  # m % 8
    d = qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 1, 0)
    assert status(d, x=0) == qnn.QNN_EINVAL
    assert status(d, t=0) == qnn.QNN_EINVAL
    assert status(d, t=FAKE + 2) == qnn.QNN_EALIGN
