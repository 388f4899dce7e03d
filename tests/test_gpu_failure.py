"""Failure detection without a GPU fault: a bounded device-side wait that can
never complete gives up, reports QNN_ETIMEOUT through the status word, and the
context keeps working."""
import numpy as np
import pytest

from paper_1908_11263_gb300 import qnn
from gpu_util import conv_gpu, conv_oracle, first_mismatch

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives():
    qnn.selftest_wait_timeout(2_000_000)  # about a millisecond at GB300 clocks
    with pytest.raises(qnn.QnnError) as e:
        qnn.device_status()
    assert e.value.status == qnn.QNN_ETIMEOUT
    qnn.device_status()  # reading the status cleared it
    # the context is intact: a layer still matches the oracle
    rng = np.random.default_rng(7)
    x = rng.integers(0, 256, size=(2, 8, 8, 32))
    w = rng.integers(-128, 128, size=(32, 3, 3, 32))
    kappa = rng.integers(1, 64, size=32)
    lam = rng.integers(-(1 << 15), 1 << 15, size=32)
    for algo in (qnn.ALGO_DIRECT, qnn.ALGO_TENSORCORE):
        got = conv_gpu(x, w, None, kappa, lam, None, 14, 8, (1, 1), (1, 1), algo)
        want = conv_oracle(x, w, None, kappa, lam, None, 14, 8, (1, 1), (1, 1))
        assert first_mismatch(got, want) is None, algo


def test_selftest_rejects_bad_limits():
    for bad in (0, -5, 1 << 31):
        with pytest.raises(qnn.QnnError) as e:
            qnn.selftest_wait_timeout(bad)
        assert e.value.status == qnn.QNN_EINVAL
