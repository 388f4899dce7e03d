"""qconv_hwc_noalloc(): the convolution entry point that allocates nothing and
keeps its scratch in a fixed array of the library's device image.  Its output
must equal qconv_hwc()'s (the entry point with a caller-owned workspace) byte
for byte, call after call, although every call reuses the same array.

The file is named to be collected last, and passes alone in a fresh process as
well as after the other tests."""
import ctypes

import numpy as np
import pytest
import torch

from paper_1908_11263_gb300 import build as qbuild
from paper_1908_11263_gb300 import qnn

GUARD = 64
FAKE = 0x10000  # 16-byte aligned, never dereferenced: validation fails first


def _layer(seed, n, h, w, c, m, k, bits, pad, shift, per_channel_shift):
    """Seeded random layer, values packed as the binding expects."""
    rng = np.random.default_rng(seed)
    top, lo, hi = (1 << bits) - 1, -(1 << (bits - 1)), (1 << (bits - 1)) - 1
    x = rng.integers(0, top + 1, size=(n, h, w, c)).astype(np.int8)
    wt = rng.integers(lo, hi + 1, size=(m, k, k, c)).astype(np.int8)
    # bias cancels the accumulators' mean (weights average -1/2) and spreads
    # over their standard deviation; lambda adds up to half the output range
    taps = k * k * c
    centre = taps * top // 4
    spread = int(np.sqrt(taps) * ((top + 1) ** 2 - 1) / 12)
    bias = (centre + rng.integers(-spread, spread + 1, size=m)).astype(np.int32)
    kappa = rng.integers(1, 400, size=m).astype(np.int16)
    lam = rng.integers(0, (top + 1) << (shift - 1), size=m).astype(np.int32)
    shifts = rng.integers(shift - 2, shift + 3, size=m).astype(np.uint8) if per_channel_shift else None
    dev = torch.device("cuda:0")
    per = 8 // bits

    def packed(v, shape):
        t = torch.from_numpy(v.reshape(-1)).to(dev)
        if bits != 8:
            t = qnn.pack_subbyte(t, bits)
        return t.view(torch.uint8).view(shape)

    return dict(
        x=packed(x, (n, h, w, c // per)),
        w=packed(wt, (m, k, k, c // per)),
        bias=torch.from_numpy(bias).to(dev),
        kappa=torch.from_numpy(kappa).to(dev),
        lam=torch.from_numpy(lam).to(dev),
        shifts=None if shifts is None else torch.from_numpy(shifts).to(dev),
        shift=shift, bits=bits, pad=pad,
        out_shape=(n, h + 2 * pad - k + 1, w + 2 * pad - k + 1, m // per),
        desc=qnn.conv_desc(n, h, w, c, m, k, k, 1, pad, bits, shift),
    )


# The first needs the most scratch; the later ones leave stale bytes of it behind.
# Shifts are scaled to each layer's accumulator spread so that outputs span [0, 2^Q-1].
LAYERS = [
    dict(seed=101, n=3, h=17, w=20, c=64, m=96, k=3, bits=8, pad=1, shift=19, per_channel_shift=True),
    dict(seed=202, n=2, h=12, w=16, c=32, m=64, k=3, bits=4, pad=1, shift=14, per_channel_shift=False),
    dict(seed=303, n=2, h=12, w=16, c=32, m=64, k=3, bits=4, pad=1, shift=14, per_channel_shift=True),
    dict(seed=404, n=1, h=9, w=64, c=64, m=32, k=5, bits=2, pad=2, shift=14, per_channel_shift=False),
]


def _guarded(shape):
    count = int(np.prod(shape))
    buf = torch.full((count + GUARD,), 0xA5, dtype=torch.uint8, device="cuda:0")
    return buf[:count].view(shape), buf


def _noalloc(layer):
    out, buf = _guarded(layer["out_shape"])
    qnn.conv_hwc_noalloc(layer["x"], layer["w"], layer["kappa"], layer["lam"], out, bias=layer["bias"],
                         shifts=layer["shifts"], shift=layer["shift"], bits=layer["bits"], pad=layer["pad"])
    return out, buf


def _with_workspace(layer):
    return qnn.conv_hwc(layer["x"], layer["w"], layer["kappa"], layer["lam"], bias=layer["bias"],
                        shifts=layer["shifts"], shift=layer["shift"], bits=layer["bits"], pad=layer["pad"],
                        algo=qnn.ALGO_TENSORCORE)


@pytest.mark.gpu
def test_noalloc_matches_qconv_hwc_on_consecutive_calls():
    layers = [_layer(**spec) for spec in LAYERS]
    for layer in layers:
        assert qnn.conv_algo(layer["desc"]) == qnn.ALGO_TENSORCORE
        assert 0 < qnn.workspace_size(layer["desc"]) <= qnn.NOALLOC_SCRATCH_BYTES
    # two passes, each a run of back-to-back no-allocation calls on one stream
    # (largest scratch first, then the reverse order); results are read only
    # after the whole run, so each call finds the previous call's scratch
    for order in (range(len(layers)), reversed(range(len(layers)))):
        order = list(order)
        got = {i: _noalloc(layers[i]) for i in order}
        qnn.device_status()  # raises on a device-side error
        for i in order:
            want = _with_workspace(layers[i])
            out, buf = got[i]
            torch.cuda.synchronize()
            assert torch.equal(out, want), f"layer {i}: {(out != want).sum().item()} bytes differ"
            assert torch.unique(want).numel() > 8, f"layer {i}: outputs nearly constant, the check is weak"
            assert bool((buf[-GUARD:] == 0xA5).all()), f"layer {i}: write past the end of the output"


@pytest.mark.gpu
def test_noalloc_allocates_no_device_memory():
    """The property the entry point exists for: once each layer has run once on the
    device (set-up done), further calls take no device memory, neither from the CUDA
    driver (free memory does not drop) nor from torch's caching allocator (its
    allocated bytes stay the same; the outputs are allocated before the count)."""
    layers = [_layer(**spec) for spec in LAYERS]
    outs = [torch.empty(layer["out_shape"], dtype=torch.uint8, device="cuda:0") for layer in layers]

    def run_all():
        for layer, out in zip(layers, outs):
            qnn.conv_hwc_noalloc(layer["x"], layer["w"], layer["kappa"], layer["lam"], out, bias=layer["bias"],
                                 shifts=layer["shifts"], shift=layer["shift"], bits=layer["bits"], pad=layer["pad"])

    run_all()  # first use on this device: set-up, and every kernel instantiation loaded
    torch.cuda.synchronize()
    free_before, _ = torch.cuda.mem_get_info()
    allocated_before = torch.cuda.memory_allocated()
    for _ in range(8):
        run_all()
    qnn.device_status()
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info()
    assert torch.cuda.memory_allocated() == allocated_before
    assert free_after >= free_before, f"device free memory dropped by {free_before - free_after} bytes"


@pytest.fixture(scope="module")
def lib():
    qbuild.build()
    return qnn.load()


def test_noalloc_rejects_what_it_cannot_run(lib):
    """Argument checks only (no CUDA call is reached), so this runs without a GPU."""
    P = ctypes.c_void_p

    def status(d, x=FAKE, y=FAKE):
        return lib.qconv_hwc_noalloc(ctypes.byref(d), P(x), P(FAKE), P(FAKE), P(FAKE), P(FAKE), None, P(y), None)

    # 3x3, 512 -> 512 channels: about 4.7 MB of re-laid-out filters
    big = qnn.conv_desc(1, 8, 8, 512, 512, 3, 3, 1, 1, 8, 10)
    assert qnn.workspace_size(big) > qnn.NOALLOC_SCRATCH_BYTES
    assert status(big) == qnn.QNN_ESCRATCH
    assert "scratch" in qnn.status_string(qnn.QNN_ESCRATCH)
    # the CUDA-core kernel has no scratch to place: qconv_hwc() with no workspace serves it
    assert status(qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 2, 1, 8, 10)) == qnn.QNN_EUNSUPPORTED
    ok = qnn.conv_desc(1, 8, 8, 32, 32, 3, 3, 1, 1, 8, 10)
    assert status(ok, x=0) == qnn.QNN_EINVAL
    assert status(ok, y=FAKE + 8) == qnn.QNN_EALIGN


def test_noalloc_empty_batch_enqueues_nothing(lib):
    """n == 0 returns QNN_OK right after validation, before any CUDA call (so it also
    runs without a GPU) and without touching the shared scratch array."""
    P = ctypes.c_void_p
    empty = qnn.conv_desc(0, 16, 16, 32, 64, 3, 3, 1, 1, 8, 12)
    assert lib.qconv_hwc_noalloc(ctypes.byref(empty), None, P(FAKE), P(FAKE), P(FAKE), P(FAKE), None, None,
                                 None) == qnn.QNN_OK
