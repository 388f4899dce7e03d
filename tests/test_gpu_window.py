"""The window tensor-core kernel (one launch per call, filters read in place, exact-chunk
count derived from the filters) and the prepared path (qconv_hwc_prepare + qconv_hwc_run) of
both tensor-core kernels, against the oracle bit for bit (Sec. III-B, Eq. 6; Sec. III-A)."""
import numpy as np
import pytest
import torch

import oracle
from paper_1908_11263_gb300 import inputs, qnn

from gpu_util import conv_gpu, conv_oracle, dev, first_mismatch, layer_tensors, pack_gpu, tc_algos, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def loaded():
    qnn.load(build_if_missing=True)
    torch.cuda.set_device(0)


def centred_requant(x, wt, bits):
    """kappa = 1, a shift matched to the accumulators' spread and a per-channel lambda that
    centres each channel in the output range: outputs spread over [0, 2^Q - 1] and every
    output changes with the accumulator at the scale of 2^shift (shift 0 where the spread
    allows it: then every output depends on the accumulator's last bit)."""
    import oracle
    acc = oracle.conv_acc(x, wt, (1, 1), (1, 1)).reshape(-1, wt.shape[0]).astype(np.int64)
    spread = float(np.percentile(acc, 90) - np.percentile(acc, 10))
    top = (1 << bits) - 1
    shift = int(max(0, np.ceil(np.log2(max(1.0, spread / (0.8 * top))))))
    lam = ((top + 1) // 2 * (1 << shift) - np.median(acc, axis=0)).astype(np.int64)
    return np.clip(lam, -(1 << 31), (1 << 31) - 1).astype(np.int32), shift


# (n, h, w, c, m, k): the benchmark layer's shape, C = 64 (K = 576) and a 5x5 window (K = 800)
SHAPES = [(2, 16, 16, 32, 64, 3), (1, 16, 16, 64, 64, 3), (2, 16, 16, 32, 32, 5)]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
@pytest.mark.parametrize("pattern", ["uniform", "extreme", "one_extreme_channel", "alternating"])
def test_chunk_count_from_filters(shape, pattern):
    """INT-8 filters whose sum |w| decides how many exact fp32 chunks the window kernel takes:
    uniform random filters allow fewer chunks than the worst case; filters at -128 throughout
    (one channel, or all) force the worst case for every channel; alternating extremes keep the
    true sum small while the chunk bound stays large.  Both tensor-core kernels equal the oracle."""
    n, h, w, c, m, k = shape
    rng = np.random.default_rng(sum(shape) * 7 + len(pattern))
    x = rng.integers(0, 256, size=(n, h, w, c))
    wt = rng.integers(-128, 128, size=(m, k, k, c))
    if pattern == "extreme":
        wt[:] = -128
        x[:] = rng.integers(0, 2, size=x.shape) * 255  # staged values at both ends
    elif pattern == "one_extreme_channel":
        wt[m // 3] = -128
    elif pattern == "alternating":
        wt[..., 0::2] = 127
        wt[..., 1::2] = -128
    lam, shift = centred_requant(x, wt, 8)
    kappa = np.ones(m, np.int16)
    want = conv_oracle(x, wt, None, kappa, lam, None, shift, 8, (1, 1), (1, 1))
    if pattern != "extreme":
        assert len(np.unique(want)) > 32, "outputs nearly constant: the check is weak"
    algos = tc_algos(n, h, w, c, m, k, k, (1, 1), (1, 1), 8)
    assert qnn.ALGO_TC_WINDOW in algos
    for algo in algos:
        got = conv_gpu(x, wt, None, kappa, lam, None, shift, 8, (1, 1), (1, 1), algo)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))


@pytest.mark.parametrize("bits", [8, 4, 2])
def test_benchmark_layer_takes_the_window_kernel(bits):
    d = qnn.conv_desc(512, 16, 16, 32, 64, 3, 3, 1, 1, bits, 12)
    assert qnn.tc_kernel(d) == qnn.ALGO_TC_WINDOW
    assert qnn.mma_operand_bits(d) == (16 if bits == 8 else 8)


@pytest.mark.parametrize("algo", [qnn.ALGO_TC_WINDOW, qnn.ALGO_TC_GENERAL])
@pytest.mark.parametrize("bits", [8, 4, 2])
@pytest.mark.parametrize("with_bias_and_shifts", [True, False])
def test_prepared_path(algo, bits, with_bias_and_shifts):
    """qconv_hwc_prepare once, then qconv_hwc_run on two different inputs: each equals the
    oracle.  Without bias and per-channel shifts the prepared workspace must stand in zeros
    and the scalar shift."""
    # INT-2 rows of a 20-pixel image are 160 B, but a window of it starts at 8-byte pixels, so
    # the window kernel needs whole-row windows there: 16 pixels wide
    n, h, w, c, m, k = 3, 14, 20 if bits != 2 else 16, 32, 48, 3
    assert algo in tc_algos(n, h, w, c, m, k, k, (1, 1), (1, 1), bits)
    rng = np.random.default_rng(bits * 11 + algo + int(with_bias_and_shifts))
    top = (1 << bits) - 1
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, k, k, c))
    taps = k * k * c
    bias = (taps * top // 4 + rng.integers(-50, 51, size=m)).astype(np.int32) if with_bias_and_shifts else None
    kappa = rng.integers(1, 300, size=m).astype(np.int16)
    shift = {8: 14, 4: 10, 2: 8}[bits]
    lam = rng.integers(0, (top + 1) << (shift - 1), size=m).astype(np.int64)
    if bias is None:  # centre the accumulators through lambda instead (weights average -1/2)
        lam += (taps * top // 4) * kappa.astype(np.int64)
    lam = lam.astype(np.int32)
    shifts = rng.integers(shift - 2, shift + 3, size=m).astype(np.uint8) if with_bias_and_shifts else None
    per = 8 // bits
    wd = pack_gpu(wt, bits).view(m, k, k, c // per)
    if bits == 8:
        wd = wd.view(torch.int8)
    prep = qnn.PreparedConv(wd, to_dev(kappa, torch.int16), to_dev(lam, torch.int32), n=n, h=h, wd=w,
                            bias=None if bias is None else to_dev(bias, torch.int32),
                            shifts=None if shifts is None else to_dev(shifts, torch.uint8), shift=shift, bits=bits,
                            stride=1, pad=1, algo=algo)
    for trial in range(2):
        x = rng.integers(0, top + 1, size=(n, h, w, c))
        want = conv_oracle(x, wt, bias, kappa, lam, shifts, shift, bits, (1, 1), (1, 1))
        got = prep(pack_gpu(x, bits).view(n, h, w, c // per)).cpu().numpy().reshape(-1)
        qnn.device_status()
        assert first_mismatch(got, want) is None, (trial, first_mismatch(got, want))
        assert len(np.unique(want)) > 4


@pytest.mark.parametrize("which", ["w2", "w4_int4", "w4_int2"])
def test_prepared_graph_full_size(which):
    """The launch configuration bench.py times, at the benchmark layer's full size (batch 512):
    filters prepared once, then qconv_hwc_run launches captured back to back in a CUDA graph on a
    side stream (consecutive launches overlap through programmatic dependent launch), alternating
    between two inputs and four outputs.  Every output byte equals the oracle's."""
    if which == "w2":
        (key, layer, wl, lid), = inputs.single_layer_workload(inputs.WORKLOAD_BATCH)
    else:
        (key, layer, wl, lid), = [t for t in inputs.single_layer_workload(inputs.WORKLOAD_SUBBYTE) if t[0] == which]
    ld = inputs.make_layer(key, layer, wl, lid)
    x, wt, bias, kappa, lam, shifts, shift = layer_tensors(ld)
    bits, n = layer.bits, layer.n
    st, pd = (layer.stride, layer.stride), (layer.pad, layer.pad)
    want = conv_oracle(x, wt, bias, kappa, lam, shifts, shift, bits, st, pd)
    want = want.reshape(n, -1)
    assert len(np.unique(want)) > 4
    per = 8 // bits
    xs = [pack_gpu(x, bits).view(n, layer.h, layer.w, layer.c // per)]
    xs.append(torch.flip(xs[0], dims=[0]).contiguous())  # the batch reversed: outputs reverse with it
    wd = pack_gpu(wt, bits).view(layer.m, layer.k, layer.k, layer.c // per)
    if bits == 8:
        wd = wd.view(torch.int8)
    stream = torch.cuda.Stream()
    prep = qnn.PreparedConv(wd, to_dev(kappa, torch.int16), to_dev(lam, torch.int32), n=n, h=layer.h, wd=layer.w,
                            bias=None if bias is None else to_dev(bias, torch.int32),
                            shifts=None if shifts is None else to_dev(shifts, torch.uint8), shift=shift, bits=bits,
                            stride=layer.stride, pad=layer.pad, stream=stream)
    assert qnn.tc_kernel(prep.desc) == qnn.ALGO_TC_WINDOW
    ys = [torch.full(prep.out_shape, 0xA5, dtype=torch.uint8, device=dev()) for _ in range(4)]
    with torch.cuda.stream(stream):
        prep(xs[0], out=ys[0], stream=stream)  # eager warm-up launch
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(8):
            prep(xs[i % 2], out=ys[i % 4], stream=stream)
    for y in ys:
        y.fill_(0xA5)
    torch.cuda.synchronize()
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    qnn.device_status()
    for i, y in enumerate(ys):
        got = y.cpu().numpy().reshape(n, -1)
        exp = want if i % 2 == 0 else want[::-1]
        assert first_mismatch(got.reshape(-1), np.ascontiguousarray(exp).reshape(-1)) is None, (which, i)


@pytest.mark.parametrize("shape", [
    (2, 32, 32, 3, 32, 5, 5, 2),    # CIFAR conv1 shape: 15 of 16 values per kernel row
    (2, 21, 32, 3, 16, 3, 3, 1),    # 9 values, a partial last tile row
    (1, 16, 48, 5, 24, 3, 3, 1),    # 15 values, three tiles across
    (2, 19, 16, 1, 8, 7, 7, 3),     # one channel, 7 wide
    (1, 20, 32, 2, 40, 5, 5, 0),    # no padding
    (3, 9, 16, 4, 32, 4, 4, 2),     # exactly 16 values, even kernel
])
@pytest.mark.parametrize("pool", [False, True])
def test_folded_kernel_columns(shape, pool):
    """Few input channels (C * kw <= 16, C not a multiple of 8): the window kernel folds the
    kernel columns into K, so a staged position carries kw neighbouring pixels' channels and an
    MMA covers one kernel row.  Every output byte equals the oracle's (and, with pool, the
    oracle's conv followed by its 2x2 max-pool), on the folded window kernel and on the general
    kernel, one-shot and prepared."""
    n, h, w, c, m, k, _, p = shape
    desc = qnn.conv_desc(n, h, w, c, m, k, k, 1, p, 8, 0)
    assert qnn.tc_kernel(desc) == qnn.ALGO_TC_WINDOW
    rng = np.random.default_rng(sum(shape) * 7 + int(pool))
    x = rng.integers(0, 256, size=(n, h, w, c))
    wt = rng.integers(-128, 128, size=(m, k, k, c))
    kappa = rng.integers(1, 64, size=m).astype(np.int16)
    bias = rng.integers(-4096, 4097, size=m).astype(np.int32)
    shift = 12
    lam = rng.integers(0, 256 << (shift - 1), size=m).astype(np.int32)
    want = conv_oracle(x, wt, bias, kappa, lam, None, shift, 8, (1, 1), (p, p))
    oh, ow = h + 2 * p - k + 1, w + 2 * p - k + 1
    if pool:
        want = oracle.maxpool(want, n, oh, ow, m, 2, 2, 8)
    assert len(np.unique(want)) > 16, "outputs nearly constant: the check is weak"
    xd, wd = to_dev(x.astype(np.uint8)), to_dev(wt.astype(np.int8))
    kd, ld_, bd = to_dev(kappa), to_dev(lam), to_dev(bias)
    for algo in (qnn.ALGO_TC_WINDOW, qnn.ALGO_TC_GENERAL):
        if pool:
            got = qnn.conv_hwc_pool2(xd, wd, kd, ld_, bias=bd, shift=shift, bits=8, pad=p, algo=algo)
        else:
            got = qnn.conv_hwc(xd, wd, kd, ld_, bias=bd, shift=shift, bits=8, stride=1, pad=p, algo=algo)
        qnn.device_status()
        got = got.cpu().numpy().reshape(-1)
        assert first_mismatch(got, want) is None, (algo, first_mismatch(got, want))
    if not pool:
        prep = qnn.PreparedConv(wd, kd, ld_, n=n, h=h, wd=w, bias=bd, shift=shift, bits=8, stride=1, pad=p)
        got = prep(xd).cpu().numpy().reshape(-1)
        qnn.device_status()
        assert first_mismatch(got, want) is None, ("prepared", first_mismatch(got, want))


@pytest.mark.parametrize("seed", range(24))
def test_random_shapes(seed):
    """Seeded random layers across the window planner's range (bit width, channels including the
    folded few-channel case, filters, kernel, padding, image size, fused pool): every tensor-core
    kernel that takes the layer equals the oracle byte for byte."""
    rng = np.random.default_rng(1000 + seed)
    bits = int(rng.choice([8, 8, 4, 2]))
    per = 8 // bits
    if bits == 8:
        c = int(rng.integers(1, 6)) if rng.integers(0, 3) == 0 else 8 * int(rng.integers(1, 9))
    else:
        c = 32 * int(rng.integers(1, 3))
    m = per * int(rng.integers(1, 96 // per + 1))
    kh, kw = int(rng.integers(1, 6)), int(rng.integers(1, 6))
    ph, pw = int(rng.integers(0, kh // 2 + 1)), int(rng.integers(0, kw // 2 + 1))
    n = int(rng.integers(1, 4))
    h = int(rng.integers(max(2, kh - 2 * ph + 1), 30))
    w = int(rng.integers(max(2, kw - 2 * pw + 1), 36))
    pool = bool(rng.integers(0, 2))
    desc = qnn.conv_desc(n, h, w, c, m, kh, kw, 1, (ph, pw), bits, 0)
    algos = tc_algos(n, h, w, c, m, kh, kw, (1, 1), (ph, pw), bits)
    if not algos:
        pytest.skip("no tensor-core kernel takes this layer")
    top = (1 << bits) - 1
    x = rng.integers(0, top + 1, size=(n, h, w, c))
    wt = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(m, kh, kw, c))
    taps = kh * kw * c
    shift = {8: 12, 4: 8, 2: 6}[bits]
    kappa = rng.integers(1, 64, size=m).astype(np.int16)
    bias = rng.integers(-(taps * top), taps * top + 1, size=m).astype(np.int32)
    lam = rng.integers(0, (top + 1) << shift, size=m).astype(np.int32)
    oh, ow = h + 2 * ph - kh + 1, w + 2 * pw - kw + 1
    want = conv_oracle(x, wt, bias, kappa, lam, None, shift, bits, (1, 1), (ph, pw))
    if pool:
        if oh < 2 or ow < 2:
            pytest.skip("no pooled pixel")
        want = oracle.maxpool(want, n, oh, ow, m, 2, 2, bits)
    xd = pack_gpu(x, bits).view(n, h, w, c // per)
    wd = pack_gpu(wt, bits).view(m, kh, kw, c // per)
    if bits == 8:
        wd = wd.view(torch.int8)
    kd, ld_, bd = to_dev(kappa), to_dev(lam), to_dev(bias)
    for algo in algos:
        if pool:
            got = qnn.conv_hwc_pool2(xd, wd, kd, ld_, bias=bd, shift=shift, bits=bits, pad=(ph, pw), algo=algo)
        else:
            got = qnn.conv_hwc(xd, wd, kd, ld_, bias=bd, shift=shift, bits=bits, stride=1, pad=(ph, pw), algo=algo)
        qnn.device_status()
        got = got.cpu().numpy().reshape(-1)
        assert first_mismatch(got, want) is None, (seed, desc_str(n, h, w, c, m, kh, kw, ph, pw, bits, pool), algo,
                                                   first_mismatch(got, want))


def desc_str(*v):
    return "n=%d h=%d w=%d c=%d m=%d k=%dx%d pad=%d,%d q%d pool=%d" % v
