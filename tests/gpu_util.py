"""Helpers shared by the GPU tests: run a layer through the C ABI (via the
binding) and through the oracle on the same integers, and compare bytes."""
from __future__ import annotations

import os

import numpy as np
import torch

import oracle
from paper_1908_11263_gb300 import inputs, qnn

THREADS = max(1, os.cpu_count() or 1)
GUARD = 64


def dev():
    return torch.device("cuda:0")


def to_dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.to(dev())


def pack_gpu(values: np.ndarray, bits: int) -> torch.Tensor:
    """Pack integer values on the GPU with the library's own pack kernel."""
    v = to_dev(values.astype(np.int8))
    if bits == 8:
        return v.view(torch.uint8)
    return qnn.pack_subbyte(v, bits)


def guarded_output(shape):
    """Output tensor followed by GUARD canary bytes; returns (view, whole buffer)."""
    n = int(np.prod(shape))
    buf = torch.full((n + GUARD,), 0xA5, dtype=torch.uint8, device=dev())
    return buf[:n].view(shape), buf


def check_guard(buf):
    tail = buf[-GUARD:].cpu().numpy()
    assert np.all(tail == 0xA5), "kernel wrote past the end of its output"


def conv_gpu(x, w, bias, kappa, lam, shifts, shift, bits, stride, pad, algo):
    """Layer through the C ABI; x [n,h,w,c] and w [m,kh,kw,c] are unpacked integers."""
    n, h, wd, c = x.shape
    m, kh, kw, _ = w.shape
    per = 8 // bits
    oh = (h + 2 * pad[0] - kh) // stride[0] + 1
    ow = (wd + 2 * pad[1] - kw) // stride[1] + 1
    xd = pack_gpu(x.reshape(n, h, wd, c), bits).view(n, h, wd, c // per)
    wdv = pack_gpu(w.reshape(m, kh, kw, c), bits).view(m, kh, kw, c // per)
    if bits == 8:
        wdv = wdv.view(torch.int8)
    out, buf = guarded_output((n, oh, ow, m // per))
    qnn.conv_hwc(xd, wdv, to_dev(kappa, torch.int16), to_dev(lam, torch.int32),
                 bias=None if bias is None else to_dev(bias, torch.int32),
                 shifts=None if shifts is None else to_dev(shifts, torch.uint8), shift=shift, bits=bits,
                 stride=stride, pad=pad, algo=algo, out=out)
    qnn.device_status()
    check_guard(buf)
    return out.cpu().numpy().reshape(-1)


def conv_oracle(x, w, bias, kappa, lam, shifts, shift, bits, stride, pad):
    n, h, wd, c = x.shape
    m, kh, kw, _ = w.shape
    shape = dict(n=n, h=h, w=wd, c=c, m=m, kh=kh, kw=kw, sh=stride[0], sw=stride[1], ph=pad[0], pw=pad[1],
                 bits=bits)
    if bits == 8:
        xp = x.astype(np.uint8).reshape(-1)
        wp = w.astype(np.int8).reshape(-1).view(np.uint8)
    else:
        xp = oracle.pack(x.reshape(-1), bits)
        wp = oracle.pack(w.reshape(-1), bits)
    return oracle.conv_hwc(xp, wp, shape, bias, kappa, lam, shifts=shifts, shift=shift, nthreads=THREADS)


def tc_algos(n, h, w, c, m, kh, kw, stride=(1, 1), pad=(0, 0), bits=8):
    """The tensor-core kernels that can run this layer, each as the algorithm value that forces it
    (the window kernel, the general kernel)."""
    out = []
    for algo in (qnn.ALGO_TC_WINDOW, qnn.ALGO_TC_GENERAL):
        try:
            qnn.conv_algo(qnn.conv_desc(n, h, w, c, m, kh, kw, stride, pad, bits, 0, algo))
            out.append(algo)
        except qnn.QnnError:
            pass
    return out


def all_algos(n, h, w, c, m, kh, kw, stride=(1, 1), pad=(0, 0), bits=8):
    """Every kernel that can run this layer: the tensor-core kernels and the CUDA-core one."""
    return tc_algos(n, h, w, c, m, kh, kw, stride, pad, bits) + [qnn.ALGO_DIRECT]


def first_mismatch(got, want):
    bad = np.nonzero(got != want)[0]
    if bad.size == 0:
        return None
    i = int(bad[0])
    return f"{bad.size} of {want.size} bytes differ; first at byte {i}: got {got[i]} want {want[i]}"


def layer_tensors(ld: inputs.LayerData):
    return ld.x, ld.w, ld.bias, ld.kappa, ld.lam, ld.shifts, ld.shift
