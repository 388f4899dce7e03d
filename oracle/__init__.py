"""CPU oracle for the quantized HWC convolution path (PULP-NN, arXiv 1908.11263).

TEST INFRASTRUCTURE ONLY.  A plain, slow, obviously correct statement of what
the GPU library computes (oracle.c, int64 throughout).  Only the tests, the
smoke check and the CPU-baseline leg of bench.py load it; the library never
does, and the two share no code.

Each wrapper takes numpy arrays and returns numpy arrays.  The arithmetic lives
in oracle.c; this module only builds it with gcc and marshals arguments.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "_build", "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, EOVERFLOW = 0, 1, 2


def build(force: bool = False) -> str:
    """Compile oracle.c into a shared library with gcc (OpenMP when available)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + ".%d.tmp" % os.getpid()
    base = ["gcc", "-O2", "-std=c99", "-shared", "-fPIC", _SRC, "-o", tmp]
    try:
        subprocess.run(base[:5] + ["-fopenmp"] + base[5:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64 = ctypes.c_int, ctypes.c_int64
            lib.oracle_unpack.argtypes = [P, i64, i32, i32, P]
            lib.oracle_pack.argtypes = [P, i64, i32, P]
            lib.oracle_conv_acc.argtypes = [i32] * 11 + [P, P, P]
            lib.oracle_floor_shift.argtypes = [i64, i32]
            lib.oracle_floor_shift.restype = i64
            lib.oracle_requant.argtypes = [i64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, i32, i32]
            lib.oracle_requant.restype = ctypes.c_int32
            lib.oracle_conv_hwc.argtypes = [i32] * 12 + [P] * 6 + [i32, P, i32]
            lib.oracle_conv_hwc_pixels.argtypes = [i32] * 12 + [P] * 6 + [i32, P, i32, P]
            lib.oracle_maxpool.argtypes = [i32] * 7 + [P, P]
            lib.oracle_conv_binary.argtypes = [i32] * 11 + [P] * 5
            lib.oracle_staircase.argtypes = [i64, P, i32]
            lib.oracle_staircase.restype = ctypes.c_int32
            lib.oracle_conv_hwc_thresholds.argtypes = [i32] * 12 + [P] * 4 + [i32]
            lib.oracle_linear.argtypes = [i32] * 3 + [P] * 4
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def _check(status, what):
    if status == EOVERFLOW:
        raise OverflowError(f"{what}: an accumulator leaves int32")
    if status != OK:
        raise ValueError(f"{what}: invalid arguments (status {status})")


def out_size(h, w, kh, kw, sh, sw, ph, pw):
    return (h + 2 * ph - kh) // sh + 1, (w + 2 * pw - kw) // sw + 1


def unpack(src, count, bits, signed):
    src = _c(src, np.uint8)
    dst = np.empty(count, np.int32)
    _check(_load().oracle_unpack(_ptr(src), count, bits, int(signed), _ptr(dst)), "unpack")
    return dst


def pack(values, bits):
    v = _c(values, np.int32).ravel()
    dst = np.empty(v.size * bits // 8, np.uint8)
    _check(_load().oracle_pack(_ptr(v), v.size, bits, _ptr(dst)), "pack")
    return dst


def conv_acc(x, w, stride=(1, 1), pad=(0, 0)):
    """int64 accumulators of Eq. 6 for unpacked x [N,H,W,C] and w [M,KH,KW,C]."""
    x = _c(x, np.int32)
    w = _c(w, np.int32)
    n, h, wd, c = x.shape
    m, kh, kw, c2 = w.shape
    assert c == c2
    oh, ow = out_size(h, wd, kh, kw, *stride, *pad)
    acc = np.empty((n, oh, ow, m), np.int64)
    _check(_load().oracle_conv_acc(n, h, wd, c, m, kh, kw, stride[0], stride[1], pad[0], pad[1],
                                   _ptr(x), _ptr(w), _ptr(acc)), "conv_acc")
    return acc


def floor_shift(t, s):
    return _load().oracle_floor_shift(int(t), int(s))


def requant(acc, bias, kappa, lam, shift, bits):
    return _load().oracle_requant(int(acc), int(bias), int(kappa), int(lam), int(shift), int(bits))


def conv_hwc(x_packed, w_packed, shape, bias, kappa, lam, shifts=None, shift=0, nthreads=1):
    """Full layer on packed buffers. shape = dict(n,h,w,c,m,kh,kw,sh,sw,ph,pw,bits). Returns packed y."""
    s = shape
    oh, ow = out_size(s["h"], s["w"], s["kh"], s["kw"], s["sh"], s["sw"], s["ph"], s["pw"])
    ny = s["n"] * oh * ow * s["m"]
    y = np.empty(ny * s["bits"] // 8, np.uint8)
    x_packed, w_packed = _c(x_packed, np.uint8), _c(w_packed, np.uint8)
    bias, kappa, lam = _c(bias, np.int32), _c(kappa, np.int16), _c(lam, np.int32)
    shifts = _c(shifts, np.uint8)
    st = _load().oracle_conv_hwc(s["n"], s["h"], s["w"], s["c"], s["m"], s["kh"], s["kw"], s["sh"], s["sw"],
                                 s["ph"], s["pw"], s["bits"], _ptr(x_packed), _ptr(w_packed), _ptr(bias),
                                 _ptr(kappa), _ptr(lam), _ptr(shifts), int(shift), _ptr(y), int(nthreads))
    _check(st, "conv_hwc")
    return y


def staircase(acc, tau, bits):
    """Staircase compression of one accumulator against one channel's thresholds (Eq. 4)."""
    t = _c(np.asarray(tau), np.int32)
    assert t.size == (1 << bits) - 1
    return int(_load().oracle_staircase(int(acc), _ptr(t), bits))


def conv_hwc_thresholds(x_packed, w_packed, shape, thresholds, nthreads=1):
    """Full layer with staircase compression; thresholds int32 [m][2^Q - 1]."""
    s = shape
    oh, ow = out_size(s["h"], s["w"], s["kh"], s["kw"], s["sh"], s["sw"], s["ph"], s["pw"])
    ny = s["n"] * oh * ow * s["m"]
    y = np.zeros(max(1, ny * s["bits"] // 8), np.uint8)
    t = _c(np.asarray(thresholds).reshape(s["m"], (1 << s["bits"]) - 1), np.int32)
    st = _load().oracle_conv_hwc_thresholds(s["n"], s["h"], s["w"], s["c"], s["m"], s["kh"], s["kw"], s["sh"], s["sw"],
                                            s["ph"], s["pw"], s["bits"], _ptr(_c(x_packed, np.uint8)),
                                            _ptr(_c(w_packed, np.uint8)), _ptr(t), _ptr(y), int(nthreads))
    _check(st, "oracle_conv_hwc_thresholds")
    return y[:ny * s["bits"] // 8]


def conv_binary(x_bits, w_bits, shape, thresholds, with_acc=False):
    """INT-1 layer (Eq. 5): x_bits / w_bits packed 8 per byte; returns packed output bits
    (and the int32 popcount accumulators when asked)."""
    s = shape
    oh, ow = out_size(s["h"], s["w"], s["kh"], s["kw"], s["sh"], s["sw"], s["ph"], s["pw"])
    ny = s["n"] * oh * ow * s["m"]
    y = np.zeros(max(1, ny // 8), np.uint8)
    acc = np.zeros(max(1, ny), np.int32) if with_acc else None
    st = _load().oracle_conv_binary(s["n"], s["h"], s["w"], s["c"], s["m"], s["kh"], s["kw"], s["sh"], s["sw"],
                                    s["ph"], s["pw"], _ptr(_c(x_bits, np.uint8)), _ptr(_c(w_bits, np.uint8)),
                                    _ptr(_c(np.asarray(thresholds), np.int32)), _ptr(y), _ptr(acc))
    _check(st, "oracle_conv_binary")
    return (y[:ny // 8], acc[:ny]) if with_acc else y[:ny // 8]


def conv_hwc_pixels(x_packed, w_packed, shape, bias, kappa, lam, pixels, shifts=None, shift=0):
    """Unpacked outputs [len(pixels), M] at the listed (n, oy, ox) output pixels."""
    s = shape
    pix = np.ascontiguousarray(np.asarray(pixels, np.int32).reshape(-1, 3))
    y = np.empty((pix.shape[0], s["m"]), np.int32)
    x_packed, w_packed = _c(x_packed, np.uint8), _c(w_packed, np.uint8)
    bias, kappa, lam = _c(bias, np.int32), _c(kappa, np.int16), _c(lam, np.int32)
    shifts = _c(shifts, np.uint8)
    st = _load().oracle_conv_hwc_pixels(s["n"], s["h"], s["w"], s["c"], s["m"], s["kh"], s["kw"], s["sh"],
                                        s["sw"], s["ph"], s["pw"], s["bits"], _ptr(x_packed), _ptr(w_packed),
                                        _ptr(bias), _ptr(kappa), _ptr(lam), _ptr(shifts), int(shift), _ptr(pix),
                                        pix.shape[0], _ptr(y))
    _check(st, "conv_hwc_pixels")
    return y


def maxpool(x_packed, n, h, w, c, k, s, bits):
    oh, ow = (h - k) // s + 1, (w - k) // s + 1
    y = np.empty(n * oh * ow * c * bits // 8, np.uint8)
    x_packed = _c(x_packed, np.uint8)
    _check(_load().oracle_maxpool(n, h, w, c, k, s, bits, _ptr(x_packed), _ptr(y)), "maxpool")
    return y


def conv_hwc_pool2(x_packed, w_packed, shape, bias, kappa, lam, shifts=None, shift=0, nthreads=1):
    """A convolution layer followed by a 2x2, stride-2 max-pooling layer over its quantized output
    (Sec. IV-A lists the pooling kernel beside the convolution), stated as the two layers in
    sequence: conv_hwc, then maxpool with window 2 and stride 2 (floor output size)."""
    y = conv_hwc(x_packed, w_packed, shape, bias, kappa, lam, shifts=shifts, shift=shift, nthreads=nthreads)
    s = shape
    oh, ow = out_size(s["h"], s["w"], s["kh"], s["kw"], s["sh"], s["sw"], s["ph"], s["pw"])
    return maxpool(y, s["n"], oh, ow, s["m"], 2, 2, s["bits"])


def linear(x, w, bias):
    """x u8 [N,K], w s8 [M,K], bias i32 [M] or None -> int32 [N,M]."""
    x = _c(x, np.uint8)
    w = _c(w, np.int8)
    bias = _c(bias, np.int32)
    n, k = x.shape
    m = w.shape[0]
    y = np.empty((n, m), np.int32)
    _check(_load().oracle_linear(n, k, m, _ptr(x), _ptr(w), _ptr(bias), _ptr(y)), "linear")
    return y
