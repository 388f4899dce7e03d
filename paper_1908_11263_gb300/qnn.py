"""Python binding of libqnn (include/qnn.h): argument marshalling only.

PyTorch provides device memory and the current stream; every step of the
computation runs in the library's CUDA kernels.  There is no fallback: when the
library is missing or fails to load, every call raises.

Tensor conventions (packed Q-bit data lives in uint8 tensors whose last
dimension counts bytes):
  activations  uint8 [n, h, w, c*Q/8]    weights  int8/uint8 [m, kh, kw, c*Q/8]
  outputs      uint8 [n, oh, ow, m*Q/8]
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

QNN_OK, QNN_EINVAL, QNN_EUNSUPPORTED, QNN_EALIGN, QNN_ECUDA, QNN_ETIMEOUT, QNN_EWORKSPACE = range(7)
QNN_ESCRATCH = 7
NOALLOC_SCRATCH_BYTES = 2 << 20  # QNN_NOALLOC_SCRATCH_BYTES
ALGO_AUTO, ALGO_DIRECT, ALGO_TENSORCORE, ALGO_TC_WINDOW, ALGO_TC_GENERAL = 0, 1, 2, 3, 4

EXPORTED = ("qconv_hwc_workspace_size", "qconv_hwc", "qconv_hwc_prepare", "qconv_hwc_run", "qconv_hwc_algo", "qlinear", "qmaxpool", "pack_subbyte",
            "unpack_subbyte", "qnn_device_status", "qnn_status_string", "qnn_version", "qconv_hwc_noalloc",
            "qnn_selftest_wait_timeout", "qconv_hwc_thresholds", "qconv_hwc_binary", "qconv_hwc_pool2", "qconv_hwc_pool2_run",
            "qconv_hwc_mma_operand_bits", "qconv_hwc_tc_kernel")


class QnnError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} (status {status})")


class ConvDesc(ctypes.Structure):
    _fields_ = [("struct_size", ctypes.c_uint32)] + [(f, ctypes.c_int32) for f in (
        "n", "h", "w", "c", "m", "kh", "kw", "stride_h", "stride_w", "pad_h", "pad_w", "bits", "shift", "algo")]


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = False):
    """Load libqnn.so (building it first only when asked)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if not os.path.exists(path):
            if not build_if_missing:
                raise RuntimeError(f"libqnn.so is not built ({path}); run paper_1908_11263_gb300.build.build()")
            _build.build()
        lib = ctypes.CDLL(path)
        P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        DP = ctypes.POINTER(ConvDesc)
        lib.qconv_hwc_workspace_size.argtypes = [DP, ctypes.POINTER(SZ)]
        lib.qconv_hwc_workspace_size.restype = I32
        lib.qconv_hwc.argtypes = [DP, P, P, P, P, P, P, P, P, SZ, P]
        lib.qconv_hwc.restype = I32
        lib.qconv_hwc_pool2.argtypes = [DP, P, P, P, P, P, P, P, P, SZ, P]
        lib.qconv_hwc_pool2.restype = I32
        lib.qconv_hwc_prepare.argtypes = [DP, P, P, P, P, P, P, SZ, P]
        lib.qconv_hwc_prepare.restype = I32
        lib.qconv_hwc_run.argtypes = [DP, P, P, P, SZ, P]
        lib.qconv_hwc_run.restype = I32
        lib.qconv_hwc_pool2_run.argtypes = [DP, P, P, P, SZ, P]
        lib.qconv_hwc_pool2_run.restype = I32
        lib.qconv_hwc_algo.argtypes = [DP]
        lib.qconv_hwc_noalloc.argtypes = [DP, P, P, P, P, P, P, P, P]
        lib.qconv_hwc_thresholds.argtypes = [DP, P, P, P, P, P, SZ, P]
        lib.qconv_hwc_binary.argtypes = [DP, P, P, P, P, P]
        lib.qconv_hwc_binary.restype = I32
        lib.qconv_hwc_thresholds.restype = I32
        lib.qconv_hwc_noalloc.restype = I32
        lib.qconv_hwc_algo.restype = I32
        lib.qconv_hwc_mma_operand_bits.argtypes = [DP]
        lib.qconv_hwc_mma_operand_bits.restype = I32
        lib.qconv_hwc_tc_kernel.argtypes = [DP]
        lib.qconv_hwc_tc_kernel.restype = I32
        lib.qlinear.argtypes = [I32, I32, I32, P, P, P, P, P]
        lib.qlinear.restype = I32
        lib.qmaxpool.argtypes = [I32] * 7 + [P, P, P]
        lib.qmaxpool.restype = I32
        lib.pack_subbyte.argtypes = [P, P, I64, I32, P]
        lib.pack_subbyte.restype = I32
        lib.unpack_subbyte.argtypes = [P, P, I64, I32, I32, P]
        lib.unpack_subbyte.restype = I32
        lib.qnn_selftest_wait_timeout.argtypes = [I64, P]
        lib.qnn_selftest_wait_timeout.restype = I32
        lib.qnn_device_status.argtypes = [P]
        lib.qnn_device_status.restype = I32
        lib.qnn_status_string.argtypes = [I32]
        lib.qnn_status_string.restype = ctypes.c_char_p
        lib.qnn_version.argtypes = []
        lib.qnn_version.restype = I32
        _lib = lib
        return lib


def status_string(status: int) -> str:
    try:
        return load().qnn_status_string(int(status)).decode()
    except Exception:
        return "unknown"


def _check(status: int, what: str):
    if status != QNN_OK:
        raise QnnError(status, what)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t: torch.Tensor, dtype, name):
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype not in (dtype if isinstance(dtype, tuple) else (dtype,)):
        raise TypeError(f"{name} must have dtype {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def conv_desc(n, h, w, c, m, kh, kw, stride=(1, 1), pad=(0, 0), bits=8, shift=0, algo=ALGO_AUTO) -> ConvDesc:
    sh, sw = (stride, stride) if isinstance(stride, int) else stride
    ph, pw = (pad, pad) if isinstance(pad, int) else pad
    return ConvDesc(ctypes.sizeof(ConvDesc), n, h, w, c, m, kh, kw, sh, sw, ph, pw, bits, shift, algo)


def workspace_size(desc: ConvDesc) -> int:
    out = ctypes.c_size_t(0)
    _check(load().qconv_hwc_workspace_size(ctypes.byref(desc), ctypes.byref(out)), "qconv_hwc_workspace_size")
    return out.value


def conv_algo(desc: ConvDesc) -> int:
    r = load().qconv_hwc_algo(ctypes.byref(desc))
    if r < 0:
        raise QnnError(-r, "qconv_hwc_algo")
    return r


def tc_kernel(desc: ConvDesc) -> int:
    """The tensor-core kernel qconv_hwc() runs for this descriptor: ALGO_TC_WINDOW or
    ALGO_TC_GENERAL (0 for the CUDA-core kernel)."""
    r = load().qconv_hwc_tc_kernel(ctypes.byref(desc))
    if r < 0:
        raise QnnError(-r, "qconv_hwc_tc_kernel")
    return r


def mma_operand_bits(desc: ConvDesc) -> int:
    """Operand width of the tensor-core MMAs for this descriptor: 16 (fp16, kind::f16),
    8 (e4m3, kind::f8f6f4) or 0 (CUDA-core kernel)."""
    r = load().qconv_hwc_mma_operand_bits(ctypes.byref(desc))
    if r < 0:
        raise QnnError(-r, "qconv_hwc_mma_operand_bits")
    return r


_workspaces: dict = {}


def _workspace(nbytes: int, device, stream):
    """Workspace per (device, stream): calls on one stream never overlap."""
    if nbytes == 0:
        return None
    key = (device.index, stream.cuda_stream if stream is not None else torch.cuda.current_stream(device).cuda_stream)
    buf = _workspaces.get(key)
    if buf is None or buf.numel() < nbytes:
        buf = torch.empty(nbytes, dtype=torch.uint8, device=device)
        _workspaces[key] = buf
    return buf


def conv_hwc(x, w, kappa, lam, *, bias=None, shifts=None, shift=0, bits=8, stride=1, pad=0, algo=ALGO_AUTO,
             out=None, workspace=None, stream=None):
    """Quantized HWC convolution with fused compression; returns uint8 [n, oh, ow, m*Q/8]."""
    _dev(x, torch.uint8, "x")
    _dev(w, (torch.int8, torch.uint8), "w")
    _dev(kappa, torch.int16, "kappa")
    _dev(lam, torch.int32, "lambda")
    if bias is not None:
        _dev(bias, torch.int32, "bias")
    if shifts is not None:
        _dev(shifts, torch.uint8, "shifts")
    per = 8 // bits
    n, h, wd, cb = x.shape
    m, kh, kw, cb2 = w.shape
    if cb != cb2:
        raise ValueError("x and w disagree on the channel count")
    desc = conv_desc(n, h, wd, cb * per, m, kh, kw, stride, pad, bits, shift, algo)
    oh = (h + 2 * desc.pad_h - kh) // desc.stride_h + 1
    ow = (wd + 2 * desc.pad_w - kw) // desc.stride_w + 1
    if out is None:
        out = torch.empty((n, oh, ow, m // per), dtype=torch.uint8, device=x.device)
    else:
        _dev(out, torch.uint8, "out")
    nbytes = workspace_size(desc)
    if workspace is None:
        workspace = _workspace(nbytes, x.device, stream)
    elif workspace.numel() < nbytes:
        raise ValueError("workspace too small")
    st = load().qconv_hwc(ctypes.byref(desc), _ptr(x), _ptr(w), _ptr(bias), _ptr(kappa), _ptr(lam), _ptr(shifts),
                          _ptr(out), _ptr(workspace), ctypes.c_size_t(nbytes), _stream(stream))
    _check(st, "qconv_hwc")
    return out


def conv_hwc_pool2(x, w, kappa, lam, *, bias=None, shifts=None, shift=0, bits=8, pad=0, algo=ALGO_AUTO, out=None,
                   workspace=None, stream=None):
    """Quantized HWC convolution (stride 1) with fused compression and 2x2 stride-2 max-pooling
    (qconv_hwc_pool2); returns uint8 [n, oh // 2, ow // 2, m*Q/8]."""
    _dev(x, torch.uint8, "x")
    _dev(w, (torch.int8, torch.uint8), "w")
    _dev(kappa, torch.int16, "kappa")
    _dev(lam, torch.int32, "lambda")
    if bias is not None:
        _dev(bias, torch.int32, "bias")
    if shifts is not None:
        _dev(shifts, torch.uint8, "shifts")
    per = 8 // bits
    n, h, wd, cb = x.shape
    m, kh, kw, cb2 = w.shape
    if cb != cb2:
        raise ValueError("x and w disagree on the channel count")
    desc = conv_desc(n, h, wd, cb * per, m, kh, kw, 1, pad, bits, shift, algo)
    oh = h + 2 * desc.pad_h - kh + 1
    ow = wd + 2 * desc.pad_w - kw + 1
    if out is None:
        out = torch.empty((n, oh // 2, ow // 2, m // per), dtype=torch.uint8, device=x.device)
    else:
        _dev(out, torch.uint8, "out")
    nbytes = workspace_size(desc)
    if workspace is None:
        workspace = _workspace(nbytes, x.device, stream)
    elif workspace.numel() < nbytes:
        raise ValueError("workspace too small")
    st = load().qconv_hwc_pool2(ctypes.byref(desc), _ptr(x), _ptr(w), _ptr(bias), _ptr(kappa), _ptr(lam),
                                _ptr(shifts), _ptr(out), _ptr(workspace), ctypes.c_size_t(nbytes), _stream(stream))
    _check(st, "qconv_hwc_pool2")
    return out


def conv_hwc_thresholds(x, w, thresholds, *, bits, stride=1, pad=0, algo=ALGO_AUTO, out=None, workspace=None,
                        stream=None):
    """Quantized HWC convolution with staircase compression (qconv_hwc_thresholds): INT-4 or INT-2
    outputs equal to the number of each channel's thresholds (int32 [m][2^Q - 1]) not above the
    accumulator; returns uint8 [n, oh, ow, m*Q/8]."""
    _dev(x, torch.uint8, "x")
    _dev(w, (torch.int8, torch.uint8), "w")
    _dev(thresholds, torch.int32, "thresholds")
    per = 8 // bits
    n, h, wd, cb = x.shape
    m, kh, kw, cb2 = w.shape
    if cb != cb2:
        raise ValueError("x and w disagree on the channel count")
    if tuple(thresholds.shape) != (m, (1 << bits) - 1):
        raise ValueError(f"thresholds must have shape {(m, (1 << bits) - 1)}")
    desc = conv_desc(n, h, wd, cb * per, m, kh, kw, stride, pad, bits, 0, algo)
    oh = (h + 2 * desc.pad_h - kh) // desc.stride_h + 1
    ow = (wd + 2 * desc.pad_w - kw) // desc.stride_w + 1
    if out is None:
        out = torch.empty((n, oh, ow, m // per), dtype=torch.uint8, device=x.device)
    else:
        _dev(out, torch.uint8, "out")
    nbytes = workspace_size(desc)
    if workspace is None:
        workspace = _workspace(nbytes, x.device, stream)
    elif workspace.numel() < nbytes:
        raise ValueError("workspace too small")
    st = load().qconv_hwc_thresholds(ctypes.byref(desc), _ptr(x), _ptr(w), _ptr(thresholds), _ptr(out),
                                     _ptr(workspace), ctypes.c_size_t(nbytes), _stream(stream))
    _check(st, "qconv_hwc_thresholds")
    return out


def conv_binary(x, w, thresholds, *, stride=1, pad=0, out=None, stream=None):
    """INT-1 convolution (qconv_hwc_binary): x uint8 [n, h, w, c/8], w uint8 [m, kh, kw, c/8] (bits,
    +1 = 1), thresholds int32 [m]; returns uint8 [n, oh, ow, m/8] output bits."""
    _dev(x, torch.uint8, "x")
    _dev(w, torch.uint8, "w")
    _dev(thresholds, torch.int32, "thresholds")
    n, h, wd, cb = x.shape
    m, kh, kw, cb2 = w.shape
    if cb != cb2:
        raise ValueError("x and w disagree on the channel count")
    desc = conv_desc(n, h, wd, cb * 8, m, kh, kw, stride, pad, 1, 0, ALGO_AUTO)
    oh = (h + 2 * desc.pad_h - kh) // desc.stride_h + 1
    ow = (wd + 2 * desc.pad_w - kw) // desc.stride_w + 1
    if out is None:
        out = torch.empty((n, oh, ow, m // 8), dtype=torch.uint8, device=x.device)
    else:
        _dev(out, torch.uint8, "out")
    _check(load().qconv_hwc_binary(ctypes.byref(desc), _ptr(x), _ptr(w), _ptr(thresholds), _ptr(out), _stream(stream)),
           "qconv_hwc_binary")
    return out


def conv_hwc_noalloc(x, w, kappa, lam, out, *, bias=None, shifts=None, shift=0, bits=8, stride=1, pad=0,
                     algo=ALGO_AUTO, stream=None):
    """conv_hwc() through qconv_hwc_noalloc(): no device memory is allocated,
    neither by the library nor here (the caller passes `out`).

    For callers that cannot allocate device memory: a runtime whose memory is
    all committed to its own arenas, a latency-critical loop where an allocation
    or free would synchronise the device, a caller with no allocator to own a
    workspace.  The layer's scratch goes to the library's fixed array of
    NOALLOC_SCRATCH_BYTES per device; larger layers raise QnnError with status
    QNN_ESCRATCH.  Only descriptors that select the tensor-core kernel.  The
    first call on a device does set-up (the array's device address, the
    kernel's shared-memory limit): make it before any stream capture.  All calls
    share the array: calls on different streams must not overlap on the GPU.
    """
    _dev(x, torch.uint8, "x")
    _dev(w, (torch.int8, torch.uint8), "w")
    _dev(kappa, torch.int16, "kappa")
    _dev(lam, torch.int32, "lambda")
    _dev(out, torch.uint8, "out")
    if bias is not None:
        _dev(bias, torch.int32, "bias")
    if shifts is not None:
        _dev(shifts, torch.uint8, "shifts")
    per = 8 // bits
    n, h, wd, cb = x.shape
    m, kh, kw, cb2 = w.shape
    if cb != cb2:
        raise ValueError("x and w disagree on the channel count")
    desc = conv_desc(n, h, wd, cb * per, m, kh, kw, stride, pad, bits, shift, algo)
    oh = (h + 2 * desc.pad_h - kh) // desc.stride_h + 1
    ow = (wd + 2 * desc.pad_w - kw) // desc.stride_w + 1
    if tuple(out.shape) != (n, oh, ow, m // per):
        raise ValueError(f"out must have shape {(n, oh, ow, m // per)}, got {tuple(out.shape)}")
    st = load().qconv_hwc_noalloc(ctypes.byref(desc), _ptr(x), _ptr(w), _ptr(bias), _ptr(kappa), _ptr(lam),
                                  _ptr(shifts), _ptr(out), _stream(stream))
    _check(st, "qconv_hwc_noalloc")
    return out


class PreparedConv:
    """A layer whose filters and compression constants were prepared once
    (qconv_hwc_prepare); calling it runs only the convolution (qconv_hwc_run)."""

    def __init__(self, w, kappa, lam, *, n, h, wd, bias=None, shifts=None, shift=0, bits=8, stride=1, pad=0,
                 algo=ALGO_TENSORCORE, stream=None):
        _dev(w, (torch.int8, torch.uint8), "w")
        _dev(kappa, torch.int16, "kappa")
        _dev(lam, torch.int32, "lambda")
        per = 8 // bits
        m, kh, kw, cb = w.shape
        self.desc = conv_desc(n, h, wd, cb * per, m, kh, kw, stride, pad, bits, shift, algo)
        self.oh = (h + 2 * self.desc.pad_h - kh) // self.desc.stride_h + 1
        self.ow = (wd + 2 * self.desc.pad_w - kw) // self.desc.stride_w + 1
        self.out_shape = (n, self.oh, self.ow, m // per)
        self.nbytes = workspace_size(self.desc)
        self.workspace = torch.empty(max(self.nbytes, 1), dtype=torch.uint8, device=w.device)
        self._keep = (w, kappa, lam, bias, shifts)
        st = load().qconv_hwc_prepare(ctypes.byref(self.desc), _ptr(w), _ptr(bias), _ptr(kappa), _ptr(lam),
                                      _ptr(shifts), _ptr(self.workspace), ctypes.c_size_t(self.nbytes),
                                      _stream(stream))
        _check(st, "qconv_hwc_prepare")

    def __call__(self, x, out=None, stream=None):
        _dev(x, torch.uint8, "x")
        if out is None:
            out = torch.empty(self.out_shape, dtype=torch.uint8, device=x.device)
        st = load().qconv_hwc_run(ctypes.byref(self.desc), _ptr(x), _ptr(out), _ptr(self.workspace),
                                  ctypes.c_size_t(self.nbytes), _stream(stream))
        _check(st, "qconv_hwc_run")
        return out

    def pool2(self, x, out=None, stream=None):
        """The convolution with its 2x2 stride-2 max-pool fused (qconv_hwc_pool2_run); returns
        uint8 [n, oh // 2, ow // 2, m*Q/8]."""
        _dev(x, torch.uint8, "x")
        if out is None:
            n, _, _, mb = self.out_shape
            out = torch.empty((n, self.oh // 2, self.ow // 2, mb), dtype=torch.uint8, device=x.device)
        st = load().qconv_hwc_pool2_run(ctypes.byref(self.desc), _ptr(x), _ptr(out), _ptr(self.workspace),
                                        ctypes.c_size_t(self.nbytes), _stream(stream))
        _check(st, "qconv_hwc_pool2_run")
        return out


def linear(x, w, bias=None, *, out=None, stream=None):
    """y[b][o] = sum_i x[b][i] * w[o][i] + bias[o]; int32 [n, m]."""
    _dev(x, torch.uint8, "x")
    _dev(w, torch.int8, "w")
    if bias is not None:
        _dev(bias, torch.int32, "bias")
    n, k = x.shape
    m, k2 = w.shape
    if k != k2:
        raise ValueError("x and w disagree on k")
    if out is None:
        out = torch.empty((n, m), dtype=torch.int32, device=x.device)
    st = load().qlinear(n, k, m, _ptr(x), _ptr(w), _ptr(bias), _ptr(out), _stream(stream))
    _check(st, "qlinear")
    return out


def maxpool(x, k=2, s=2, bits=8, *, out=None, stream=None):
    """Max-pool packed NHWC activations; returns uint8 [n, oh, ow, c*Q/8]."""
    _dev(x, torch.uint8, "x")
    n, h, wd, cb = x.shape
    c = cb * 8 // bits
    oh, ow = (h - k) // s + 1, (wd - k) // s + 1
    if out is None:
        out = torch.empty((n, oh, ow, cb), dtype=torch.uint8, device=x.device)
    st = load().qmaxpool(n, h, wd, c, k, s, bits, _ptr(x), _ptr(out), _stream(stream))
    _check(st, "qmaxpool")
    return out


def pack_subbyte(src, bits, *, out=None, stream=None):
    """int8 values [..., L] -> packed uint8 [..., L*Q/8] (low Q bits of each value)."""
    _dev(src, torch.int8, "src")
    shape = tuple(src.shape[:-1]) + (src.shape[-1] * bits // 8,)
    if out is None:
        out = torch.empty(shape, dtype=torch.uint8, device=src.device)
    st = load().pack_subbyte(_ptr(src), _ptr(out), src.numel(), bits, _stream(stream))
    _check(st, "pack_subbyte")
    return out


def unpack_subbyte(src, bits, signed, *, out=None, stream=None):
    """packed uint8 [..., B] -> int8 [..., B*8/Q] (sign-extended when signed)."""
    _dev(src, (torch.uint8, torch.int8), "src")
    shape = tuple(src.shape[:-1]) + (src.shape[-1] * 8 // bits,)
    if out is None:
        out = torch.empty(shape, dtype=torch.int8, device=src.device)
    st = load().unpack_subbyte(_ptr(src), _ptr(out), out.numel(), bits, int(bool(signed)), _stream(stream))
    _check(st, "unpack_subbyte")
    return out


def selftest_wait_timeout(limit_cycles: int, stream=None):
    """Enqueue the bounded-wait failure self-test (see qnn_selftest_wait_timeout)."""
    _check(load().qnn_selftest_wait_timeout(int(limit_cycles), _stream(stream)), "qnn_selftest_wait_timeout")


def device_status(stream=None):
    """Synchronise and raise if a bounded device-side wait gave up since the last check."""
    _check(load().qnn_device_status(_stream(stream)), "device status")
