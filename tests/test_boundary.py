"""C-ABI boundary checks that need no GPU: the library builds and loads, exports
every function include/qnn.h declares, and rejects invalid arguments before
launching anything (only argument checks run, no CUDA call is reached)."""
import ctypes
import os
import re
import shutil
import subprocess

import pytest

from paper_1908_11263_gb300 import build as qbuild
from paper_1908_11263_gb300 import qnn

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "qnn.h")


@pytest.fixture(scope="module")
def lib():
    qbuild.build()
    return qnn.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(\w+)\s*\([^;{]*\)\s*;", text)) - {"sizeof"})


def test_header_declares_the_expected_surface():
    names = declared_functions()
    for f in ("qconv_hwc", "qlinear", "qmaxpool", "pack_subbyte", "unpack_subbyte", "qconv_hwc_workspace_size"):
        assert f in names


def test_header_is_plain_c():
    """The boundary is a C ABI: include/qnn.h compiles as pedantic C99 (no C++ or torch types)."""
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-fsyntax-only", "-x", "c", HEADER],
                   check=True)


def test_library_exports_every_declared_function(lib):
    missing = [f for f in declared_functions() if not hasattr(lib, f)]
    assert not missing, missing
    assert set(qnn.EXPORTED) <= set(declared_functions())


def test_version_and_status_strings(lib):
    assert lib.qnn_version() == 100
    for s in range(7):
        assert qnn.status_string(s) not in ("", "unknown status")
    assert qnn.status_string(99) == "unknown status"


def desc(**kw):
    base = dict(n=2, h=16, w=16, c=32, m=64, kh=3, kw=3, stride=(1, 1), pad=(1, 1), bits=8, shift=12)
    base.update(kw)
    return qnn.conv_desc(base["n"], base["h"], base["w"], base["c"], base["m"], base["kh"], base["kw"],
                         base["stride"], base["pad"], base["bits"], base["shift"], base.get("algo", 0))


FAKE = 0x10000  # 16-byte aligned, never dereferenced: every case below fails validation first


def conv_status(lib, d, x=FAKE, w=FAKE, bias=FAKE, kappa=FAKE, lam=FAKE, shifts=None, y=FAKE, ws=FAKE, wsb=1 << 30):
    P = ctypes.c_void_p
    return lib.qconv_hwc(ctypes.byref(d), P(x), P(w), P(bias), P(kappa), P(lam), P(shifts), P(y), P(ws),
                         ctypes.c_size_t(wsb), P(0))


@pytest.mark.parametrize("kw,code", [
    (dict(h=0), qnn.QNN_EINVAL), (dict(c=-1), qnn.QNN_EINVAL), (dict(m=0), qnn.QNN_EINVAL),
    (dict(n=-1), qnn.QNN_EINVAL), (dict(stride=(0, 1)), qnn.QNN_EINVAL), (dict(pad=(-1, 0)), qnn.QNN_EINVAL),
    (dict(h=1, pad=(0, 0)), qnn.QNN_EINVAL),  # kernel taller than the padded input
    (dict(shift=63), qnn.QNN_EINVAL), (dict(shift=-1), qnn.QNN_EINVAL),
    (dict(bits=3), qnn.QNN_EUNSUPPORTED), (dict(bits=1), qnn.QNN_EUNSUPPORTED),
    (dict(bits=4, c=33), qnn.QNN_EUNSUPPORTED), (dict(bits=2, m=62), qnn.QNN_EUNSUPPORTED),
    (dict(c=40000, kh=1, kw=1, pad=(0, 0)), qnn.QNN_EUNSUPPORTED),  # accumulator bound
    (dict(algo=7), qnn.QNN_EINVAL), (dict(stride=(2, 2), algo=qnn.ALGO_TENSORCORE), qnn.QNN_EUNSUPPORTED),
    # the window kernel: stride 1, whole 8-channel chunks at INT-8, at most 128 output channels
    (dict(stride=(2, 2), algo=qnn.ALGO_TC_WINDOW), qnn.QNN_EUNSUPPORTED),
    (dict(c=12, algo=qnn.ALGO_TC_WINDOW), qnn.QNN_EUNSUPPORTED),
    (dict(m=136, algo=qnn.ALGO_TC_WINDOW), qnn.QNN_EUNSUPPORTED),
    (dict(stride=(2, 2), algo=qnn.ALGO_TC_GENERAL), qnn.QNN_EUNSUPPORTED),
])
def test_conv_descriptor_validation(lib, kw, code):
    assert conv_status(lib, desc(**kw)) == code


def test_conv_pointer_and_alignment_validation(lib):
    d = desc()
    assert conv_status(lib, d, x=0) == qnn.QNN_EINVAL
    assert conv_status(lib, d, w=0) == qnn.QNN_EINVAL
    assert conv_status(lib, d, kappa=0) == qnn.QNN_EINVAL
    assert conv_status(lib, d, lam=0) == qnn.QNN_EINVAL
    assert conv_status(lib, d, y=0) == qnn.QNN_EINVAL
    assert conv_status(lib, d, x=FAKE + 8) == qnn.QNN_EALIGN
    assert conv_status(lib, d, y=FAKE + 1) == qnn.QNN_EALIGN
    assert conv_status(lib, d, w=FAKE + 4) == qnn.QNN_EALIGN
    assert conv_status(lib, d, bias=FAKE + 2) == qnn.QNN_EALIGN
    assert conv_status(lib, d, kappa=FAKE + 1) == qnn.QNN_EALIGN
    # the general tensor-core kernel needs its workspace (the window kernel, which this layer
    # takes by default, reads the filters in place and needs none)
    g = desc(algo=qnn.ALGO_TC_GENERAL)
    assert conv_status(lib, g, ws=0) == qnn.QNN_EWORKSPACE
    assert conv_status(lib, g, wsb=16) == qnn.QNN_EWORKSPACE
    assert conv_status(lib, g, ws=FAKE + 16) == qnn.QNN_EWORKSPACE
    bad = desc()
    bad.struct_size = 8
    assert conv_status(lib, bad) == qnn.QNN_EINVAL
    assert lib.qconv_hwc(None, *([None] * 8), ctypes.c_size_t(0), None) == qnn.QNN_EINVAL


def test_prepare_and_run_validation(lib):
    """qconv_hwc_prepare / qconv_hwc_run on the window kernel: the workspace (the prepared image,
    qconv_hwc_workspace_size bytes, 256-byte aligned) is required by both; run needs x and y,
    16-byte aligned; a descriptor that only the CUDA-core kernel takes has nothing to run.  No
    CUDA call is reached."""
    P, SZ = ctypes.c_void_p, ctypes.c_size_t
    d = desc()
    need = qnn.workspace_size(d)
    assert need > 0

    def prep(ws=FAKE, nbytes=need, w=FAKE, kappa=FAKE, lam=FAKE):
        return lib.qconv_hwc_prepare(ctypes.byref(d), P(w), None, P(kappa), P(lam), None, P(ws), SZ(nbytes), None)

    def run(dd=d, x=FAKE, y=FAKE, ws=FAKE, nbytes=need):
        return lib.qconv_hwc_run(ctypes.byref(dd), P(x), P(y), P(ws), SZ(nbytes), None)

    assert prep(ws=0) == qnn.QNN_EWORKSPACE
    assert prep(nbytes=need - 1) == qnn.QNN_EWORKSPACE
    assert prep(ws=FAKE + 16) == qnn.QNN_EWORKSPACE
    assert prep(w=0) == qnn.QNN_EINVAL
    assert prep(kappa=0) == qnn.QNN_EINVAL
    assert run(ws=0) == qnn.QNN_EWORKSPACE
    assert run(nbytes=need - 1) == qnn.QNN_EWORKSPACE
    assert run(ws=FAKE + 128) == qnn.QNN_EWORKSPACE
    assert run(x=0) == qnn.QNN_EINVAL
    assert run(y=FAKE + 4) == qnn.QNN_EALIGN
    assert run(dd=desc(stride=(2, 2))) == qnn.QNN_EUNSUPPORTED  # the CUDA-core kernel only


def test_algo_selection_and_workspace(lib):
    assert qnn.conv_algo(desc()) == qnn.ALGO_TENSORCORE
    assert qnn.conv_algo(desc(stride=(2, 2))) == qnn.ALGO_DIRECT
    assert qnn.conv_algo(desc(algo=qnn.ALGO_DIRECT)) == qnn.ALGO_DIRECT
    assert qnn.workspace_size(desc(algo=qnn.ALGO_DIRECT)) == 0
    ws = qnn.workspace_size(desc(algo=qnn.ALGO_TC_GENERAL))
    # general kernel: fp16 filters (64 x 3*3*32) plus 16 bytes of constants per channel
    assert ws >= 64 * 288 * 2 + 64 * 16
    for bits in (4, 2):
        assert qnn.conv_algo(desc(bits=bits)) == qnn.ALGO_TENSORCORE
    with pytest.raises(qnn.QnnError):
        qnn.conv_algo(desc(bits=5))


def test_subbyte_layers_with_c_multiple_of_32_plan_e4m3_filters(lib):
    """The general kernel: INT-4/INT-2 layers whose C is a multiple of 32 stage e4m3 bytes (one
    byte per filter element in the workspace); INT-8 and C = 16 keep fp16 (two bytes). Its
    workspace is the filters plus 96 bytes of per-channel constants and thresholds."""
    consts = 64 * (32 + 64)
    g = qnn.ALGO_TC_GENERAL
    assert qnn.workspace_size(desc(algo=g)) == 64 * 3 * 3 * 32 * 2 + consts
    for bits in (4, 2):
        assert qnn.workspace_size(desc(bits=bits, algo=g)) == 64 * 3 * 3 * 32 * 1 + consts
        d16 = qnn.conv_desc(1, 8, 8, 16, 64, 3, 3, 1, 1, bits, 10, g)
        assert qnn.workspace_size(d16) == 64 * 3 * 3 * 16 * 2 + consts
        # the operand-format query agrees: e4m3 (8 bits) with C = 32, fp16 with C = 16
        assert qnn.mma_operand_bits(desc(bits=bits)) == 8
        assert qnn.mma_operand_bits(d16) == 16
    assert qnn.mma_operand_bits(desc()) == 16
    assert qnn.mma_operand_bits(desc(stride=(2, 2))) == 0
    with pytest.raises(qnn.QnnError):
        qnn.mma_operand_bits(desc(bits=5))


def test_window_kernel_selection_and_prepared_workspace(lib):
    """Tensor-core requests take the window kernel where its plan fits (the benchmark layer at
    every Q, the CIFAR-shaped conv1 with its kernel columns folded into K, conv2 / conv3) and the
    general kernel elsewhere (C * kw above 16 at C = 3, more than 128 output channels).  The window kernel's prepared workspace holds the image qconv_hwc_prepare
    builds: the filters as the B operand (taps x 4 K-chunks x 64 rows x 16 bytes), then the
    records (2 x 64 x 16 bytes + flags), the tap sums ((taps + 3) x 64 int32), the MMA table
    (2 strips x 9 taps x 2 k-steps x 8 bytes) and the pre-load operands (4 KB + 64 x 32 bytes)."""
    for bits in (8, 4, 2):
        assert qnn.tc_kernel(desc(bits=bits)) == qnn.ALGO_TC_WINDOW
    assert qnn.tc_kernel(qnn.conv_desc(1024, 16, 16, 32, 32, 5, 5, 1, 2, 8, 10)) == qnn.ALGO_TC_WINDOW
    assert qnn.tc_kernel(qnn.conv_desc(1024, 8, 8, 32, 64, 5, 5, 1, 2, 8, 10)) == qnn.ALGO_TC_WINDOW
    # C = 3: the kernel columns fold into K (kw * C = 15 values per position and kernel row)
    assert qnn.tc_kernel(qnn.conv_desc(1024, 32, 32, 3, 32, 5, 5, 1, 2, 8, 10)) == qnn.ALGO_TC_WINDOW
    assert qnn.tc_kernel(qnn.conv_desc(4, 32, 32, 3, 32, 7, 7, 1, 3, 8, 10)) == qnn.ALGO_TC_GENERAL  # 21 > 16
    assert qnn.tc_kernel(qnn.conv_desc(64, 14, 14, 256, 512, 1, 1, 1, 0, 8, 10)) == qnn.ALGO_TC_GENERAL
    assert qnn.tc_kernel(desc(algo=qnn.ALGO_TC_GENERAL)) == qnn.ALGO_TC_GENERAL
    assert qnn.tc_kernel(desc(stride=(2, 2))) == 0
    parts = 9 * 4 * 64 * 16 + (2 * 64 * 16 + 16) + 12 * 64 * 4 + 2 * 9 * 2 * 8 + 4096 + 64 * 32
    size = qnn.workspace_size(desc())
    assert size % 256 == 0 and parts <= size <= parts + 256 + 128  # 16- and 128-byte region alignment


def test_other_entry_points_validate(lib):
    P = ctypes.c_void_p
    assert lib.qlinear(-1, 4, 4, P(FAKE), P(FAKE), None, P(FAKE), None) == qnn.QNN_EINVAL
    assert lib.qlinear(4, 0, 4, P(FAKE), P(FAKE), None, P(FAKE), None) == qnn.QNN_EINVAL
    assert lib.qlinear(4, 4, 4, None, P(FAKE), None, P(FAKE), None) == qnn.QNN_EINVAL
    assert lib.qlinear(4, 1 << 20, 4, P(FAKE), P(FAKE), None, P(FAKE), None) == qnn.QNN_EUNSUPPORTED
    assert lib.qlinear(4, 4, 4, P(FAKE), P(FAKE), None, P(FAKE + 2), None) == qnn.QNN_EALIGN
    assert lib.qmaxpool(1, 4, 4, 8, 5, 2, 8, P(FAKE), P(FAKE), None) == qnn.QNN_EINVAL
    assert lib.qmaxpool(1, 4, 4, 8, 2, 0, 8, P(FAKE), P(FAKE), None) == qnn.QNN_EINVAL
    assert lib.qmaxpool(1, 4, 4, 8, 2, 2, 3, P(FAKE), P(FAKE), None) == qnn.QNN_EUNSUPPORTED
    assert lib.qmaxpool(1, 4, 4, 3, 2, 2, 4, P(FAKE), P(FAKE), None) == qnn.QNN_EUNSUPPORTED
    assert lib.pack_subbyte(P(FAKE), P(FAKE), 7, 4, None) == qnn.QNN_EUNSUPPORTED
    assert lib.pack_subbyte(P(FAKE), P(FAKE), -4, 4, None) == qnn.QNN_EINVAL
    assert lib.pack_subbyte(P(FAKE), P(FAKE), 8, 6, None) == qnn.QNN_EUNSUPPORTED
    assert lib.unpack_subbyte(None, P(FAKE), 8, 2, 1, None) == qnn.QNN_EINVAL
    assert lib.unpack_subbyte(P(FAKE), P(FAKE), 6, 2, 1, None) == qnn.QNN_EUNSUPPORTED
