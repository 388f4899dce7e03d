"""Host-side bounds of the tensor-core planner, without a GPU: tests/plan_bounds.cpp is compiled
with the host C++ compiler, linked against the built library (which exports qnn::plan_conv_tc),
and run. For every layer shape of the parity tests and workloads, with and without the fused
pool, it checks that each address the kernel derives from the plan stays inside the buffers the
plan sizes. It also checks the accumulator chunks' exactness bound and the reciprocal division
the kernel uses."""
import os
import shutil
import subprocess

import pytest

from paper_1908_11263_gb300 import build as qbuild

HERE = os.path.dirname(os.path.abspath(__file__))


def _cuda_root():
    nvcc = qbuild.nvcc()
    return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))


def test_plans_keep_every_access_in_bounds(tmp_path):
    lib = qbuild.build()
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    cuda = _cuda_root()
    exe = str(tmp_path / "plan_bounds")
    subprocess.run([cxx, "-std=c++17", "-O1", f"-I{os.path.join(cuda, 'include')}", os.path.join(HERE, "plan_bounds.cpp"),
                    "-o", exe, lib, f"-Wl,-rpath,{os.path.dirname(lib)}", f"-L{os.path.join(cuda, 'lib64')}",
                    "-lcudart"], check=True)
    out = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert out.returncode == 0 and out.stdout.rstrip().endswith("fails=0"), out.stdout[-4000:]
    # the planner chose both tile shapes and both staging formats somewhere in the list
    text = out.stdout
    for word in ("strips", "rows", "e4m3", "fp16"):
        assert f" {word} " in text, word
