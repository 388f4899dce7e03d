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
    # and the documented choices for the workloads' layers
    plans = {line.split(": ok=")[0]: line.split(": ok=")[1] for line in text.splitlines() if ": ok=" in line}
    expect = {
        "512x16x16x32->64 k3x3 p1,1 q8 pool0": "rows fp16",    # whole output rows per row tile, kernel 3 wide
        "512x16x16x32->64 k3x3 p1,1 q4 pool0": "rows e4m3",
        "512x16x16x32->64 k3x3 p1,1 q2 pool0": "rows e4m3",
        "64x56x56x64->64 k3x3 p1,1 q8 pool0": "strips fp16",
        "64x28x28x128->128 k3x3 p1,1 q8 pool0": "strips fp16",
        "64x14x14x256->256 k3x3 p1,1 q8 pool0": "strips fp16",
        "64x14x14x256->512 k1x1 p0,0 q8 pool0": "rows fp16",   # a 1x1 kernel needs no copies
        "1024x32x32x3->32 k5x5 p2,2 q8 pool0": "strips fp16",
        "1024x16x16x32->32 k5x5 p2,2 q8 pool0": "strips fp16",
        "1024x8x8x32->64 k5x5 p2,2 q8 pool0": "strips fp16",
        "512x16x16x32->64 k3x3 p1,1 q8 pool1": "strips fp16",  # the fused pool always takes strips
    }
    for key, want in expect.items():
        assert plans[key].split(" nt=")[0] == "1 " + want, (key, plans[key])


def test_window_plans_keep_every_access_in_bounds(tmp_path):
    """The same for the window kernel's planner (tests/win_bounds.cpp): shared-memory layout,
    every bulk copy, converter load and store, MMA operand row and the exact-chunk bound."""
    lib = qbuild.build()
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    cuda = _cuda_root()
    exe = str(tmp_path / "win_bounds")
    subprocess.run([cxx, "-std=c++17", "-O1", f"-I{os.path.join(cuda, 'include')}", os.path.join(HERE, "win_bounds.cpp"),
                    "-o", exe, lib, f"-Wl,-rpath,{os.path.dirname(lib)}", f"-L{os.path.join(cuda, 'lib64')}",
                    "-lcudart"], check=True)
    out = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert out.returncode == 0 and out.stdout.rstrip().endswith("fails=0"), out.stdout[-4000:]
    text = out.stdout
    for word in ("S=1", "S=2", "e4m3", "fp16", "full-rows", "row-segments"):
        assert f" {word} " in text or f" {word}\n" in text, word
    plans = {line.split(": ok=")[0]: line.split(": ok=")[1] for line in text.splitlines() if ": ok=" in line}
    # the benchmark layer at every bit width: whole images (two strips) per tile, one bulk copy each
    for q, fmt in ((8, "fp16"), (4, "e4m3"), (2, "e4m3")):
        got = plans[f"512x16x16x32->64 k3x3 p1,1 q{q} pool0"]
        assert got.startswith(f"1 S=2 {fmt} nt=64") and got.endswith("full-rows"), (q, got)
    # CIFAR conv1 (C = 3): kernel columns folded into K, whole rows, one 16-value K-step per kernel row
    got = plans["1024x32x32x3->32 k5x5 p2,2 q8 pool0"]
    assert got.startswith("1 S=2 fp16 nt=32 sp=16 wh=20") and got.endswith("full-rows folded"), got
    assert " folded" in text and text.count(" folded") >= 10
    # a layer the window kernel leaves to the general kernel: more than 128 output channels
    assert plans["64x14x14x256->512 k1x1 p0,0 q8 pool0"] == "0"
