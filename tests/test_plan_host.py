"""Invariants of the host launch planner, compiled with the host compiler and
run on the CPU (no GPU): score splits cover the whole cache and fit the
workspace, the tensor-core kernel's weighted splits partition every
sequence's tiles within the page-id staging bound, gather chunks stay within
the chunk kernel's limit, the slice gather is chosen only for kept sets it
can hold, every benchmarked call shape gets the expected select form
(fused select + gather and its slice width, select only, or the
shared-memory select), and the chunk gather's benchmarked shapes get their
expected chunk count, text-merge slices and CTAs per (sequence, kv-head)
(tests/plan_invariants.cpp)."""

import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA_INC = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")


def test_planner_invariants(tmp_path):
    cxx = shutil.which("g++")
    if cxx is None or not os.path.exists(os.path.join(CUDA_INC, "cuda.h")):
        pytest.skip("needs g++ and the CUDA headers")
    exe = tmp_path / "plan_invariants"
    subprocess.run([cxx, "-std=c++17", "-O2", "-I", os.path.join(ROOT, "paper_2605_31457_gb300", "csrc"),
                    "-I", CUDA_INC, os.path.join(ROOT, "tests", "plan_invariants.cpp"), "-o", str(exe)],
                   check=True, capture_output=True, text=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "0 violations" in r.stdout
