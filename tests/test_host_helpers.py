"""Host-side logic of the library checked on the CPU (no GPU, no kernel launch).

aligned_prefetch_range: logq_linear_grouped accepts an L2 prefetch hint at any
alignment, and the bulk prefetch it issues wants a 16-byte aligned start and a
whole number of 16-byte units.  The helper is compiled with the host compiler
from the library's own header and checked over every start offset and length
in a window, against the largest aligned range inside the caller's range.
"""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA_INC = "/usr/local/cuda/include"


def test_aligned_prefetch_range(tmp_path):
    cxx = shutil.which("g++")
    if cxx is None or not os.path.isdir(CUDA_INC):
        pytest.skip("host compiler or CUDA headers missing")
    exe = tmp_path / "prefetch_range_check"
    subprocess.run([cxx, "-std=c++17", "-I", os.path.join(ROOT, "include"),
                    "-I", os.path.join(ROOT, "paper_2607_01127_gb300", "csrc"), "-I", CUDA_INC,
                    os.path.join(ROOT, "tests", "host", "prefetch_range_check.cpp"), "-o", str(exe)],
                   check=True, capture_output=True, text=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr
