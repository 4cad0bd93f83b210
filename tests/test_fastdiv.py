"""The multiply-based division of the tensor-core contraction's epilogue
(paper_2609_19611_gb300/csrc/fastdiv.h) equals integer division: compiled
with the host compiler and run over every divisor up to 4096, sampled larger
divisors up to 2^31, and dividends near multiples of each divisor."""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2609_19611_gb300", "csrc")


def test_fast_division_matches_integer_division(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    exe = str(tmp_path / "fastdiv_check")
    subprocess.run([cxx, "-O2", "-std=c++17", "-I", CSRC, os.path.join(HERE, "fastdiv_check.cpp"),
                    "-o", exe], check=True)
    out = subprocess.run([exe], capture_output=True, text=True)
    assert out.returncode == 0 and out.stdout.strip().endswith("ok"), out.stdout[-2000:]
