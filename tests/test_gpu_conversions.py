"""The integer-only conversions of the kernels' decisions (sjd_device.cuh:
u64 to fp32 and fp64 with ties to even, fl32(fl64(total) 2^-47), the exact
widening of fp32 to fp64) give the bits of CUDA's own casts, on 2^26 values:
edge values (powers of two and their neighbours, exact ties at 24 and 53
bits, the largest values) and seeded random ones of every magnitude. The
check program is built with nvcc for this GPU and run in a child process."""

import os
import shutil
import subprocess
import tempfile

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_integer_conversions_match_the_casts():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "conv_check")
        subprocess.run([nvcc, "-gencode=arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
                        "-I", os.path.join(ROOT, "include"), "-I", os.path.join(ROOT, "paper_2603_18599_gb300", "csrc"),
                        os.path.join(HERE, "conv_check.cu"), "-o", exe], check=True, capture_output=True, timeout=600)
        r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "mismatches u64_to_f32_rn 0 u64_to_f64_rn 0 fix_to_f32 0 f32_to_f64 0" in r.stdout, r.stdout
