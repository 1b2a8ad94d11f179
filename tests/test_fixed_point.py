"""fix_rn and fix_rn_small, the float-to-fixed-point conversions of the least-squares
statistics, equal the fp64 route (llrint of the exact product q * 2^e, saturated) bit for bit
(fix_rn_small in its range: 2^e a normal fp32 number, |q 2^e| < 2^31): compiled for the host
with g++ from the same header the kernels include. No GPU needed."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.skipif(shutil.which("g++") is None, reason="g++ not available")
def test_fix_rn_matches_the_fp64_conversion(tmp_path):
    exe = tmp_path / "fixed_point_check"
    subprocess.run(["g++", "-O2", "-std=c++17", "-I",
                    os.path.join(ROOT, "paper_2412_09282_gb300", "csrc"),
                    os.path.join(ROOT, "tests", "fixed_point_check.cpp"), "-o", str(exe)],
                   check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "disagreements=0" in r.stdout
