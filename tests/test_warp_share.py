"""The host rule that shares one sweep launch's warps among the element-type /
alignment classes (csrc/warp_share.h), compiled with the host C++ compiler
and checked by tests/c/warp_share_test.cc: warp counts sum to the launch,
follow the weighted block counts, give every class at least one warp, and
every CTA gets an even share of every class; within a class the ranges are
cut by estimated segment cost (monotone boundaries covering every segment,
the equal-count split for unit costs).  No GPU."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.skipif(shutil.which("g++") is None, reason="g++ not available")
def test_warp_share_rule(tmp_path):
    exe = str(tmp_path / "warp_share_test")
    src = os.path.join(ROOT, "tests", "c", "warp_share_test.cc")
    inc = os.path.join(ROOT, "paper_2509_03047_gb300", "csrc")
    r = subprocess.run(["g++", "-std=c++17", "-O1", "-Wall", "-I", inc, src, "-o", exe], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr[-3000:]
    r = subprocess.run([exe], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "warp_share ok" in r.stdout
