"""The C ABI from plain C (tests/c/abi_restore.c): it builds and links against
libflashrec.so with nothing but flashrec.h and the CUDA runtime (CPU test),
and on a GPU it runs a whole restore -- fingerprint, pack, transit damage,
unpack_verify, re-send, diff -- and checks every byte (GPU test)."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "abi_restore.c")


def _build(tmp_path):
    from paper_2509_03047_gb300 import build

    lib = build.build()
    nvcc = build.nvcc()
    exe = str(tmp_path / "abi_restore")
    libdir = os.path.dirname(lib)
    cmd = [nvcc, "-O2", SRC, "-I", os.path.join(ROOT, "include"), "-L", libdir,
           "-lflashrec", "-Xlinker", "-rpath," + libdir, "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr[-3000:]
    return exe


@pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                    reason="nvcc not available")
def test_c_program_builds_against_the_library(tmp_path):
    exe = _build(tmp_path)
    assert os.path.exists(exe)


@pytest.mark.gpu
def test_c_program_restores_a_state(tmp_path):
    exe = _build(tmp_path)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "abi_restore ok" in r.stdout
