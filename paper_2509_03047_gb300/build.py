"""Build libflashrec.so in-tree with nvcc for sm_103a (GB300).

The translation units compile in parallel; the result is linked with the
static CUDA runtime into ``paper_2509_03047_gb300/libflashrec.so``.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
OUT_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libflashrec.so")
SOURCES = ["sweep_fp.cu", "sweep_pack.cu", "sweep_unpack.cu", "sweep_unpack_fp.cu", "finalize.cu", "api.cu",
           "static_fingerprint.cu"]
HEADERS = ["gf2.cuh", "layout.h", "kernels.h", "sweep_impl.cuh", "warp_share.h"]

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              "-Xptxas", "-v", "-I", os.path.join(ROOT, "include")]


def nvcc() -> str:
    for cand in [os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"]:
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: libflashrec needs the CUDA 13 toolkit to build")


def _stale(target: str, deps) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


# Files that define the device kernels (the sweep, finalize, compaction and
# diff kernels); host-only planning and API code is not among them.
KERNEL_FILES = ["sweep_fp.cu", "sweep_pack.cu", "sweep_unpack.cu", "sweep_unpack_fp.cu", "finalize.cu", "gf2.cuh",
                "layout.h", "kernels.h", "sweep_impl.cuh"]


def _code_only(text: str) -> str:
    """`text` without its C/C++ comments, trailing blanks and blank lines:
    what the compiler sees, so an edit to a comment leaves the digest alone.
    (String literals in these sources contain no comment markers.)"""
    import re

    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"//[^\n]*", "", text)
    return "\n".join(line.rstrip() for line in text.splitlines() if line.strip())


def source_digest(kernels_only: bool = False) -> str:
    """Hash of the sources' code (comments left out) and the compile flags:
    identifies what a profile measured.  With `kernels_only`, of the
    device-kernel files alone."""
    import hashlib

    h = hashlib.sha256(" ".join(a for a in ARCH + NVCC_FLAGS if not os.path.isabs(a)).encode())
    names = KERNEL_FILES if kernels_only else SOURCES + HEADERS
    for name in sorted(names):
        with open(os.path.join(CSRC, name), encoding="utf-8") as f:
            h.update(name.encode() + b"\0" + _code_only(f.read()).encode())
    if not kernels_only:
        with open(os.path.join(ROOT, "include", "flashrec.h"), encoding="utf-8") as f:
            h.update(_code_only(f.read()).encode())
    return h.hexdigest()[:16]


def build(force: bool = False, verbose: bool = False) -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    headers = [os.path.join(CSRC, h) for h in HEADERS] + [os.path.join(ROOT, "include", "flashrec.h")]
    exe = nvcc()

    def compile_one(src):
        path = os.path.join(CSRC, src)
        obj = os.path.join(OUT_DIR, src.replace(".cu", ".o"))
        if force or _stale(obj, [path] + headers):
            cmd = [exe] + ARCH + NVCC_FLAGS + ["-c", path, "-o", obj]
            r = subprocess.run(cmd, capture_output=True, text=True)
            with open(obj + ".log", "w") as f:
                f.write(" ".join(cmd) + "\n" + r.stdout + r.stderr)
            if r.returncode != 0:
                raise RuntimeError("nvcc failed for %s:\n%s" % (src, r.stderr[-4000:]))
            if verbose:
                sys.stderr.write(r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(compile_one, SOURCES))
    if force or _stale(LIB, objs):
        tmp = LIB + ".tmp%d" % os.getpid()
        cmd = [exe] + ARCH + ["-shared", "-o", tmp] + objs + ["-cudart", "static"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("link failed:\n%s" % r.stderr[-4000:])
        os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True))
