"""The C-ABI library builds, loads without a GPU, and exports every function
that include/flashrec.h declares (no compute calls here)."""
import ctypes
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "flashrec.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*(fr_[a-z_0-9]+)\s*\(", src, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ["fr_plan_create", "fr_plan_info", "fr_plan_destroy", "fr_fingerprint", "fr_pack",
                 "fr_unpack_verify", "fr_diff", "fr_sync_status", "fr_status_str"]:
        assert want in names


def test_library_exports_every_declared_symbol():
    from paper_2509_03047_gb300 import build

    path = build.build()
    lib = ctypes.CDLL(path)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings_without_gpu():
    from paper_2509_03047_gb300 import flashrec as fr

    assert fr.fr_status_str(fr.FR_ERR_CAPACITY) == "FR_ERR_CAPACITY"
    assert fr.fr_version() >= 10000
