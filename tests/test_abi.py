"""The C-ABI library builds for sm_103a, loads, and exports every entry point
that include/kvprm.h declares (no compute calls: runs without a GPU)."""
import ctypes
import os
import re

import paper_2607_09153_gb300 as kp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "kvprm.h")).read()
    return sorted(set(re.findall(r"KVPRM_API\s+[\w\s\*]+?\b(kvprm_\w+)\s*\(", src)))


def test_header_declares_entry_points():
    names = declared_symbols()
    for must in ("kvprm_create", "kvprm_score", "kvprm_destroy"):
        assert must in names


def test_library_exports_every_declared_symbol():
    lib = kp.lib()
    for name in declared_symbols():
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


def test_no_oracle_in_product():
    """The scoring library neither links nor names the oracle."""
    csrc = os.path.join(ROOT, "paper_2607_09153_gb300")
    for dirpath, _, files in os.walk(csrc):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "from oracle" not in text, f
                assert "kvprm_oracle" not in text, f
