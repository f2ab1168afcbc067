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


def test_create_rejects_bad_qk_norm():
    """Host-side validation of the q/k norm flag happens before any device call."""
    L = kp.lib()
    one = (ctypes.c_void_p * 1)(0x1000)
    for flag, qn in ((1, None), (2, one), (-1, one)):
        cfg = kp.KvprmConfig(1, 256, 4, 2, 64, 1024, 16, 1e4, 1e-6, flag, 4, 8)
        cast = lambda a: ctypes.cast(a, kp.kvprm._VPP) if a is not None else None  # noqa: E731
        w = kp.KvprmWeights(0x1000, 0x1000, 0x1000, 0x1000, cast(one), cast(one), cast(one), cast(one), cast(one),
                            cast(one), cast(qn), cast(qn))
        ctx = ctypes.c_void_p()
        assert L.kvprm_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(ctx)) == kp.KVPRM_EINVAL
        assert not ctx.value
