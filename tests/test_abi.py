"""The C ABI: liblmgc.so builds for sm_103a and exports every entry point include/lmgc.h
declares (no GPU needed; nothing is computed)."""
import ctypes
import os
import re

from paper_2409_17836_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "lmgc.h")).read()
    return sorted(set(re.findall(r"^lmgc_status\s+(lmgc_\w+)\s*\(", text, flags=re.M)))


def test_library_exports_every_declared_symbol():
    path = B.build()
    lib = ctypes.CDLL(path)
    syms = declared_symbols()
    assert len(syms) >= 16
    missing = [s for s in syms if not hasattr(lib, s)]
    assert not missing, missing


def test_binding_names_match_header():
    from paper_2409_17836_gb300 import lmgc
    assert sorted(lmgc.SYMBOLS) == declared_symbols()
    for s in declared_symbols():
        assert callable(getattr(lmgc, s)), s
