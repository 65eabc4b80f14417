"""The C-ABI library builds, loads and exports every symbol include/dlmz.h declares (no GPU needed)."""
import ctypes
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    txt = open(os.path.join(ROOT, "include", "dlmz.h")).read()
    return sorted(set(re.findall(r"DLMZ_API\s+[\w\s\*]*?\b(dlmz_\w+)\s*\(", txt)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("dlmz_model_create", "dlmz_model_destroy", "dlmz_compress", "dlmz_decompress", "dlmz_free",
              "dlmz_strerror", "dlmz_quantize", "dlmz_forward_logits", "dlmz_encode_step", "dlmz_decode_step"):
        assert n in names


def test_library_builds_loads_and_exports_all_symbols():
    from paper_2608_11249_gb300 import build
    path = build.build()
    lib = ctypes.CDLL(path)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing
    lib.dlmz_strerror.restype = ctypes.c_char_p
    assert lib.dlmz_strerror(-3) == b"corrupt container"


def test_binding_imports_with_same_names():
    from paper_2608_11249_gb300 import build
    build.build()
    from paper_2608_11249_gb300 import dlmz
    for n in _declared():
        assert hasattr(dlmz.lib, n)
