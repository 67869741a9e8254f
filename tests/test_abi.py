"""CPU checks of the C ABI library: it builds, loads, exports every symbol the
header declares, and rejects bad arguments without touching a GPU."""
import ctypes
import os
import re

import pytest

from paper_2603_08957_gb300 import _lib

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    text = open(os.path.join(ROOT, "include", "ucl.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ucl_[a-z_]+)\s*\(", text)))


def test_header_declares_the_binding_exports():
    assert _declared() == sorted(_lib.EXPORTS)


def test_library_exports_every_declared_symbol():
    lib = _lib.load()
    for name in _declared():
        assert hasattr(lib, name), name


def test_status_strings():
    lib = _lib.load()
    for code, name in _lib.STATUS_NAMES.items():
        assert lib.ucl_status_str(code).decode() == name


def test_null_arguments_are_rejected():
    lib = _lib.load()
    h = ctypes.c_void_p()
    assert lib.ucl_ctx_create(0, None, ctypes.cast(None, _lib.ALLOC_FN), ctypes.cast(None, _lib.FREE_FN), None,
                              None) == 1
    assert lib.ucl_ctx_destroy(None) == 1
    assert lib.ucl_relation_destroy(None) == 1
    assert lib.ucl_einsum(None, b"Ij,jK->IK", 2, None, None, ctypes.byref(h)) == 1
    assert h.value is None
    assert lib.ucl_last_error(None) == b"NULL context"


@pytest.mark.skipif(os.path.exists("/dev/nvidia0"), reason="only meaningful without a GPU")
def test_context_without_gpu_fails_cleanly():
    lib = _lib.load()
    h = ctypes.c_void_p()
    st = lib.ucl_ctx_create(0, None, ctypes.cast(None, _lib.ALLOC_FN), ctypes.cast(None, _lib.FREE_FN), None,
                            ctypes.byref(h))
    assert st in (0, 7)
    if st == 0:
        lib.ucl_ctx_destroy(h)
