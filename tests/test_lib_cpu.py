"""The C-ABI library builds for sm_103a, loads, and exports every entry point include/atspeed.h
declares (no compute calls: this runs without a GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "atspeed.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(atspeed_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2410_05165_gb300.build import build
    path = build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("atspeed_create", "atspeed_prefill", "atspeed_draft_step", "atspeed_verify", "atspeed_beam_search"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for n in _declared():
        assert hasattr(lib, n), n


def test_binding_names_match_header(lib):
    from paper_2410_05165_gb300 import EXPORTS
    assert sorted(EXPORTS) == _declared()


def test_create_rejects_null_arguments(lib):
    """Host-side validation runs before any device work; no GPU needed for a null argument."""
    lib.atspeed_create.restype = ctypes.c_int
    out = ctypes.c_void_p()
    st = lib.atspeed_create(None, None, None, None, ctypes.byref(out))
    assert st == -1
    lib.atspeed_last_error.restype = ctypes.c_char_p
    assert b"null" in lib.atspeed_last_error(None)
