"""Host-side checks of the C-ABI library (no GPU): it loads, exports every symbol that
include/mixflow.h declares, and rejects bad arguments before touching the device."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mixflow.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2505_00793_gb300 import build, native
    build.build()
    return native.load()


def _declared():
    txt = open(HEADER).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(mf_[a-z0-9_]+)\s*\(", txt)))


def test_header_matches_binding_exports():
    from paper_2505_00793_gb300 import native
    assert _declared() == sorted(native.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    assert lib.mf_status_string(0) == b"ok"
    assert lib.mf_status_string(6) == b"device wait timed out"


def test_rejects_bad_arguments_on_host(lib):
    from paper_2505_00793_gb300 import native
    h = C.c_void_p()
    assert lib.mf_create(None, C.byref(h)) == 1
    d = native.mf_model_desc()
    d.arch, d.n_layers = 0, 0
    assert lib.mf_create(C.byref(d), C.byref(h)) == 1          # no layers
    d.arch = 1
    assert lib.mf_create(C.byref(d), C.byref(h)) == 1          # decoder without a shape
    # empty GEMM and bad term masks are rejected before any launch
    assert lib.mf_dual_gemm_bf16(0, 8, 8, None, 8, None, 8, None, 8, None, 8, None, 8, None,
                                 None, 8, None, 1, None) == 1
    assert lib.mf_dual_gemm_bf16(8, 8, 8, None, 8, None, 8, None, 8, None, 8, None, 8, None,
                                 None, 8, None, 64, None) == 1
    assert lib.mf_destroy(None) == 1
    assert lib.mf_sync(None) == 1
