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


def test_binding_checks_tensor_arguments():
    """The binding refuses, before any library call, tensors the ABI cannot take: a wrong
    element type, a non-contiguous layout, or host memory (whose pointer a kernel would
    dereference as a device address)."""
    import torch
    from paper_2505_00793_gb300 import native, synth
    assert native._dev(None, "d_theta0", torch.float32) is None
    with pytest.raises(ValueError, match="dtype"):
        native._dev(torch.zeros(4, dtype=torch.float64), "theta0", torch.float32)
    with pytest.raises(ValueError, match="contiguous"):
        native._dev(torch.zeros(4, 4).t(), "theta0", torch.float32)
    with pytest.raises(ValueError, match="unit stride"):
        native._dev(torch.zeros(4, 4, dtype=torch.bfloat16).t(), "A0", torch.bfloat16, rows=True)
    with pytest.raises(ValueError, match="CUDA"):
        native._dev(torch.zeros(4), "theta0", torch.float32)
    with pytest.raises(ValueError, match="CUDA"):    # strided rows are fine, host memory is not
        native._dev(torch.zeros(4, 8, dtype=torch.bfloat16)[:, :6], "A0", torch.bfloat16,
                    rows=True)
    expect = {"tiny": (torch.float32, torch.float32), "wide": (torch.bfloat16, torch.int32),
              "deep": (torch.bfloat16, torch.float32), "toy": (torch.bfloat16, torch.float32),
              "decoder_small": (torch.int32, torch.int32)}
    for name, dt in expect.items():
        assert native.io_dtypes(native.model_desc_for(synth.WORKLOADS[name])) == dt, name
    # the host-side input conversion gives exactly those dtypes (small shapes of each kind)
    for w in (synth.WORKLOADS["tiny"],
              synth.Workload("c", [8, 16, 4], "gelu", "ce", "bf16", B=4, T=2, B_outer=3),
              synth.toy("t", 8, 4, 2, T=2),
              synth.decoder("d", 16, 2, 32, 1, 24, 8, B=2, T=2, B_outer=2)):
        d = native.to_device_inputs(w, synth.make_inputs(w), device="cpu")
        x_dt, y_dt = native.io_dtypes(native.model_desc_for(w))
        for k in ("inner_x", "outer_x"):
            assert d[k].dtype == x_dt and d[k].is_contiguous(), (w.name, k)
        for k in ("inner_y", "outer_y"):
            assert d[k].dtype == y_dt and d[k].is_contiguous(), (w.name, k)
        for k in ("theta0", "eta"):
            assert d[k].dtype == torch.float32, (w.name, k)
