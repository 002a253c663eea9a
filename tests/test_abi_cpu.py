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


def _header_enums():
    """Every `NAME = value` of the header's enums (comments stripped)."""
    txt = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    vals = {}
    for body in re.findall(r"enum\s*\{(.*?)\}", txt, flags=re.S):
        for name, v in re.findall(r"\b(MF_[A-Z0-9_]+)\s*=\s*(\d+)", body):
            vals[name] = int(v)
    for name, v in re.findall(r"\b(MF_[A-Z_]+)\s*=\s*(\d+)\s*[,}]", txt):
        vals.setdefault(name, int(v))
    return vals


def test_binding_constants_match_header():
    """The binding's enum values (options, losses, activations, meta kinds, modes) are the
    header's."""
    from paper_2505_00793_gb300 import native
    h = _header_enums()
    pairs = {"MF_ARCH_MLP": native.MF_ARCH_MLP, "MF_ARCH_DECODER": native.MF_ARCH_DECODER,
             "MF_ACT_IDENT": native.ACTS["ident"], "MF_ACT_TANH": native.ACTS["tanh"],
             "MF_ACT_GELU": native.ACTS["gelu"], "MF_ACT_SILU": native.ACTS["silu"],
             "MF_LOSS_SQUARED": native.LOSSES["squared"], "MF_LOSS_SOFTMAX_CE": native.LOSSES["ce"],
             "MF_LOSS_NEXT_TOKEN_CE": native.LOSSES["next_token_ce"],
             "MF_LOSS_CHAIN_MSE": native.LOSSES["chain_mse"],
             "MF_PREC_FP32": native.PRECISIONS["fp32"], "MF_PREC_BF16": native.PRECISIONS["bf16"],
             "MF_OPTIM_SGD": native.OPTIMIZERS["sgd"], "MF_OPTIM_ADAM": native.OPTIMIZERS["adam"],
             "MF_META_EXAMPLE_WEIGHTS": native.MF_META_EXAMPLE_WEIGHTS,
             "MF_META_PARAM_LOGLR": native.MF_META_PARAM_LOGLR,
             "MF_META_SCALAR_LOGLR": native.MF_META_SCALAR_LOGLR,
             "MF_HVP_MIXED_FOR": native.MF_HVP_MIXED_FOR, "MF_HVP_REV_REV": native.MF_HVP_REV_REV}
    for name, value in pairs.items():
        assert h[name] == value, name
    opts = {k: v for k, v in h.items() if k.startswith("MF_OPT_")}
    assert opts and all(getattr(native, k) == v for k, v in opts.items())
    status = {v: k for k, v in h.items() if k == "MF_OK" or k.startswith("MF_ERR_")}
    assert status == native.STATUS


def test_binding_structs_match_header():
    """ctypes structures have the header's fields, in order, with the header's C types."""
    from paper_2505_00793_gb300 import native
    txt = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    ctype = {"int": C.c_int, "float": C.c_float}
    for name, cls in (("mf_model_desc", native.mf_model_desc),
                      ("mf_loop_desc", native.mf_loop_desc)):
        body = re.search(r"typedef struct\s*\{([^{}]*)\}\s*" + name + ";", txt).group(1)
        fields = []
        for decl in body.split(";"):
            decl = decl.strip()
            if not decl:
                continue
            typ, rest = decl.split(None, 1)
            for item in rest.split(","):
                item = item.strip()
                m = re.match(r"(\w+)\s*\[(.*)\]", item)
                if m:
                    n = eval(m.group(2).replace("MF_MAX_LAYERS", str(native.MF_MAX_LAYERS)))
                    fields.append((m.group(1), ctype[typ] * n))
                else:
                    fields.append((item, ctype[typ]))
        got = [(f, t) for f, t in cls._fields_]
        assert [f for f, _ in got] == [f for f, _ in fields], name
        for (f, t), (_, u) in zip(got, fields):
            assert C.sizeof(t) == C.sizeof(u), (name, f)
            assert getattr(t, "_type_", t) == getattr(u, "_type_", u), (name, f)
