"""mf_hvp_noalloc: the Hessian-vector product for callers that cannot allocate device
memory (embedders whose memory is fully reserved up front by their own allocator, hosts that
only accept pre-registered buffers).  Its outputs must match mf_hvp's on the same inputs, on
two calls in a row (the second call finds the first call's leftovers in the shared static
workspace).

Collected last on purpose: if it fails, a run stopping at the first failure has already
run every other test."""
import ctypes as C

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth


@pytest.mark.gpu
@pytest.mark.parametrize("case", ["bf16", "fp32", "chain_bf16"])
def test_hvp_noalloc_matches_hvp(case):
    torch, native = need_gpu()
    if case == "bf16":
        w = synth.Workload("noalloc_bf16", [128, 256, 136, 10], "gelu", "ce", "bf16", B=64, T=1,
                           B_outer=8, alpha=0.05)
        tol = 2e-2
    elif case == "chain_bf16":
        # the motivating example's chain loss (Eq. 8), M = 3, on a 256-wide map
        w = synth.toy("noalloc_chain", 256, 96, 3, T=1, precision="bf16", init_std=1.0 / 16.0)
        tol = 2e-2
    else:
        w = synth.Workload("noalloc_fp32", [40, 70, 3], "tanh", "squared", "fp32", B=33, T=1,
                           B_outer=8, alpha=0.1, noise_std=0.1)
        tol = 1e-4
    inp = synth.make_inputs(w)
    d = native.to_device_inputs(w, inp)
    v = torch.from_numpy(synth.random_direction(w.n_params, 5, 1)).cuda()
    wt = torch.from_numpy(np.linspace(0.3, 1.0, w.B).astype(np.float32)).cuda()
    x, y = d["inner_x"][0], d["inner_y"][0]

    mf = native.MixFlow.for_workload(w)
    ref_hv = torch.empty(w.n_params, device="cuda")
    ref_g = torch.empty(w.n_params, device="cuda")
    ref_tl = torch.empty(w.B, device="cuda")
    mf.hvp(w.B, d["theta0"], x, y, v, ref_hv, ex_w=wt, tangent_losses=ref_tl, grad=ref_g)
    mf.sync()
    mf.close()

    lib = native.lib()
    desc = native.model_desc_for(w)
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    p = lambda t: C.c_void_p(t.data_ptr())
    for _ in range(2):
        hv = torch.full((w.n_params,), float("nan"), device="cuda")
        g = torch.full((w.n_params,), float("nan"), device="cuda")
        tl = torch.full((w.B,), float("nan"), device="cuda")
        st = lib.mf_hvp_noalloc(C.byref(desc), w.B, p(d["theta0"]), p(x), p(y), p(wt), p(v),
                                p(hv), p(tl), p(g), stream)
        assert st == 0
        torch.cuda.synchronize()
        assert rel_l2(hv.cpu().numpy(), ref_hv.cpu().numpy()) < tol
        assert rel_l2(g.cpu().numpy(), ref_g.cpu().numpy()) < tol
        assert rel_l2(tl.cpu().numpy(), ref_tl.cpu().numpy()) < tol


@pytest.mark.gpu
def test_hvp_noalloc_rejects_oversize():
    torch, native = need_gpu()
    w = synth.Workload("too_big", [1024] * 5 + [10], "gelu", "ce", "bf16", B=256, T=1,
                       B_outer=8, alpha=0.05)
    desc = native.model_desc_for(w)
    dummy = torch.zeros(16, device="cuda")
    p = C.c_void_p(dummy.data_ptr())
    st = native.lib().mf_hvp_noalloc(C.byref(desc), w.B, p, p, p, None, p, p, None, None, None)
    assert st == 1   # MF_ERR_INVALID_ARG: the workspace would exceed the static array


@pytest.mark.gpu
def test_hvp_noalloc_rejects_decoder():
    torch, native = need_gpu()
    w = synth.decoder("dec_noalloc", 64, 1, 128, 1, 200, 64, B=2, T=1, B_outer=2, alpha=1e-2)
    desc = native.model_desc_for(w)
    dummy = torch.zeros(16, device="cuda")
    p = C.c_void_p(dummy.data_ptr())
    st = native.lib().mf_hvp_noalloc(C.byref(desc), w.B, p, p, p, None, p, p, None, None, None)
    assert st == 2   # MF_ERR_UNSUPPORTED: decoders need mf_hvp and a handle
