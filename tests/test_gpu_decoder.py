"""Decoder-only transformer through the C ABI against the float64 oracle.

float32 decoders (SIMT path) at relative L2 1e-4; bf16 decoders (tensor-core path, batched
attention GEMMs, cluster split-K) at 2e-2.  Sizes span several tiles of every GEMM with the
causal softmax, RoPE, RMSNorm, GELU MLP, embedding scatter and next-token loss."""
import math

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, SLR = synth.EXAMPLE_WEIGHTS, synth.SCALAR_LOGLR

FP32 = {
    "dec32_a": synth.decoder("dec32_a", 16, 2, 32, 2, 32, 8, B=3, T=2, B_outer=2,
                             alpha=0.1).with_(precision="fp32"),
    "dec32_mom": synth.decoder("dec32_mom", 32, 4, 48, 2, 40, 16, B=2, T=3, B_outer=3,
                               momentum=0.9, meta_kind=EX | SLR,
                               extra={"scalar_loglr": math.log(0.1)}).with_(precision="fp32"),
}

BF16 = {
    "dec16_small": synth.decoder("dec16_small", 128, 2, 256, 2, 256, 64, B=4, T=2, B_outer=4,
                                 alpha=1e-2),
    "dec16_mom": synth.decoder("dec16_mom", 64, 1, 128, 1, 200, 128, B=2, T=3, B_outer=2,
                               momentum=0.9, meta_kind=EX | SLR,
                               extra={"scalar_loglr": math.log(1e-2)}),
}


def _run(w, inp):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.full((w.n_eta,), float("nan"), device="cuda")
    d_th = torch.full((w.n_params,), float("nan"), device="cuda")
    V = torch.full((1,), float("nan"), device="cuda")
    mf.meta_grad(native.loop_desc_for(w), d["theta0"], d["eta"], d["inner_x"], d["inner_y"],
                 d["outer_x"], d["outer_y"], d_eta, d_th, V)
    mf.sync()
    out = dict(d_eta=d_eta.cpu().numpy(), d_theta0=d_th.cpu().numpy(), V=float(V.cpu()))
    mf.close()
    return out


def _check(w, tol):
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    got = _run(w, inp)
    assert np.isfinite(got["d_eta"]).all() and np.isfinite(got["d_theta0"]).all()
    assert abs(got["V"] - ref["V"]) <= tol * abs(ref["V"]), (got["V"], ref["V"])
    e1 = rel_l2(got["d_theta0"], ref["d_theta0"])
    e0 = rel_l2(got["d_eta"], ref["d_eta"])
    assert e1 < tol, (w.name, "d_theta0", e1)
    assert e0 < tol, (w.name, "d_eta", e0)


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(FP32))
def test_decoder_meta_grad_fp32(name):
    _check(FP32[name], 1e-4)


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(BF16))
def test_decoder_meta_grad_bf16(name):
    _check(BF16[name], 2e-2)


@pytest.mark.gpu
@pytest.mark.parametrize("name,tol", [("dec32_mom", 1e-4), ("dec16_small", 2e-2)])
def test_decoder_hvp(name, tol):
    torch, native = need_gpu()
    w = FP32.get(name) or BF16[name]
    inp = synth.make_inputs(w)
    ids = inp.inner_x[0]
    v = synth.random_direction(w.n_params, 2, 3)
    wt = np.linspace(0.3, 1.0, w.B).astype(np.float32)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    Hv = torch.full((w.n_params,), float("nan"), device="cuda")
    g = torch.full((w.n_params,), float("nan"), device="cuda")
    tl = torch.full((w.B,), float("nan"), device="cuda")
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], torch.from_numpy(v).cuda(), Hv,
           ex_w=torch.from_numpy(wt).cuda(), tangent_losses=tl, grad=g)
    mf.sync()
    assert rel_l2(g.cpu().numpy(), om.grad(w, inp.theta0, ids, ids, wt)) < tol
    assert rel_l2(Hv.cpu().numpy(), om.hvp(w, inp.theta0, ids, ids, v, wt)) < tol
    assert rel_l2(tl.cpu().numpy(), om.tangent_losses(w, inp.theta0, ids, ids, v)) < tol
    mf.close()


@pytest.mark.gpu
def test_decoder_small_full_size_single_step():
    """The 27M-parameter decoder (d 512, 8 heads, MLP 2048, 6 blocks, vocabulary 8192,
    16 sequences of 256 tokens) at T = 1, every output against the oracle."""
    _check(synth.WORKLOADS["decoder_small"].with_(T=1), 2e-2)
