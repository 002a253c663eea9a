"""Adam inner loops (Section 5's optimiser) on the GPU against the float64 oracle.

The sweep reverses each Adam step elementwise inside the fused adjoint update; the tangent
of every HVP is the gradient cotangent.  Covered: MLPs at float32 (1e-4) and bf16 (2e-2) with
every meta-parameter kind, the decoder, both HVP modes, segment checkpoints (bit-identical
to the full store), the rollout entry point, and argument checks.

Adam's step is close to lr sign(g), with a derivative spike of height ~1/eps where a
gradient component crosses zero, so eps sets the meta-gradient's conditioning.  Measured on
the oracle: with eps = 1e-8 a relative change of 1e-7 in theta_0 moves the multi-tile MLP's
meta-gradient by 8e-4, and rounding theta_0 to bf16 moves the bf16 cases' by 1.5-90%; at
eps = 1e-3 those shifts are below 3e-7 and 6e-3.  The small float32 cases keep eps from
1e-8 (amplification below 100); the multi-tile and bf16 cases use eps = 1e-3."""
import math

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, PLR, SLR = synth.EXAMPLE_WEIGHTS, synth.PARAM_LOGLR, synth.SCALAR_LOGLR

FP32 = {
    "ce_gelu_ex": synth.Workload("a_ce", [6, 8, 8, 4], "gelu", "ce", "fp32", B=5, T=4, B_outer=7,
                                 alpha=0.01, optimizer="adam"),
    "tanh_plr": synth.Workload("a_plr", [4, 6, 3], "tanh", "squared", "fp32", B=6, T=4,
                               B_outer=5, meta_kind=PLR, optimizer="adam", beta1=0.8,
                               beta2=0.95, adam_eps=1e-4, loglr_mean=math.log(0.01),
                               loglr_std=0.1, noise_std=0.1),
    "silu_ex_slr": synth.Workload("a_slr", [5, 7, 2], "silu", "squared", "fp32", B=4, T=5,
                                  B_outer=6, meta_kind=EX | SLR, optimizer="adam",
                                  adam_eps=1e-6, noise_std=0.1,
                                  extra={"scalar_loglr": math.log(0.01)}),
    "ex_plr": synth.Workload("a_explr", [5, 7, 3], "tanh", "squared", "fp32", B=5, T=3,
                             B_outer=4, meta_kind=EX | PLR, optimizer="adam", adam_eps=1e-3,
                             loglr_mean=math.log(0.01), loglr_std=0.1, noise_std=0.1),
    "multi_tile": synth.Workload("a_mt", [40, 136, 70, 3], "tanh", "squared", "fp32", B=90, T=3,
                                 B_outer=70, alpha=0.005, optimizer="adam", adam_eps=1e-3,
                                 noise_std=0.1),
    "dec32": synth.decoder("a_dec", 32, 4, 48, 2, 40, 16, B=2, T=3, B_outer=3, alpha=1e-3,
                           meta_kind=EX | SLR, optimizer="adam",
                           extra={"scalar_loglr": math.log(1e-3)}).with_(precision="fp32"),
}

BF16 = {
    "wide_small": synth.Workload("a_wide", [128, 256, 256, 10], "gelu", "ce", "bf16", B=64, T=4,
                                 B_outer=96, alpha=1e-3, optimizer="adam", adam_eps=1e-3),
    "deep_small": synth.Workload("a_deep", [256] * 4, "silu", "squared", "bf16", B=64, T=4,
                                 B_outer=64, meta_kind=PLR, optimizer="adam", adam_eps=1e-3,
                                 loglr_mean=math.log(1e-3), loglr_std=0.1),
    "dec16": synth.decoder("a_dec16", 64, 1, 128, 1, 200, 128, B=2, T=3, B_outer=2,
                           alpha=1e-3, optimizer="adam", adam_eps=1e-3),
}


def _meta(w, inp, mode=0, k=1, calls=1):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    loop = native.loop_desc_for(w, mode, ckpt_every=k)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.full((w.n_eta,), float("nan"), device="cuda")
    d_th = torch.full((w.n_params,), float("nan"), device="cuda")
    V = torch.full((1,), float("nan"), device="cuda")
    outs = []
    for _ in range(calls):
        mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th, V)
        mf.sync()
        outs.append((d_eta.cpu().numpy().copy(), d_th.cpu().numpy().copy(),
                     V.cpu().numpy().copy()))
    mf.close()
    for o in outs[1:]:
        assert all(np.array_equal(a, b) for a, b in zip(o, outs[0]))
    return outs[0]


def _check(w, tol, mode=0):
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    de, dt, V = _meta(w, inp, mode, calls=3)
    assert np.isfinite(de).all() and np.isfinite(dt).all()
    if w.n_eta:
        assert rel_l2(de, ref["d_eta"]) < tol, rel_l2(de, ref["d_eta"])
    assert rel_l2(dt, ref["d_theta0"]) < tol, rel_l2(dt, ref["d_theta0"])
    assert abs(float(V[0]) - ref["V"]) <= tol * abs(ref["V"])


@pytest.mark.gpu
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("name", list(FP32))
def test_adam_fp32(name, mode):
    _check(FP32[name], 1e-4, mode)


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(BF16))
def test_adam_bf16(name):
    _check(BF16[name], 2e-2)


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["silu_ex_slr", "tanh_plr", "dec32"])
def test_adam_segments_bit_identical(name):
    w = FP32[name]
    inp = synth.make_inputs(w)
    ref = _meta(w, inp, 0, 1)
    for k in (2, 3, w.T):
        out = _meta(w, inp, 0, k, calls=3 if k == 2 else 1)
        for a, b in zip(out, ref):
            assert np.array_equal(a, b), (name, k)


@pytest.mark.gpu
def test_adam_modes_agree():
    w = FP32["silu_ex_slr"]
    inp = synth.make_inputs(w)
    a = _meta(w, inp, 0)
    b = _meta(w, inp, 1)
    for x, y in zip(a, b):
        assert rel_l2(x, y) < 1e-5


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["ce_gelu_ex", "tanh_plr"])
def test_adam_rollout(name):
    torch, native = need_gpu()
    w = FP32[name]
    inp = synth.make_inputs(w)
    thetas, _ = om.rollout(w, inp)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    thT = torch.full((w.n_params,), float("nan"), device="cuda")
    mf.inner_rollout(native.loop_desc_for(w), d["theta0"], d["eta"], d["inner_x"],
                     d["inner_y"], thT)
    mf.sync()
    out = thT.cpu().numpy()
    mf.close()
    assert rel_l2(out, thetas[-1].numpy()) < 1e-5


@pytest.mark.gpu
def test_adam_arguments_checked():
    torch, native = need_gpu()
    w = FP32["ce_gelu_ex"]
    mf = native.MixFlow.for_workload(w)
    for field, value in (("momentum", 0.9), ("beta1", 1.0), ("beta2", -0.1),
                         ("adam_eps", 0.0), ("optimizer", 7)):
        loop = native.loop_desc_for(w)
        setattr(loop, field, value)
        with pytest.raises(native.MixflowError):
            mf.workspace_bytes(loop)
    mf.close()
