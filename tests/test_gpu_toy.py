"""The motivating example of Section 3 (Eq. 8) on the GPU: a D x D linear map followed by the
M-step recursion y_i = i (2 + sin y_{i-1})^cos y_{i-1} inside the loss kernel, theta_0 as the
meta-parameter (MAML-style), against the float64 oracle in both HVP modes.  The mixed mode
carries the recursion's derivatives and stores nothing of it; reverse-over-reverse records
the chain's tape (2 M floats per output element), so only its workspace grows with M."""
import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

CASES = {
    # float32 (SIMT GEMMs), theta_0 ~ N(0, 1) as in the paper's listing
    "toy32_m3": (synth.toy("toy32_m3", 24, 20, 3, T=2, precision="fp32"), 1e-4),
    # the recursion's derivatives grow like M!; at M = 8 a relative change of 1e-7 in theta_0
    # already moves the float64 meta-gradient by tens of percent, so the deep float32 case
    # keeps M = 6 with y_0 of unit scale (theta_0 ~ N(0, 1/D)), where it moves by 7e-6
    "toy32_m6": (synth.toy("toy32_m6", 40, 33, 6, T=2, precision="fp32",
                           init_std=1.0 / np.sqrt(40.0)), 1e-4),
    "toy32_m0": (synth.toy("toy32_m0", 16, 12, 0, T=3, precision="fp32"), 1e-4),
    # bf16 tensor cores, theta_0 scaled by 1/sqrt(D) (several tiles, ragged tails).  Rounding
    # theta and v to bf16 alone moves the exact HVP by 0.9% at M = 3 and by 2.1% at M = 4,
    # so parity against the unrounded oracle at 2e-2 uses M = 3; test_toy_hvp_bf16_operands
    # checks deeper chains against the oracle on the same bf16 operands
    "toy16_m3": (synth.toy("toy16_m3", 264, 150, 3, T=2, init_std=1.0 / 16.0), 2e-2),
}


def _run(w, inp, mode=0):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.zeros(0, device="cuda")
    d_th = torch.full((w.n_params,), float("nan"), device="cuda")
    V = torch.full((1,), float("nan"), device="cuda")
    mf.meta_grad(native.loop_desc_for(w, mode), d["theta0"], d["eta"], d["inner_x"],
                 d["inner_y"], d["outer_x"], d["outer_y"], d_eta, d_th, V)
    mf.sync()
    ws = mf.workspace_bytes(native.loop_desc_for(w, mode))
    out = d_th.cpu().numpy(), float(V.cpu()), ws
    mf.close()
    return out


@pytest.mark.gpu
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("name", list(CASES))
def test_toy_meta_grad(name, mode):
    w, tol = CASES[name]
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    dth, V, _ = _run(w, inp, mode)
    assert np.isfinite(dth).all()
    assert rel_l2(dth, ref["d_theta0"]) < tol, rel_l2(dth, ref["d_theta0"])
    assert abs(V - ref["V"]) <= tol * abs(ref["V"])


@pytest.mark.gpu
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("name", ["toy32_m3", "toy32_m6", "toy16_m3"])
def test_toy_hvp(name, mode):
    """H v, grad L and the tangent losses of one inner step through the chain."""
    w, tol = CASES[name]
    inp = synth.make_inputs(w)
    x, y = inp.inner_x[0], inp.inner_y[0]
    v = synth.random_direction(w.n_params, 6, 2) * np.float32(w.init_std)
    wt = np.linspace(0.25, 1.0, w.B).astype(np.float32)
    hv, gg, tt = _hvp(w, inp, v, wt, mode)
    assert rel_l2(hv, om.hvp(w, inp.theta0, x, y, v, wt)) < tol
    assert rel_l2(gg, om.grad(w, inp.theta0, x, y, wt)) < tol
    assert rel_l2(tt, om.tangent_losses(w, inp.theta0, x, y, v)) < tol


@pytest.mark.gpu
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("M", [4, 6])
def test_toy_hvp_bf16_operands(M, mode):
    """Deeper chains on the bf16 path against the oracle evaluated on the same bf16-rounded
    theta and v (the GEMM operands); what remains is the kernel's own error: float32
    accumulation, the float32 chain, and the bf16 seeds of the weight product."""
    w = synth.toy("toy16_ops", 264, 150, M, T=2, init_std=1.0 / 16.0)
    inp = synth.make_inputs(w)
    x, y = inp.inner_x[0], inp.inner_y[0]
    v = synth.random_direction(w.n_params, 6, 2) * np.float32(w.init_std)
    wt = np.linspace(0.25, 1.0, w.B).astype(np.float32)
    hv, gg, tt = _hvp(w, inp, v, wt, mode)
    th_r, v_r = synth.round_bf16(inp.theta0), synth.round_bf16(v)
    assert rel_l2(hv, om.hvp(w, th_r, x, y, v_r, wt)) < 5e-3
    assert rel_l2(gg, om.grad(w, th_r, x, y, wt)) < 5e-3
    assert rel_l2(tt, om.tangent_losses(w, th_r, x, y, v_r)) < 5e-3


def _hvp(w, inp, v, wt, mode):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    Hv = torch.full((w.n_params,), float("nan"), device="cuda")
    g = torch.full((w.n_params,), float("nan"), device="cuda")
    tl = torch.full((w.B,), float("nan"), device="cuda")
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], torch.from_numpy(v).cuda(), Hv,
           ex_w=torch.from_numpy(wt).cuda(), tangent_losses=tl, grad=g, hvp_mode=mode)
    mf.sync()
    out = Hv.cpu().numpy(), g.cpu().numpy(), tl.cpu().numpy()
    mf.close()
    return out


@pytest.mark.gpu
def test_toy_workspace_against_steps():
    """Mixed mode: the workspace does not depend on M (the axis of the paper's Fig. 3).
    Reverse-over-reverse: it grows by exactly the chain's tape, 2 M floats per element of
    the B x D output (up to the allocator's 256-byte alignment)."""
    torch, native = need_gpu()
    B, D = 256, 512
    mixed, rr = [], []
    for M in (1, 8, 64):
        w = synth.toy("toy_ws", D, B, M)
        mf = native.MixFlow.for_workload(w)
        mixed.append(mf.workspace_bytes(native.loop_desc_for(w, 0)))
        rr.append(mf.workspace_bytes(native.loop_desc_for(w, 1)))
        mf.close()
    assert mixed[0] == mixed[1] == mixed[2]
    assert rr[0] > mixed[0]
    for M, r in zip((8, 64), rr[1:]):
        assert abs((r - rr[0]) - 2 * (M - 1) * B * D * 4) <= 256


@pytest.mark.gpu
def test_toy_full_size_hvp_symmetry():
    """Full-size example (B = 1024, D = 4096, M = 8, bf16): u^T (H v) = v^T (H u) through mf_hvp."""
    torch, native = need_gpu()
    w = synth.WORKLOADS["toy"]
    inp = synth.make_inputs(w.with_(T=1))
    d = native.to_device_inputs(w.with_(T=1), inp)
    mf = native.MixFlow.for_workload(w)
    u = torch.from_numpy(synth.random_direction(w.n_params, 1, 1)).cuda() / 64.0
    v = torch.from_numpy(synth.random_direction(w.n_params, 1, 2)).cuda() / 64.0
    Hu, Hv = torch.empty_like(u), torch.empty_like(v)
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], u, Hu)
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], v, Hv)
    mf.sync()
    a = float(torch.dot(u.double(), Hv.double()))
    b = float(torch.dot(v.double(), Hu.double()))
    assert np.isfinite(a) and np.isfinite(b)
    assert abs(a - b) <= 2e-2 * float(u.double().norm() * Hv.double().norm())
    mf.close()
