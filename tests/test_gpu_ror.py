"""Reverse-over-reverse Hessian-vector products (Algorithm 1's schedule) on the GPU.

The two modes compute the same mathematical object (Eqs. 6-7: the Hessian is symmetric, so
differentiating the backward pass in reverse equals pushing a tangent forward through it).
Checked here: each mode against the float64 oracle, the two modes against each other at
float32 (where only the summation order differs), the full meta-gradient in both modes for
MLPs and the decoder, graph replay, and that the stored backward graph makes
reverse-over-reverse need more workspace than the mixed-mode sweep."""
import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

from test_gpu_parity import BF16_CASES, FP32_CASES

MIXED, REVREV = 0, 1


def _hvp(w, inp, mode, v, wt):
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
@pytest.mark.parametrize("name", ["tiny", "tiny_ce_gelu", "tiny_mom_plr_silu", "fp32_multi_tile"])
def test_ror_hvp_fp32(name):
    w = FP32_CASES[name]
    inp = synth.make_inputs(w)
    x, y = inp.inner_x[0], inp.inner_y[0]
    v = synth.random_direction(w.n_params, 3, 11)
    wt = np.linspace(0.25, 1.0, w.B).astype(np.float32)
    hv_r, g_r, tl_r = _hvp(w, inp, REVREV, v, wt)
    hv_m, g_m, tl_m = _hvp(w, inp, MIXED, v, wt)
    assert np.isfinite(hv_r).all() and np.isfinite(g_r).all() and np.isfinite(tl_r).all()
    ref_hv = om.hvp(w, inp.theta0, x, y, v, wt)
    assert rel_l2(hv_r, ref_hv) < 1e-4
    assert rel_l2(g_r, om.grad(w, inp.theta0, x, y, wt)) < 1e-4
    assert rel_l2(tl_r, om.tangent_losses(w, inp.theta0, x, y, v)) < 1e-4
    # same float32 arithmetic up to summation order
    assert rel_l2(hv_r, hv_m) < 1e-5
    assert rel_l2(g_r, g_m) < 1e-5
    assert rel_l2(tl_r, tl_m) < 1e-5


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["wide_small", "wide_ragged", "deep_small"])
def test_ror_hvp_bf16(name):
    w = BF16_CASES[name]
    inp = synth.make_inputs(w)
    x, y = inp.inner_x[0], inp.inner_y[0]
    v = synth.random_direction(w.n_params, 4, 11)
    wt = np.linspace(0.25, 1.0, w.B).astype(np.float32)
    hv_r, g_r, tl_r = _hvp(w, inp, REVREV, v, wt)
    assert rel_l2(hv_r, om.hvp(w, inp.theta0, x, y, v, wt)) < 2e-2
    assert rel_l2(g_r, om.grad(w, inp.theta0, x, y, wt)) < 2e-2
    assert rel_l2(tl_r, om.tangent_losses(w, inp.theta0, x, y, v)) < 2e-2


def _meta(w, inp, mode):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    loop = native.loop_desc_for(w, hvp_mode=mode)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.full((w.n_eta,), float("nan"), device="cuda")
    d_th = torch.full((w.n_params,), float("nan"), device="cuda")
    V = torch.full((1,), float("nan"), device="cuda")
    outs = []
    for _ in range(3):   # the third call replays a captured graph
        mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th, V)
        mf.sync()
        outs.append((d_eta.cpu().numpy().copy(), d_th.cpu().numpy().copy(), float(V.cpu())))
    ws = mf.workspace_bytes(loop)
    mf.close()
    for o in outs[1:]:
        assert np.array_equal(o[0], outs[0][0]) and np.array_equal(o[1], outs[0][1])
    return outs[0], ws


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(FP32_CASES))
def test_ror_meta_grad_fp32(name):
    w = FP32_CASES[name]
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    (de_r, dt_r, V_r), _ = _meta(w, inp, REVREV)
    (de_m, dt_m, _), _ = _meta(w, inp, MIXED)
    assert rel_l2(de_r, ref["d_eta"]) < 1e-4
    assert rel_l2(dt_r, ref["d_theta0"]) < 1e-4
    assert abs(V_r - ref["V"]) <= 1e-4 * abs(ref["V"])
    assert rel_l2(de_r, de_m) < 1e-5
    assert rel_l2(dt_r, dt_m) < 1e-5


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["wide_small", "deep_small", "mlp_ex_slr", "wide_split"])
def test_ror_meta_grad_bf16(name):
    w = BF16_CASES[name]
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    (de_r, dt_r, _), _ = _meta(w, inp, REVREV)
    assert rel_l2(de_r, ref["d_eta"]) < 2e-2
    assert rel_l2(dt_r, ref["d_theta0"]) < 2e-2


@pytest.mark.gpu
def test_ror_needs_more_workspace():
    """The stored inner backward graph (every layer's dz and da, their adjoints) is what
    reverse-over-reverse keeps beyond the mixed-mode sweep."""
    torch, native = need_gpu()
    for w in (synth.WORKLOADS["wide"], synth.WORKLOADS["deep"]):
        mf = native.MixFlow.for_workload(w)
        a = mf.workspace_bytes(native.loop_desc_for(w, hvp_mode=MIXED))
        b = mf.workspace_bytes(native.loop_desc_for(w, hvp_mode=REVREV))
        mf.close()
        assert b > a


@pytest.mark.gpu
@pytest.mark.parametrize("name,tol,tol_modes", [("dec32_a", 1e-4, 1e-5), ("dec32_mom", 1e-4, 1e-5),
                                               ("dec16_small", 2e-2, 5e-3), ("dec16_mom", 2e-2, 5e-3)])
def test_ror_decoder_meta_grad(name, tol, tol_modes):
    """Decoder reverse-over-reverse (block-granular reverse graph): against the oracle, and
    against the mixed-mode sweep (float32: same arithmetic up to summation order; bf16: the
    primal-only and dual GEMMs may tile differently)."""
    from test_gpu_decoder import BF16 as DBF16, FP32 as DFP32
    w = DFP32.get(name) or DBF16[name]
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    (de_r, dt_r, V_r), ws_r = _meta(w, inp, REVREV)
    (de_m, dt_m, _), ws_m = _meta(w, inp, MIXED)
    assert rel_l2(de_r, ref["d_eta"]) < tol
    assert rel_l2(dt_r, ref["d_theta0"]) < tol
    assert abs(V_r - ref["V"]) <= tol * abs(ref["V"])
    assert rel_l2(de_r, de_m) < tol_modes
    assert rel_l2(dt_r, dt_m) < tol_modes
    assert ws_r > ws_m


@pytest.mark.gpu
def test_ror_decoder_hvp():
    torch, native = need_gpu()
    from test_gpu_decoder import FP32 as DFP32
    w = DFP32["dec32_mom"]
    inp = synth.make_inputs(w)
    v = synth.random_direction(w.n_params, 5, 11)
    wt = np.linspace(0.25, 1.0, w.B).astype(np.float32)
    hv_r, g_r, tl_r = _hvp(w, inp, REVREV, v, wt)
    hv_m, g_m, tl_m = _hvp(w, inp, MIXED, v, wt)
    x, y = inp.inner_x[0], inp.inner_y[0]
    assert rel_l2(hv_r, om.hvp(w, inp.theta0, x, y, v, wt)) < 1e-4
    assert rel_l2(hv_r, hv_m) < 1e-5
    assert rel_l2(g_r, g_m) < 1e-5
    assert rel_l2(tl_r, tl_m) < 1e-5
