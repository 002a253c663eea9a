"""CUDA path against the float64 oracle, element by element, through the C ABI.

Tolerances (relative L2): 1e-4 for float32-precision workloads, 2e-2 for bf16-GEMM
workloads (bf16 operands with float32 accumulation, against exact float64 on the same
bf16-rounded inputs).  Sizes span several GEMM tiles with ragged tails; the full-size
"wide" workload (the benchmark's) is compared in full, the full-size "deep" workload at
T = 1 (where the oracle finishes in seconds) and through properties at T = 32."""
import math

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, PLR, SLR = synth.EXAMPLE_WEIGHTS, synth.PARAM_LOGLR, synth.SCALAR_LOGLR

FP32_CASES = {
    "tiny": synth.WORKLOADS["tiny"],
    "tiny_ce_gelu": synth.Workload("tiny_ce_gelu", [6, 8, 8, 4], "gelu", "ce", "fp32", B=5, T=3,
                                   B_outer=7, alpha=0.3),
    "tiny_mom_plr_silu": synth.Workload("tiny_mom_plr_silu", [4, 6, 3], "silu", "squared", "fp32",
                                        B=6, T=3, B_outer=5, momentum=0.9, meta_kind=PLR,
                                        loglr_mean=math.log(0.2), loglr_std=0.1),
    "tiny_ex_slr_mom": synth.Workload("tiny_ex_slr_mom", [5, 7, 2], "tanh", "squared", "fp32",
                                      B=4, T=3, B_outer=6, momentum=0.5, meta_kind=EX | SLR,
                                      noise_std=0.1, extra={"scalar_loglr": math.log(0.3)}),
    "fp32_multi_tile": synth.Workload("fp32_multi_tile", [40, 136, 70, 3], "tanh", "squared",
                                      "fp32", B=90, T=3, B_outer=70, alpha=0.2, noise_std=0.1),
    # weight logits and per-parameter log-lrs together: d eta_lr starts T*B = 15 floats into
    # eta, so the fused update takes its element-wise (unaligned) path
    "tiny_ex_plr_mom": synth.Workload("tiny_ex_plr_mom", [5, 7, 3], "tanh", "squared", "fp32",
                                      B=5, T=3, B_outer=4, momentum=0.5, meta_kind=EX | PLR,
                                      loglr_mean=math.log(0.1), loglr_std=0.1, noise_std=0.1),
}

BF16_CASES = {
    # several 128-row/column tiles plus ragged tails on every GEMM dimension
    "wide_small": synth.Workload("wide_small", [128, 256, 256, 10], "gelu", "ce", "bf16", B=64,
                                 T=4, B_outer=96, alpha=0.05),
    "wide_ragged": synth.Workload("wide_ragged", [72, 200, 136, 10], "gelu", "ce", "bf16", B=40,
                                  T=3, B_outer=56, alpha=0.05),
    "deep_small": synth.Workload("deep_small", [256] * 5, "silu", "squared", "bf16", B=64, T=6,
                                 B_outer=64, momentum=0.9, meta_kind=PLR,
                                 loglr_mean=math.log(1e-2), loglr_std=0.1),
    # K large enough for the cluster split-K path (S = 2 and 4) with ragged M = 100 / 120
    "wide_split": synth.Workload("wide_split", [1024, 384, 200, 10], "gelu", "ce", "bf16", B=100,
                                 T=3, B_outer=120, alpha=0.05),
    "mlp_ex_slr": synth.Workload("mlp_ex_slr", [64, 192, 130, 8], "tanh", "squared", "bf16",
                                 B=48, T=4, B_outer=32, momentum=0.5, meta_kind=EX | SLR,
                                 noise_std=0.1, extra={"scalar_loglr": math.log(0.05)}),
}


def run_meta_grad(w, inp):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    loop = native.loop_desc_for(w)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.full((w.n_eta,), float("nan"), device="cuda")
    d_th = torch.full((w.n_params,), float("nan"), device="cuda")
    V = torch.full((1,), float("nan"), device="cuda")
    mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                 d["outer_y"], d_eta, d_th, V)
    mf.sync()
    out = dict(d_eta=d_eta.cpu().numpy(), d_theta0=d_th.cpu().numpy(), V=float(V.cpu()))
    mf.close()
    return out


def _check(w, tol):
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    got = run_meta_grad(w, inp)
    assert np.isfinite(got["d_eta"]).all() and np.isfinite(got["d_theta0"]).all()
    e_eta = rel_l2(got["d_eta"], ref["d_eta"])
    e_th = rel_l2(got["d_theta0"], ref["d_theta0"])
    assert e_eta < tol, (w.name, e_eta)
    assert e_th < tol, (w.name, e_th)
    assert abs(got["V"] - ref["V"]) <= tol * abs(ref["V"])
    return e_eta, e_th


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(FP32_CASES))
def test_meta_grad_fp32(name):
    _check(FP32_CASES[name], 1e-4)


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(BF16_CASES))
def test_meta_grad_bf16(name):
    _check(BF16_CASES[name], 2e-2)


@pytest.mark.gpu
def test_meta_grad_wide_full_size():
    """The benchmark workload at its full size, every output against the oracle."""
    _check(synth.WORKLOADS["wide"], 2e-2)


@pytest.mark.gpu
def test_meta_grad_deep_full_size_single_step():
    """The 134M-parameter per-parameter-lr workload at full width with T = 1: the oracle
    computes every d eta_lr (= -lr * grad L_0 * grad V(theta_1))."""
    _check(synth.WORKLOADS["deep"].with_(T=1), 2e-2)


def _hvp_case(w, tol, seed=0):
    torch, native = need_gpu()
    inp = synth.make_inputs(w)
    x, y = inp.inner_x[0], inp.inner_y[0]
    v = synth.random_direction(w.n_params, seed, 11)
    wt = np.linspace(0.25, 1.0, w.B).astype(np.float32)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    tv = torch.from_numpy(v).cuda()
    tw = torch.from_numpy(wt).cuda()
    Hv = torch.full((w.n_params,), float("nan"), device="cuda")
    g = torch.full((w.n_params,), float("nan"), device="cuda")
    tl = torch.full((w.B,), float("nan"), device="cuda")
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], tv, Hv, ex_w=tw,
           tangent_losses=tl, grad=g)
    mf.sync()
    ref_hv = om.hvp(w, inp.theta0, x, y, v, wt)
    ref_g = om.grad(w, inp.theta0, x, y, wt)
    ref_tl = om.tangent_losses(w, inp.theta0, x, y, v)
    assert rel_l2(Hv.cpu().numpy(), ref_hv) < tol
    assert rel_l2(g.cpu().numpy(), ref_g) < tol
    assert rel_l2(tl.cpu().numpy(), ref_tl) < tol
    mf.close()


@pytest.mark.gpu
def test_hvp_fp32():
    _hvp_case(FP32_CASES["fp32_multi_tile"], 1e-4)
    _hvp_case(FP32_CASES["tiny_ce_gelu"], 1e-4)


@pytest.mark.gpu
def test_hvp_bf16():
    _hvp_case(BF16_CASES["wide_small"], 2e-2)
    _hvp_case(BF16_CASES["deep_small"], 2e-2)


@pytest.mark.gpu
def test_hvp_symmetry_full_width():
    """u^T (H v) = v^T (H u) (Eqs. 6-7) at the full wide-workload size, through mf_hvp."""
    torch, native = need_gpu()
    w = synth.WORKLOADS["wide"]
    inp = synth.make_inputs(w.with_(T=1))
    d = native.to_device_inputs(w.with_(T=1), inp)
    mf = native.MixFlow.for_workload(w)
    u = torch.from_numpy(synth.random_direction(w.n_params, 1, 1)).cuda()
    v = torch.from_numpy(synth.random_direction(w.n_params, 1, 2)).cuda()
    Hu = torch.empty_like(u)
    Hv = torch.empty_like(v)
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], u, Hu)
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], v, Hv)
    mf.sync()
    a = float(torch.dot(u.double(), Hv.double()))
    b = float(torch.dot(v.double(), Hu.double()))
    scale = float(u.double().norm() * Hv.double().norm())
    assert abs(a - b) <= 2e-2 * scale
    mf.close()


@pytest.mark.gpu
def test_inner_rollout_matches_oracle():
    torch, native = need_gpu()
    for w, tol in ((FP32_CASES["tiny_mom_plr_silu"], 1e-5), (BF16_CASES["deep_small"], 1e-2)):
        inp = synth.make_inputs(w)
        thetas, _ = om.rollout(w, inp)
        mf = native.MixFlow.for_workload(w)
        d = native.to_device_inputs(w, inp)
        out = torch.empty(w.n_params, device="cuda")
        mf.inner_rollout(native.loop_desc_for(w), d["theta0"], d["eta"], d["inner_x"],
                         d["inner_y"], out)
        mf.sync()
        ref = thetas[-1].numpy()
        assert rel_l2(out.cpu().numpy() - inp.theta0, ref - inp.theta0) < tol
        mf.close()


@pytest.mark.gpu
def test_special_cases_on_gpu():
    """alpha = 0: zero weight meta-gradient and dV/dtheta_0 = grad V(theta_0)."""
    w = FP32_CASES["tiny"].with_(alpha=0.0)
    inp = synth.make_inputs(w)
    got = run_meta_grad(w, inp)
    assert np.abs(got["d_eta"]).max() == 0.0
    gV = om.grad(w, inp.theta0, inp.outer_x, inp.outer_y)
    assert rel_l2(got["d_theta0"], gV) < 1e-5


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["mlp_ex_slr", "wide_split"])
def test_deterministic_repeat(name):
    """Two calls on the same inputs give bit-identical meta-gradients (fixed-order sums,
    including the cluster split-K reduction)."""
    w = BF16_CASES[name]
    inp = synth.make_inputs(w)
    a = run_meta_grad(w, inp)
    b = run_meta_grad(w, inp)
    assert np.array_equal(a["d_eta"], b["d_eta"])
    assert np.array_equal(a["d_theta0"], b["d_theta0"])


@pytest.mark.gpu
def test_graph_replay_matches_eager():
    """Repeated calls with the same pointers run eagerly, then capture a CUDA graph, then
    replay it; new input values behind the same pointers must be picked up by the replay."""
    torch, native = need_gpu()
    w = BF16_CASES["wide_split"]
    inp = synth.make_inputs(w)
    mf = native.MixFlow.for_workload(w)
    loop = native.loop_desc_for(w)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.empty(w.n_eta, device="cuda")
    d_th = torch.empty(w.n_params, device="cuda")
    outs = []
    for call in range(4):
        if call == 3:   # new inputs behind the same pointers
            d["eta"].mul_(-0.5)
        mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th)
        mf.sync()
        outs.append((d_eta.cpu().numpy().copy(), d_th.cpu().numpy().copy()))
    for k in (1, 2):
        assert np.array_equal(outs[0][0], outs[k][0]) and np.array_equal(outs[0][1], outs[k][1])
    eta2 = (inp.eta.astype(np.float64) * -0.5).astype(np.float32)
    ref = om.meta_grad(w, synth.Inputs(inp.theta0, eta2, inp.inner_x, inp.inner_y, inp.outer_x,
                                       inp.outer_y))
    assert rel_l2(outs[3][0], ref["d_eta"]) < 2e-2
    # graphs off: same numbers as the eager first call
    mf.set_option(native.MF_OPT_CUDA_GRAPHS, 0)
    d["eta"].mul_(-2.0)
    mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                 d["outer_y"], d_eta, d_th)
    mf.sync()
    assert np.array_equal(d_eta.cpu().numpy(), outs[0][0])
    mf.close()


@pytest.mark.gpu
@pytest.mark.parametrize("option", ["MF_OPT_PDL", "MF_OPT_CONCURRENT"])
def test_launch_options_bit_identical(option):
    """Programmatic dependent launch and the two-stream backward change when kernels may
    run, not what they compute or the order of dependent memory effects: the meta-gradient
    is bit-identical with the option on and off, eager and replayed."""
    torch, native = need_gpu()
    opt = getattr(native, option)
    w = BF16_CASES["wide_ragged"]
    inp = synth.make_inputs(w)
    outs = []
    for val in (1, 0, 1):
        mf = native.MixFlow.for_workload(w)
        mf.set_option(opt, val)
        loop = native.loop_desc_for(w)
        d = native.to_device_inputs(w, inp)
        d_eta = torch.empty(w.n_eta, device="cuda")
        d_th = torch.empty(w.n_params, device="cuda")
        for _ in range(3):   # eager, capture, replay
            mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                         d["outer_y"], d_eta, d_th)
        mf.sync()
        outs.append((d_eta.cpu().numpy(), d_th.cpu().numpy()))
        mf.close()
    for k in (1, 2):
        assert np.array_equal(outs[0][0], outs[k][0]) and np.array_equal(outs[0][1], outs[k][1])


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["wide_small", "wide_split", "mlp_ex_slr"])
def test_meta_grad_bf16_pair_tiles(name):
    """Every GEMM with more than 128 rows on 256-row CTA-pair tiles."""
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(synth.WORKLOADS["tiny"])
    mf.set_option(native.MF_OPT_GEMM_2SM, 2)
    try:
        _check(BF16_CASES[name], 2e-2)
    finally:
        mf.set_option(native.MF_OPT_GEMM_2SM, 1)
        mf.close()
