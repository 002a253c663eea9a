"""Option paths, each against the default path or the oracle.

- MF_OPT_GEMM_PERSISTENT (on by default, mode 2): the persistent CTA-pair GEMM in modes 1
  and 3 against float64 products of the same bf16 operands, on grids with several tiles per
  CTA pair (both TMEM accumulator sets and the stage ring reused across tiles), and bf16
  meta-gradients against the oracle.
- MF_OPT_FUSED_HEAD (off by default): the narrow output layer, loss and data product in one kernel;
  meta-gradients, HVPs with gradient and tangent losses, and the label check, against the
  oracle at the default path's tolerances.
- MF_OPT_LAYER_UPDATES (off by default): per-layer updates on the update stream; the same update element for
  element, so meta-gradients are bit-identical to the single update (eager, captured and
  replayed calls)."""
import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om
import test_gpu_adam as ta
import test_gpu_gemm as tg
import test_gpu_parity as tp

def _set(native, option, value):
    """Process-wide options; any handle can set them."""
    mf = native.MixFlow.for_workload(synth.WORKLOADS["tiny"])
    mf.set_option(option, value)
    mf.close()


# ---- persistent CTA-pair GEMM ------------------------------------------------------------

@pytest.fixture(params=[1, 3])
def persistent(request):
    """Mode 1 (dual products at 128-wide tiles, two TMEM sets) and mode 3 (256-wide dual
    tiles, one set: the default mode's path for dual products with K > 2048)."""
    torch, native = need_gpu()
    _set(native, native.MF_OPT_GEMM_2SM, 2)
    _set(native, native.MF_OPT_GEMM_PERSISTENT, request.param)
    yield
    _set(native, native.MF_OPT_GEMM_PERSISTENT, 2)   # the default
    _set(native, native.MF_OPT_GEMM_2SM, 1)


MANY_TILES = [(2048, 1024, 64), (4096, 512, 136), (1280, 2304, 200)]


@pytest.mark.gpu
@pytest.mark.parametrize("shape", tg.PAIR_SHAPES + MANY_TILES)
@pytest.mark.parametrize("mask", tg.MASKS)
def test_persistent_dual_gemm(persistent, shape, mask):
    tg.test_dual_gemm(shape, mask)


@pytest.mark.gpu
@pytest.mark.parametrize("shape", tg.MN_SHAPES + MANY_TILES[:1])
@pytest.mark.parametrize("layout", [1, 2, 3])
@pytest.mark.parametrize("mask", [1, 1 | 8 | 16, 2 | 4])
def test_persistent_dual_gemm_mn_major(persistent, shape, layout, mask):
    torch, native = need_gpu()
    tg.test_dual_gemm_mn_major(shape, layout, mask, 2)
    _set(native, native.MF_OPT_GEMM_2SM, 2)   # the helper resets the pair mode on exit


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["wide_small", "wide_split", "deep_small", "mlp_ex_slr"])
def test_persistent_meta_grad_bf16(persistent, name):
    tp._check(tp.BF16_CASES[name], 2e-2)


# ---- fused narrow head ---------------------------------------------------------------------

@pytest.fixture
def fused():
    torch, native = need_gpu()
    _set(native, native.MF_OPT_FUSED_HEAD, 1)
    yield
    _set(native, native.MF_OPT_FUSED_HEAD, 0)


LINEAR = synth.Workload("linear_fused", [12, 3], "ident", "squared", "fp32", B=9, T=3,
                        B_outer=5, alpha=0.1, noise_std=0.1)


@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(tp.FP32_CASES))
def test_fused_head_fp32(fused, name):
    tp._check(tp.FP32_CASES[name], 1e-4)


@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(tp.BF16_CASES))
def test_fused_head_bf16(fused, name):
    tp._check(tp.BF16_CASES[name], 2e-2)


@pytest.mark.gpu
def test_fused_head_single_layer(fused):
    tp._check(LINEAR, 1e-4)


@pytest.mark.gpu
def test_fused_head_wide_full(fused):
    tp._check(synth.WORKLOADS["wide"], 2e-2)


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["wide_small", "tiny_ce_gelu"])
def test_fused_head_hvp(fused, name):
    torch, native = need_gpu()
    w = tp.BF16_CASES.get(name) or tp.FP32_CASES[name]
    tol = 2e-2 if w.precision == "bf16" else 1e-4
    inp = synth.make_inputs(w)
    d = native.to_device_inputs(w, inp)
    mf = native.MixFlow.for_workload(w)
    v = synth.random_direction(w.n_params, 7, 1)
    wt = np.linspace(0.2, 1.0, w.B).astype(np.float32)
    Hv = torch.empty(w.n_params, device="cuda")
    g = torch.empty(w.n_params, device="cuda")
    tl = torch.empty(w.B, device="cuda")
    mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], torch.from_numpy(v).cuda(), Hv,
           ex_w=torch.from_numpy(wt).cuda(), tangent_losses=tl, grad=g)
    mf.sync()
    mf.close()
    x, y = inp.inner_x[0], inp.inner_y[0]
    assert rel_l2(Hv.cpu().numpy(), om.hvp(w, inp.theta0, x, y, v, wt)) < tol
    assert rel_l2(g.cpu().numpy(), om.grad(w, inp.theta0, x, y, wt)) < tol
    assert rel_l2(tl.cpu().numpy(), om.tangent_losses(w, inp.theta0, x, y, v)) < tol


@pytest.mark.gpu
def test_fused_head_reports_bad_label(fused):
    import test_gpu_errors as te
    te.test_out_of_range_class_label_is_reported()


# ---- per-layer updates --------------------------------------------------------------------

def _runs(w, layer_updates, ckpt_every=1):
    torch, native = need_gpu()
    inp = synth.make_inputs(w)
    d = native.to_device_inputs(w, inp)
    mf = native.MixFlow.for_workload(w)
    mf.set_option(native.MF_OPT_LAYER_UPDATES, 1 if layer_updates else 0)
    loop = native.loop_desc_for(w, ckpt_every=ckpt_every)
    outs = []
    for _ in range(3):   # eager, captured, replayed
        d_eta = torch.full((w.n_eta,), float("nan"), device="cuda")
        d_th = torch.full((w.n_params,), float("nan"), device="cuda")
        V = torch.full((1,), float("nan"), device="cuda")
        mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th, V)
        mf.sync()
        outs.append((d_eta.cpu().numpy(), d_th.cpu().numpy(), V.cpu().numpy()))
    mf.close()
    return outs


UPD_CASES = dict(tp.FP32_CASES)
UPD_CASES.update(tp.BF16_CASES)
UPD_CASES.update({"adam_" + k: v for k, v in ta.FP32.items() if v.arch != "decoder"})


def _same(a, b):
    for x, y in zip(a, b):
        for p, q in zip(x, y):
            assert np.array_equal(p, q)


@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(UPD_CASES))
def test_layer_updates_bit_identical(name):
    w = UPD_CASES[name]
    _same(_runs(w, False), _runs(w, True))


@pytest.mark.gpu
@pytest.mark.parametrize("k", [2, 3])
def test_layer_updates_with_segments(k):
    w = tp.BF16_CASES["deep_small"]
    _same(_runs(w, False, ckpt_every=k), _runs(w, True, ckpt_every=k))


@pytest.mark.gpu
def test_layer_updates_with_fused_head(fused):
    w = tp.BF16_CASES["wide_small"]
    _same(_runs(w, False), _runs(w, True))
