"""Fused dual attention (MF_OPT_FLASH_ATTN) against the float64 oracle and against the
materialised attention of the same library.

The fused path serves bf16 decoders with 64-wide heads and sequences of whole 64-token
tiles; it keeps only per-row statistics instead of the S x S probabilities.  Cases span one
to four query/key tiles per head (the causal diagonal, off-diagonal tiles and the skipped
upper triangle), one and several heads, both HVP modes, HVPs, and the workspace saving."""
import math

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, SLR = synth.EXAMPLE_WEIGHTS, synth.SCALAR_LOGLR

CASES = {
    # d, H, F, L, V, S
    "one_tile": synth.decoder("f1", 128, 2, 256, 2, 256, 64, B=4, T=2, B_outer=4, alpha=1e-2),
    "three_tiles": synth.decoder("f3", 64, 1, 128, 1, 200, 192, B=2, T=3, B_outer=2,
                                 momentum=0.9, meta_kind=EX | SLR,
                                 extra={"scalar_loglr": math.log(1e-2)}),
    "four_tiles_4h": synth.decoder("f4", 256, 4, 512, 1, 304, 256, B=2, T=2, B_outer=2,
                                   alpha=1e-2),
}


def _run(w, inp, flash, mode=0):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    mf.set_option(native.MF_OPT_FLASH_ATTN, 1 if flash else 0)
    loop = native.loop_desc_for(w, mode)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.full((w.n_eta,), float("nan"), device="cuda")
    d_th = torch.full((w.n_params,), float("nan"), device="cuda")
    V = torch.full((1,), float("nan"), device="cuda")
    outs = []
    for _ in range(3):   # eager, capture, replay
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
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("name", list(CASES))
def test_flash_meta_grad(name, mode):
    w = CASES[name]
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    (de_f, dt_f, V_f), ws_f = _run(w, inp, True, mode)
    (de_m, dt_m, V_m), ws_m = _run(w, inp, False, mode)
    assert np.isfinite(de_f).all() and np.isfinite(dt_f).all()
    assert rel_l2(de_f, ref["d_eta"]) < 2e-2
    assert rel_l2(dt_f, ref["d_theta0"]) < 2e-2
    assert abs(V_f - ref["V"]) <= 2e-2 * abs(ref["V"])
    # the two attention forms round different intermediates to bf16; both sit at the same
    # distance from the oracle, far closer to each other than the bf16 bound
    assert rel_l2(dt_f, dt_m) < 1e-2
    assert rel_l2(de_f, de_m) < 1e-2
    assert ws_f < ws_m


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["three_tiles", "four_tiles_4h"])
def test_flash_hvp(name):
    torch, native = need_gpu()
    w = CASES[name]
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
    assert rel_l2(g.cpu().numpy(), om.grad(w, inp.theta0, ids, ids, wt)) < 2e-2
    assert rel_l2(Hv.cpu().numpy(), om.hvp(w, inp.theta0, ids, ids, v, wt)) < 2e-2
    assert rel_l2(tl.cpu().numpy(), om.tangent_losses(w, inp.theta0, ids, ids, v)) < 2e-2
    mf.close()


@pytest.mark.gpu
def test_flash_workspace_saving():
    """Without P and P' per block and the score scratch: the decoder_small workspace shrinks
    by (2 L + 2) B H S^2 bf16 values (P, P' per block; dS, dS') and 4 B H S^2 float32 values
    (scores, score gradients and their tangents) and the per-head float32 outputs O, O'
    (2 B H S d_head values; the fused forward writes them head-merged in bf16), less the row
    statistics (lse and rbar per block, D and D') of 2 (L + 1) B H S float32 values."""
    torch, native = need_gpu()
    w = synth.WORKLOADS["decoder_small"]
    mf = native.MixFlow.for_workload(w)
    loop = native.loop_desc_for(w)
    mf.set_option(native.MF_OPT_FLASH_ATTN, 0)
    ws_m = mf.workspace_bytes(loop)
    mf.set_option(native.MF_OPT_FLASH_ATTN, 1)
    ws_f = mf.workspace_bytes(loop)
    mf.close()
    S, L = w.seq, w.n_blocks
    BH = max(w.B, w.B_outer) * w.n_heads
    ss = BH * S * S
    dh = w.d_model // w.n_heads
    saved = (2 * L + 2) * ss * 2 + 4 * ss * 4 + 2 * BH * S * dh * 4 - (L + 1) * 2 * BH * S * 4
    assert abs((ws_m - ws_f) - saved) <= 256 * (4 * L + 16), (ws_m - ws_f, saved)


@pytest.mark.gpu
def test_decoder_large_full_size_hvp_symmetry():
    """The 218M-parameter decoder (12 blocks, d 1024, 16 heads, S = 1024, fused attention)
    at full size: u^T (H v) = v^T (H u) through mf_hvp (Eqs. 6-7), and H is linear in its
    direction.  Directions are scaled like the weights (0.02)."""
    torch, native = need_gpu()
    w = synth.WORKLOADS["decoder_large"]
    w1 = w.with_(T=1)
    inp = synth.make_inputs(w1)
    d = native.to_device_inputs(w1, inp)
    mf = native.MixFlow.for_workload(w)
    u = torch.from_numpy(synth.random_direction(w.n_params, 4, 1)).cuda() * 0.02
    v = torch.from_numpy(synth.random_direction(w.n_params, 4, 2)).cuda() * 0.02
    Hu, Hv, Hs = torch.empty_like(u), torch.empty_like(v), torch.empty_like(u)
    for vec, out in ((u, Hu), (v, Hv), (u + v, Hs)):
        mf.hvp(w.B, d["theta0"], d["inner_x"][0], d["inner_y"][0], vec, out)
    mf.sync()
    mf.close()
    a = float(torch.dot(u.double(), Hv.double()))
    b = float(torch.dot(v.double(), Hu.double()))
    assert np.isfinite(a) and np.isfinite(b)
    scale = float(u.double().norm() * Hv.double().norm())
    assert abs(a - b) <= 2e-2 * scale, (a, b, scale)
    assert rel_l2(Hs.cpu().numpy(), (Hu + Hv).cpu().numpy()) < 2e-2
