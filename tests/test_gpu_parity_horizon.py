"""Oracle parity at the per-block shapes of the larger workloads and at their full horizons.

Mixed-mode meta-gradients are exact (Proposition 3.1), so Algorithm 2 on the GPU must give
Algorithm 1's dV/d eta, dV/d theta_0 and V (the oracle, float64) up to bf16 rounding of the
GEMM operands: relative L2 2e-2 on every output, the same bar as every bf16 case.

- Larger transformer (Section 5's long-horizon language model): its exact block shapes
  (d 1024, 16 heads of 64, MLP 4096, vocabulary 32768, S = 1024, i.e. 16 attention tiles per
  head on the fused attention path), heavy ball 0.9, per-sequence weight logits plus the
  scalar log learning rate, with 2 blocks, 2 sequences and T = 2 so the oracle finishes in
  well under a minute.
- Deep MLP with learned per-parameter learning rates: 4096-wide SiLU layers, heavy ball 0.9,
  at the full horizon T = 32, where bf16 errors of 32 momentum steps accumulate in theta_t
  and in the adjoint.
- Small transformer at its full horizon T = 8 and full shapes, with 4 of its 16 sequences."""
import math

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, PLR, SLR = synth.EXAMPLE_WEIGHTS, synth.PARAM_LOGLR, synth.SCALAR_LOGLR
TOL = 2e-2

LARGE_BLOCKS = synth.decoder("decoder_large_2blk", 1024, 16, 4096, 2, 32768, 1024, B=2, T=2,
                             B_outer=2, momentum=0.9, meta_kind=EX | SLR,
                             extra={"scalar_loglr": math.log(1e-3)})
DEEP_T32 = synth.Workload("deep_3x4096_T32", [4096] * 4, "silu", "squared", "bf16", B=128,
                          T=32, B_outer=128, momentum=0.9, meta_kind=PLR,
                          loglr_mean=math.log(1e-2), loglr_std=0.1)
SMALL_T8 = synth.WORKLOADS["decoder_small"].with_(name="decoder_small_B4", B=4, B_outer=4)


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
    del d, d_eta, d_th, V
    torch.cuda.empty_cache()
    return out


def _compare(w):
    need_gpu()
    inp = synth.make_inputs(w)
    got = _run(w, inp)
    ref = om.meta_grad(w, inp)
    assert np.isfinite(got["d_eta"]).all() and np.isfinite(got["d_theta0"]).all()
    errs = {"V": abs(got["V"] - ref["V"]) / abs(ref["V"]),
            "d_theta0": rel_l2(got["d_theta0"], ref["d_theta0"]),
            "d_eta": rel_l2(got["d_eta"], ref["d_eta"])}
    o = 0
    if w.meta_kind & EX:     # the weight logits and the learning-rate part, each on its own
        n = w.T * w.B
        errs["d_eta_weights"] = rel_l2(got["d_eta"][:n], ref["d_eta"][:n])
        o = n
    if w.meta_kind & (PLR | SLR):
        errs["d_eta_lr"] = rel_l2(got["d_eta"][o:], ref["d_eta"][o:])
    print(w.name, {k: f"{v:.2e}" for k, v in errs.items()})
    for k, e in errs.items():
        assert e < TOL, (w.name, k, e)


@pytest.mark.gpu
def test_decoder_large_blocks_meta_grad():
    _compare(LARGE_BLOCKS)


@pytest.mark.gpu
def test_deep_full_horizon_meta_grad():
    _compare(DEEP_T32)


@pytest.mark.gpu
def test_decoder_small_full_horizon_meta_grad():
    _compare(SMALL_T8)
