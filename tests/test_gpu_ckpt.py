"""Segment rematerialisation of the checkpoint store (ckpt_every = k, Section 4).

With k > 1 the store keeps theta_t (and m_t) only at multiples of k; the sweep re-runs each
earlier segment's rollout from its checkpoint with the same kernels.  The tests require the
meta-gradient to be bit-identical to k = 1 for every segment length (ragged last segments,
k = T, k > T), every optimiser state (plain SGD, momentum without a learning-rate
meta-parameter, per-parameter and scalar log learning rates), both HVP modes, both
architectures and the toy example, plus the store's size."""
import math

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, PLR, SLR = synth.EXAMPLE_WEIGHTS, synth.PARAM_LOGLR, synth.SCALAR_LOGLR

CASES = {
    "sgd_ex": synth.WORKLOADS["tiny"].with_(T=7),
    "mom_ex": synth.Workload("mom_ex", [6, 8, 3], "tanh", "squared", "fp32", B=5, T=7,
                             B_outer=4, momentum=0.9, alpha=0.1, noise_std=0.1),
    "mom_plr": synth.Workload("mom_plr", [4, 6, 3], "silu", "squared", "fp32", B=6, T=7,
                              B_outer=5, momentum=0.9, meta_kind=PLR,
                              loglr_mean=math.log(0.2), loglr_std=0.1),
    "mom_ex_slr": synth.Workload("mom_ex_slr", [5, 7, 2], "tanh", "squared", "fp32", B=4, T=8,
                                 B_outer=6, momentum=0.5, meta_kind=EX | SLR, noise_std=0.1,
                                 extra={"scalar_loglr": math.log(0.3)}),
    "bf16_deep": synth.Workload("bf16_deep", [256] * 4, "silu", "squared", "bf16", B=64, T=6,
                                B_outer=64, momentum=0.9, meta_kind=PLR,
                                loglr_mean=math.log(1e-2), loglr_std=0.1),
    "bf16_wide": synth.Workload("bf16_wide", [128, 256, 10], "gelu", "ce", "bf16", B=64, T=5,
                                B_outer=32, alpha=0.05),
    "dec32_mom": synth.decoder("dec32_mom", 32, 4, 48, 2, 40, 16, B=2, T=5, B_outer=3,
                               momentum=0.9, meta_kind=EX | SLR,
                               extra={"scalar_loglr": math.log(0.1)}).with_(precision="fp32"),
    "dec16": synth.decoder("dec16", 64, 1, 128, 1, 200, 128, B=2, T=4, B_outer=2, alpha=1e-2),
    "toy32": synth.toy("toy32", 24, 20, 3, T=5, precision="fp32"),
}


def _meta(w, inp, k, mode=0, calls=1):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    loop = native.loop_desc_for(w, mode, ckpt_every=k)
    d = native.to_device_inputs(w, inp)
    d_eta = torch.full((w.n_eta,), float("nan"), device="cuda")
    d_th = torch.full((w.n_params,), float("nan"), device="cuda")
    V = torch.full((1,), float("nan"), device="cuda")
    outs = []
    for _ in range(calls):   # the third call replays a captured graph
        mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th, V)
        mf.sync()
        outs.append((d_eta.cpu().numpy().copy(), d_th.cpu().numpy().copy(),
                     V.cpu().numpy().copy()))
    ws = mf.workspace_bytes(loop)
    mf.close()
    for o in outs[1:]:
        assert all(np.array_equal(a, b) for a, b in zip(o, outs[0]))
    return outs[0], ws


def _slots(w, k):
    """|theta|-sized store slots for segment length k, as include/mixflow.h states them:
    floor(T/k) + k for theta; m alike when the sweep reads it (log-lr meta-parameters), or
    at the checkpoints plus one running slot when only a recompute needs it (momentum)."""
    T = w.T
    k = min(max(k, 1), T)
    n_ck = T // k + 1
    lr_meta = bool(w.meta_kind & (PLR | SLR))
    if lr_meta:
        m = n_ck - 1 + k - 1
    elif w.momentum != 0 and k > 1:
        m = n_ck
    else:
        m = 0
    return n_ck + k - 1 + m


def _ks(T):
    return sorted({2, 3, T - 1 if T > 2 else 2, T, T + 4})


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(CASES))
def test_segments_bit_identical(name):
    w = CASES[name]
    inp = synth.make_inputs(w)
    ref, ws1 = _meta(w, inp, 1)
    for k in _ks(w.T):
        out, ws = _meta(w, inp, k, calls=3 if k == 2 else 1)
        for a, b in zip(out, ref):
            assert np.array_equal(a, b), (name, k)
        expect = (_slots(w, k) - _slots(w, 1)) * w.n_params * 4
        assert abs((ws - ws1) - expect) <= 512, (name, k, ws - ws1, expect)


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["mom_ex_slr", "bf16_deep", "dec32_mom"])
def test_segments_reverse_over_reverse(name):
    w = CASES[name]
    inp = synth.make_inputs(w)
    ref, _ = _meta(w, inp, 1, mode=1)
    for k in (2, 3):
        out, _ = _meta(w, inp, k, mode=1)
        for a, b in zip(out, ref):
            assert np.array_equal(a, b), (name, k)


@pytest.mark.gpu
def test_segments_against_oracle():
    w = CASES["mom_plr"]
    inp = synth.make_inputs(w)
    (de, dt, V), _ = _meta(w, inp, 3)
    ref = om.meta_grad(w, inp)
    assert rel_l2(de, ref["d_eta"]) < 1e-4
    assert rel_l2(dt, ref["d_theta0"]) < 1e-4


@pytest.mark.gpu
def test_store_size():
    """floor(T/k) + k parameter slots (and as many momentum slots, less the one for m_0),
    against T + 1 and T: the deep workload's T = 32 store at k = 6 shrinks by 44 of 65
    |theta|-sized slots."""
    torch, native = need_gpu()
    w = synth.WORKLOADS["deep"].with_(dims=[512] * 3, B=64, B_outer=64)
    P4 = w.n_params * 4
    mf = native.MixFlow.for_workload(w)
    ws = {k: mf.workspace_bytes(native.loop_desc_for(w, 0, ckpt_every=k)) for k in (1, 4, 6, 32)}
    mf.close()
    T = w.T
    for k in (4, 6):
        slots = (T + 1 + T) - ((T // k + k) + (T // k + k - 1))
        assert abs((ws[1] - ws[k]) - slots * P4) <= 512, (k, ws[1] - ws[k], slots * P4)
    assert ws[32] == ws[1]


@pytest.mark.gpu
def test_negative_ckpt_every_is_rejected():
    torch, native = need_gpu()
    w = CASES["sgd_ex"]
    mf = native.MixFlow.for_workload(w)
    with pytest.raises(native.MixflowError):
        mf.workspace_bytes(native.loop_desc_for(w, 0, ckpt_every=-1))
    mf.close()
