"""Binomial checkpointing of the theta_t store (ckpt_slots = s, Section 4's binomial
checkpointing): the rollout leaves the schedule's snapshots, and the sweep recomputes every
other state from a snapshot with the rollout's own kernels before reversing it.  The
meta-gradient must be bit-identical to the full store (ckpt_every = 1) for every slot count
(one snapshot: the most recomputation; s >= T - 1: none), every optimiser state (plain SGD,
momentum, per-parameter and scalar log learning rates, Adam, whose reverse of a step waits
for the recompute of the state before it), both HVP modes, both architectures and the
motivating example, on eager, captured and replayed calls; and the store holds s + 3 states."""
import math

import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om
import test_gpu_ckpt as tc

CASES = dict(tc.CASES)
CASES["adam_plr"] = synth.Workload("adam_plr", [4, 6, 3], "tanh", "squared", "fp32", B=5, T=7,
                                   B_outer=4, optimizer="adam", adam_eps=1e-3,
                                   meta_kind=synth.PARAM_LOGLR, loglr_mean=math.log(0.05),
                                   loglr_std=0.1, noise_std=0.1)
CASES["adam_ex_bf16"] = synth.Workload("adam_ex_bf16", [128, 256, 10], "gelu", "ce", "bf16",
                                       B=64, T=6, B_outer=32, optimizer="adam", adam_eps=1e-3,
                                       alpha=1e-3)


def _meta(w, inp, k=1, s=0, mode=0, calls=1):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    loop = native.loop_desc_for(w, mode, ckpt_every=k, ckpt_slots=s)
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


def _slots(w, s):
    """|theta|-sized buffers of the binomial store: s + 3 states of theta, plus m for each
    when kept (momentum, learned learning rate, Adam), v with Adam, and Adam's moment
    cotangents and the two buffers of a deferred step."""
    n = min(s, max(w.T - 1, 1)) + 3
    lr_meta = bool(w.meta_kind & (synth.PARAM_LOGLR | synth.SCALAR_LOGLR))
    if w.optimizer == "adam":
        return n + 2 * n + 4
    return n + (n if (lr_meta or w.momentum != 0) else 0)


def _ss(T):
    return sorted({1, 2, max(T // 2, 1), max(T - 2, 1), T + 3})


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(CASES))
def test_binomial_bit_identical(name):
    w = CASES[name]
    inp = synth.make_inputs(w)
    ref, _ = _meta(w, inp)
    for s in _ss(w.T):
        out, ws = _meta(w, inp, s=s, calls=3 if s == 2 else 1)
        for a, b in zip(out, ref):
            assert np.array_equal(a, b), (name, s)


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["mom_ex_slr", "bf16_deep", "dec32_mom", "adam_plr"])
def test_binomial_reverse_over_reverse(name):
    w = CASES[name]
    inp = synth.make_inputs(w)
    ref, _ = _meta(w, inp, mode=1)
    for s in (1, 3):
        out, _ = _meta(w, inp, s=s, mode=1)
        for a, b in zip(out, ref):
            assert np.array_equal(a, b), (name, s)


@pytest.mark.gpu
def test_binomial_against_oracle():
    w = CASES["mom_plr"]
    inp = synth.make_inputs(w)
    (de, dt, V), _ = _meta(w, inp, s=2)
    ref = om.meta_grad(w, inp)
    assert rel_l2(de, ref["d_eta"]) < 1e-4
    assert rel_l2(dt, ref["d_theta0"]) < 1e-4


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["sgd_ex", "mom_plr", "adam_plr"])
def test_binomial_store_size(name):
    torch, native = need_gpu()
    w = CASES[name]
    mf = native.MixFlow.for_workload(w)
    ws1 = mf.workspace_bytes(native.loop_desc_for(w, 0))
    lr_meta = bool(w.meta_kind & (synth.PARAM_LOGLR | synth.SCALAR_LOGLR))
    full = (w.T + 1) + (w.T if lr_meta else 0)     # momentum alone runs in a buffer at k = 1
    if w.optimizer == "adam":
        full = (w.T + 1) + 2 * w.T + 2
    for s in (1, 2, 4):
        ws = mf.workspace_bytes(native.loop_desc_for(w, 0, ckpt_slots=s))
        assert abs((ws - ws1) - (_slots(w, s) - full) * w.n_params * 4) <= 1024, (name, s)
    mf.close()


@pytest.mark.gpu
def test_binomial_descriptor_checks():
    torch, native = need_gpu()
    w = CASES["sgd_ex"]
    mf = native.MixFlow.for_workload(w)
    for k, s in ((2, 1), (1, -1), (1, 2000)):
        with pytest.raises(native.MixflowError):
            mf.workspace_bytes(native.loop_desc_for(w, 0, ckpt_every=k, ckpt_slots=s))
    mf.close()
