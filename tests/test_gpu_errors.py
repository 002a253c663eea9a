"""Error paths and degenerate sizes on the GPU.

Failures are made on the host or through inputs the kernels check themselves: invalid loop
descriptors, the host-side fault injector (a failed workspace allocation, a device wait
reported as expired), device waits that really expire under a zero wait limit, a NaN in theta_0 (caught by the update kernel's finiteness check),
and out-of-range class labels and token ids (bounds-checked, clamped and reported by the
loss and embedding kernels).  After every error the handle stays usable and the next call
gives the same result as a fresh handle.  Degenerate sizes (one example, one inner step,
one-row GEMMs, a single attention tile) are checked against the oracle."""
import numpy as np
import pytest

from gpu_util import need_gpu, rel_l2
from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, PLR, SLR = synth.EXAMPLE_WEIGHTS, synth.PARAM_LOGLR, synth.SCALAR_LOGLR
INVALID, OOM, NONFINITE, TIMEOUT = 1, 3, 5, 6


def _buffers(torch, w):
    return (torch.full((w.n_eta,), float("nan"), device="cuda"),
            torch.full((w.n_params,), float("nan"), device="cuda"),
            torch.full((1,), float("nan"), device="cuda"))


def _call(mf, native, w, d, bufs, sync=True):
    d_eta, d_th, V = bufs
    mf.meta_grad(native.loop_desc_for(w), d["theta0"], d["eta"], d["inner_x"], d["inner_y"],
                 d["outer_x"], d["outer_y"], d_eta, d_th, V)
    if sync:
        mf.sync()
    return d_eta.cpu().numpy().copy(), d_th.cpu().numpy().copy()


def _fresh(w, inp):
    torch, native = need_gpu()
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    out = _call(mf, native, w, d, _buffers(torch, w))
    mf.close()
    return out


@pytest.mark.gpu
def test_invalid_loop_descriptors():
    torch, native = need_gpu()
    w = synth.WORKLOADS["tiny"]
    mf = native.MixFlow.for_workload(w)
    for field, value in (("T", 0), ("B", 0), ("B_outer", 0), ("meta_kind", 8),
                         ("meta_kind", PLR | SLR), ("momentum", 1.0), ("momentum", -0.5),
                         ("hvp_mode", 7), ("ckpt_every", -1), ("optimizer", 2)):
        loop = native.loop_desc_for(w)
        setattr(loop, field, value)
        with pytest.raises(native.MixflowError) as e:
            mf.workspace_bytes(loop)
        assert e.value.status == INVALID, (field, value)
    mf.close()


@pytest.mark.gpu
def test_injected_allocation_failure_then_recovery():
    torch, native = need_gpu()
    w = synth.WORKLOADS["tiny"]
    inp = synth.make_inputs(w)
    ref = _fresh(w, inp)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    bufs = _buffers(torch, w)
    mf.inject_fault(1)
    with pytest.raises(native.MixflowError) as e:
        _call(mf, native, w, d, bufs)
    assert e.value.status == OOM
    out = _call(mf, native, w, d, bufs)
    mf.close()
    assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


@pytest.mark.gpu
def test_injected_timeout_then_recovery():
    torch, native = need_gpu()
    w = synth.WORKLOADS["tiny"]
    inp = synth.make_inputs(w)
    ref = _fresh(w, inp)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    bufs = _buffers(torch, w)
    _call(mf, native, w, d, bufs, sync=False)
    mf.inject_fault(2)
    with pytest.raises(native.MixflowError) as e:
        mf.sync()
    assert e.value.status == TIMEOUT
    out = _call(mf, native, w, d, bufs)
    mf.close()
    assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


@pytest.mark.gpu
@pytest.mark.parametrize("persistent", [False, True])
def test_device_wait_expiry_then_recovery(persistent):
    """A real device-side timeout, no injection: with MF_OPT_WAIT_LIMIT_US = 0 the
    tensor-core GEMMs' MMA issuer and epilogue give up at their first wait that does not
    complete at once, record the timeout, let the loads and MMAs they issued complete and
    end.  mf_sync reports MF_ERR_TIMEOUT (no trap; the context stays usable), and with the
    default limit back the same handle reproduces a fresh handle's meta-gradient bit for bit.
    The persistent variant sends every GEMM of more than 128 rows (the weight products here)
    through the persistent CTA-pair kernel."""
    torch, native = need_gpu()
    w = synth.Workload("wait_bf16", [128, 256, 136, 10], "gelu", "ce", "bf16", B=64, T=2,
                       B_outer=64, alpha=0.05)
    inp = synth.make_inputs(w)
    ref = _fresh(w, inp)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    bufs = _buffers(torch, w)
    try:
        mf.set_option(native.MF_OPT_WAIT_LIMIT_US, 0)
        if persistent:
            mf.set_option(native.MF_OPT_GEMM_2SM, 2)
            mf.set_option(native.MF_OPT_GEMM_PERSISTENT, 1)
        with pytest.raises(native.MixflowError) as e:
            _call(mf, native, w, d, bufs)
        assert e.value.status == TIMEOUT
    finally:
        mf.set_option(native.MF_OPT_WAIT_LIMIT_US, 2000000)
        mf.set_option(native.MF_OPT_GEMM_PERSISTENT, 2)   # the default
        mf.set_option(native.MF_OPT_GEMM_2SM, 1)
    out = _call(mf, native, w, d, bufs)
    mf.close()
    assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["tiny", "wide_bf16"])
def test_nonfinite_theta_is_reported(name):
    torch, native = need_gpu()
    w = synth.WORKLOADS["tiny"] if name == "tiny" else synth.Workload(
        "e_wide", [64, 128, 10], "gelu", "ce", "bf16", B=32, T=2, B_outer=16, alpha=0.05)
    inp = synth.make_inputs(w)
    ref = _fresh(w, inp)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    bad = dict(d)
    bad["theta0"] = d["theta0"].clone()
    bad["theta0"][3] = float("nan")
    bufs = _buffers(torch, w)
    with pytest.raises(native.MixflowError) as e:
        _call(mf, native, w, bad, bufs)
    assert e.value.status == NONFINITE
    out = _call(mf, native, w, d, bufs)
    mf.close()
    assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


@pytest.mark.gpu
def test_out_of_range_class_label_is_reported():
    torch, native = need_gpu()
    w = synth.Workload("e_ce", [6, 8, 4], "tanh", "ce", "fp32", B=5, T=2, B_outer=3, alpha=0.2)
    inp = synth.make_inputs(w)
    ref = _fresh(w, inp)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    bad = dict(d)
    bad["inner_y"] = d["inner_y"].clone()
    bad["inner_y"].view(-1)[2] = 4          # classes are 0..3
    bufs = _buffers(torch, w)
    with pytest.raises(native.MixflowError) as e:
        _call(mf, native, w, bad, bufs)
    assert e.value.status == INVALID
    out = _call(mf, native, w, d, bufs)
    mf.close()
    assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


@pytest.mark.gpu
def test_out_of_range_token_id_is_reported():
    torch, native = need_gpu()
    w = synth.decoder("e_dec", 64, 1, 128, 1, 200, 64, B=2, T=1, B_outer=2, alpha=1e-2)
    inp = synth.make_inputs(w)
    ref = _fresh(w, inp)
    mf = native.MixFlow.for_workload(w)
    d = native.to_device_inputs(w, inp)
    bad = dict(d)
    bad["inner_x"] = d["inner_x"].clone()
    bad["inner_x"].view(-1)[7] = w.vocab    # ids are 0..V-1
    bad["inner_y"] = bad["inner_x"]
    bufs = _buffers(torch, w)
    with pytest.raises(native.MixflowError) as e:
        _call(mf, native, w, bad, bufs)
    assert e.value.status == INVALID
    out = _call(mf, native, w, d, bufs)
    mf.close()
    assert np.array_equal(out[0], ref[0]) and np.array_equal(out[1], ref[1])


DEGENERATE = {
    # one example, one inner step, one outer example; one-row GEMMs on the bf16 path
    "mlp32_b1_t1": (synth.Workload("g1", [5, 7, 3], "tanh", "squared", "fp32", B=1, T=1,
                                   B_outer=1, alpha=0.3, noise_std=0.1), 1e-4),
    "mlp16_b1_t1": (synth.Workload("g2", [64, 128, 10], "gelu", "ce", "bf16", B=1, T=1,
                                   B_outer=1, alpha=0.05), 2e-2),
    "mlp16_b1_t3_mom_plr": (synth.Workload("g3", [64, 96, 8], "silu", "squared", "bf16", B=1,
                                           T=3, B_outer=2, momentum=0.9, meta_kind=PLR,
                                           loglr_mean=np.log(1e-2), loglr_std=0.1), 2e-2),
    # a single sequence of a single 64-token attention tile (fused attention)
    "dec16_b1_t1": (synth.decoder("g4", 64, 1, 128, 1, 200, 64, B=1, T=1, B_outer=1,
                                  alpha=1e-2), 2e-2),
}


@pytest.mark.gpu
@pytest.mark.parametrize("name", list(DEGENERATE))
def test_degenerate_sizes(name):
    w, tol = DEGENERATE[name]
    inp = synth.make_inputs(w)
    ref = om.meta_grad(w, inp)
    de, dt = _fresh(w, inp)
    assert np.isfinite(de).all() and np.isfinite(dt).all()
    assert rel_l2(de, ref["d_eta"]) < tol
    assert rel_l2(dt, ref["d_theta0"]) < tol
