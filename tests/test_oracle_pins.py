"""Pins of the CPU oracle against facts other than itself (no GPU needed).

* P1  central finite differences of V(eta) (the meta-gradient is the exact derivative of
      the unrolled program, Eq. 2 / Proposition 3.1), on several small MLP workloads
      covering every activation, both losses, momentum and all meta-parameter kinds.
* P2  linear model with squared loss: Hessian = kron(X^T W X / (B*O), I_O) in closed form,
      and the whole meta-gradient through the explicit-matrix adjoint recurrence of Eq. 5.
* P3  Hessian symmetry u^T (H v) = v^T (H u) (Schwarz, Eqs. 6-7) and linearity.
* P4  explicit Hessian of a 8->16->1 tanh MLP by finite differences of the gradient, which
      is itself pinned to finite differences of the plain forward loss.
* P5  special cases: alpha = 0 gives zero weight meta-gradient and dV/dtheta_0 = grad V;
      T = 1 gives d eta_b = -(alpha/B) sigma'(eta_b) grad l_b(theta_0) . grad V(theta_1);
      Adam's first step from zero moments is theta_1 = theta_0 - lr g / (|g| + eps) exactly,
      so d eta_b = (sigma'(eta_b)/B) grad l_b . (-lr eps / (|g| + eps)^2 (*) grad V(theta_1)).
* tangent losses dl_b/dtheta . v against finite differences of l_b.
"""
import math

import numpy as np
import pytest

from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

EX, PLR, SLR = synth.EXAMPLE_WEIGHTS, synth.PARAM_LOGLR, synth.SCALAR_LOGLR


def _rel(a, b):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _fd_eta(w, inp, idx, h=1e-5, dirs=None):
    eta = inp.eta.astype(np.float64)
    out = []
    for i in idx:
        e = np.zeros_like(eta)
        e[i] = h
        out.append((om.value(w, inp, eta + e) - om.value(w, inp, eta - e)) / (2 * h))
    return np.array(out)


SMALL = {
    "tiny": synth.WORKLOADS["tiny"],
    "ce_gelu": synth.Workload("ce_gelu", [6, 8, 8, 4], "gelu", "ce", "fp32", B=5, T=3,
                              B_outer=7, alpha=0.3),
    "mom_plr_silu": synth.Workload("mom_plr_silu", [4, 6, 3], "silu", "squared", "fp32", B=6,
                                   T=3, B_outer=5, momentum=0.9, meta_kind=PLR,
                                   loglr_mean=math.log(0.2), loglr_std=0.1),
    "ex_slr_tanh_mom": synth.Workload("ex_slr_tanh_mom", [5, 7, 2], "tanh", "squared", "fp32",
                                      B=4, T=3, B_outer=6, momentum=0.5, meta_kind=EX | SLR,
                                      noise_std=0.1, extra={"scalar_loglr": math.log(0.3)}),
    # Adam inner loops (eps large enough that its derivative terms are not negligible)
    "adam_ex_gelu": synth.Workload("adam_ex_gelu", [5, 6, 3], "gelu", "ce", "fp32", B=4, T=3,
                                   B_outer=5, alpha=0.05, optimizer="adam", adam_eps=1e-3),
    "adam_plr_tanh": synth.Workload("adam_plr_tanh", [4, 5, 2], "tanh", "squared", "fp32", B=5,
                                    T=3, B_outer=4, meta_kind=PLR, optimizer="adam",
                                    beta1=0.8, beta2=0.95, adam_eps=1e-2,
                                    loglr_mean=math.log(0.02), loglr_std=0.1, noise_std=0.1),
}


@pytest.mark.parametrize("name", list(SMALL))
def test_p1_finite_differences(name):
    w = SMALL[name]
    inp = synth.make_inputs(w)
    res = om.meta_grad(w, inp)
    n = w.n_eta
    idx = list(range(n)) if n <= 64 else list(np.random.default_rng(0).choice(n, 40, replace=False))
    fd = _fd_eta(w, inp, idx)
    assert _rel(res["d_eta"][idx], fd) < 1e-6, (res["d_eta"][idx], fd)
    assert np.abs(res["d_eta"][idx]).max() > 1e-6  # non-trivial


def test_p1_theta0_finite_differences():
    w = SMALL["ce_gelu"]
    inp = synth.make_inputs(w)
    res = om.meta_grad(w, inp)
    rng = np.random.default_rng(1)
    for k in rng.choice(w.n_params, 6, replace=False):
        h = 1e-5
        ip = synth.Inputs(inp.theta0.astype(np.float64).copy(), inp.eta, inp.inner_x, inp.inner_y,
                          inp.outer_x, inp.outer_y)
        im = synth.Inputs(inp.theta0.astype(np.float64).copy(), inp.eta, inp.inner_x, inp.inner_y,
                          inp.outer_x, inp.outer_y)
        ip.theta0[k] += h
        im.theta0[k] -= h
        fd = (om.value(w, ip) - om.value(w, im)) / (2 * h)
        assert abs(res["d_theta0"][k] - fd) <= 1e-6 * (abs(fd) + 1e-3)


def _linear_workload(B=6, T=3, din=4, dout=3):
    return synth.Workload("lin", [din, dout], "ident", "squared", "fp32", B=B, T=T, B_outer=5,
                          alpha=0.2, noise_std=0.1)


def _xt(x):
    return np.concatenate([x, np.ones((x.shape[0], 1))], axis=1)


def test_p2_linear_hessian_closed_form():
    w = _linear_workload()
    inp = synth.make_inputs(w)
    ex = 1.0 / (1.0 + np.exp(-inp.eta.astype(np.float64).reshape(w.T, w.B)))
    X = _xt(inp.inner_x[0].astype(np.float64))
    O = w.dims[-1]
    H = np.kron(X.T @ np.diag(ex[0]) @ X / (w.B * O), np.eye(O))
    v = synth.random_direction(w.n_params, 3)
    hv = om.hvp(w, inp.theta0, inp.inner_x[0], inp.inner_y[0], v, ex[0])
    assert _rel(hv, H @ v) < 1e-12


def test_p2_linear_meta_grad_closed_form():
    w = _linear_workload()
    inp = synth.make_inputs(w)
    O, B = w.dims[-1], w.B
    eta = inp.eta.astype(np.float64).reshape(w.T, B)
    wts = 1.0 / (1.0 + np.exp(-eta))
    theta = inp.theta0.astype(np.float64)
    Xs = [_xt(inp.inner_x[t].astype(np.float64)) for t in range(w.T)]
    Ys = [inp.inner_y[t].astype(np.float64) for t in range(w.T)]

    def resid(theta, X, Y):  # f - y, with theta as [(din+1), O]
        return X @ theta.reshape(-1, O) - Y

    thetas = [theta]
    for t in range(w.T):
        r = resid(thetas[-1], Xs[t], Ys[t])
        g = (Xs[t].T @ (wts[t][:, None] * r) / (B * O)).reshape(-1)
        thetas.append(thetas[-1] - w.alpha * g)
    Xo = _xt(inp.outer_x.astype(np.float64))
    ro = resid(thetas[-1], Xo, inp.outer_y.astype(np.float64))
    tb = (Xo.T @ ro / (w.B_outer * O)).reshape(-1)
    d_eta = np.zeros((w.T, B))
    for t in range(w.T - 1, -1, -1):
        X = Xs[t]
        H = np.kron(X.T @ np.diag(wts[t]) @ X / (B * O), np.eye(O))
        r = resid(thetas[t], X, Ys[t])
        for b in range(B):
            grad_lb = np.outer(X[b], r[b]).reshape(-1) / O
            d_eta[t, b] = wts[t, b] * (1 - wts[t, b]) * (-w.alpha / B) * grad_lb @ tb
        tb = tb - w.alpha * H @ tb
    res = om.meta_grad(w, inp)
    assert _rel(res["d_eta"], d_eta.reshape(-1)) < 1e-12
    assert _rel(res["d_theta0"], tb) < 1e-12


def _mlp8():
    return synth.Workload("h8", [8, 16, 1], "tanh", "squared", "fp32", B=10, T=1, B_outer=4,
                          alpha=0.1, noise_std=0.1)


def test_p3_symmetry_and_linearity():
    for w in (_mlp8(), SMALL["ce_gelu"], SMALL["mom_plr_silu"]):
        inp = synth.make_inputs(w)
        u = synth.random_direction(w.n_params, 0, 1).astype(np.float64)
        v = synth.random_direction(w.n_params, 0, 2).astype(np.float64)
        wt = np.linspace(0.2, 1.0, w.B)
        args = (inp.theta0, inp.inner_x[0], inp.inner_y[0])
        hu = om.hvp(w, *args, u, wt)
        hv = om.hvp(w, *args, v, wt)
        assert abs(u @ hv - v @ hu) <= 1e-12 * (abs(u @ hv) + 1e-12)
        huv = om.hvp(w, *args, 2.0 * u - 3.0 * v, wt)
        assert _rel(huv, 2.0 * hu - 3.0 * hv) < 1e-12


def test_p4_explicit_hessian():
    w = _mlp8()
    inp = synth.make_inputs(w)
    P = w.n_params
    assert P == 161
    x, y = inp.inner_x[0], inp.inner_y[0]
    theta = inp.theta0.astype(np.float64)
    # gradient vs finite differences of the plain forward loss
    from oracle import model
    import torch

    def L(th):
        return float(model.weighted_inner_loss(w, torch.from_numpy(th), torch.from_numpy(x.astype(np.float64)),
                                               torch.from_numpy(y.astype(np.float64)),
                                               torch.ones(w.B, dtype=torch.float64)))
    g = om.grad(w, theta, x, y)
    h = 1e-6
    gfd = np.array([(L(theta + h * e) - L(theta - h * e)) / (2 * h) for e in np.eye(P)])
    assert _rel(g, gfd) < 1e-7
    # Hessian column by column from finite differences of the gradient
    h = 1e-5
    Hfd = np.stack([(om.grad(w, theta + h * e, x, y) - om.grad(w, theta - h * e, x, y)) / (2 * h)
                    for e in np.eye(P)], axis=1)
    assert _rel(Hfd, Hfd.T) < 1e-7
    v = synth.random_direction(P, 0, 5)
    assert _rel(om.hvp(w, theta, x, y, v), Hfd @ v) < 1e-7


def test_p5_alpha_zero():
    w = SMALL["tiny"].with_(alpha=0.0)
    inp = synth.make_inputs(w)
    res = om.meta_grad(w, inp)
    assert np.abs(res["d_eta"]).max() == 0.0
    gV = om.grad(w, inp.theta0, inp.outer_x, inp.outer_y)
    assert _rel(res["d_theta0"], gV) < 1e-14


def test_p5_single_step():
    w = SMALL["tiny"].with_(T=1)
    inp = synth.make_inputs(w)
    res = om.meta_grad(w, inp)
    thetas, _ = om.rollout(w, inp)
    gV = om.grad(w, thetas[1].numpy(), inp.outer_x, inp.outer_y)
    eta = inp.eta.astype(np.float64)
    s = 1 / (1 + np.exp(-eta))
    expect = []
    for b in range(w.B):
        glb = om.grad(w, inp.theta0, inp.inner_x[0][b:b + 1], inp.inner_y[0][b:b + 1])
        expect.append(-(w.alpha / w.B) * s[b] * (1 - s[b]) * glb @ gV)
    assert _rel(res["d_eta"], expect) < 1e-12


def test_p5_adam_single_step():
    w = synth.Workload("adam1", [4, 6, 2], "tanh", "squared", "fp32", B=5, T=1, B_outer=4,
                       alpha=0.05, optimizer="adam", adam_eps=1e-2, noise_std=0.1)
    inp = synth.make_inputs(w)
    eta = inp.eta.astype(np.float64)
    s = 1 / (1 + np.exp(-eta))
    g = om.grad(w, inp.theta0, inp.inner_x[0], inp.inner_y[0], s)
    theta1 = inp.theta0.astype(np.float64) - w.alpha * g / (np.abs(g) + w.adam_eps)
    thetas, _ = om.rollout(w, inp)
    assert _rel(thetas[1].numpy(), theta1) < 1e-14
    gV = om.grad(w, theta1, inp.outer_x, inp.outer_y)
    dthdg = -w.alpha * w.adam_eps / (np.abs(g) + w.adam_eps) ** 2
    expect = []
    for b in range(w.B):
        glb = om.grad(w, inp.theta0, inp.inner_x[0][b:b + 1], inp.inner_y[0][b:b + 1])
        expect.append(s[b] * (1 - s[b]) / w.B * glb @ (dthdg * gV))
    res = om.meta_grad(w, inp)
    assert _rel(res["d_eta"], expect) < 1e-12
    assert np.abs(expect).max() > 1e-6


def test_tangent_losses_fd():
    for w in (SMALL["ce_gelu"], _mlp8()):
        inp = synth.make_inputs(w)
        v = synth.random_direction(w.n_params, 0, 7)
        theta = inp.theta0.astype(np.float64)
        x, y = inp.inner_x[0], inp.inner_y[0]
        ld = om.tangent_losses(w, theta, x, y, v)
        h = 1e-6
        fd = (om.per_example_losses(w, theta + h * v, x, y)
              - om.per_example_losses(w, theta - h * v, x, y)) / (2 * h)
        assert _rel(ld, fd) < 1e-7


# ---- decoder-only transformer -------------------------------------------------------------
DEC = {
    "dec_ex": synth.decoder("dec_ex", 16, 2, 32, 2, 32, 8, B=3, T=2, B_outer=2, alpha=0.1),
    "dec_mom_slr": synth.decoder("dec_mom_slr", 16, 4, 24, 1, 24, 6, B=2, T=3, B_outer=2,
                                 momentum=0.9, meta_kind=EX | SLR,
                                 extra={"scalar_loglr": math.log(0.2)}),
}


@pytest.mark.parametrize("name", list(DEC))
def test_p1_decoder_finite_differences(name):
    w = DEC[name]
    inp = synth.make_inputs(w)
    res = om.meta_grad(w, inp)
    idx = list(range(w.n_eta))
    fd = _fd_eta(w, inp, idx)
    assert _rel(res["d_eta"], fd) < 1e-6, (res["d_eta"], fd)
    assert np.abs(res["d_eta"]).max() > 1e-7


def test_decoder_model_properties():
    """Semantics of the oracle's decoder: RoPE keeps norms and makes q.k depend on the
    position difference only; attention is causal; RMSNorm is scale invariant."""
    import torch
    from oracle import model
    g = torch.Generator().manual_seed(0)
    q = torch.randn(1, 1, 1, 8, generator=g, dtype=torch.float64)
    k = torch.randn(1, 1, 1, 8, generator=g, dtype=torch.float64)
    S = 12
    qs = model.rope(q.expand(1, 1, S, 8).clone(), 10000.0)[0, 0]
    ks = model.rope(k.expand(1, 1, S, 8).clone(), 10000.0)[0, 0]
    assert torch.allclose(qs.norm(dim=-1), q.norm().expand(S), rtol=1e-12)
    dots = qs @ ks.T
    for shift in range(S):
        diag = torch.diagonal(dots, offset=shift)
        assert torch.allclose(diag, diag[0].expand_as(diag), rtol=1e-10, atol=1e-12)
    x = torch.randn(4, 8, generator=g, dtype=torch.float64)
    gain = torch.rand(8, generator=g, dtype=torch.float64) + 0.5
    assert torch.allclose(model.rmsnorm(3.7 * x, gain, 0.0), model.rmsnorm(x, gain, 0.0))
    w = DEC["dec_ex"]
    inp = synth.make_inputs(w)
    theta = torch.from_numpy(inp.theta0.astype(np.float64))
    ids = torch.from_numpy(inp.inner_x[0].astype(np.int64))
    ids2 = ids.clone()
    ids2[:, 5:] = (ids2[:, 5:] + 7) % w.vocab           # change the future only
    f1 = model.decoder_logits(w, theta, ids)
    f2 = model.decoder_logits(w, theta, ids2)
    assert torch.equal(f1[:, :5], f2[:, :5])
    assert not torch.allclose(f1[:, 5:], f2[:, 5:])


def test_zipf_ids_law():
    """Token ids follow the truncated Zipf(1.1) law (inverse-CDF sampling)."""
    g = np.random.default_rng(3)
    V = 50
    ids = synth.zipf_ids(g, (200000,), V, 1.1)
    assert ids.min() >= 0 and ids.max() < V
    p = np.arange(1, V + 1, dtype=np.float64) ** -1.1
    p /= p.sum()
    emp = np.bincount(ids, minlength=V) / ids.size
    assert np.abs(emp - p).max() < 4e-3


# ---- motivating example of Section 3 (Eq. 8): theta_0 meta-gradient through the recursion
TOY = synth.toy("toy_tiny", 4, 3, 3, precision="fp32")


def test_toy_theta0_finite_differences():
    """Every component of dV/dtheta_0 (MAML-style meta-parameter) against central finite
    differences of the unrolled program, through the 3-step recursion."""
    w = TOY
    inp = synth.make_inputs(w)
    res = om.meta_grad(w, inp)
    h = 1e-6
    fd = []
    for k in range(w.n_params):
        th_p = inp.theta0.astype(np.float64).copy()
        th_m = th_p.copy()
        th_p[k] += h
        th_m[k] -= h
        vp = om.value(w, synth.Inputs(th_p, inp.eta, inp.inner_x, inp.inner_y, inp.outer_x, inp.outer_y))
        vm = om.value(w, synth.Inputs(th_m, inp.eta, inp.inner_x, inp.inner_y, inp.outer_x, inp.outer_y))
        fd.append((vp - vm) / (2 * h))
    assert _rel(res["d_theta0"], fd) < 1e-6
    assert np.abs(res["d_theta0"]).max() > 1e-3


def test_toy_zero_steps_is_linear_closed_form():
    """With M = 0 the example is a linear model with L = mean((x W - y)^2): gradient
    (2/(B O)) X^T (X W - Y), Hessian (2/(B O)) X^T X (x) I, adjoint recurrence of Eq. 5."""
    w = synth.toy("toy_lin", 5, 4, 0, T=3, precision="fp32")
    inp = synth.make_inputs(w)
    D, B = w.dims[0], w.B
    W = inp.theta0.astype(np.float64).reshape(D, D)
    Xs = [inp.inner_x[t].astype(np.float64) for t in range(w.T)]
    Ys = [inp.inner_y[t].astype(np.float64) for t in range(w.T)]
    Ws = [W]
    for t in range(w.T):
        g = 2.0 / (B * D) * Xs[t].T @ (Xs[t] @ Ws[-1] - Ys[t])
        Ws.append(Ws[-1] - w.alpha * g)
    Xo, Yo = inp.outer_x.astype(np.float64), inp.outer_y.astype(np.float64)
    tb = (2.0 / (w.B_outer * D) * Xo.T @ (Xo @ Ws[-1] - Yo)).reshape(-1)
    for t in range(w.T - 1, -1, -1):
        H = np.kron(2.0 / (B * D) * Xs[t].T @ Xs[t], np.eye(D))
        tb = tb - w.alpha * H @ tb
    res = om.meta_grad(w, inp)
    assert _rel(res["d_theta0"], tb) < 1e-12


def test_oracle_matches_its_golden_values():
    """The oracle reproduces the values tests/golden/make_oracle_golden.py wrote with it (a
    regression anchor for its own arithmetic; the paper prints no worked values)."""
    import json
    import os
    import sys
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    sys.path.insert(0, here)
    import make_oracle_golden as g
    with open(os.path.join(here, "oracle_golden.json")) as f:
        gold = json.load(f)
    assert set(gold) == set(g.CASES)
    for name, w in g.CASES.items():
        r = om.meta_grad(w, synth.make_inputs(w))
        assert abs(r["V"] - gold[name]["V"]) <= 1e-12 * abs(gold[name]["V"])
        for key in ("d_eta", "d_theta0"):
            ref = np.array(gold[name][key])
            if ref.size:
                assert _rel(r[key], ref) < 1e-12, (name, key)


def _decoder_losses_by_loops(w, theta, ids):
    """The decoder's per-sequence next-token losses written out position by position in plain
    Python floats from the model's definition: embedding lookup; per block a pre-RMSNorm
    (x / sqrt(mean x^2 + eps), times the gain), the q | k | v projection with heads in
    contiguous column groups, RoPE as a rotation of each coordinate pair (j, j + dh/2) by the
    angle s * base^(-2j/dh), causal attention with scores scaled by 1/sqrt(dh), the output
    projection and a residual add, then a pre-RMSNorm GELU MLP and a residual add; a final
    RMSNorm, the untied head, and the cross-entropy of token s+1 given tokens 0..s, averaged
    over the S positions."""
    d, H, F, V, eps = w.d_model, w.n_heads, w.d_ff, w.vocab, w.rms_eps
    dh, half = d // H, d // H // 2
    th = [float(v) for v in theta]
    pos = [0]

    def take(rows, cols=None):
        o = pos[0]
        if cols is None:
            pos[0] += rows
            return th[o:o + rows]
        pos[0] += rows * cols
        return [th[o + r * cols:o + (r + 1) * cols] for r in range(rows)]

    def norm(x, g):
        r = 1.0 / math.sqrt(sum(v * v for v in x) / len(x) + eps)
        return [gi * xi * r for gi, xi in zip(g, x)]

    def matvec(x, W):
        return [sum(x[r] * W[r][c] for r in range(len(x))) for c in range(len(W[0]))]

    def rotate(vec, s):
        out = list(vec)
        for j in range(half):
            a = s * w.rope_base ** (-2.0 * j / dh)
            x1, x2 = vec[j], vec[j + half]
            out[j] = x1 * math.cos(a) - x2 * math.sin(a)
            out[j + half] = x1 * math.sin(a) + x2 * math.cos(a)
        return out

    E = take(V, d)
    blocks = []
    for _ in range(w.n_blocks):
        blocks.append((take(d), take(d, 3 * d), take(d, d), take(d), take(d, F), take(F, d)))
    gf, Wh = take(d), take(d, V)
    assert pos[0] == len(th)
    out = []
    for seq in ids:
        S = len(seq) - 1
        xs = [list(E[int(seq[s])]) for s in range(S)]
        for g1, Wqkv, Wo, g2, W1, W2 in blocks:
            qkv = [matvec(norm(x, g1), Wqkv) for x in xs]
            att = [[0.0] * d for _ in range(S)]
            for h in range(H):
                q = [rotate(r[h * dh:(h + 1) * dh], s) for s, r in enumerate(qkv)]
                k = [rotate(r[d + h * dh:d + (h + 1) * dh], s) for s, r in enumerate(qkv)]
                v = [r[2 * d + h * dh:2 * d + (h + 1) * dh] for r in qkv]
                for i in range(S):
                    sc = [sum(a * b for a, b in zip(q[i], k[j])) / math.sqrt(dh)
                          for j in range(i + 1)]
                    mx = max(sc)
                    p = [math.exp(c - mx) for c in sc]
                    z = sum(p)
                    for c in range(dh):
                        att[i][h * dh + c] = sum(p[j] / z * v[j][c] for j in range(i + 1))
            xs = [[a + b for a, b in zip(x, matvec(o, Wo))] for x, o in zip(xs, att)]
            for i in range(S):
                hid = matvec(norm(xs[i], g2), W1)
                hid = [0.5 * a * (1.0 + math.erf(a / math.sqrt(2.0))) for a in hid]
                xs[i] = [a + b for a, b in zip(xs[i], matvec(hid, W2))]
        ce = 0.0
        for s in range(S):
            f = matvec(norm(xs[s], gf), Wh)
            mx = max(f)
            ce += mx + math.log(sum(math.exp(c - mx) for c in f)) - f[int(seq[s + 1])]
        out.append(ce / S)
    return np.array(out)


def test_decoder_forward_by_scalar_loops():
    """The oracle's decoder losses against the model written out position by position, with
    random gains so that every gain, the attention scale, the RoPE pairing and the
    next-token shift are exercised (a second route from the definition)."""
    import torch
    from oracle import model
    w = synth.decoder("dec_loops", 8, 2, 12, 2, 11, 5, B=3, T=1, B_outer=1)
    g = np.random.default_rng(11)
    theta = np.concatenate([g.uniform(0.5, 1.5, n) if name.startswith("g")
                            else 0.4 * g.standard_normal(n)
                            for name, n in w.decoder_layout()])
    ids = synth.zipf_ids(g, (3, 6), w.vocab, 1.1)
    ref = _decoder_losses_by_loops(w, theta, ids)
    got = model.decoder_losses(w, torch.from_numpy(theta), torch.from_numpy(ids.astype(np.int64)))
    assert _rel(got.numpy(), ref) < 1e-13, (got, ref)
    assert ref.std() > 1e-3
