"""Oracle pins by an independent route: symbolic derivatives and 60-digit arithmetic.

Each small workload is written out again from its definition (the inner model, the
per-example losses, the weighted inner loss L_t of Eq. 1, the momentum-SGD update of Eq. 2,
the outer loss V), and sympy differentiates the inner loss symbolically.  The unrolled
program then runs in mpmath at 60 significant digits, and the meta-gradient dV/d(eta,
theta_0) is taken by central differences with step 1e-20, which is exact to far below
float64 resolution.  None of this touches the oracle's autograd tape, its per-step
checkpointing or its reverse-over-reverse sweep (Algorithm 1), so a wrong term, sign, index
or transposition there fails here at the 1e-10 level, 10^4 times tighter than float64
finite differences allow.
"""
import math

import numpy as np
import pytest

from paper_2505_00793_gb300 import synth
from oracle import metagrad as om

sp = pytest.importorskip("sympy")
mp = pytest.importorskip("mpmath")

EX, PLR, SLR = synth.EXAMPLE_WEIGHTS, synth.PARAM_LOGLR, synth.SCALAR_LOGLR
DPS = 60
H = "1e-20"


def _act(name, z):
    if name == "ident":
        return z
    if name == "tanh":
        return sp.tanh(z)
    if name == "gelu":
        return z / 2 * (1 + sp.erf(z / sp.sqrt(2)))
    if name == "silu":
        return z / (1 + sp.exp(-z))
    raise ValueError(name)


def _example_losses(w, th, X, Y):
    """Per-example losses of an MLP on symbolic inputs X [B][din] and targets Y [B][dout]
    (for cross-entropy Y is the one-hot label)."""
    layers, o = [], 0
    for i in range(w.n_layers):
        din, dout = w.dims[i], w.dims[i + 1]
        W = [[th[o + r * dout + c] for c in range(dout)] for r in range(din)]
        o += din * dout
        b = None
        if w.has_bias:
            b = th[o:o + dout]
            o += dout
        layers.append((W, b))
    assert o == w.n_params
    out = []
    for xb, yb in zip(X, Y):
        h = list(xb)
        for i, (W, b) in enumerate(layers):
            z = [sum(h[r] * W[r][c] for r in range(len(h))) + (b[c] if b is not None else 0)
                 for c in range(len(W[0]))]
            h = [_act(w.act, v) for v in z] if i + 1 < len(layers) else z
        n = len(h)
        if w.loss == "squared":
            out.append(sum((h[c] - yb[c]) ** 2 for c in range(n)) / (2 * n))
        elif w.loss == "ce":
            out.append(sp.log(sum(sp.exp(v) for v in h)) - sum(yb[c] * h[c] for c in range(n)))
        elif w.loss == "chain_mse":
            ys = h
            for i in range(1, w.extra["chain_steps"] + 1):
                ys = [i * (2 + sp.sin(v)) ** sp.cos(v) for v in ys]
            out.append(sum((ys[c] - yb[c]) ** 2 for c in range(n)) / n)
        else:
            raise ValueError(w.loss)
    return out


class Unrolled:
    """The inner loop and the outer loss of workload w at DPS digits."""

    def __init__(self, w, inp):
        self.w, P, B = w, w.n_params, w.B
        din, dout = w.dims[0], w.dims[-1]
        th = sp.symbols(f"th0:{P}")
        c = sp.symbols(f"c0:{B}")
        X = [sp.symbols(f"x{b}_0:{din}") for b in range(B)]
        Y = [sp.symbols(f"y{b}_0:{dout}") for b in range(B)]
        L = sum(cb * lb for cb, lb in zip(c, _example_losses(w, th, X, Y))) / B
        grad = [sp.diff(L, v) for v in th]
        flat = lambda rows: [v for r in rows for v in r]
        args = list(th) + list(c) + flat(X) + flat(Y)
        self.grad = sp.lambdify(args, grad, modules="mpmath", cse=True)
        self.losses = sp.lambdify(list(th) + flat(X) + flat(Y), _example_losses(w, th, X, Y),
                                  modules="mpmath", cse=True)
        Bo = w.B_outer
        Xo = [sp.symbols(f"u{b}_0:{din}") for b in range(Bo)]
        Yo = [sp.symbols(f"v{b}_0:{dout}") for b in range(Bo)]
        V = sum(_example_losses(w, th, Xo, Yo)) / Bo
        self.outer = sp.lambdify(list(th) + flat(Xo) + flat(Yo), V, modules="mpmath", cse=True)
        mpf = lambda a: [mp.mpf(float(v)) for v in np.asarray(a, np.float64).reshape(-1)]
        self.x = [mpf(inp.inner_x[t]) for t in range(w.T)]
        self.y = [self._targets(inp.inner_y[t]) for t in range(w.T)]
        self.ox, self.oy = mpf(inp.outer_x), self._targets(inp.outer_y)
        self.theta0 = mpf(inp.theta0)
        self.eta = mpf(inp.eta)

    def _targets(self, y):
        if self.w.loss == "ce":
            n = self.w.dims[-1]
            return [mp.mpf(1 if k == int(lab) else 0) for lab in np.asarray(y).reshape(-1)
                    for k in range(n)]
        return [mp.mpf(float(v)) for v in np.asarray(y, np.float64).reshape(-1)]

    def value(self, eta, theta0):
        w, P, B = self.w, self.w.n_params, self.w.B
        o, ex, lr = 0, None, [mp.mpf(w.alpha)] * P
        if w.meta_kind & EX:
            ex = eta[:w.T * B]
            o = w.T * B
        if w.meta_kind & PLR:
            lr = [mp.exp(v) for v in eta[o:o + P]]
            o += P
        if w.meta_kind & SLR:
            lr = [mp.exp(eta[o])] * P
        th, m, v = list(theta0), [mp.mpf(0)] * P, [mp.mpf(0)] * P
        for t in range(w.T):
            c = [1 / (1 + mp.exp(-v)) for v in ex[t * B:(t + 1) * B]] if ex else [mp.mpf(1)] * B
            g = self.grad(*th, *c, *self.x[t], *self.y[t])
            if w.optimizer == "adam":   # Kingma & Ba with bias correction
                b1, b2 = mp.mpf(w.beta1), mp.mpf(w.beta2)
                m = [b1 * mi + (1 - b1) * gi for mi, gi in zip(m, g)]
                v = [b2 * vi + (1 - b2) * gi * gi for vi, gi in zip(v, g)]
                c1, c2 = 1 - b1 ** (t + 1), 1 - b2 ** (t + 1)
                th = [ti - li * (mi / c1) / (mp.sqrt(vi / c2) + mp.mpf(w.adam_eps))
                      for ti, li, mi, vi in zip(th, lr, m, v)]
            else:
                m = [w.momentum * mi + gi for mi, gi in zip(m, g)]
                th = [ti - li * mi for ti, li, mi in zip(th, lr, m)]
        return self.outer(*th, *self.ox, *self.oy)

    def meta_grad(self):
        h = mp.mpf(H)
        def d(vec, i, which):
            vp, vm = list(vec), list(vec)
            vp[i] += h
            vm[i] -= h
            if which == "eta":
                return (self.value(vp, self.theta0) - self.value(vm, self.theta0)) / (2 * h)
            return (self.value(self.eta, vp) - self.value(self.eta, vm)) / (2 * h)
        de = [d(self.eta, i, "eta") for i in range(len(self.eta))]
        dt = [d(self.theta0, i, "theta") for i in range(len(self.theta0))]
        return (np.array([float(v) for v in de]), np.array([float(v) for v in dt]),
                float(self.value(self.eta, self.theta0)))


CASES = {
    # tanh, bias, momentum, per-example weight logits and per-parameter log learning rates
    "tanh_mom_ex_plr": synth.Workload("s1", [2, 3, 2], "tanh", "squared", "fp32", B=2, T=2,
                                      B_outer=3, momentum=0.9, meta_kind=EX | PLR,
                                      loglr_mean=math.log(0.3), loglr_std=0.2, noise_std=0.1,
                                      eta_std=1.0),
    # GELU, cross-entropy, momentum, weight logits and a scalar log learning rate
    "gelu_ce_ex_slr": synth.Workload("s2", [3, 3, 3], "gelu", "ce", "fp32", B=3, T=2, B_outer=2,
                                     momentum=0.5, meta_kind=EX | SLR, eta_std=1.0,
                                     extra={"scalar_loglr": math.log(0.5)}),
    # SiLU, plain SGD over three steps, weight logits
    "silu_sgd_ex": synth.Workload("s3", [2, 2, 1], "silu", "squared", "fp32", B=2, T=3,
                                  B_outer=2, alpha=0.4, noise_std=0.2, eta_std=1.0),
    # the motivating example of Section 3 (Eq. 8), M = 2, theta_0 the meta-parameter
    "toy_chain": synth.toy("s4", 2, 2, 2, T=2, precision="fp32", init_std=0.7),
    # Adam inner loops: weight logits with cross-entropy, per-parameter log learning rates
    "adam_ex_ce": synth.Workload("s5", [3, 3, 3], "tanh", "ce", "fp32", B=3, T=3, B_outer=2,
                                 alpha=0.05, optimizer="adam", adam_eps=1e-3, eta_std=1.0),
    "adam_plr": synth.Workload("s6", [2, 3, 2], "silu", "squared", "fp32", B=2, T=2, B_outer=3,
                               meta_kind=PLR, optimizer="adam", beta1=0.8, beta2=0.95,
                               adam_eps=1e-2, loglr_mean=math.log(0.03), loglr_std=0.2,
                               noise_std=0.1),
}


@pytest.mark.parametrize("name", list(CASES))
def test_meta_grad_symbolic(name):
    w = CASES[name]
    inp = synth.make_inputs(w)
    with mp.workdps(DPS):
        de, dt, V = Unrolled(w, inp).meta_grad()
    ref = om.meta_grad(w, inp)
    assert abs(ref["V"] - V) <= 1e-13 * abs(V)
    if de.size:
        scale_e = np.abs(de).max()
        assert np.abs(ref["d_eta"] - de).max() <= 1e-10 * scale_e, (ref["d_eta"], de)
        assert scale_e > 1e-6
    assert np.abs(ref["d_theta0"] - dt).max() <= 1e-10 * np.abs(dt).max(), (ref["d_theta0"], dt)
    assert np.abs(dt).max() > 1e-6


@pytest.mark.parametrize("name", ["tanh_mom_ex_plr", "gelu_ce_ex_slr", "toy_chain"])
def test_hvp_and_tangent_losses_symbolic(name):
    """H v as the derivative of the symbolic gradient along v (Eq. 6), and the per-example
    tangent losses dl_b/dtheta . v (the mixed term of Eq. 7), at 60 digits."""
    w = CASES[name]
    inp = synth.make_inputs(w)
    v = synth.random_direction(w.n_params, 9, 3).astype(np.float64)
    wt = np.linspace(0.3, 0.9, w.B)
    with mp.workdps(DPS):
        u = Unrolled(w, inp)
        h = mp.mpf(H)
        vm = [mp.mpf(float(a)) for a in v]
        cw = [mp.mpf(float(a)) for a in wt]
        tp = [a + h * b for a, b in zip(u.theta0, vm)]
        tm = [a - h * b for a, b in zip(u.theta0, vm)]
        gp = u.grad(*tp, *cw, *u.x[0], *u.y[0])
        gm = u.grad(*tm, *cw, *u.x[0], *u.y[0])
        hv = np.array([float((a - b) / (2 * h)) for a, b in zip(gp, gm)])
        lp = u.losses(*tp, *u.x[0], *u.y[0])
        lm = u.losses(*tm, *u.x[0], *u.y[0])
        ld = np.array([float((a - b) / (2 * h)) for a, b in zip(lp, lm)])
    x, y = inp.inner_x[0], inp.inner_y[0]
    ref_hv = om.hvp(w, inp.theta0, x, y, v, wt)
    assert np.abs(ref_hv - hv).max() <= 1e-11 * np.abs(hv).max()
    ref_ld = om.tangent_losses(w, inp.theta0, x, y, v)
    assert np.abs(ref_ld - ld).max() <= 1e-11 * np.abs(ld).max()
