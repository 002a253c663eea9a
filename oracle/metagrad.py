"""Oracle meta-gradient: Algorithm 1 (standard Truncated-BPTT) in float64 on the CPU.

Test infrastructure only (see ``oracle/__init__.py``).

Inner loop (Eq. 2; the optimiser state upsilon is the momentum, or Adam's two moments):
    SGD / heavy ball:  m_{t+1} = mu * m_t + g_t,   theta_{t+1} = theta_t - lr (*) m_{t+1}
    Adam (Kingma & Ba, with bias correction; the optimiser of Section 5's inner loops):
        m_{t+1} = b1 m_t + (1 - b1) g_t,   v_{t+1} = b2 v_t + (1 - b2) g_t^2
        theta_{t+1} = theta_t - lr (*) (m_{t+1} / c1) / (sqrt(v_{t+1} / c2) + eps),
        c1 = 1 - b1^(t+1),  c2 = 1 - b2^(t+1)
with g_t = grad L_t(theta_t), zero initial state, lr = alpha, or exp(eta_lr) per parameter,
or exp(eta_s) for a scalar log-lr, and
L_t = (1/B) sum_b sigmoid(eta_{t,b}) l_b when per-example weight logits are meta-parameters.
Outer loss V(theta_T) is the unweighted mean loss on the held-out batch.

``meta_grad`` differentiates V through the unrolled loop by reverse mode at both levels
(Algorithm 1): the inner gradient is recorded with ``create_graph`` so that the outer
backward pass runs reverse-over-reverse through it.  Per-inner-step checkpointing
(Section 4): the rollout keeps (theta_t, m_t); the backward sweep rebuilds the tape of one
step at a time and pulls the cotangent (theta_bar_{t+1}, m_bar_{t+1}) through it.

Index convention (the algorithm listings mix 0- and 1-based ranges): steps t = 0..T-1, and
the weight logits eta_{t,.} act at step t.
"""
from __future__ import annotations

import numpy as np
import torch

from . import model

F64 = torch.float64
EXAMPLE_WEIGHTS, PARAM_LOGLR, SCALAR_LOGLR = 1, 2, 4


def t64(a) -> torch.Tensor:
    if isinstance(a, torch.Tensor):
        return a.detach().to(F64) if a.is_floating_point() else a.detach()
    a = np.asarray(a)
    if a.dtype.kind in "iu":
        return torch.from_numpy(a.astype(np.int64))
    return torch.from_numpy(a.astype(np.float64))


def split_eta(w, eta: torch.Tensor):
    """Split the flat meta-parameter vector: [T*B example logits][P log-lrs][1 scalar log-lr]."""
    o, ex, plr, slr = 0, None, None, None
    if w.meta_kind & EXAMPLE_WEIGHTS:
        ex = eta[o:o + w.T * w.B].reshape(w.T, w.B)
        o += w.T * w.B
    if w.meta_kind & PARAM_LOGLR:
        plr = eta[o:o + w.n_params]
        o += w.n_params
    if w.meta_kind & SCALAR_LOGLR:
        slr = eta[o]
        o += 1
    return ex, plr, slr


def learning_rate(w, eta: torch.Tensor):
    _, plr, slr = split_eta(w, eta)
    if plr is not None:
        return torch.exp(plr)
    if slr is not None:
        return torch.exp(slr)
    return torch.tensor(w.alpha, dtype=F64)


def example_weights(w, eta: torch.Tensor, t: int):
    ex, _, _ = split_eta(w, eta)
    if ex is None:
        return torch.ones(w.B, dtype=F64)
    return torch.sigmoid(ex[t])


def _safe_sqrt(v):
    """sqrt(v) whose derivative at v = 0 is taken as 0.  v_{t+1} = 0 only where every
    gradient so far was exactly 0, and there m_{t+1} = 0 and dv/dg = 2 (1 - b2) g = 0 too, so
    every path through that derivative is multiplied by 0 (the limit of the product)."""
    pos = v > 0
    return torch.where(pos, torch.sqrt(torch.where(pos, v, torch.ones_like(v))),
                       torch.zeros_like(v))


def n_state(w) -> int:
    """Number of optimiser state tensors: m for SGD / heavy ball, (m, v) for Adam."""
    return 2 if getattr(w, "optimizer", "sgd") == "adam" else 1


def _step(w, theta, state, eta, x, y, t, create_graph):
    """One inner update Phi(theta_t, upsilon_t, eta, x_t) -> (theta_{t+1}, upsilon_{t+1})."""
    L = model.weighted_inner_loss(w, theta, x, y, example_weights(w, eta, t))
    (g,) = torch.autograd.grad(L, theta, create_graph=create_graph)
    lr = learning_rate(w, eta)
    if n_state(w) == 2:
        m, v = state
        m_next = w.beta1 * m + (1.0 - w.beta1) * g
        v_next = w.beta2 * v + (1.0 - w.beta2) * g * g
        c1 = 1.0 - w.beta1 ** (t + 1)
        c2 = 1.0 - w.beta2 ** (t + 1)
        theta_next = theta - lr * (m_next / c1) / (_safe_sqrt(v_next / c2) + w.adam_eps)
        return theta_next, (m_next, v_next)
    (m,) = state
    m_next = w.momentum * m + g
    theta_next = theta - lr * m_next
    return theta_next, (m_next,)


def rollout(w, inp, eta=None):
    """Inner rollout storing every (theta_t, upsilon_t), t = 0..T.  Returns (thetas, states)
    with states[t] a tuple of state tensors."""
    eta = t64(inp.eta if eta is None else eta)
    X, Y = t64(inp.inner_x), t64(inp.inner_y)
    theta = t64(inp.theta0)
    state = tuple(torch.zeros_like(theta) for _ in range(n_state(w)))
    thetas, states = [theta], [state]
    for t in range(w.T):
        th = theta.clone().requires_grad_(True)
        with torch.enable_grad():
            tn, sn = _step(w, th, state, eta, X[t], Y[t], t, create_graph=False)
        theta, state = tn.detach(), tuple(v.detach() for v in sn)
        thetas.append(theta)
        states.append(state)
    return thetas, states


def value(w, inp, eta=None) -> float:
    """V(theta_T(eta)): the outer loss after the unrolled inner loop (first-order only)."""
    thetas, _ = rollout(w, inp, eta)
    return float(model.outer_loss(w, thetas[-1], t64(inp.outer_x), t64(inp.outer_y)))


def meta_grad(w, inp, eta=None):
    """dV/d eta, dV/d theta_0 and V by Algorithm 1 with per-step checkpointing.

    Returns a dict with numpy float64 arrays 'd_eta' [n_eta], 'd_theta0' [P] and float 'V'.
    """
    eta0 = t64(inp.eta if eta is None else eta)
    X, Y = t64(inp.inner_x), t64(inp.inner_y)
    thetas, states = rollout(w, inp, eta0)
    # Outer gradient (Eq. 4): cotangent (dV/d theta_T, 0) on (theta_T, upsilon_T).
    thT = thetas[-1].clone().requires_grad_(True)
    with torch.enable_grad():
        V = model.outer_loss(w, thT, t64(inp.outer_x), t64(inp.outer_y))
        (theta_bar,) = torch.autograd.grad(V, thT)
    s_bar = tuple(torch.zeros_like(theta_bar) for _ in range(n_state(w)))
    d_eta = torch.zeros_like(eta0)
    for t in range(w.T - 1, -1, -1):
        theta_bar, s_bar, ge = reverse_step(w, eta0, X[t], Y[t], t, thetas[t], states[t],
                                            theta_bar, s_bar)
        if ge is not None:
            d_eta = d_eta + ge
    return {"d_eta": d_eta.numpy(), "d_theta0": theta_bar.numpy(), "V": float(V.detach())}


def reverse_step(w, eta, x, y, t, theta_t, state_t, theta_bar, s_bar):
    """One step of Algorithm 1's backward loop: rebuild inner step t at (theta_t, upsilon_t)
    on a tape whose inner gradient is itself taped (create_graph), and pull the cotangent
    (theta_bar_{t+1}, upsilon_bar_{t+1}) back through it.  Returns (theta_bar_t,
    upsilon_bar_t, this step's contribution to d eta, or None)."""
    th = theta_t.clone().requires_grad_(True)
    st = tuple(v.clone().requires_grad_(True) for v in state_t)
    et = eta.clone().requires_grad_(True)
    with torch.enable_grad():
        tn, sn = _step(w, th, st, et, x, y, t, create_graph=True)
        grads = torch.autograd.grad((tn, *sn), (th, *st, et), (theta_bar, *s_bar),
                                    allow_unused=True)
    theta_bar = grads[0]
    s_bar = tuple(gs if gs is not None else torch.zeros_like(theta_bar) for gs in grads[1:-1])
    return theta_bar, s_bar, grads[-1]


def grad(w, theta, x, y, weights=None):
    """grad_theta L with L = (1/B) sum_b weights_b l_b (weights default to 1)."""
    th = t64(theta).clone().requires_grad_(True)
    x, y = t64(x), t64(y)
    wt = torch.ones(x.shape[0], dtype=F64) if weights is None else t64(weights)
    with torch.enable_grad():
        L = model.weighted_inner_loss(w, th, x, y, wt)
        (g,) = torch.autograd.grad(L, th)
    return g.numpy()


def hvp(w, theta, x, y, v, weights=None):
    """H v with H = d^2 L / d theta^2, by reverse-over-reverse (grad of <grad L, v>)."""
    th = t64(theta).clone().requires_grad_(True)
    x, y, v = t64(x), t64(y), t64(v)
    wt = torch.ones(x.shape[0], dtype=F64) if weights is None else t64(weights)
    with torch.enable_grad():
        L = model.weighted_inner_loss(w, th, x, y, wt)
        (g,) = torch.autograd.grad(L, th, create_graph=True)
        (hv,) = torch.autograd.grad((g * v).sum(), th)
    return hv.numpy()


def tangent_losses(w, theta, x, y, v):
    """Per-example directional derivatives dl_b/d theta . v (the mixed term of Eq. 7 for
    per-example weights), via the transpose of the per-example-loss VJP."""
    th = t64(theta).clone().requires_grad_(True)
    x, y, v = t64(x), t64(y), t64(v)
    c = torch.zeros(x.shape[0], dtype=F64, requires_grad=True)
    with torch.enable_grad():
        l = model.losses(w, th, x, y)
        (jtc,) = torch.autograd.grad(l, th, c, create_graph=True)
        (ldot,) = torch.autograd.grad((jtc * v).sum(), c)
    return ldot.numpy()


def per_example_losses(w, theta, x, y):
    with torch.no_grad():
        return model.losses(w, t64(theta), t64(x), t64(y)).numpy()
