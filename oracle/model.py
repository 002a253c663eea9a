"""Inner models and per-example losses of the oracle, in plain float64 PyTorch CPU ops.

Test infrastructure only (see ``oracle/__init__.py``).

The paper leaves the inner model abstract (L(theta, eta, x) in Eq. 1); the workloads fix it
as a multilayer perceptron with a flat parameter vector laid out per layer as W_l
[d_l, d_{l+1}] row-major followed by b_l [d_{l+1}].  Per-example losses:

* squared:  l_b = 1/2 * mean_o (f_bo - y_bo)^2
* ce:       l_b = logsumexp(f_b) - f_{b, y_b}     (natural log)

The weighted inner loss of the loss-weighting task (Section 5, L = alpha(eta, x) * NTP) is
L_t = (1/B) sum_b sigmoid(eta_{t,b}) l_b, normalised by B, not by the sum of weights.
"""
from __future__ import annotations

import math

import torch

F64 = torch.float64


def act(name: str, z: torch.Tensor) -> torch.Tensor:
    """Hidden activation: identity, tanh, exact-erf GELU x*Phi(x), or SiLU x*sigmoid(x)."""
    if name == "ident":
        return z
    if name == "tanh":
        return torch.tanh(z)
    if name == "gelu":
        return 0.5 * z * (1.0 + torch.erf(z / math.sqrt(2.0)))
    if name == "silu":
        return z * torch.sigmoid(z)
    raise ValueError(name)


def unpack(w, theta: torch.Tensor):
    """Views (W_l, b_l) into the flat parameter vector (layout of ``Workload.layer_offsets``)."""
    out = []
    for i, (ow, ob) in enumerate(w.layer_offsets()):
        din, dout = w.dims[i], w.dims[i + 1]
        W = theta[ow:ow + din * dout].reshape(din, dout)
        b = theta[ob:ob + dout] if ob >= 0 else None
        out.append((W, b))
    return out


def mlp_forward(w, theta: torch.Tensor, x: torch.Tensor) -> torch.Tensor:
    """f = W_L phi(... phi(x W_1 + b_1) ...) + b_L; activation after every layer but the last."""
    h = x
    layers = unpack(w, theta)
    for i, (W, b) in enumerate(layers):
        h = h @ W
        if b is not None:
            h = h + b
        if i + 1 < len(layers):
            h = act(w.act, h)
    return h


def per_example_loss(w, f: torch.Tensor, y: torch.Tensor) -> torch.Tensor:
    """Vector of per-example losses l_b (shape [B])."""
    if w.loss == "squared":
        return 0.5 * ((f - y) ** 2).mean(dim=1)
    if w.loss == "ce":
        lse = torch.logsumexp(f, dim=1)
        return lse - f.gather(1, y.long().view(-1, 1)).view(-1)
    raise ValueError(w.loss)


def losses(w, theta, x, y):
    return per_example_loss(w, mlp_forward(w, theta, x), y)


def weighted_inner_loss(w, theta, x, y, weights):
    """L_t(theta) = (1/B) sum_b weights_b l_b(theta)."""
    l = losses(w, theta, x, y)
    return (weights * l).sum() / l.shape[0]


def outer_loss(w, theta, x, y):
    """V(theta_T) = mean_b l_b(theta_T) on the held-out batch (unweighted)."""
    return losses(w, theta, x, y).mean()
