"""Inner models and per-example losses of the oracle, in plain float64 PyTorch CPU ops.

Test infrastructure only (see ``oracle/__init__.py``).

The paper leaves the inner model abstract (L(theta, eta, x) in Eq. 1); the workloads fix it
as a multilayer perceptron with a flat parameter vector laid out per layer as W_l
[d_l, d_{l+1}] row-major followed by b_l [d_{l+1}].  The decoder-only transformer of the language-modelling tasks (Section 5: Chinchilla-style
models with RoPE) is written out in ``decoder_logits``.  Per-example losses:

* squared:  l_b = 1/2 * mean_o (f_bo - y_bo)^2
* ce:       l_b = logsumexp(f_b) - f_{b, y_b}     (natural log)
* chain_mse (the motivating example of Section 3): l_b = mean_o (y_M(f_bo) - y_bo)^2 with the
  recursion y_0 = f, y_i = i * (2 + sin y_{i-1}) ** cos y_{i-1}, i = 1..M (Eq. 8).

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


def chain(f: torch.Tensor, M: int) -> torch.Tensor:
    """The M-step elementwise recursion of the motivating example (Eq. 8)."""
    y = f
    for i in range(1, M + 1):
        y = i * (2.0 + torch.sin(y)) ** torch.cos(y)
    return y


def per_example_loss(w, f: torch.Tensor, y: torch.Tensor) -> torch.Tensor:
    """Vector of per-example losses l_b (shape [B])."""
    if w.loss == "squared":
        return 0.5 * ((f - y) ** 2).mean(dim=1)
    if w.loss == "chain_mse":
        return ((chain(f, w.extra["chain_steps"]) - y) ** 2).mean(dim=1)
    if w.loss == "ce":
        lse = torch.logsumexp(f, dim=1)
        return lse - f.gather(1, y.long().view(-1, 1)).view(-1)
    raise ValueError(w.loss)


def decoder_unpack(w, theta):
    """Named views into the flat decoder parameter vector (``Workload.decoder_layout``)."""
    out, o = {}, 0
    for name, n in w.decoder_layout():
        out[name] = theta[o:o + n]
        o += n
    return out


def rmsnorm(x, g, eps):
    """y = g * x / sqrt(mean(x^2) + eps) over the last axis (pre-norm of the decoder blocks)."""
    return g * x * torch.rsqrt((x * x).mean(dim=-1, keepdim=True) + eps)


def rope(x, base):
    """Rotary position embedding, rotate-half form, over the last axis of [B, H, S, dh]:
    out = x cos(p w) + rot(x) sin(p w), rot(x) = [-x2, x1], w_j = base^(-2 (j mod dh/2) / dh)."""
    S, dh = x.shape[-2], x.shape[-1]
    half = dh // 2
    j = torch.arange(half, dtype=F64)
    inv = base ** (-2.0 * j / dh)
    ang = torch.arange(S, dtype=F64)[:, None] * inv[None, :]       # [S, half]
    cos = torch.cat([torch.cos(ang), torch.cos(ang)], dim=-1)
    sin = torch.cat([torch.sin(ang), torch.sin(ang)], dim=-1)
    rot = torch.cat([-x[..., half:], x[..., :half]], dim=-1)
    return x * cos + rot * sin


def decoder_logits(w, theta, ids):
    """Decoder-only transformer: token embedding, n_blocks pre-RMSNorm blocks (causal
    multi-head attention with RoPE, GELU MLP, residual connections), final RMSNorm, untied
    head.  ids [B, S+1]; returns logits [B, S, V] for positions 0..S-1."""
    P = decoder_unpack(w, theta)
    d, H, F, V = w.d_model, w.n_heads, w.d_ff, w.vocab
    dh = d // H
    B, S = ids.shape[0], ids.shape[1] - 1
    x = P["E"].reshape(V, d)[ids[:, :S]]                            # [B, S, d]
    mask = torch.triu(torch.ones(S, S, dtype=torch.bool), diagonal=1)
    for l in range(w.n_blocks):
        h = rmsnorm(x, P[f"g1.{l}"], w.rms_eps)
        qkv = h @ P[f"Wqkv.{l}"].reshape(d, 3 * d)
        q, k, v = (t.reshape(B, S, H, dh).transpose(1, 2) for t in qkv.split(d, dim=-1))
        q, k = rope(q, w.rope_base), rope(k, w.rope_base)
        s = (q @ k.transpose(-1, -2)) / math.sqrt(dh)
        s = s.masked_fill(mask, float("-inf"))
        o = torch.softmax(s, dim=-1) @ v                             # [B, H, S, dh]
        x = x + o.transpose(1, 2).reshape(B, S, d) @ P[f"Wo.{l}"].reshape(d, d)
        h2 = rmsnorm(x, P[f"g2.{l}"], w.rms_eps)
        x = x + act("gelu", h2 @ P[f"W1.{l}"].reshape(d, F)) @ P[f"W2.{l}"].reshape(F, d)
    return rmsnorm(x, P["gf"], w.rms_eps) @ P["Wh"].reshape(d, V)


def decoder_losses(w, theta, ids):
    """Per-sequence next-token cross-entropy, mean over the S predicted positions."""
    f = decoder_logits(w, theta, ids)
    tgt = ids[:, 1:].long()
    ce = torch.logsumexp(f, dim=-1) - f.gather(-1, tgt[..., None])[..., 0]
    return ce.mean(dim=1)


def losses(w, theta, x, y):
    if getattr(w, "arch", "mlp") == "decoder":
        return decoder_losses(w, theta, x.long())
    return per_example_loss(w, mlp_forward(w, theta, x), y)


def weighted_inner_loss(w, theta, x, y, weights):
    """L_t(theta) = (1/B) sum_b weights_b l_b(theta)."""
    l = losses(w, theta, x, y)
    return (weights * l).sum() / l.shape[0]


def outer_loss(w, theta, x, y):
    """V(theta_T) = mean_b l_b(theta_T) on the held-out batch (unweighted)."""
    return losses(w, theta, x, y).mean()
