"""Seeded synthetic workloads for the Truncated-BPTT meta-gradient (shared input recipe).

This module is the only code shared by the CPU oracle and the CUDA path.  It holds the
workload shapes and draws their inputs; it contains none of the meta-gradient arithmetic
(no loss, no gradient, no update rule).  The one model evaluation in here is the random
*teacher* network that labels regression inputs, i.e. data generation.

Every random array comes from ``numpy.random.Generator(PCG64(SeedSequence([seed, k])))``
with a fixed stream index ``k`` per role, so the oracle and the GPU path see bit-identical
inputs.  Values that the bf16 path consumes are rounded to bf16 (round-to-nearest-even)
here, once, and handed to both sides as float32 arrays holding bf16-representable values.

Workloads (problem statement: bilevel problem of Eq. 1 unrolled as Eq. 2; meta-parameters
as in the loss-weighting and learned-learning-rate tasks of Section 5):

* ``tiny``  - 16->32->1 tanh MLP, squared loss, B=8, T=4 SGD steps, alpha=0.1, per-example
  weight logits, fp32.
* ``wide``  - 1024-wide 4-hidden-layer GELU MLP with a 10-class softmax head, B=256, T=16,
  alpha=0.05, per-example weight logits, outer batch 1024, bf16 GEMMs.
* ``deep``  - 8 Linear 4096->4096 layers (SiLU after the first 7), regression onto a random
  teacher, per-parameter log learning rates, SGD with momentum 0.9, B=512, T=32, bf16 GEMMs.
* ``decoder_small`` - decoder-only transformer, 6 layers, d_model 512, 8 heads, MLP 2048
  GELU, pre-RMSNorm, RoPE, causal attention, vocabulary 8192, sequences of 256 tokens with
  ids drawn from a Zipf(1.1) law truncated to the vocabulary, batch 16, T=8 SGD steps,
  alpha=1e-3, per-sequence weight logits, next-token cross-entropy.
* ``decoder_large`` - 12 layers, d_model 1024, 16 heads, MLP 4096, sequences of 1024, batch 8,
  vocabulary 32768, T=16 heavy-ball (0.9) steps, per-sequence weights plus a scalar log-lr.
* ``toy`` - the motivating example of Section 3: one D x D linear map followed by an M-step
  elementwise recursion, mean-squared error on random targets, B=1024, D=4096, T=2 SGD steps
  with lr 1e-3; the meta-parameter is the initial point theta_0 (MAML-style), so the
  meta-gradient is d V / d theta_0 (meta_kind 0).  Inputs, targets and theta_0 are standard
  normal; ``toy_bf16`` scales theta_0 by 1/sqrt(D) so that the recursion sees O(1) inputs
  and bf16 GEMM operands stay meaningful.
"""
from __future__ import annotations

import copy
import math
from dataclasses import dataclass, field, replace
from typing import Optional

import numpy as np

# Stream indices (one per role).  Changing one changes every stored expected value.
_STREAMS = {"x": 1, "teacher": 2, "noise": 3, "theta0": 4, "eta": 5, "outer": 6,
            "tokens": 7, "labels": 8, "outer_noise": 9, "outer_labels": 10, "dir": 11,
            "targets": 12}


def rng(seed: int, stream: str) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, _STREAMS[stream]])))


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round float values to the nearest bf16 (ties to even); returned as float32."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


# meta-parameter kinds (bit mask, same values as the C header)
EXAMPLE_WEIGHTS = 1
PARAM_LOGLR = 2
SCALAR_LOGLR = 4


@dataclass
class Workload:
    name: str
    dims: list                      # MLP layer widths [d_in, h1, ..., d_out] (MLP only)
    act: str                        # hidden activation: ident|tanh|gelu|silu
    loss: str                       # squared | ce | chain_mse (toy task; extra["chain_steps"])
    precision: str                  # fp32 | bf16
    B: int
    T: int
    B_outer: int
    alpha: float = 0.0              # constant lr (when no log-lr meta-parameter)
    momentum: float = 0.0           # heavy-ball coefficient (optimizer "sgd")
    optimizer: str = "sgd"          # sgd (plain or heavy-ball) | adam
    beta1: float = 0.9              # Adam moment decays and epsilon
    beta2: float = 0.999
    adam_eps: float = 1e-8
    meta_kind: int = EXAMPLE_WEIGHTS
    loglr_mean: float = 0.0
    loglr_std: float = 0.0
    eta_std: float = 1.0            # example-logit std
    noise_std: float = 0.0          # regression-target noise std
    seed: int = 0
    has_bias: bool = True
    extra: dict = field(default_factory=dict)
    # decoder-only transformer (arch == "decoder"); dims/act/has_bias unused there
    arch: str = "mlp"
    d_model: int = 0
    n_heads: int = 0
    d_ff: int = 0
    vocab: int = 0
    seq: int = 0
    n_blocks: int = 0
    zipf_s: float = 1.1
    init_std: float = 0.02
    rope_base: float = 10000.0
    rms_eps: float = 1e-6

    @property
    def n_layers(self) -> int:
        return len(self.dims) - 1

    @property
    def n_params(self) -> int:
        if self.arch == "decoder":
            return sum(n for _, n in self.decoder_layout())
        return sum(self.dims[i] * self.dims[i + 1] + (self.dims[i + 1] if self.has_bias else 0)
                   for i in range(self.n_layers))

    def decoder_layout(self):
        """(name, size) of each decoder tensor in flat-parameter order: embedding E [V][d];
        per block g1 [d], Wqkv [d][3d], Wo [d][d], g2 [d], W1 [d][dff], W2 [dff][d]; final gain
        gf [d]; head Wh [d][V]."""
        d, V, F = self.d_model, self.vocab, self.d_ff
        out = [("E", V * d)]
        for l in range(self.n_blocks):
            out += [(f"g1.{l}", d), (f"Wqkv.{l}", d * 3 * d), (f"Wo.{l}", d * d),
                    (f"g2.{l}", d), (f"W1.{l}", d * F), (f"W2.{l}", F * d)]
        out += [("gf", d), ("Wh", d * V)]
        return out

    @property
    def n_eta(self) -> int:
        n = 0
        if self.meta_kind & EXAMPLE_WEIGHTS:
            n += self.T * self.B
        if self.meta_kind & PARAM_LOGLR:
            n += self.n_params
        if self.meta_kind & SCALAR_LOGLR:
            n += 1
        return n

    def layer_offsets(self):
        """(W offset, b offset) of each layer in the flat parameter vector.

        Layout: for each layer l, W_l as [d_l][d_{l+1}] row-major, then b_l [d_{l+1}].
        """
        offs, o = [], 0
        for i in range(self.n_layers):
            din, dout = self.dims[i], self.dims[i + 1]
            ow = o
            o += din * dout
            ob = o if self.has_bias else -1
            if self.has_bias:
                o += dout
            offs.append((ow, ob))
        return offs

    def with_(self, **kw) -> "Workload":
        return replace(copy.deepcopy(self), **kw)


def decoder(name, d, H, F, L, V, S, B, T, B_outer, alpha=0.0, momentum=0.0,
            meta_kind=EXAMPLE_WEIGHTS, **kw):
    return Workload(name, [], "gelu", "next_token_ce", "bf16", B=B, T=T, B_outer=B_outer,
                    alpha=alpha, momentum=momentum, meta_kind=meta_kind, has_bias=False,
                    arch="decoder", d_model=d, n_heads=H, d_ff=F, vocab=V, seq=S, n_blocks=L,
                    **kw)


WORKLOADS = {
    "tiny": Workload("tiny", [16, 32, 1], "tanh", "squared", "fp32", B=8, T=4, B_outer=8,
                     alpha=0.1, noise_std=0.1),
    "wide": Workload("wide", [1024] * 5 + [10], "gelu", "ce", "bf16", B=256, T=16,
                     B_outer=1024, alpha=0.05),
    "deep": Workload("deep", [4096] * 9, "silu", "squared", "bf16", B=512, T=32,
                     B_outer=512, momentum=0.9, meta_kind=PARAM_LOGLR,
                     loglr_mean=math.log(1e-2), loglr_std=0.1),
    "decoder_small": decoder("decoder_small", 512, 8, 2048, 6, 8192, 256, B=16, T=8, B_outer=16,
                             alpha=1e-3),
    "decoder_large": decoder("decoder_large", 1024, 16, 4096, 12, 32768, 1024, B=8, T=16,
                             B_outer=8, momentum=0.9, meta_kind=EXAMPLE_WEIGHTS | SCALAR_LOGLR,
                             extra={"scalar_loglr": math.log(1e-3)}),
}


def toy(name, D, B, M, T=2, precision="bf16", init_std=None, **kw):
    """Motivating example: x theta followed by the M-step recursion, MSE, theta_0 meta-gradient."""
    return Workload(name, [D, D], "ident", "chain_mse", precision, B=B, T=T, B_outer=B,
                    alpha=1e-3, meta_kind=0, has_bias=False,
                    init_std=1.0 if init_std is None else init_std,
                    extra={"chain_steps": M}, **kw)


WORKLOADS["toy"] = toy("toy", 4096, 1024, 8, precision="bf16", init_std=1.0 / 64.0)
WORKLOADS["toy_fp32"] = toy("toy_fp32", 4096, 1024, 8, precision="fp32")


def glorot_params(w: Workload, g: np.random.Generator) -> np.ndarray:
    """Glorot-uniform weights, zero biases, in the flat layout of ``layer_offsets``."""
    theta = np.zeros(w.n_params, dtype=np.float64)
    for i, (ow, ob) in enumerate(w.layer_offsets()):
        din, dout = w.dims[i], w.dims[i + 1]
        lim = math.sqrt(6.0 / (din + dout))
        theta[ow:ow + din * dout] = g.uniform(-lim, lim, size=din * dout)
    return theta.astype(np.float32)


def _teacher_outputs(w: Workload, x: np.ndarray) -> np.ndarray:
    """Labels for regression workloads: a Glorot-initialised copy of the architecture
    (own stream) evaluated in float32.  Data generation only."""
    tw = glorot_params(w, rng(w.seed, "teacher"))
    h = x.astype(np.float32)
    for i, (ow, ob) in enumerate(w.layer_offsets()):
        din, dout = w.dims[i], w.dims[i + 1]
        W = tw[ow:ow + din * dout].reshape(din, dout)
        h = h @ W
        if ob >= 0:
            h = h + tw[ob:ob + dout]
        if i + 1 < w.n_layers:
            if w.act == "tanh":
                h = np.tanh(h)
            elif w.act == "gelu":
                from scipy.special import erf
                h = (0.5 * h * (1.0 + erf(h / math.sqrt(2.0)))).astype(np.float32)
            elif w.act == "silu":
                h = h / (1.0 + np.exp(-h))
    return h.astype(np.float32)


@dataclass
class Inputs:
    theta0: np.ndarray      # [P] float32
    eta: np.ndarray         # [n_eta] float32
    inner_x: np.ndarray     # [T, B, d_in] float32 (bf16-representable for bf16 workloads)
    inner_y: np.ndarray     # [T, B] int32 labels or [T, B, d_out] float32 targets
    outer_x: np.ndarray     # [B_outer, d_in]
    outer_y: np.ndarray     # [B_outer] int32 or [B_outer, d_out] float32


def zipf_ids(g: np.random.Generator, shape, V: int, s: float) -> np.ndarray:
    """Token ids from p(k) ~ k^-s on k = 1..V (truncated Zipf), id = k - 1, by inverse CDF."""
    p = np.arange(1, V + 1, dtype=np.float64) ** (-s)
    cdf = np.cumsum(p / p.sum())
    u = g.random(size=shape)
    return np.minimum(np.searchsorted(cdf, u, side="right"), V - 1).astype(np.int32)


def decoder_params(w: Workload, g: np.random.Generator) -> np.ndarray:
    """N(0, init_std) matrices, unit RMSNorm gains, in the layout of ``decoder_layout``."""
    parts = []
    for name, n in w.decoder_layout():
        if name.startswith("g"):
            parts.append(np.ones(n))
        else:
            parts.append(w.init_std * g.standard_normal(n))
    return np.concatenate(parts).astype(np.float32)


def make_inputs(w: Workload) -> Inputs:
    """Draw every input of one meta-gradient call for workload ``w``."""
    if w.arch == "decoder":
        ids = zipf_ids(rng(w.seed, "tokens"), (w.T, w.B, w.seq + 1), w.vocab, w.zipf_s)
        oids = zipf_ids(rng(w.seed, "outer"), (w.B_outer, w.seq + 1), w.vocab, w.zipf_s)
        theta0 = decoder_params(w, rng(w.seed, "theta0"))
        ge = rng(w.seed, "eta")
        parts = []
        if w.meta_kind & EXAMPLE_WEIGHTS:
            parts.append(w.eta_std * ge.standard_normal(w.T * w.B))
        if w.meta_kind & PARAM_LOGLR:
            parts.append(w.loglr_mean + w.loglr_std * ge.standard_normal(w.n_params))
        if w.meta_kind & SCALAR_LOGLR:
            parts.append(np.array([w.extra.get("scalar_loglr", math.log(1e-3))]))
        eta = np.concatenate(parts).astype(np.float32)
        # token ids double as inputs (positions 0..S-1) and targets (positions 1..S)
        return Inputs(theta0, eta, ids, ids, oids, oids)
    din, dout = w.dims[0], w.dims[-1]
    rd = round_bf16 if w.precision == "bf16" else (lambda a: np.asarray(a, np.float32))
    x = rd(rng(w.seed, "x").standard_normal((w.T, w.B, din)))
    ox = rd(rng(w.seed, "outer").standard_normal((w.B_outer, din)))
    if w.loss == "chain_mse":
        # motivating example: standard-normal targets and theta_0 (scaled by init_std)
        gt = rng(w.seed, "targets")
        y = gt.standard_normal((w.T, w.B, dout)).astype(np.float32)
        oy = gt.standard_normal((w.B_outer, dout)).astype(np.float32)
        theta0 = (w.init_std * rng(w.seed, "theta0").standard_normal(w.n_params)).astype(np.float32)
        return Inputs(theta0, np.zeros(0, np.float32), np.ascontiguousarray(x, np.float32), y,
                      np.ascontiguousarray(ox, np.float32), oy)
    if w.loss == "ce":
        y = rng(w.seed, "labels").integers(0, dout, size=(w.T, w.B)).astype(np.int32)
        oy = rng(w.seed, "outer_labels").integers(0, dout, size=(w.B_outer,)).astype(np.int32)
    else:
        y = _teacher_outputs(w, x.reshape(-1, din)).reshape(w.T, w.B, dout)
        oy = _teacher_outputs(w, ox)
        if w.noise_std > 0:
            y = (y + w.noise_std * rng(w.seed, "noise").standard_normal(y.shape)).astype(np.float32)
            oy = (oy + w.noise_std * rng(w.seed, "outer_noise").standard_normal(oy.shape)).astype(np.float32)
    theta0 = glorot_params(w, rng(w.seed, "theta0"))
    ge = rng(w.seed, "eta")
    parts = []
    if w.meta_kind & EXAMPLE_WEIGHTS:
        parts.append(w.eta_std * ge.standard_normal(w.T * w.B))
    if w.meta_kind & PARAM_LOGLR:
        parts.append(w.loglr_mean + w.loglr_std * ge.standard_normal(w.n_params))
    if w.meta_kind & SCALAR_LOGLR:
        parts.append(np.array([w.extra.get("scalar_loglr", math.log(1e-3))]))
    eta = np.concatenate(parts).astype(np.float32)
    return Inputs(theta0, eta, np.ascontiguousarray(x, np.float32), y,
                  np.ascontiguousarray(ox, np.float32), oy)


def random_direction(n: int, seed: int = 0, k: int = 0) -> np.ndarray:
    """A seeded Gaussian direction of length n (HVP tangents, directional checks)."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, _STREAMS["dir"], k])))
    return g.standard_normal(n).astype(np.float32)
