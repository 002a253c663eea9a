"""ctypes binding of ``libmixflow.so`` (the C ABI of ``include/mixflow.h``).

Argument marshalling only: every step of the meta-gradient runs in the library's CUDA
kernels.  Functions keep the C names; ``MixFlow`` wraps a handle and takes torch tensors
(device memory and streams come from PyTorch).  Creating a handle (or any call) raises if
the library has not been built - there is no fallback implementation.  Tensor arguments are
checked before the call: a CUDA tensor, contiguous, of the dtype the ABI states; the library
itself only sees pointers and cannot tell a host pointer or a wrong element type.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libmixflow.so")

MF_MAX_LAYERS = 32
MF_ARCH_MLP, MF_ARCH_DECODER = 0, 1
ACTS = {"ident": 0, "tanh": 1, "gelu": 2, "silu": 3}
LOSSES = {"squared": 0, "ce": 1, "next_token_ce": 2, "chain_mse": 3}
PRECISIONS = {"fp32": 0, "bf16": 1}
OPTIMIZERS = {"sgd": 0, "adam": 1}
MF_META_EXAMPLE_WEIGHTS, MF_META_PARAM_LOGLR, MF_META_SCALAR_LOGLR = 1, 2, 4
MF_HVP_MIXED_FOR, MF_HVP_REV_REV = 0, 1
(MF_OPT_CUDA_GRAPHS, MF_OPT_PDL, MF_OPT_CONCURRENT, MF_OPT_GEMM_2SM, MF_OPT_FLASH_ATTN,
 MF_OPT_GEMM_PERSISTENT, MF_OPT_FUSED_HEAD, MF_OPT_LAYER_UPDATES,
 MF_OPT_WAIT_LIMIT_US) = 1, 2, 3, 4, 5, 6, 7, 8, 9
STATUS = {0: "MF_OK", 1: "MF_ERR_INVALID_ARG", 2: "MF_ERR_UNSUPPORTED", 3: "MF_ERR_OOM",
          4: "MF_ERR_CUDA", 5: "MF_ERR_NONFINITE", 6: "MF_ERR_TIMEOUT"}

# Every symbol include/mixflow.h declares (checked by the CPU test suite).
EXPORTS = ["mf_create", "mf_destroy", "mf_set_allocator", "mf_param_count",
           "mf_workspace_bytes", "mf_release_workspace", "mf_inner_rollout", "mf_hvp",
           "mf_meta_grad", "mf_sync", "mf_status_string", "mf_last_error", "mf_stats",
           "mf_set_kernel_timing", "mf_kernel_time", "mf_inject_fault", "mf_dual_gemm_bf16",
           "mf_hvp_noalloc", "mf_set_option", "mf_replay_gemms", "mf_checkpoint_plan"]


class mf_model_desc(C.Structure):
    _fields_ = [("arch", C.c_int), ("n_layers", C.c_int), ("dims", C.c_int * (MF_MAX_LAYERS + 1)),
                ("act", C.c_int), ("has_bias", C.c_int), ("loss", C.c_int), ("precision", C.c_int),
                ("d_model", C.c_int), ("n_heads", C.c_int), ("d_ff", C.c_int), ("vocab", C.c_int),
                ("seq_len", C.c_int), ("rope_base", C.c_float), ("rms_eps", C.c_float),
                ("chain_steps", C.c_int)]


class mf_loop_desc(C.Structure):
    _fields_ = [("T", C.c_int), ("B", C.c_int), ("B_outer", C.c_int), ("alpha", C.c_float),
                ("momentum", C.c_float), ("meta_kind", C.c_int), ("hvp_mode", C.c_int),
                ("ckpt_every", C.c_int), ("optimizer", C.c_int), ("beta1", C.c_float),
                ("beta2", C.c_float), ("adam_eps", C.c_float), ("ckpt_slots", C.c_int)]


class MixflowError(RuntimeError):
    def __init__(self, status, msg=""):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


def load(path: str = LIB_PATH) -> C.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"native library missing: {path} (run __graft_entry__.build())")
    lib = C.CDLL(path)
    vp, i64p, u64p, szp, dblp = C.c_void_p, C.POINTER(C.c_int64), C.POINTER(C.c_uint64), \
        C.POINTER(C.c_size_t), C.POINTER(C.c_double)
    H = C.c_void_p
    sig = {
        "mf_create": ([C.POINTER(mf_model_desc), C.POINTER(H)], C.c_int),
        "mf_destroy": ([H], C.c_int),
        "mf_set_allocator": ([H, vp, vp, vp], C.c_int),
        "mf_param_count": ([H, C.POINTER(mf_loop_desc), i64p, i64p], C.c_int),
        "mf_workspace_bytes": ([H, C.POINTER(mf_loop_desc), szp], C.c_int),
        "mf_release_workspace": ([H], C.c_int),
        "mf_inner_rollout": ([H, C.POINTER(mf_loop_desc), vp, vp, vp, vp, vp, vp], C.c_int),
        "mf_hvp": ([H, C.c_int, vp, vp, vp, vp, vp, vp, vp, vp, C.c_int, vp], C.c_int),
        "mf_meta_grad": ([H, C.POINTER(mf_loop_desc), vp, vp, vp, vp, vp, vp, vp, vp, vp, vp], C.c_int),
        "mf_sync": ([H], C.c_int),
        "mf_status_string": ([C.c_int], C.c_char_p),
        "mf_last_error": ([H], C.c_char_p),
        "mf_stats": ([H, u64p, szp], C.c_int),
        "mf_set_kernel_timing": ([H, C.c_int], C.c_int),
        "mf_kernel_time": ([H, dblp, u64p, dblp], C.c_int),
        "mf_replay_gemms": ([H, C.c_int, vp, dblp, u64p, dblp], C.c_int),
        "mf_checkpoint_plan": ([C.c_int, C.c_int, C.c_int, C.POINTER(C.c_int), i64p], C.c_int),
        "mf_inject_fault": ([H, C.c_int], C.c_int),
        "mf_set_option": ([H, C.c_int, C.c_int], C.c_int),
        "mf_hvp_noalloc": ([C.POINTER(mf_model_desc), C.c_int, vp, vp, vp, vp, vp, vp, vp, vp, vp],
                           C.c_int),
        "mf_dual_gemm_bf16": ([C.c_int, C.c_int, C.c_int, vp, C.c_int, vp, C.c_int, vp, C.c_int, vp,
                               C.c_int, vp, C.c_int, vp, vp, C.c_int, vp, C.c_uint, vp], C.c_int),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    return lib


_lib = None


def lib() -> C.CDLL:
    global _lib
    if _lib is None:
        _lib = load()
    return _lib


def _dev(t, name, dtype, rows=False):
    """Device pointer of tensor argument ``name`` (None -> NULL) after checking its dtype,
    layout (contiguous; with ``rows``, only unit stride along the last axis, the leading
    dimension being passed separately) and that it lives on a CUDA device."""
    if t is None:
        return None
    if t.dtype != dtype:
        raise ValueError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if rows:
        if t.dim() != 2 or (t.shape[1] > 1 and t.stride(1) != 1):
            raise ValueError(f"{name}: expected a 2-D tensor with unit stride along its rows")
    elif not t.is_contiguous():
        raise ValueError(f"{name}: expected a contiguous tensor")
    if not t.is_cuda:
        raise ValueError(f"{name}: expected a CUDA tensor, got one on {t.device}")
    return C.c_void_p(t.data_ptr())


def io_dtypes(desc: mf_model_desc):
    """torch dtypes of (x, y) for a model: token ids for decoders; for MLPs bf16 or float32
    inputs (the model's precision) and int32 class labels (cross-entropy) or float32 targets."""
    import torch
    if desc.arch == MF_ARCH_DECODER:
        return torch.int32, torch.int32
    x = torch.bfloat16 if desc.precision == PRECISIONS["bf16"] else torch.float32
    y = torch.int32 if desc.loss == LOSSES["ce"] else torch.float32
    return x, y


def _stream(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


def model_desc_for(w) -> mf_model_desc:
    """mf_model_desc of a ``synth.Workload`` (MLP or decoder-only transformer)."""
    d = mf_model_desc()
    if getattr(w, "arch", "mlp") == "decoder":
        d.arch = MF_ARCH_DECODER
        d.n_layers = w.n_blocks
        d.d_model, d.n_heads, d.d_ff, d.vocab, d.seq_len = w.d_model, w.n_heads, w.d_ff, w.vocab, w.seq
        d.rope_base, d.rms_eps = w.rope_base, w.rms_eps
        d.loss = LOSSES["next_token_ce"]
        d.precision = PRECISIONS[w.precision]
        return d
    d.arch = MF_ARCH_MLP
    d.n_layers = len(w.dims) - 1
    for i, v in enumerate(w.dims):
        d.dims[i] = v
    d.act = ACTS[w.act]
    d.has_bias = 1 if w.has_bias else 0
    d.loss = LOSSES[w.loss]
    d.precision = PRECISIONS[w.precision]
    d.chain_steps = int(w.extra.get("chain_steps", 0))
    return d


def checkpoint_plan(T: int, ckpt_every: int = 1, ckpt_slots: int = 0):
    """(stored states, inner steps re-run) of a sweep's checkpoint plan (mf_checkpoint_plan)."""
    n, r = C.c_int(), C.c_int64()
    st = lib().mf_checkpoint_plan(T, ckpt_every, ckpt_slots, C.byref(n), C.byref(r))
    if st != 0:
        raise MixflowError(st, "mf_checkpoint_plan")
    return n.value, r.value


def loop_desc_for(w, hvp_mode: int = MF_HVP_MIXED_FOR, ckpt_every: int = 1,
                  ckpt_slots: int = 0) -> mf_loop_desc:
    l = mf_loop_desc()
    l.T, l.B, l.B_outer = w.T, w.B, w.B_outer
    l.alpha, l.momentum = w.alpha, w.momentum
    l.meta_kind = w.meta_kind
    l.hvp_mode = hvp_mode
    l.ckpt_every = ckpt_every
    l.ckpt_slots = ckpt_slots
    l.optimizer = OPTIMIZERS[getattr(w, "optimizer", "sgd")]
    l.beta1, l.beta2, l.adam_eps = w.beta1, w.beta2, w.adam_eps
    return l


def mf_dual_gemm_bf16(M, N, K, A0, A1, B0, B1, C0, C1, terms, bias0=None, bias1=None,
                      stream=None):
    """C0/C1 (float32) = selected products of bf16 K-major operands (see mixflow.h)."""
    import torch
    bf, f32 = torch.bfloat16, torch.float32
    ld = lambda t: (t.stride(0) if t is not None else 0)
    st = lib().mf_dual_gemm_bf16(M, N, K, _dev(A0, "A0", bf, True), ld(A0),
                                 _dev(A1, "A1", bf, True), ld(A1), _dev(B0, "B0", bf, True),
                                 ld(B0), _dev(B1, "B1", bf, True), ld(B1),
                                 _dev(C0, "C0", f32, True), ld(C0), _dev(bias0, "bias0", f32),
                                 _dev(C1, "C1", f32, True), ld(C1), _dev(bias1, "bias1", f32),
                                 terms, _stream(stream))
    if st != 0:
        raise MixflowError(st, "mf_dual_gemm_bf16")


class MixFlow:
    """One library handle for one inner-model architecture."""

    def __init__(self, desc: mf_model_desc):
        self._lib = lib()
        self.desc = desc
        h = C.c_void_p()
        st = self._lib.mf_create(C.byref(desc), C.byref(h))
        if st != 0:
            raise MixflowError(st, "mf_create")
        self.h = h
        self.x_dtype, self.y_dtype = io_dtypes(desc)

    @classmethod
    def for_workload(cls, w):
        return cls(model_desc_for(w))

    def close(self):
        if getattr(self, "h", None):
            self._lib.mf_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, st, what):
        if st != 0:
            raise MixflowError(st, f"{what}: {self._lib.mf_last_error(self.h).decode()}")

    def param_count(self, loop=None):
        n, e = C.c_int64(), C.c_int64()
        self._check(self._lib.mf_param_count(self.h, C.byref(loop) if loop else None,
                                             C.byref(n), C.byref(e)), "mf_param_count")
        return n.value, e.value

    def workspace_bytes(self, loop):
        b = C.c_size_t()
        self._check(self._lib.mf_workspace_bytes(self.h, C.byref(loop), C.byref(b)),
                    "mf_workspace_bytes")
        return b.value

    def release_workspace(self):
        self._check(self._lib.mf_release_workspace(self.h), "mf_release_workspace")

    def meta_grad(self, loop, theta0, eta, inner_x, inner_y, outer_x, outer_y, d_eta,
                  d_theta0=None, outer_loss=None, stream=None):
        import torch
        f32, xd, yd = torch.float32, self.x_dtype, self.y_dtype
        st = self._lib.mf_meta_grad(self.h, C.byref(loop), _dev(theta0, "theta0", f32),
                                    _dev(eta, "eta", f32), _dev(inner_x, "inner_x", xd),
                                    _dev(inner_y, "inner_y", yd), _dev(outer_x, "outer_x", xd),
                                    _dev(outer_y, "outer_y", yd), _dev(d_eta, "d_eta", f32),
                                    _dev(d_theta0, "d_theta0", f32),
                                    _dev(outer_loss, "outer_loss", f32), _stream(stream))
        self._check(st, "mf_meta_grad")

    def inner_rollout(self, loop, theta0, eta, inner_x, inner_y, thetaT, stream=None):
        import torch
        f32 = torch.float32
        st = self._lib.mf_inner_rollout(self.h, C.byref(loop), _dev(theta0, "theta0", f32),
                                        _dev(eta, "eta", f32),
                                        _dev(inner_x, "inner_x", self.x_dtype),
                                        _dev(inner_y, "inner_y", self.y_dtype),
                                        _dev(thetaT, "thetaT", f32), _stream(stream))
        self._check(st, "mf_inner_rollout")

    def hvp(self, B, theta, x, y, v, Hv, ex_w=None, tangent_losses=None, grad=None,
            hvp_mode=MF_HVP_MIXED_FOR, stream=None):
        import torch
        f32 = torch.float32
        st = self._lib.mf_hvp(self.h, B, _dev(theta, "theta", f32), _dev(x, "x", self.x_dtype),
                              _dev(y, "y", self.y_dtype), _dev(ex_w, "ex_w", f32),
                              _dev(v, "v", f32), _dev(Hv, "Hv", f32),
                              _dev(tangent_losses, "tangent_losses", f32),
                              _dev(grad, "grad", f32), hvp_mode, _stream(stream))
        self._check(st, "mf_hvp")

    def sync(self):
        self._check(self._lib.mf_sync(self.h), "mf_sync")

    def stats(self):
        n, p = C.c_uint64(), C.c_size_t()
        self._check(self._lib.mf_stats(self.h, C.byref(n), C.byref(p)), "mf_stats")
        return n.value, p.value

    def set_kernel_timing(self, on: bool):
        self._check(self._lib.mf_set_kernel_timing(self.h, 1 if on else 0), "mf_set_kernel_timing")

    def kernel_time(self):
        ms, n, fl = C.c_double(), C.c_uint64(), C.c_double()
        self._check(self._lib.mf_kernel_time(self.h, C.byref(ms), C.byref(n), C.byref(fl)),
                    "mf_kernel_time")
        return ms.value, n.value, fl.value

    def record_gemms(self):
        """Record the bf16 dual GEMM launches of the next call (mf_set_kernel_timing(h, 2))."""
        self._check(self._lib.mf_set_kernel_timing(self.h, 2), "mf_set_kernel_timing")

    def replay_gemms(self, reps: int = 1, stream=None):
        """(ms of one back-to-back replay of the recorded GEMMs, launches, flops)."""
        ms, n, fl = C.c_double(), C.c_uint64(), C.c_double()
        self._check(self._lib.mf_replay_gemms(self.h, reps, _stream(stream), C.byref(ms),
                                              C.byref(n), C.byref(fl)), "mf_replay_gemms")
        return ms.value, n.value, fl.value

    def set_torch_allocator(self):
        """Route the handle's workspace through PyTorch's caching allocator (mf_set_allocator),
        so that torch.cuda.max_memory_allocated() sees it."""
        import torch

        @C.CFUNCTYPE(C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p)
        def _alloc(nbytes, stream, ctx):
            try:
                return torch.cuda.caching_allocator_alloc(int(nbytes), stream=stream or 0)
            except Exception:
                return None

        @C.CFUNCTYPE(None, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p)
        def _free(ptr, nbytes, stream, ctx):
            torch.cuda.caching_allocator_delete(ptr)

        self._alloc_cbs = (_alloc, _free)   # kept alive with the handle
        self._check(self._lib.mf_set_allocator(self.h, C.cast(_alloc, C.c_void_p),
                                               C.cast(_free, C.c_void_p), None),
                    "mf_set_allocator")

    def set_option(self, option: int, value: int):
        self._check(self._lib.mf_set_option(self.h, option, value), "mf_set_option")

    def inject_fault(self, kind: int):
        self._check(self._lib.mf_inject_fault(self.h, kind), "mf_inject_fault")


def to_device_inputs(w, inp, device="cuda"):
    """Move a ``synth.Inputs`` to the device with the dtypes the ABI expects."""
    import torch
    if getattr(w, "arch", "mlp") == "decoder":
        ids = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(device)
        f = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(device)
        ix, ox = ids(inp.inner_x), ids(inp.outer_x)
        return dict(theta0=f(inp.theta0), eta=f(inp.eta), inner_x=ix, inner_y=ix, outer_x=ox,
                    outer_y=ox)
    xdt = torch.bfloat16 if w.precision == "bf16" else torch.float32

    def xt(a):
        return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(device).to(xdt).contiguous()

    def yt(a):
        if a.dtype.kind in "iu":
            return torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(device)
        return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(device)

    f = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(device)
    return dict(theta0=f(inp.theta0), eta=f(inp.eta), inner_x=xt(inp.inner_x),
                inner_y=yt(inp.inner_y), outer_x=xt(inp.outer_x), outer_y=yt(inp.outer_y))
