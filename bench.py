"""Benchmark: mixed-mode (forward-over-reverse) Truncated-BPTT meta-gradient steps per second.

One step = one full ``mf_meta_grad`` call on the "decoder_large" workload, the largest
configuration: a 12-block decoder-only transformer (d_model 1024, 16 heads, MLP 4096 GELU,
pre-RMSNorm, RoPE, causal attention, vocabulary 32768, sequences of 1024 Zipf(1.1) token
ids), B = 8 sequences per inner step, T = 16 heavy-ball (0.9) steps, per-sequence weight
logits plus a scalar log learning rate (129 meta-parameters), outer batch 8, bf16
tensor-core GEMMs with float32 accumulation and float32 parameters/adjoints (218M
parameters).  Inputs are seeded synthetic data resident in HBM when the timed region starts.

Prints one JSON line (rank 0) with, next to the step rate:
- ``roofline``: the tcgen05 dual GEMM (the dominant kernel); its launches of one call are
  recorded and replayed back to back as a graph under CUDA events (``mf_replay_gemms``);
- ``hbm``: peak HBM of the call, measured with ``torch.cuda.max_memory_allocated`` while the
  library's workspace comes from PyTorch's allocator, split into the static part (theta_t
  and m_t store, inputs, eta, d eta) and the sweep's dynamic part, for the mixed-mode sweep
  and for the reverse-over-reverse sweep of the same library (Section 5's memory ratio);
- ``cpu_baseline``: the float64 oracle on the host cores, on a bounded sample;
- ``e2e``: the same metric through the public API from pinned host buffers.

``--impl reference`` times the CPU float64 oracle instead (a bounded sample per step).
Multi-GPU runs are independent replicas (weak scaling), one process per GPU under torchrun.

``--workload`` measures another configuration the same way (wide and deep MLPs, the small
transformer, the motivating example of Section 3 with ``--chain-steps M``).
``--hvp-mode rr`` runs the reverse-over-reverse sweep instead of the mixed-mode one.
``--ckpt-every k`` keeps the theta_t store in segments of k steps, ``--ckpt-slots s`` in the
binomial schedule with s snapshots, and ``--optimizer adam``
replaces the workload's SGD / momentum by Adam. Those lines skip the CPU baseline unless
``--cpu-baseline`` is given.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "decoder_large"
WORKLOAD_DESCS = {
    "wide": ("wide MLP 1024-1024x4-10 GELU, softmax-CE, B=256, T=16 SGD alpha=0.05, "
             "per-example weight logits (4096), outer batch 1024, bf16 GEMMs / fp32 state"),
    "deep": ("deep MLP 8 x 4096 SiLU, squared loss on a teacher, B=512, T=32 momentum 0.9, "
             "per-parameter log learning rates (134M), outer batch 512, bf16 GEMMs / fp32 state"),
    "decoder_small": ("decoder-only transformer 6 x d512, 8 heads, MLP 2048 GELU, vocab 8192, "
                      "S=256, B=16 sequences, T=8 SGD alpha=1e-3, per-sequence weights, outer 16, "
                      "Zipf(1.1) token ids, bf16 GEMMs / fp32 state"),
    "decoder_large": ("decoder-only transformer 12 x d1024, 16 heads, MLP 4096 GELU, vocab 32768, "
                      "S=1024, B=8, T=16 momentum 0.9, per-sequence weights + scalar log-lr, outer 8, "
                      "Zipf(1.1) token ids, bf16 GEMMs / fp32 state"),
    "toy": ("motivating example of Section 3: y_0 = x theta (4096 x 4096, no bias), M = 8 steps "
            "of y_i = i (2 + sin y_{i-1})^cos y_{i-1}, MSE on N(0,1) targets, B=1024, T=2 SGD "
            "alpha=1e-3, theta_0 meta-gradient (16.8M), outer batch 1024, bf16 GEMMs / fp32 state"),
}
WORKLOAD_DESC = WORKLOAD_DESCS[WORKLOAD]


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _max_over_ranks(x: float, ws: int, device) -> float:
    """The largest of the ranks' values (the slowest replica sets the job's time)."""
    if ws <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t)


def _job_rate(total_ms: float, steps: int, ws: int, device):
    """(ms per step of the slowest rank, whole-job meta-steps/s over all ranks)."""
    ms = _max_over_ranks(total_ms, ws, device) / steps
    return ms, ws * 1000.0 / ms


def _replica_workload(w, rank: int):
    """Replica r solves its own problem: the same shapes and distributions, seed + r."""
    return w if rank == 0 else w.with_(seed=w.seed + rank)


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return None
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm, smax, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax = max(smax, float(r[2]))
            except ValueError:
                continue
            for n, v in zip(names, r[5:9]):
                if v.lower() in ("active", "1", "yes"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


TRAFFIC_FILES = {
    "decoder_large": "tc_dual_gemm_decoder_large_traffic.json",
}


def _dram_traffic(workload):
    """Mean DRAM bytes per launch of the dominant kernel (all its launches in one call of
    the workload) from the committed ncu capture, or None when there is no capture for the
    workload or the kernel's sources changed since the counters were taken."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", TRAFFIC_FILES[workload])) as f:
            rec = json.load(f)
        h = hashlib.sha256()
        for name in rec["source_files"]:
            with open(os.path.join(ROOT, name), "rb") as src:
                h.update(src.read())
        if h.hexdigest() != rec["source_sha256"]:
            return None
        return rec["traffic_bytes_per_launch"]
    except Exception:
        return None


# ---- the float64 oracle on a bounded sample ------------------------------------------------
# The oracle's meta-gradient (Algorithm 1) is a sum of per-sequence (per-example) pieces:
# per inner step t and sequence b, the forward + backward of the rollout (inner gradient) and
# the reverse step through that sequence's part of step t (taped inner gradient); plus, once
# per meta-step, the outer gradient over the B_outer held-out sequences.  One sample unit is
# one of these pieces on ONE sequence of the workload (same shapes, same draws), and
#     oracle time per meta-step = B T (rollout + reverse) + B_outer outer.
UNIT_KINDS = ("rollout", "reverse", "outer")


_SAMPLE_INPUTS = {}


def _sample_inputs(w):
    """One-sequence, one-step inputs of workload w, drawn once per process."""
    from paper_2505_00793_gb300 import synth
    if w.name not in _SAMPLE_INPUTS:
        w1 = w.with_(B=1, T=1, B_outer=1)
        # the cotangent pulled back by the reverse unit: a seeded direction
        bar = synth.random_direction(w1.n_params, 0, 0).astype("float64")
        _SAMPLE_INPUTS[w.name] = (w1, synth.make_inputs(w1), bar)
    return _SAMPLE_INPUTS[w.name]


def oracle_unit(w, kind):
    """Wall seconds of one sample unit of the oracle on one sequence of workload w."""
    import torch
    from paper_2505_00793_gb300 import synth
    from oracle import metagrad as om
    w1, inp, bar_np = _sample_inputs(w)
    if kind == "rollout":
        t0 = time.perf_counter()
        om.rollout(w1, inp)
        return time.perf_counter() - t0
    if kind == "outer":
        t0 = time.perf_counter()
        om.grad(w1, inp.theta0, inp.outer_x, inp.outer_y)
        return time.perf_counter() - t0
    eta = om.t64(inp.eta)
    X, Y = om.t64(inp.inner_x), om.t64(inp.inner_y)
    th = om.t64(inp.theta0)
    state = tuple(torch.zeros_like(th) for _ in range(om.n_state(w1)))
    bar = torch.from_numpy(bar_np)
    s_bar = tuple(torch.zeros_like(th) for _ in range(om.n_state(w1)))
    t0 = time.perf_counter()
    om.reverse_step(w1, eta, X[0], Y[0], 0, th, state, bar, s_bar)
    return time.perf_counter() - t0


def oracle_meta_step_seconds(w, unit_s):
    """Oracle seconds per meta-step from the mean time of each unit kind."""
    return w.B * w.T * (unit_s["rollout"] + unit_s["reverse"]) + w.B_outer * unit_s["outer"]


# Workloads whose full oracle meta-gradient takes minutes are sampled by units; the others
# (the MLPs of a few million parameters, the motivating example) run whole.  One sequence is
# a GEMM-sized piece of a decoder step (1024 tokens), so the units scale; the one-sequence
# unit also repeats the parameter-sized work of a step (taped update, cotangent sums) once
# per sequence, so the estimate over-states the oracle's time somewhat.
SAMPLED = ("decoder_large", "decoder_small", "deep")


def oracle_full(w):
    """Wall seconds of the whole oracle meta-gradient of workload w."""
    from paper_2505_00793_gb300 import synth
    from oracle import metagrad as om
    inp = synth.make_inputs(w)
    t0 = time.perf_counter()
    om.meta_grad(w, inp)
    return time.perf_counter() - t0


def cpu_baseline(w, min_seconds=10.0):
    """Each unit once (about 25 s of CPU work on decoder_large), scaled to one meta-step; or,
    for the small workloads, whole oracle meta-gradients repeated for at least min_seconds."""
    import torch
    if w.name not in SAMPLED:
        runs = []
        while not runs or sum(runs) < min_seconds:
            runs.append(oracle_full(w))
        return {"value": 1.0 / statistics.mean(runs), "unit": "meta-steps/s",
                "cores": torch.get_num_threads(), "kind": "oracle",
                "sample": f"{len(runs)} whole oracle meta-gradients of the workload (T={w.T}), "
                          f"{sum(runs):.1f} s of CPU work, mean time per meta-gradient"}
    unit_s = {k: oracle_unit(w, k) for k in UNIT_KINDS}
    spent = sum(unit_s.values())
    per_step = oracle_meta_step_seconds(w, unit_s)
    return {"value": 1.0 / per_step, "unit": "meta-steps/s", "cores": torch.get_num_threads(),
            "kind": "oracle",
            "sample": (f"one sequence of the workload through one inner step of the float64 "
                       f"oracle: rollout forward+backward {unit_s['rollout']:.2f} s, reverse step "
                       f"of Algorithm 1 (taped inner gradient) {unit_s['reverse']:.2f} s, outer "
                       f"gradient {unit_s['outer']:.2f} s ({spent:.1f} s of CPU work); meta-step "
                       f"time = B*T*(rollout + reverse) + B_outer*outer = {per_step:.0f} s")}


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    import torch
    from paper_2505_00793_gb300 import synth
    w = synth.WORKLOADS[args.workload]
    if w.name in SAMPLED:
        _sample_inputs(w)
    if w.name not in SAMPLED:     # whole oracle meta-gradients, one per step
        for _ in range(args.warmup):
            oracle_full(w)
        step_s = [oracle_full(w) for _ in range(args.steps)]
        ms = 1000.0 * statistics.mean(step_s)
        value = 1000.0 / ms
        print(json.dumps({
            "impl": "reference", "metric": "meta-grad steps/s", "value": value,
            "unit": "meta-steps/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD_DESCS[args.workload]},
            "cpu_baseline": {"value": value, "unit": "meta-steps/s",
                             "cores": torch.get_num_threads(), "kind": "oracle",
                             "sample": "one whole oracle meta-gradient per step"},
            "e2e": {"value": value, "unit": "meta-steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}), flush=True)
        return 0
    # step i times sample unit UNIT_KINDS[i % 3] (a bounded piece of the oracle's work)
    for i in range(args.warmup):
        oracle_unit(w, UNIT_KINDS[i % 3])
    times = {k: [] for k in UNIT_KINDS}
    step_s = []
    t_start = time.perf_counter()
    for i in range(args.steps):
        k = UNIT_KINDS[i % 3]
        dt = oracle_unit(w, k)
        times[k].append(dt)
        step_s.append(dt)
    wall = time.perf_counter() - t_start
    for k in UNIT_KINDS:          # fewer than three timed steps: the missing kinds once more
        if not times[k]:
            times[k].append(oracle_unit(w, k))
    unit_s = {k: statistics.mean(v) for k, v in times.items()}
    per_step = oracle_meta_step_seconds(w, unit_s)
    value = 1.0 / per_step
    ms = 1000.0 * statistics.mean(step_s)
    sample = (f"step i times one sample unit, cycling rollout / reverse / outer: one sequence "
              f"of the workload through one inner step of the float64 oracle (mean s: "
              + ", ".join(f"{k} {unit_s[k]:.2f}" for k in UNIT_KINDS)
              + f"); value = 1 / (B*T*(rollout + reverse) + B_outer*outer) = 1 / {per_step:.0f} s; "
              f"ms_per_step is the measured time of one sample unit")
    print(json.dumps({
        "impl": "reference", "metric": "meta-grad steps/s", "value": value, "unit": "meta-steps/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": WORKLOAD_DESCS[args.workload]},
        "timed_wall_s": wall,
        "cpu_baseline": {"value": value, "unit": "meta-steps/s", "cores": torch.get_num_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "meta-steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)
    return 0


def _static_bytes(w, ckpt_every, inputs_bytes, out_bytes, ckpt_slots=0):
    """Section 4's static memory: the theta_t store (and the m_t store when the learning rate
    is a meta-parameter, m_t and v_t with Adam), the inputs, eta and the meta-gradient.  With
    the binomial store: its s + 3 states (theta, m when kept, v with Adam)."""
    from paper_2505_00793_gb300 import synth
    lr_meta = bool(w.meta_kind & (synth.PARAM_LOGLR | synth.SCALAR_LOGLR))
    if ckpt_slots > 0:
        n = min(ckpt_slots, max(w.T - 1, 1)) + 3
        per = 1 + (1 if (lr_meta or w.momentum != 0 or w.optimizer == "adam") else 0) + \
            (1 if w.optimizer == "adam" else 0)
        return n * per * w.n_params * 4 + inputs_bytes + out_bytes
    k = min(max(ckpt_every, 1), w.T)
    if w.optimizer == "adam":       # m_t and v_t for every t (their cotangents are dynamic)
        m_slots = 2 * (w.T // k + k - 1)
    elif lr_meta:
        m_slots = w.T // k + k - 1
    else:
        m_slots = (w.T // k + 1) if (w.momentum != 0 and k > 1) else 0
    store = ((w.T // k + k) + m_slots) * w.n_params * 4
    return store + inputs_bytes + out_bytes


def run_gpu(args):
    import torch
    import torch.distributed as dist
    from paper_2505_00793_gb300 import native, synth

    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    if ws > 1:
        dist.init_process_group("nccl")
    w = synth.WORKLOADS[args.workload]
    if args.chain_steps is not None:
        w = w.with_(extra={**w.extra, "chain_steps": args.chain_steps})
    if args.optimizer == "adam":
        w = w.with_(optimizer="adam", momentum=0.0, adam_eps=args.adam_eps)
    w = _replica_workload(w, rank)
    inp = synth.make_inputs(w)
    d = native.to_device_inputs(w, inp)
    mf = native.MixFlow.for_workload(w)
    mf.set_torch_allocator()        # the workspace shows in torch's memory statistics
    if args.gemm_persistent is not None:
        mf.set_option(native.MF_OPT_GEMM_PERSISTENT, args.gemm_persistent)
    if args.flash_attn is not None:
        mf.set_option(native.MF_OPT_FLASH_ATTN, args.flash_attn)
    if args.fused_head:
        mf.set_option(native.MF_OPT_FUSED_HEAD, 1)
    if args.layer_updates:
        mf.set_option(native.MF_OPT_LAYER_UPDATES, 1)
    rr = args.hvp_mode == "rr"
    mode = native.MF_HVP_REV_REV if rr else native.MF_HVP_MIXED_FOR
    loop = native.loop_desc_for(w, mode, ckpt_every=args.ckpt_every, ckpt_slots=args.ckpt_slots)
    d_eta = torch.empty(w.n_eta, device="cuda")
    # the meta-gradient lands in d_eta, or in d theta_0 when theta_0 is the meta-parameter
    d_th = torch.empty(w.n_params, device="cuda") if w.n_eta == 0 else None
    d_out = d_eta if d_th is None else d_th
    V = torch.empty(1, device="cuda")
    stream = torch.cuda.current_stream()
    # decoders pass the same token-id tensor as x and y: count it once
    inputs_bytes = sum(v.numel() * v.element_size() for k, v in d.items()
                       if not (k.endswith("_y") and v is d[k[:-1] + "x"]))

    def step(lp=loop):
        mf.meta_grad(lp, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th, V, stream=stream)

    # ---- peak HBM of one call (first call: eager, allocates the workspace) ---------------
    torch.cuda.synchronize()
    torch.cuda.reset_peak_memory_stats()
    base_first = torch.cuda.memory_allocated()    # inputs and outputs
    step()
    mf.sync()
    total_b = torch.cuda.max_memory_allocated()
    static_b = _static_bytes(w, args.ckpt_every, inputs_bytes, d_out.numel() * 4 + 4,
                             args.ckpt_slots)

    flush = torch.empty(256 * 1024 * 1024 // 4, device="cuda")   # > 129 MB L2
    for _ in range(max(args.warmup, 3)):
        step()
    mf.sync()

    def barrier():
        if ws > 1:
            dist.barrier()
        torch.cuda.synchronize()

    # ---- timed region: K steps, L2 flushed before each (outside the step's events) -------
    clk = ClockSampler(local)
    time.sleep(0.3)
    launches0, _ = mf.stats()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    barrier()
    for e0, e1 in evs:
        flush.fill_(1.0)
        e0.record(stream)
        step()
        e1.record(stream)
    barrier()
    clocks = clk.stop()
    mf.sync()
    launches1, _ = mf.stats()
    total_ms = sum(e0.elapsed_time(e1) for e0, e1 in evs)
    ms_per_step, value = _job_rate(total_ms, args.steps, ws, "cuda")

    # ---- dominant kernel (tcgen05 dual GEMM): the launches of one call, recorded and then
    # replayed back to back as one graph under one CUDA event pair, K times ----------------
    mf.record_gemms()
    step()
    mf.sync()
    g_ms_list, g_n, g_flops = [], 0, 0.0
    for _ in range(args.steps):
        flush.fill_(1.0)
        ms_, g_n, g_flops = mf.replay_gemms(1, stream=stream)
        g_ms_list.append(ms_)
    g_ms = statistics.mean(g_ms_list)
    peaks, peak_src = _peaks()
    g_tflops = g_flops / (g_ms * 1e-3) / 1e12 if g_ms > 0 else 0.0
    peak_tc = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])

    # ---- end to end through the public API with host buffers -------------------------------
    uniq = [k for k in d if not (k.endswith("_y") and d[k] is d[k[:-1] + "x"])]
    pin = {k: d[k].cpu().pin_memory() for k in uniq}
    h_out = torch.empty(d_out.numel(), pin_memory=True)
    h_V = torch.empty(1, pin_memory=True)
    h2d = sum(v.numel() * v.element_size() for v in pin.values())
    d2h = h_out.numel() * 4 + 4
    for _ in range(2):
        for k in uniq:
            d[k].copy_(pin[k], non_blocking=True)
        step()
        h_out.copy_(d_out, non_blocking=True)
        h_V.copy_(V, non_blocking=True)
    barrier()
    e_evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
             for _ in range(args.steps)]
    for e0, e1 in e_evs:
        flush.fill_(1.0)
        e0.record(stream)
        for k in uniq:
            d[k].copy_(pin[k], non_blocking=True)
        step()
        h_out.copy_(d_out, non_blocking=True)
        h_V.copy_(V, non_blocking=True)
        e1.record(stream)
    barrier()
    _, e2e_value = _job_rate(sum(e0.elapsed_time(e1) for e0, e1 in e_evs), args.steps, ws,
                             "cuda")
    mf.sync()
    out_main = h_out.clone()

    # ---- the other sweep of the same library, for Section 5's memory ratio: one call of the
    # reverse-over-reverse sweep (or of the mixed mode, when rr is the benchmarked one) with
    # peak HBM measured the same way, and its meta-gradient next to this one ----------------
    other = native.MF_HVP_MIXED_FOR if rr else native.MF_HVP_REV_REV
    loop_o = native.loop_desc_for(w, other, ckpt_every=args.ckpt_every,
                                  ckpt_slots=args.ckpt_slots)
    del flush
    mf.release_workspace()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    torch.cuda.reset_peak_memory_stats()
    base_b = torch.cuda.memory_allocated()
    step(loop_o)
    mf.sync()
    other_total_b = torch.cuda.max_memory_allocated() - base_b + base_first
    agree = float(torch.linalg.vector_norm(d_out.cpu() - out_main) /
                  torch.linalg.vector_norm(out_main).clamp_min(1e-30))
    dyn_main = total_b - static_b
    dyn_other = other_total_b - static_b
    mixed_dyn, ror_dyn = (dyn_other, dyn_main) if rr else (dyn_main, dyn_other)
    mixed_tot, ror_tot = (other_total_b, total_b) if rr else (total_b, other_total_b)

    out = None
    if rank == 0:
        cpu = None
        default = args.workload == WORKLOAD and not rr
        if ws == 1 and not args.no_cpu_baseline and (default or args.cpu_baseline):
            cpu = cpu_baseline(w)
        traffic = _dram_traffic(args.workload) if default and not (
            args.gemm_persistent is not None or args.fused_head or args.layer_updates) else None
        flash_desc = {0: "attention materialised per block", 1: "", 2: "warp-level fused attention only",
                      3: "tcgen05 primal attention forward too",
                      4: "warp-level fused attention backward"}
        out = {
            "metric": "meta-grad steps/s", "value": value, "unit": "meta-steps/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_DESCS[args.workload]
                       + ("; reverse-over-reverse HVPs" if rr else "")
                       + (f"; M overridden to {args.chain_steps}"
                          if args.chain_steps is not None else "")
                       + (f"; checkpoint store in segments of {args.ckpt_every} steps"
                          if args.ckpt_every > 1 else "")
                       + (f"; binomial checkpoint store with {args.ckpt_slots} snapshots "
                          f"({native.checkpoint_plan(w.T, 1, args.ckpt_slots)[1]} inner steps "
                          "recomputed)" if args.ckpt_slots > 0 else "")
                       + (f"; Adam inner optimiser (b1 0.9, b2 0.999, eps {args.adam_eps:g}) "
                          "in place of SGD" if args.optimizer == "adam" else "")
                       + (f"; persistent CTA-pair GEMM mode {args.gemm_persistent}"
                          if args.gemm_persistent is not None else "")
                       + (f"; {flash_desc[args.flash_attn]}"
                          if args.flash_attn not in (None, 1) else "")
                       + ("; output layer, loss and data product fused"
                          if args.fused_head else "")
                       + ("; per-layer updates overlapping the backward pass"
                          if args.layer_updates else ""),
                       "parallelism": f"replicas x{ws}",
                       "l2": "flushed before every timed step (256 MB write outside the step events)"},
            "roofline": {"bound": "tensor", "kernel": "tcgen05 dual GEMM (tc_dual_gemm / tc2_dual_gemm)",
                         "achieved": g_tflops, "peak": peak_tc, "unit": "TFLOP/s",
                         "frac": g_tflops / peak_tc, "traffic": traffic,
                         "peak_source": f"{peak_src} bf16_tflops_sustained",
                         "method": "the call's GEMM launches recorded, then replayed back to back "
                                   "as one graph between two CUDA events (L2 flushed before each "
                                   f"replay), mean of {args.steps} replays",
                         "launches_per_step": g_n, "flops_per_step": g_flops,
                         "ms_per_step": g_ms, "avg_launch_us": 1000.0 * g_ms / max(g_n, 1),
                         "share_of_step": g_ms / ms_per_step,
                         "within_step": g_ms <= ms_per_step},
            "hvp_tflops": g_tflops,
            "peak_hbm_gb": total_b / 1e9,
            "hbm": {"method": "torch.cuda.max_memory_allocated over one call, library workspace "
                              "routed through torch's allocator (mf_set_allocator)",
                    "total_gb": total_b / 1e9, "static_gb": static_b / 1e9,
                    "dynamic_gb": dyn_main / 1e9,
                    "hvp_mode": "reverse-over-reverse" if rr else "mixed forward-over-reverse",
                    "mixed_total_gb": mixed_tot / 1e9, "mixed_dynamic_gb": mixed_dyn / 1e9,
                    "ror_total_gb": ror_tot / 1e9, "ror_dynamic_gb": ror_dyn / 1e9,
                    "ror_over_mixed_dynamic": ror_dyn / max(mixed_dyn, 1),
                    "ror_vs_mixed_meta_grad_rel_l2": agree},
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "meta-steps/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": int(launches1 - launches0),
            "clocks": clocks,
        }
        print(json.dumps(out), flush=True)
    mf.close()
    if ws > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="mixflow", choices=["mixflow", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-baseline", action="store_true",
                    help="also time the oracle for a non-default workload or mode")
    ap.add_argument("--workload", default=WORKLOAD, choices=sorted(WORKLOAD_DESCS))
    ap.add_argument("--chain-steps", type=int, default=None,
                    help="M of the motivating example's recursion (--workload toy)")
    ap.add_argument("--hvp-mode", default="for", choices=["for", "rr"])
    ap.add_argument("--optimizer", default="sgd", choices=["sgd", "adam"],
                    help="inner optimiser (adam replaces the workload's SGD / momentum)")
    ap.add_argument("--adam-eps", type=float, default=1e-8)
    ap.add_argument("--ckpt-slots", type=int, default=0,
                    help="binomial checkpointing with this many snapshots (0 = off)")
    ap.add_argument("--ckpt-every", type=int, default=1,
                    help="segment length of the theta_t store (1 = keep every theta_t)")
    ap.add_argument("--gemm-persistent", type=int, nargs="?", const=1, default=None,
                    help="MF_OPT_GEMM_PERSISTENT mode (0 off; 1 all, duals 128-wide; 2 as 1 "
                         "but duals with K > 2048 256-wide, the library default; "
                         "3 all, duals 256-wide)")
    ap.add_argument("--flash-attn", type=int, default=None, choices=[0, 1, 2, 3, 4],
                    help="MF_OPT_FLASH_ATTN (library default 1)")
    ap.add_argument("--fused-head", action="store_true",
                    help="output layer, loss and data product in one kernel (MF_OPT_FUSED_HEAD)")
    ap.add_argument("--layer-updates", action="store_true",
                    help="per-layer updates overlapping the backward pass (MF_OPT_LAYER_UPDATES)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
