"""Benchmark: mixed-mode (forward-over-reverse) Truncated-BPTT meta-gradient steps per second.

One step = one full ``mf_meta_grad`` call on the "wide" workload: a 1024-wide, 4-hidden-layer
GELU MLP with a 10-class softmax head, B = 256 examples per inner step, T = 16 SGD steps
(alpha = 0.05), per-example weight logits (T*B = 4096 meta-parameters), outer batch 1024,
bf16 tensor-core GEMMs with float32 accumulation and float32 parameters/adjoints.  Inputs are
seeded synthetic data resident in HBM when the timed region starts.

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU float64 oracle instead.
Multi-GPU runs are independent replicas (weak scaling), one process per GPU under torchrun.

``--workload`` measures another configuration the same way (deep MLP, the two decoder-only
transformers, the motivating example of Section 3 with ``--chain-steps M``).
``--hvp-mode rr`` runs the reverse-over-reverse sweep instead of the mixed-mode one, for the
memory comparison. ``--ckpt-every k`` keeps the theta_t store in segments of k steps, and
``--optimizer adam`` replaces the workload's SGD / momentum by Adam. Those lines skip the
CPU baseline unless ``--cpu-baseline`` is given.
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

WORKLOAD = "wide"
REF_T_SAMPLE = 4
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


def _dram_traffic():
    """DRAM bytes per launch of the dominant kernel from the committed ncu capture, or None
    when the kernel's sources changed since the counters were taken."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "tc_dual_gemm_wide_traffic.json")) as f:
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


def cpu_oracle_time(w, t_sample=None, min_seconds=0.0):
    """Wall time of the float64 oracle meta-gradient on workload w, run on the first
    ``t_sample`` inner steps (all T when None) and scaled by T / t_sample.  Scaling also
    multiplies the outer-gradient part, so a sampled figure over-states the oracle's time
    slightly.  The oracle runs again until ``min_seconds`` of CPU work are spent; the time is
    the mean over the runs.  Returns (seconds for the full workload, seconds spent, threads,
    runs)."""
    import torch
    from paper_2505_00793_gb300 import synth
    from oracle import metagrad as om
    ts = w.T if t_sample is None else min(t_sample, w.T)
    ws = w.with_(T=ts)
    inp = synth.make_inputs(ws)
    spent, runs = 0.0, 0
    while runs == 0 or spent < min_seconds:
        t0 = time.perf_counter()
        om.meta_grad(ws, inp)
        spent += time.perf_counter() - t0
        runs += 1
    return spent / runs * w.T / ts, spent, torch.get_num_threads(), runs


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    from paper_2505_00793_gb300 import synth
    w = synth.WORKLOADS[WORKLOAD]
    for _ in range(args.warmup):
        cpu_oracle_time(w, REF_T_SAMPLE)
    est = []
    for _ in range(args.steps):
        full, spent, cores, _ = cpu_oracle_time(w, REF_T_SAMPLE)
        est.append(full)
    ms = 1000.0 * statistics.mean(est)
    value = 1000.0 / ms
    sample = (f"per step: oracle meta-gradient over the first {REF_T_SAMPLE} of the 16 inner "
              f"steps of the same workload, time scaled by 16/{REF_T_SAMPLE}")
    print(json.dumps({
        "impl": "reference", "metric": "meta-grad steps/s", "value": value, "unit": "meta-steps/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": WORKLOAD_DESC},
        "cpu_baseline": {"value": value, "unit": "meta-steps/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "meta-steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)
    return 0


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
    if args.gemm_persistent:
        mf.set_option(native.MF_OPT_GEMM_PERSISTENT, 1)
    if args.fused_head:
        mf.set_option(native.MF_OPT_FUSED_HEAD, 1)
    if args.layer_updates:
        mf.set_option(native.MF_OPT_LAYER_UPDATES, 1)
    rr = args.hvp_mode == "rr"
    loop = native.loop_desc_for(w, native.MF_HVP_REV_REV if rr else native.MF_HVP_MIXED_FOR,
                                ckpt_every=args.ckpt_every)
    d_eta = torch.empty(w.n_eta, device="cuda")
    # the meta-gradient lands in d_eta, or in d theta_0 when theta_0 is the meta-parameter
    d_th = torch.empty(w.n_params, device="cuda") if w.n_eta == 0 else None
    d_out = d_eta if d_th is None else d_th
    V = torch.empty(1, device="cuda")
    stream = torch.cuda.current_stream()
    flush = torch.empty(256 * 1024 * 1024 // 4, device="cuda")   # > 129 MB L2

    def step():
        mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th, V, stream=stream)

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
    launches1, peak_ws = mf.stats()
    total_ms = sum(e0.elapsed_time(e1) for e0, e1 in evs)
    ms_per_step, value = _job_rate(total_ms, args.steps, ws, "cuda")

    # ---- dominant kernel (tcgen05 dual GEMM): CUDA events around each of its launches,
    # recorded inside the replayed graph, over K more steps of the same workload ---------
    mf.set_kernel_timing(True)
    for _ in range(3):        # eager run, graph capture, first replay with timing events
        step()
    mf.sync()
    mf.kernel_time()
    g_ms = g_n = g_flops = 0.0
    t_ms = 0.0   # step time of this pass (its event nodes slow the step down a little)
    for _ in range(args.steps):
        flush.fill_(1.0)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        e1.synchronize()
        ms_, n_, fl_ = mf.kernel_time()
        g_ms += ms_; g_n += n_; g_flops += fl_
        t_ms += e0.elapsed_time(e1)
    mf.set_kernel_timing(False)
    peaks, peak_src = _peaks()
    g_tflops = g_flops / (g_ms * 1e-3) / 1e12 if g_ms > 0 else 0.0
    peak_tc = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])

    # ---- end to end through the public API with host buffers -------------------------------
    pin = {k: v.cpu().pin_memory() for k, v in d.items()}
    h_eta = torch.empty(d_out.numel(), pin_memory=True)
    h_V = torch.empty(1, pin_memory=True)
    h2d = sum(v.numel() * v.element_size() for v in pin.values())
    d2h = h_eta.numel() * 4 + 4
    for _ in range(2):
        for k in d:
            d[k].copy_(pin[k], non_blocking=True)
        step()
        h_eta.copy_(d_out, non_blocking=True)
        h_V.copy_(V, non_blocking=True)
    barrier()
    e_evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
             for _ in range(args.steps)]
    for e0, e1 in e_evs:
        flush.fill_(1.0)
        e0.record(stream)
        for k in d:
            d[k].copy_(pin[k], non_blocking=True)
        step()
        h_eta.copy_(d_out, non_blocking=True)
        h_V.copy_(V, non_blocking=True)
        e1.record(stream)
    barrier()
    _, e2e_value = _job_rate(sum(e0.elapsed_time(e1) for e0, e1 in e_evs), args.steps, ws,
                             "cuda")
    mf.sync()

    inputs_bytes = h2d
    peak_hbm_gb = (peak_ws + inputs_bytes + d_out.numel() * 4) / 1e9
    # static part (Section 4's accounting): the theta_t store (and m_t store when the learning
    # rate is a meta-parameter), the inputs, eta and d eta; the rest is the sweep's dynamic memory
    lr_meta = bool(w.meta_kind & (synth.PARAM_LOGLR | synth.SCALAR_LOGLR))
    k = min(max(args.ckpt_every, 1), w.T)
    if w.optimizer == "adam":       # m_t and v_t for every t (their cotangents are dynamic)
        m_slots = 2 * (w.T // k + k - 1)
    elif lr_meta:
        m_slots = w.T // k + k - 1
    else:
        m_slots = (w.T // k + 1) if (w.momentum != 0 and k > 1) else 0
    store = ((w.T // k + k) + m_slots) * w.n_params * 4
    static_gb = (store + inputs_bytes + d_out.numel() * 4) / 1e9

    out = None
    if rank == 0:
        cpu = None
        default = args.workload == WORKLOAD and not rr
        if ws == 1 and not args.no_cpu_baseline and (default or args.cpu_baseline):
            full_s, spent, cores, runs = cpu_oracle_time(w, min_seconds=10.0)
            cpu = {"value": 1.0 / full_s, "unit": "meta-steps/s", "cores": cores, "kind": "oracle",
                   "sample": f"{runs} full oracle meta-gradients of the workload (T={w.T}), "
                             f"{spent:.1f} s of CPU work, mean time per meta-gradient"}
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
                       + (f"; Adam inner optimiser (b1 0.9, b2 0.999, eps {args.adam_eps:g}) "
                          "in place of SGD" if args.optimizer == "adam" else "")
                       + ("; CTA-pair GEMMs as persistent kernels"
                          if args.gemm_persistent else "")
                       + ("; output layer, loss and data product fused"
                          if args.fused_head else "")
                       + ("; per-layer updates overlapping the backward pass"
                          if args.layer_updates else ""),
                       "parallelism": f"replicas x{ws}",
                       "l2": "flushed before every timed step (256 MB write outside the step events)"},
            "roofline": {"bound": "tensor", "kernel": "tc_dual_gemm_kernel (tcgen05 dual GEMM)",
                         "achieved": g_tflops, "peak": peak_tc, "unit": "TFLOP/s",
                         "frac": g_tflops / peak_tc,
                         "traffic": _dram_traffic() if args.workload == WORKLOAD else None,
                         "peak_source": f"{peak_src} bf16_tflops_sustained",
                         "launches_per_step": g_n / max(args.steps, 1),
                         "avg_launch_us": 1000.0 * g_ms / max(g_n, 1),
                         "share_of_step": g_ms / max(t_ms, 1e-9)},
            "hvp_tflops": g_tflops,
            "peak_hbm_gb": peak_hbm_gb,
            "hbm": {"total_gb": peak_hbm_gb, "static_gb": static_gb,
                    "dynamic_gb": peak_hbm_gb - static_gb,
                    "hvp_mode": "reverse-over-reverse" if rr else "mixed forward-over-reverse"},
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
    ap.add_argument("--ckpt-every", type=int, default=1,
                    help="segment length of the theta_t store (1 = keep every theta_t)")
    ap.add_argument("--gemm-persistent", action="store_true",
                    help="run CTA-pair GEMMs as persistent kernels (MF_OPT_GEMM_PERSISTENT)")
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
