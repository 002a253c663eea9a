"""Run mf_meta_grad a few times on a named case, for capturing kernels under ncu.

``python profile_run.py --case NAME [--calls N]`` prints the kernel
launches of one call (from mf_stats) and runs N eager calls (CUDA graphs off, so every launch
is visible).  The cases keep the device footprint at a few GB while the HBM-bound kernels
still move far more than the 129 MB L2 per launch:

* deep_4k       two 4096 x 4096 SiLU layers (33.6M parameters), B = 512, T = 2, momentum 0.9,
                per-parameter log learning rates: the fused update kernels (K4/K5)
* deep_4k_adam  the same with the Adam inner optimiser
* decoder_small the bench's 6 x d512 decoder (row kernels: RMSNorm, RoPE, softmax, CE)
* toy           the motivating example, M = 8 (chain loss kernels), either HVP mode
* decoder_s1024 two blocks of the larger decoder (d 1024, 16 heads, S = 1024), two
                sequences: the fused attention at the larger decoder's sequence length
* wide_small    the wide workload's shapes at T = 2 (256-row GEMMs, the 10-class head)
* decoder_large_T2  the bench workload (12 x d1024, 16 heads, S = 1024, B = 8, heavy ball,
                weights + scalar log-lr) at T = 2: every kernel of a step at full size

``--gemm-persistent``, ``--fused-head``, ``--layer-updates`` and ``--flash-attn`` set the
opt-in paths, so that
their kernels can be captured on the same cases.
"""
from __future__ import annotations

import argparse
import math


def case(name: str):
    from paper_2505_00793_gb300 import synth
    if name == "deep_4k":
        return synth.Workload("deep_4k", [4096] * 3, "silu", "squared", "bf16", B=512, T=2,
                              B_outer=512, momentum=0.9, meta_kind=synth.PARAM_LOGLR,
                              loglr_mean=math.log(1e-2), loglr_std=0.1)
    if name == "deep_4k_adam":
        return case("deep_4k").with_(name="deep_4k_adam", momentum=0.0, optimizer="adam",
                                     loglr_mean=math.log(1e-4))
    if name in ("decoder_small", "toy"):
        return synth.WORKLOADS[name]
    if name == "wide_small":
        return synth.WORKLOADS["wide"].with_(name="wide_small", T=2)
    if name == "decoder_large_T2":
        return synth.WORKLOADS["decoder_large"].with_(name="decoder_large_T2", T=2)
    if name == "decoder_s1024":
        return synth.decoder("decoder_s1024", 1024, 16, 4096, 2, 32768, 1024, B=2, T=2,
                             B_outer=2, alpha=1e-3)
    raise ValueError(name)


def main() -> None:
    import torch
    from paper_2505_00793_gb300 import native, synth

    ap = argparse.ArgumentParser()
    ap.add_argument("--case", required=True,
                    choices=["deep_4k", "deep_4k_adam", "decoder_small", "toy",
                             "decoder_s1024", "wide_small", "decoder_large_T2"])
    ap.add_argument("--calls", type=int, default=3)
    ap.add_argument("--hvp-mode", type=int, default=0)
    ap.add_argument("--gemm-persistent", type=int, nargs="?", const=1, default=None,
                    help="MF_OPT_GEMM_PERSISTENT mode (library default when absent)")
    ap.add_argument("--fused-head", action="store_true")
    ap.add_argument("--layer-updates", action="store_true")
    ap.add_argument("--flash-attn", type=int, default=None, choices=[0, 1, 2, 3, 4],
                    help="MF_OPT_FLASH_ATTN (library default when absent)")
    args = ap.parse_args()
    torch.cuda.set_device(0)
    w = case(args.case)
    inp = synth.make_inputs(w)
    d = native.to_device_inputs(w, inp)
    mf = native.MixFlow.for_workload(w)
    mf.set_option(native.MF_OPT_CUDA_GRAPHS, 0)
    if args.gemm_persistent is not None:
        mf.set_option(native.MF_OPT_GEMM_PERSISTENT, args.gemm_persistent)
    mf.set_option(native.MF_OPT_FUSED_HEAD, 1 if args.fused_head else 0)
    mf.set_option(native.MF_OPT_LAYER_UPDATES, 1 if args.layer_updates else 0)
    if args.flash_attn is not None:
        mf.set_option(native.MF_OPT_FLASH_ATTN, args.flash_attn)
    loop = native.loop_desc_for(w, args.hvp_mode)
    d_eta = torch.empty(w.n_eta, device="cuda")
    d_th = torch.empty(w.n_params, device="cuda")
    V = torch.empty(1, device="cuda")
    n0, _ = mf.stats()
    for i in range(args.calls):
        mf.meta_grad(loop, d["theta0"], d["eta"], d["inner_x"], d["inner_y"], d["outer_x"],
                     d["outer_y"], d_eta, d_th, V)
        mf.sync()
        if i == 0:
            n1, peak = mf.stats()
            print(f"{args.case}: {n1 - n0} launches per call, workspace {peak / 1e9:.2f} GB",
                  flush=True)
    mf.close()


if __name__ == "__main__":
    main()
