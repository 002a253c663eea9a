"""Throughput of the tcgen05 dual GEMM (``mf_dual_gemm_bf16``) on the shapes of the
workloads, next to cuBLAS on one product of the same shape.

``python gemm_bench.py`` prints one JSON line per shape.  TF/s counts
2*M*N*K per product term; times are CUDA events over back-to-back launches with warm L2.
"""
from __future__ import annotations

import argparse
import json

# (name, M, N, K, product-term mask); masks as in include/mixflow.h
SHAPES = [
    ("wide dual forward", 256, 1024, 1024, 25),
    ("wide weight tangent", 1025, 1024, 256, 6),
    ("deep forward", 512, 4096, 4096, 1),
    ("deep dual forward", 512, 4096, 4096, 25),
    ("deep weight tangent", 4097, 4096, 512, 6),
    ("large transformer qkv dual", 8192, 3072, 1024, 25),
    ("large transformer W1 dual", 8192, 4096, 1024, 25),
    ("large transformer W2 dual", 8192, 1024, 4096, 25),
    ("large transformer Wo dual", 8192, 1024, 1024, 25),
    ("large transformer Wqkv data dual", 8192, 1024, 3072, 25),
    ("large transformer head dual", 8192, 32768, 1024, 25),
    ("large transformer head weight tangent", 1024, 32768, 8192, 6),
    ("square 8192", 8192, 8192, 8192, 1),
]


def main() -> None:
    import torch
    from paper_2505_00793_gb300 import native

    ap = argparse.ArgumentParser()
    ap.add_argument("--only", default="", help="substring of the shape names to run")
    ap.add_argument("--persistent", type=int, nargs="?", const=1, default=None,
                    help="MF_OPT_GEMM_PERSISTENT mode (library default when absent)")
    ap.add_argument("--split", action="store_true",
                    help="dual products (terms 25) as two single-accumulator launches: "
                         "C0 = A0 B0^T, then C1 = A1 B0^T + A0 B1^T")
    args = ap.parse_args()
    torch.cuda.set_device(0)
    if args.persistent is not None:   # a process-wide option, set through any handle
        from paper_2505_00793_gb300 import synth
        h = native.MixFlow.for_workload(synth.WORKLOADS["tiny"])
        h.set_option(native.MF_OPT_GEMM_PERSISTENT, args.persistent)
        h.close()
    s = torch.cuda.current_stream()
    for name, M, N, K, t in SHAPES:
        if args.only and args.only not in name:
            continue
        mk = lambda r: (torch.randn(r, K, device="cuda") * 0.1).to(torch.bfloat16)
        A0, A1, B0, B1 = mk(M), mk(M), mk(N), mk(N)
        C0 = torch.empty(M, N, device="cuda")
        C1 = torch.empty(M, N, device="cuda")
        def run():
            if args.split and t == 25:
                native.mf_dual_gemm_bf16(M, N, K, A0, A1, B0, B1, C0, None, 1, stream=s)
                native.mf_dual_gemm_bf16(M, N, K, A0, A1, B0, B1, C1, None, 2 | 4, stream=s)
            else:
                native.mf_dual_gemm_bf16(M, N, K, A0, A1, B0, B1, C0, C1, t, stream=s)
        for _ in range(3):
            run()
        torch.cuda.synchronize()
        n = 20 if M * N * K < 1e11 else 10
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(s)
        for _ in range(n):
            run()
        e1.record(s)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / n
        terms = bin(t).count("1")
        for _ in range(3):
            torch.matmul(A0, B0.t())
        torch.cuda.synchronize()
        e0.record(s)
        for _ in range(n):
            torch.matmul(A0, B0.t())
        e1.record(s)
        torch.cuda.synchronize()
        cb = e0.elapsed_time(e1) / n
        print(json.dumps({"name": name, "M": M, "N": N, "K": K, "terms": t,
                          "persistent": args.persistent, "split": args.split, "us": ms * 1e3,
                          "tflops": 2.0 * M * N * K * terms / ms / 1e9,
                          "cublas_one_product_tflops": 2.0 * M * N * K / cb / 1e9}), flush=True)
        del A0, A1, B0, B1, C0, C1
        torch.cuda.empty_cache()


if __name__ == "__main__":
    main()
