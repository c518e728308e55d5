"""One tcgen05 GEMM shape in isolation, for kernel profiling (ncu) and timing.

  python -m paper_2608_12703_gb300.profile_gemm --M 5120 --N 448 --K 1280 --impl 4 --reps 20

impl as in asr_spec_test_gemm (0 one pass, 2 workspace split, 4 cluster split
with wide N tiles).  Prints the mean time per call (CUDA events, each call
synchronous) and the achieved TFLOP/s.
"""
from __future__ import annotations

import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--M", type=int, default=5120)
    ap.add_argument("--N", type=int, default=448)
    ap.add_argument("--K", type=int, default=1280)
    ap.add_argument("--impl", type=int, default=4)
    ap.add_argument("--reps", type=int, default=20)
    args = ap.parse_args()
    import torch
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300 import build as B
    B.build()
    g = torch.Generator(device="cpu").manual_seed(0)
    a = torch.randn(args.M, args.K, generator=g).to(torch.bfloat16).cuda()
    b = torch.randn(args.N, args.K, generator=g).to(torch.bfloat16).cuda()
    c = torch.empty(args.M, args.N, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    for _ in range(3):
        A.asr_spec_test_gemm(args.impl, a, b, c, args.M, args.N, args.K, st)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.reps):
        A.asr_spec_test_gemm(args.impl, a, b, c, args.M, args.N, args.K, st)
    e1.record()
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / args.reps
    err = (c - a.float() @ b.float().T).abs().max().item()
    print(f"M={args.M} N={args.N} K={args.K} impl={args.impl}: {us:.1f} us per call (incl. host sync), "
          f"{2 * args.M * args.N * args.K / us / 1e6:.1f} TFLOP/s, max err {err:.3g}")


if __name__ == "__main__":
    main()
