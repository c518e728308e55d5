"""Small, fixed verify workload for kernel profiling (ncu) and quick timing.

Builds one workload's decoder and utterances, prefills, then runs `--warmup`
and `--rounds` verify rounds with k drafts per utterance (all rows scored
every round, the heaviest round shape), and prints the per-round time from
CUDA events on the library's stream.

  python -m paper_2608_12703_gb300.profile_run --config large-bf16-b1-k8 --warmup 2 --rounds 3

Kernel launches per round (bf16 decoders): 2 + 12 per layer + 4.
"""
from __future__ import annotations

import argparse
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workload as W  # noqa: E402


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--config", default="large-bf16-b1-k8", choices=sorted(W.CONFIGS))
    ap.add_argument("--warmup", type=int, default=2)
    ap.add_argument("--rounds", type=int, default=3)
    ap.add_argument("--no-graphs", action="store_true")
    ap.add_argument("--classes", action="store_true",
                    help="also time each kernel class with CUDA events (direct launches)")
    args = ap.parse_args()

    import torch
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300 import build as B
    from paper_2608_12703_gb300.session import Session

    B.build()
    wl = W.CONFIGS[args.config]
    dims = wl.dims
    sess = Session(dims, W.make_weights(dims), max_batch=wl.batch, max_draft=wl.k)
    if args.no_graphs:
        A.asr_spec_set_graphs(sess.h, False)
    sess.encode_cache(W.make_encoder_states(dims, wl.enc_lens, wl.t_max), list(wl.enc_lens))
    sess.prefill(W.make_prompt(dims, wl.batch))
    rng = np.random.default_rng(5)
    with torch.cuda.stream(sess.stream):
        drafts = [torch.from_numpy(rng.integers(0, dims.vocab, size=(wl.batch, wl.k)).astype(np.int32)).cuda()
                  for _ in range(args.warmup + args.rounds)]
        lens = torch.full((wl.batch,), wl.k, dtype=torch.int32, device="cuda")
    sess.stream.synchronize()
    times = []
    for i in range(args.warmup + args.rounds):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(sess.stream)
        sess.verify_device(drafts[i], lens, wl.k)
        e1.record(sess.stream)
        if i >= args.warmup:
            times.append((e0, e1))
    torch.cuda.synchronize()
    us = [a.elapsed_time(b) * 1e3 for a, b in times]
    st = sess.status()
    print(f"{wl.name}: verify rounds {len(us)}, us per round: " + " ".join(f"{u:.1f}" for u in us)
          + f"; status {st}")
    if args.classes:
        A.asr_spec_profile_read(sess.h)
        A.asr_spec_profile(sess.h, True)
        for i in range(args.rounds):
            sess.verify_device(drafts[i], lens, wl.k)
        ms, launches, _ = A.asr_spec_profile_read(sess.h)
        A.asr_spec_profile(sess.h, False)
        print("  per round (us, event-bracketed direct launches): " + ", ".join(
            f"{n} {1e3 * m / args.rounds:.0f}" for n, m in zip(A.PROF_CLASSES, ms)))
    sess.close()
    if st:
        sys.exit(1)


if __name__ == "__main__":
    main()
