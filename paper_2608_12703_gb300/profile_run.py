"""Small, fixed verify workload for kernel profiling (ncu) and quick timing.

Builds one workload's decoder and utterances, prefills, then runs `--warmup`
and `--rounds` verify rounds with k drafts per utterance (all rows scored
every round, the heaviest round shape), and prints the per-round time from
CUDA events on the library's stream.

  python -m paper_2608_12703_gb300.profile_run --config large-bf16-b1-k8 --warmup 2 --rounds 3

Options: --classes (CUDA-event time per kernel class), --timeline (the launch
timeline per launch kind), --fewrow-trace (per-CTA phase stamps of the
few-row launches), --tree-nodes N (tree verifies beside the linear one), --enc-len T
(encoder memories of T frames), --batch-sweep 1,4,16,64 (verification cost and
anchor-readout share against batch size), --gemm IMPL,M,N,K (one GEMM shape
through the kernel test entry, for captures of a single kernel).

Kernel launches per round (bf16 decoders): at most 9 rows (e.g. batch 1):
2 + 6 per layer + 3 (few-row layers, final LayerNorm, LM head, accept);
more rows: 2 + 8 per layer + 2 (tensor-core chain, LayerNorm folded).
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


def timeline_summary(ns, kinds, rounds):
    """Per launch kind: launches per round, mean busy time (end - past the wait),
    its part up to the kernel's midpoint (GEMM: MMAs done; attention: key loop
    done), the mean gap from the previous launch's end to this one's
    past-the-wait point, and the shares of the recorded span."""
    from paper_2608_12703_gb300 import asrspec as A
    ns = ns.astype(np.int64)
    ok = ns[:, 3] > 0
    t0 = ns[ok, 0].min() if ok.any() else 0
    span = (ns[ok, 3].max() - t0) / 1e3 if ok.any() else 0.0
    rows = {}
    prev_end = None
    for (s, w, m, e), k in zip(ns, kinds):
        if e == 0:
            continue
        w = w or s
        r = rows.setdefault(int(k), [0, 0.0, 0.0, 0.0])
        r[0] += 1
        r[1] += (e - w) / 1e3
        r[2] += (m - w) / 1e3 if m else 0.0
        if prev_end is not None:
            r[3] += (w - prev_end) / 1e3
        prev_end = e
    lines = [f"  launch timeline over {rounds} rounds: span {span:.1f} us ({span / max(rounds, 1):.1f} us per round), "
             f"{int(ok.sum())} launches recorded"]
    lines.append(f"  {'kind':<20}{'per round':>10}{'busy us':>10}{'to mid':>9}{'gap us':>9}{'busy %':>9}{'gap %':>8}")
    for k, (n, busy, mid, gap) in sorted(rows.items(), key=lambda kv: -(kv[1][1] + kv[1][3])):
        lines.append(f"  {A.tl_kind_name(k):<20}{n / rounds:>10.1f}{busy / n:>10.2f}{mid / n:>9.2f}{gap / n:>9.2f}"
                     f"{100 * busy / span:>9.1f}{100 * gap / span:>8.1f}")
    return "\n".join(lines)


FEWROW_KINDS = ["qkv_self", "self_out", "query_cross", "cross_out", "mlp_up", "mlp_down"]
FEWROW_PHASES = ["entry", "past_wait", "rows", "weights", "reduced", "exchange", "attention", "exit", "kv_in",
                 "combined", "merge_in", "inputs_in"]


def fewrow_trace_summary(tr):
    """Per few-row launch kind (averaged over layers): each phase's median and
    maximum over CTAs, in us after the previous launch's last exit (negative:
    the CTA was resident before it), and the launch's span from that exit to
    its own last exit."""
    tr = tr.astype(np.int64)
    n = tr.shape[0]
    lines = [f"  few-row trace: {n} launches; us after the previous launch's last CTA exit, median / max over CTAs"]
    lines.append("  " + f"{'kind':<12}" + "".join(f"{p:>16}" for p in FEWROW_PHASES) + f"{'span':>9}")
    acc = {k: [] for k in FEWROW_KINDS}
    for i in range(1, n):
        prev_exit = tr[i - 1][:, 7].max()
        cta = tr[i][:, 0] > 0
        with np.errstate(all="ignore"):
            rel = np.where(tr[i][cta] > 0, (tr[i][cta] - prev_exit) / 1e3, np.nan)
        acc[FEWROW_KINDS[i % 6]].append(rel)
    import warnings
    warnings.simplefilter("ignore", RuntimeWarning)
    for k in FEWROW_KINDS:
        if not acc[k]:
            continue
        med = np.nanmean([np.nanmedian(r, axis=0) for r in acc[k]], axis=0)
        mx = np.nanmean([np.nanmax(r, axis=0) for r in acc[k]], axis=0)
        cells = "".join(f"{a:>8.2f}/{b:<7.2f}" if np.isfinite(a) else f"{'-':>16}"
                        for a, b in zip(med[:12], mx[:12]))
        lines.append(f"  {k:<12}{cells}{mx[7]:>9.2f}")
    return "\n".join(lines)


GEMM_KINDS = ["qkv", "self_out", "cross_query", "cross_out", "mlp_up", "mlp_down"]
GEMM_PHASES = ["setup", "past_wait", "first_full", "loads_out", "mma_done", "staged", "landed", "epi_ready",
               "first_rows", "reduced", "end"]


def gemm_trace_summary(tr):
    """Per many-row projection (averaged over layers): each phase's median and
    maximum over CTAs, in us after the launch's first CTA entry (phases 1, 8,
    2, 9, 3, 5, 6, 10, 11, 7, 4 of the GEMM's stamps)."""
    tr = tr.astype(np.int64)
    lines = [f"  GEMM trace: {tr.shape[0]} launches; us after the launch's first CTA entry, median / max over CTAs"]
    lines.append("  " + f"{'kind':<12}{'CTAs':>6}" + "".join(f"{p:>16}" for p in GEMM_PHASES))
    acc = {k: [] for k in GEMM_KINDS}
    for i in range(tr.shape[0]):
        cta = tr[i][:, 0] > 0
        if not cta.any():
            continue
        t0 = tr[i][cta, 0].min()
        with np.errstate(all="ignore"):
            rel = np.where(tr[i][cta] > 0, (tr[i][cta] - t0) / 1e3, np.nan)
        acc[GEMM_KINDS[i % 6]].append(rel)
    import warnings
    warnings.simplefilter("ignore", RuntimeWarning)
    for k in GEMM_KINDS:
        if not acc[k]:
            continue
        cols = [1, 8, 2, 9, 3, 5, 6, 10, 11, 7, 4]
        med = np.nanmean([np.nanmedian(r, axis=0) for r in acc[k]], axis=0)
        mx = np.nanmean([np.nanmax(r, axis=0) for r in acc[k]], axis=0)
        cells = "".join(f"{med[c]:>8.2f}/{mx[c]:<7.2f}" if np.isfinite(med[c]) else f"{'-':>16}" for c in cols)
        lines.append(f"  {k:<12}{acc[k][0].shape[0]:>6}{cells}")
    return "\n".join(lines)


def gemm_only(args):
    """One GEMM shape through the kernel test entry, timed with CUDA events."""
    import torch
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300 import build as B
    B.build()
    impl, M, N, K = (int(x) for x in args.gemm.split(","))
    g = torch.Generator(device="cpu").manual_seed(0)
    a = (0.25 * torch.randn(M, K, generator=g)).to(torch.bfloat16).cuda()
    b = torch.randn(N, K, generator=g).to(torch.bfloat16).cuda()
    c = torch.empty((max(M, N), max(M, N)), device="cuda")
    st = torch.cuda.current_stream()
    us = []
    for i in range(args.warmup + args.rounds):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        A.asr_spec_test_gemm(impl, a, b, c, M, N, K, st.cuda_stream)
        e1.record(st)
        torch.cuda.synchronize()
        if i >= args.warmup:
            us.append(e0.elapsed_time(e1) * 1e3)
    print(f"gemm impl {impl} M {M} N {N} K {K}: us per call (with the entry's set-up) "
          + " ".join(f"{u:.1f}" for u in us))


def batch_sweep(batches, k, rounds, warmup):
    """Verification cost against batch size on the large decoder: the first B
    utterances of the 64-utterance workload (ragged encoder lengths), k drafts
    each, all rows scored; per round the CUDA-event time of the verify call
    (graph replay) and, from the launch timeline, the time of the acceptance +
    anchor-readout kernel, whose ratio to the verify call is the runtime
    correction's cost on the scale of one target verification (the quantity
    the paper's cost condition compares with the gain in accepted length)."""
    import torch
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300.session import Session
    base = W.CONFIGS["large-bf16-b64-k6"]
    dims = base.dims
    blob = W.make_weights(dims)
    rng = np.random.default_rng(5)
    lines = [f"  {'batch':>6}{'rows':>6}{'verify us':>11}{'per utt us':>12}{'accept+anchor us':>18}{'readout / verify':>18}"]
    for B in batches:
        enc_lens = list(base.enc_lens[:B])
        t_max = max(enc_lens)
        sess = Session(dims, blob, max_batch=B, max_draft=k)
        sess.encode_cache(W.make_encoder_states(dims, enc_lens, t_max), enc_lens)
        sess.prefill(W.make_prompt(dims, B))
        with torch.cuda.stream(sess.stream):
            drafts = [torch.from_numpy(rng.integers(0, dims.vocab, size=(B, k)).astype(np.int32)).cuda()
                      for _ in range(warmup + rounds)]
            lens = torch.full((B,), k, dtype=torch.int32, device="cuda")
        sess.stream.synchronize()
        times = []
        for i in range(warmup + rounds):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(sess.stream)
            sess.verify_device(drafts[i], lens, k)
            e1.record(sess.stream)
            if i >= warmup:
                times.append((e0, e1))
        torch.cuda.synchronize()
        us = float(np.median([a.elapsed_time(b) * 1e3 for a, b in times]))
        A.asr_spec_timeline(sess.h, True)
        for i in range(rounds):
            sess.verify_device(drafts[i], lens, k)
        ns, kinds = A.asr_spec_timeline_read(sess.h)
        A.asr_spec_timeline(sess.h, False)
        ns = ns.astype(np.int64)
        acc = ns[kinds == 6]
        acc_us = float(np.median((acc[:, 3] - np.where(acc[:, 1] > 0, acc[:, 1], acc[:, 0])) / 1e3))
        st = sess.status()
        sess.close()
        if st:
            raise RuntimeError(f"status {st} at batch {B}")
        lines.append(f"  {B:>6}{B * (k + 1):>6}{us:>11.1f}{us / B:>12.1f}{acc_us:>18.2f}{acc_us / us:>18.4f}")
    return "\n".join(lines)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--config", default="large-bf16-b1-k8", choices=sorted(W.CONFIGS))
    ap.add_argument("--warmup", type=int, default=2)
    ap.add_argument("--rounds", type=int, default=3)
    ap.add_argument("--no-graphs", action="store_true")
    ap.add_argument("--classes", action="store_true",
                    help="also time each kernel class with CUDA events (direct launches)")
    ap.add_argument("--timeline", action="store_true",
                    help="also record the launch timeline of the rounds (direct launches) and summarise it per kind")
    ap.add_argument("--fewrow-trace", action="store_true",
                    help="also record the per-CTA phase stamps of one verify's few-row launches (more rows: its "
                         "tensor-core projections) and summarise them")
    ap.add_argument("--batch-sweep", default="",
                    help="comma-separated batch sizes: verification cost and anchor-readout share of the large "
                         "decoder at each (replaces the single-workload run)")
    ap.add_argument("--k", type=int, default=6, help="drafts per utterance of --batch-sweep")
    ap.add_argument("--enc-len", type=int, default=0,
                    help="encoder frames of every utterance instead of the workload's (long-form audio: > 1500)")
    ap.add_argument("--tree-nodes", type=int, default=0,
                    help="also time tree verifies of this many nodes per utterance (random trees whose first k "
                         "nodes form one branch) beside the linear verify")
    ap.add_argument("--gemm", default="",
                    help="IMPL,M,N,K: run only the GEMM test entry (asr_spec_test_gemm) with random bf16 operands, "
                         "--warmup + --rounds times, and print the per-call time")
    args = ap.parse_args()
    if args.gemm:
        return gemm_only(args)
    if args.batch_sweep:
        from paper_2608_12703_gb300 import build as B
        B.build()
        batches = [int(b) for b in args.batch_sweep.split(",")]
        print(f"large decoder, k = {args.k}, median of {args.rounds} verify rounds after {args.warmup} warm-up:")
        print(batch_sweep(batches, args.k, args.rounds, args.warmup))
        return

    import torch
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300 import build as B
    from paper_2608_12703_gb300.session import Session

    B.build()
    wl = W.CONFIGS[args.config]
    if args.enc_len:
        import dataclasses
        dims = dataclasses.replace(wl.dims, max_enc=max(wl.dims.max_enc, args.enc_len))
        wl = dataclasses.replace(wl, dims=dims, enc_lens=(args.enc_len,) * wl.batch, t_max=args.enc_len)
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
    if args.timeline:
        A.asr_spec_timeline(sess.h, True)
        for i in range(args.rounds):
            sess.verify_device(drafts[i], lens, wl.k)
        ns, kinds = A.asr_spec_timeline_read(sess.h)
        A.asr_spec_timeline(sess.h, False)
        print(timeline_summary(ns, kinds, args.rounds))
    if args.fewrow_trace:
        A.asr_spec_fewrow_trace(sess.h, True)
        sess.verify_device(drafts[0], lens, wl.k)
        tr = A.asr_spec_fewrow_trace_read(sess.h)
        A.asr_spec_fewrow_trace(sess.h, False)
        if dims.dtype == "bf16" and wl.batch * (wl.k + 1) > 9:
            print(gemm_trace_summary(tr))
        else:
            print(fewrow_trace_summary(tr))
    if args.tree_nodes:
        n = args.tree_nodes
        trng = np.random.default_rng(9)
        tsess = Session(dims, W.make_weights(dims), max_batch=wl.batch, max_draft=max(n, wl.k))
        tsess.encode_cache(W.make_encoder_states(dims, wl.enc_lens, wl.t_max), list(wl.enc_lens))
        tsess.prefill(W.make_prompt(dims, wl.batch))
        parent = np.array([[trng.integers(0, i + 1) if i >= wl.k else i for i in range(n)]
                           for _ in range(wl.batch)], dtype=np.int32)
        with torch.cuda.stream(tsess.stream):
            tok_d = [torch.from_numpy(trng.integers(0, dims.vocab, size=(wl.batch, n)).astype(np.int32)).cuda()
                     for _ in range(args.warmup + args.rounds)]
            par_d = torch.from_numpy(parent).cuda()
            lens_t = torch.full((wl.batch,), n, dtype=torch.int32, device="cuda")
            path_d = torch.zeros((wl.batch, n), dtype=torch.int32, device="cuda")
        tsess.stream.synchronize()
        o = tsess.out[:, :wl.batch]
        tt = []
        for i in range(args.warmup + args.rounds):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(tsess.stream)
            A.asr_spec_verify_tree(tsess.h, tok_d[i], par_d, lens_t, n, o[0], o[1], o[2], o[3], path_d)
            e1.record(tsess.stream)
            if i >= args.warmup:
                tt.append((e0, e1))
        torch.cuda.synchronize()
        tus = [a.elapsed_time(b) * 1e3 for a, b in tt]
        print(f"  tree verify, {n} nodes per utterance: us per round " + " ".join(f"{u:.1f}" for u in tus)
              + f"; status {tsess.status()}")
        tsess.close()
    sess.close()
    if st:
        sys.exit(1)


if __name__ == "__main__":
    main()
