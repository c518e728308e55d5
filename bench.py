#!/usr/bin/env python
"""Benchmark of the speculative draft-verify step on GB300.

One step = one whole speculative decode of the workload's batch: the
encoder-cache build for every utterance, the prompt prefill, then verify
rounds (drafts from the synthetic draft source, longest-prefix acceptance,
commit, re-anchoring) until every utterance has its target length.
value = emitted tokens (accepted drafts + bonus tokens) per second over the
timed steps, with weights and encoder states resident in HBM.

Also reported, on the same workload: per-verify-call latency (CUDA events) over
the decode and at a fixed state (verify, rollback, verify: 20 + 100 calls), the
encoder-cache build alone,
the dominant kernel against its roofline, an end-to-end number through
host buffers, the CPU oracle on a bounded sample, and the batch-1 workload.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]

N > 1 runs under torchrun as independent replicas (one per GPU, no collective
on the data path); value is the sum over ranks divided by the slowest rank.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workload as W  # noqa: E402

MAIN_CONFIG = "large-bf16-b64-k6"
BATCH1_CONFIG = "large-bf16-b1-k8"
# the other workloads, reported as extra keys: the tiny fp32 decoder, the
# small decoder at batch 16 and one point of the batch-32 acceptance/rollback sweep
EXTRA_CONFIGS = ("small-bf16-b16-k8", "small-bf16-b32-k16-p0.2", "tiny-fp32-b1-k4")
METRIC = "accepted tokens/s"


def max_over_ranks(dist, x: float, device="cuda") -> float:
    """The largest value of x over the ranks (every rank gets it): the slowest
    replica's time bounds the whole job.  dist = torch.distributed or None."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world: int, steps: int, tokens_per_step: int, seconds_max: float) -> float:
    """Tokens of all replicas (weak scaling: each rank decodes its own batch)
    divided by the slowest rank's time."""
    return world * steps * tokens_per_step / seconds_max


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=float(d["hbm_gbs"]), bf16=float(d["bf16_tflops"]),
                    bf16_sus=float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------
class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out = ""

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------
_WEIGHTS = {}


def weights(dims):
    if dims not in _WEIGHTS:
        _WEIGHTS.clear()
        _WEIGHTS[dims] = W.make_weights(dims)
    return _WEIGHTS[dims]


class DecodeRun:
    """One workload resident on one GPU, plus the reference transcript that
    drives the synthetic draft source."""

    def __init__(self, wl: W.Workload):
        import torch
        from paper_2608_12703_gb300 import asrspec as A
        from paper_2608_12703_gb300.session import DeviceDrafts, Session
        self.torch, self.A = torch, A
        self.wl = wl
        dims = wl.dims
        self.sess = Session(dims, weights(dims), max_batch=wl.batch, max_draft=wl.k)
        enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
        self.enc_host = torch.from_numpy(enc).to(self.sess.storage_dtype).pin_memory()
        self.enc_lens = np.array(wl.enc_lens, dtype=np.int32)
        self.prompt = W.make_prompt(dims, wl.batch)
        with torch.cuda.stream(self.sess.stream):
            self.enc = self.enc_host.to("cuda")
            self.enc_lens_d = torch.from_numpy(self.enc_lens).cuda()
            self.prompt_d = torch.from_numpy(self.prompt).cuda()
        self.sess.stream.synchronize()
        self.total = np.array(wl.total_lens, dtype=np.int64)
        self.corr = W.make_corruption(wl)
        # The reference transcript that drives the drafts: the target's greedy
        # output under this workload's batching.  One-token rounds give a first
        # transcript; one speculative decode driven by it gives the transcript
        # of the speculative batching itself (a fixed point: its own greedy path).
        truth0 = self._greedy_transcript()
        self.truth, self.changed_tokens = self._speculative_transcript(DeviceDrafts, truth0)
        self.drafts = DeviceDrafts(self.sess, self.truth, self.total, self.corr, wl.k)
        self.tokens_per_decode = int(sum(wl.n_out))
        self.rounds = self._count_rounds()

    def _begin(self):
        A, s = self.A, self.sess
        A.asr_spec_encode_cache(s.h, self.wl.batch, self.enc, self.wl.t_max, self.enc_lens_d)
        s.B = self.wl.batch
        A.asr_spec_prefill(s.h, self.prompt_d, self.prompt.shape[1])

    def _greedy_transcript(self):
        """The GPU target's own greedy transcript (one token per round)."""
        B = self.wl.batch
        self._begin()
        truth = np.zeros((B, self.wl.dims.max_pos), dtype=np.int64)
        truth[:, :self.prompt.shape[1]] = self.prompt
        kv = np.full(B, self.prompt.shape[1] - 1)
        zeros = np.zeros((B, 1), dtype=np.int32)
        while True:
            active = kv + 1 < self.total
            if not active.any():
                break
            out = self.sess.verify(zeros, np.where(active, 0, -1).astype(np.int32), k=0)
            for b in np.nonzero(active)[0]:
                truth[b, kv[b] + 1] = out.bonus[b]
            kv = out.kv_len.astype(np.int64)
        assert self.sess.status() == 0
        return truth

    def _speculative_transcript(self, DeviceDrafts, truth0):
        B, k = self.wl.batch, self.wl.k
        drafts = DeviceDrafts(self.sess, truth0, self.total, self.corr, k)
        self._begin()
        seq = [list(self.prompt[b]) for b in range(B)]
        while True:
            d, l = drafts.next()
            lh = self.sess.host(l)
            if (lh < 0).all():
                break
            dh = self.sess.host(d)
            o = self.sess.host(self.sess.verify_device(d, l, k))
            for b in np.nonzero(lh >= 0)[0]:
                seq[b] += [int(t) for t in dh[b, :o[0][b]]] + [int(o[1][b])]
        truth = np.zeros_like(truth0)
        changed = 0
        for b in range(B):
            assert len(seq[b]) == self.total[b], (b, len(seq[b]), self.total[b])
            truth[b, :len(seq[b])] = seq[b]
            changed += int((truth[b, :len(seq[b])] != truth0[b, :len(seq[b])]).sum())
        assert self.sess.status() == 0
        return truth, changed

    def _count_rounds(self):
        self._begin()
        n = 0
        while True:
            d, l = self.drafts.next()
            if (self.sess.host(l) < 0).all():
                break
            self.sess.verify_device(d, l, self.wl.k)
            n += 1
        kv, _ = self.sess.state()
        assert np.array_equal(kv + 1, self.total), (kv, self.total)
        assert self.sess.status() == 0
        return n

    def decode(self, ev=None):
        """One whole decode, enqueued without host synchronisation."""
        self._begin()
        k = self.wl.k
        for _ in range(self.rounds):
            d, l = self.drafts.next()
            if ev is not None:
                e0 = self.torch.cuda.Event(enable_timing=True)
                e0.record(self.sess.stream)
            self.sess.verify_device(d, l, k)
            if ev is not None:
                e1 = self.torch.cuda.Event(enable_timing=True)
                e1.record(self.sess.stream)
                ev.append((e0, e1))

    def launches(self):
        _, launches, _ = self.A.asr_spec_profile_read(self.sess.h)
        return int(launches.sum())

    def timed(self, steps, warmup, dist=None, gpu_index=0):
        torch = self.torch
        for _ in range(warmup):
            self.decode()
        torch.cuda.synchronize()
        self.A.asr_spec_profile_read(self.sess.h)          # reset counters
        verify_ev = []
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with ClockSampler(gpu_index) as clk:
            start.record(self.sess.stream)
            for _ in range(steps):
                self.decode(verify_ev)
            end.record(self.sess.stream)
            torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
        ms = start.elapsed_time(end)
        _, launches, traffic = self.A.asr_spec_profile_read(self.sess.h)
        per_call = np.array([a.elapsed_time(b) for a, b in verify_ev]) * 1e3
        assert self.sess.status() == 0
        return dict(ms=ms, launches=int(launches.sum()) + 0, traffic=traffic, clocks=clk.summary(),
                    verify_us=dict(median=float(np.median(per_call)), p10=float(np.percentile(per_call, 10)),
                                   p90=float(np.percentile(per_call, 90)), calls=int(len(per_call))))

    def fixed_state(self, reps=100, warm=20):
        """The paper's per-step protocol: one verify call repeated at a fixed
        committed state (verify, rollback to the state, verify again), here the
        state after half of the decode's rounds.  Per-call CUDA-event times of
        `reps` calls after `warm` warm-up calls."""
        torch, A, s = self.torch, self.A, self.sess
        self._begin()
        for _ in range(self.rounds // 2):
            d, l = self.drafts.next()
            s.verify_device(d, l, self.wl.k)
        d, l = self.drafts.next()
        with torch.cuda.stream(s.stream):
            kv = torch.zeros(self.wl.batch, dtype=torch.int32, device="cuda")
            pe = torch.zeros(self.wl.batch, dtype=torch.int32, device="cuda")
        A.asr_spec_state(s.h, kv, pe)
        ev = []
        for i in range(warm + reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s.stream)
            s.verify_device(d, l, self.wl.k)
            e1.record(s.stream)
            A.asr_spec_rollback(s.h, kv, pe)
            if i >= warm:
                ev.append((e0, e1))
        torch.cuda.synchronize()
        us = np.array([a.elapsed_time(b) for a, b in ev]) * 1e3
        assert s.status() == 0
        return {"median": float(np.median(us)), "p10": float(np.percentile(us, 10)),
                "p90": float(np.percentile(us, 90)), "reps": reps, "warmup": warm,
                "state": f"after {self.rounds // 2} of {self.rounds} rounds"}

    def encode_ms(self, reps=5):
        """asr_spec_encode_cache alone (all layers' encoder K/V), CUDA events."""
        torch, A, s = self.torch, self.A, self.sess
        ev = []
        for i in range(reps + 1):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s.stream)
            A.asr_spec_encode_cache(s.h, self.wl.batch, self.enc, self.wl.t_max, self.enc_lens_d)
            e1.record(s.stream)
            if i:
                ev.append((e0, e1))
        torch.cuda.synchronize()
        return float(np.mean([a.elapsed_time(b) for a, b in ev]))

    def launch_timeline(self):
        """One decode with the launch timeline recorded (direct launches)."""
        A = self.A
        A.asr_spec_timeline(self.sess.h, True)
        self.decode()
        tl = A.asr_spec_timeline_read(self.sess.h)
        A.asr_spec_timeline(self.sess.h, False)
        return tl

    def profile(self):
        """One decode with per-kernel-class CUDA events (direct launches)."""
        A = self.A
        A.asr_spec_profile_read(self.sess.h)
        A.asr_spec_profile(self.sess.h, True)
        self.decode()
        ms, launches, traffic = A.asr_spec_profile_read(self.sess.h)
        A.asr_spec_profile(self.sess.h, False)
        return ms, launches, traffic

    def e2e(self, steps, dist=None):
        """The same decodes through host buffers: encoder states copied from pinned
        host memory every step, drafts built on the host and passed with every
        verify call, outputs read back every round.  Returns this rank's
        seconds with the rest; the caller combines the ranks."""
        torch, A = self.torch, self.A
        s = self.sess
        wl = self.wl
        h2d = d2h = 0
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(steps):
            with torch.cuda.stream(s.stream):
                enc = self.enc_host.to("cuda", non_blocking=True)
            h2d += self.enc_host.numel() * self.enc_host.element_size()
            s.set_host_io(True)
            A.asr_spec_encode_cache(s.h, wl.batch, enc, wl.t_max, self.enc_lens)
            A.asr_spec_prefill(s.h, self.prompt.astype(np.int32), self.prompt.shape[1])
            h2d += self.enc_lens.nbytes + self.prompt.astype(np.int32).nbytes
            kv = np.full(wl.batch, self.prompt.shape[1] - 1)
            while True:
                draft, lens = W.make_drafts(self.truth, self.total, kv, wl.k, self.corr)
                if np.all(lens < 0):
                    break
                out = s.verify(draft, lens)
                h2d += draft.nbytes + lens.nbytes
                d2h += 4 * out.accepted.nbytes
                kv = out.kv_len.astype(np.int64)
            s.set_host_io(False)
            del enc
        torch.cuda.synchronize()
        dt = time.perf_counter() - t0
        if dist is not None:
            dist.barrier()
        return dict(value=steps * self.tokens_per_decode / dt, unit="tokens/s",
                    h2d_bytes_per_step=int(h2d // steps), d2h_bytes_per_step=int(d2h // steps), seconds=dt)


class DraftLoop:
    """The real cached loop on the device (Sec. 3 "Speculative Loop"): each
    round the library's one-block draft proposes (catch-up of the last
    verification, restart, k - 1 continuations, audio window around the last
    anchor), the target verifies, nothing is read back in between.  The draft
    is random-init (no trained weights): its acceptance is not the paper's,
    its cost is.  rho = one draft step / one verification (Eq. breakeven),
    one draft step = a round's drafting time / k."""

    def __init__(self, wl: W.Workload, window="anchor"):
        import torch
        from paper_2608_12703_gb300.session import DraftModel, Session
        self.torch, self.wl = torch, wl
        dims = wl.dims
        self.sess = Session(dims, weights(dims), max_batch=wl.batch, max_draft=wl.k)
        self.dm = DraftModel(self.sess, W.make_draft_weights(dims), wl.total_lens, wl.k, window)
        enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
        self.prompt = W.make_prompt(dims, wl.batch)
        with torch.cuda.stream(self.sess.stream):
            self.enc = torch.from_numpy(enc).to("cuda").to(self.sess.storage_dtype)
            self.enc_lens_d = torch.from_numpy(np.array(wl.enc_lens, dtype=np.int32)).cuda()
            self.prompt_d = torch.from_numpy(self.prompt).cuda()
        self.sess.stream.synchronize()
        self.rounds, self.emitted, self.acc_sum, self.offered = self._count_rounds()

    def _begin(self):
        from paper_2608_12703_gb300 import asrspec as A
        s = self.sess
        A.asr_spec_encode_cache(s.h, self.wl.batch, self.enc, self.wl.t_max, self.enc_lens_d)
        s.B = self.wl.batch
        A.asr_spec_prefill(s.h, self.prompt_d, self.prompt.shape[1])

    def _count_rounds(self):
        self._begin()
        n = emitted = acc = offered = 0
        while True:
            d, l = self.dm.propose()
            lh = self.sess.host(l)
            if (lh < 0).all():
                break
            o = self.sess.host(self.sess.verify_device(d, l, self.wl.k))
            live = lh >= 0
            emitted += int(o[0][live].sum() + live.sum())
            acc += int(o[0][live].sum())
            offered += int(lh[live].sum())
            n += 1
        kv, _ = self.sess.state()
        assert np.array_equal(kv + 1, self.wl.total_lens), (kv, self.wl.total_lens)
        assert self.sess.status() == 0
        return n, emitted, acc, offered

    def decode(self, ev=None):
        self._begin()
        torch, k = self.torch, self.wl.k
        for _ in range(self.rounds):
            e = [torch.cuda.Event(enable_timing=True) for _ in range(3)] if ev is not None else None
            if e:
                e[0].record(self.sess.stream)
            d, l = self.dm.propose()
            if e:
                e[1].record(self.sess.stream)
            self.sess.verify_device(d, l, k)
            if e:
                e[2].record(self.sess.stream)
                ev.append(e)

    def timed(self, steps, warmup):
        torch = self.torch
        for _ in range(warmup):
            self.decode()
        torch.cuda.synchronize()
        ev = []
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(self.sess.stream)
        for _ in range(steps):
            self.decode(ev)
        end.record(self.sess.stream)
        torch.cuda.synchronize()
        assert self.sess.status() == 0
        ms = start.elapsed_time(end)
        draft_us = np.array([a.elapsed_time(b) for a, b, _ in ev]) * 1e3
        verify_us = np.array([b.elapsed_time(c) for _, b, c in ev]) * 1e3
        k = self.wl.k
        step_us = float(np.median(draft_us)) / k
        return {"workload": self.wl.name, "window": "anchor", "draft": "one-block, random-init (seeded)",
                "value": steps * self.emitted / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms / steps,
                "rounds_per_step": self.rounds, "emitted_per_step": self.emitted,
                "mean_accepted_per_round": self.acc_sum / max(self.rounds, 1),
                "acceptance_of_offered": self.acc_sum / max(self.offered, 1),
                "draft_round_us": {"median": float(np.median(draft_us)), "p10": float(np.percentile(draft_us, 10)),
                                   "p90": float(np.percentile(draft_us, 90))},
                "verify_us": {"median": float(np.median(verify_us)), "p10": float(np.percentile(verify_us, 10)),
                              "p90": float(np.percentile(verify_us, 90))},
                "draft_step_us": step_us, "rho": step_us / float(np.median(verify_us)),
                "draft_share_of_loop": float(draft_us.sum() / (draft_us.sum() + verify_us.sum())),
                "steps": steps, "warmup": warmup}


# Launch kinds of the timeline (ASR_TL_*; a LayerNorm-fused GEMM counts with its
# GEMM) and the profile class (CUDA events) that times the same kernel.
TL_KIND_CLASS = {17: "qkv", 18: "resid", 19: "query", 20: "mlp_up", 22: "lm_head", 4: "self_attn",
                 5: "cross_attn", 3: "layernorm", 8: "qkv_self", 9: "query_cross"}

# launches of a kernel class per verify call that runs it
CLASS_PER_CALL = {"qkv": 1, "resid": 3, "query": 1, "mlp_up": 1, "lm_head": 0, "self_attn": 1, "cross_attn": 1,
                  "layernorm": 3, "qkv_self": 1, "query_cross": 1}


def kind_class(kind: int):
    return TL_KIND_CLASS.get(kind - 32 if kind >= 48 else kind)


def algorithmic_work(dims, cls, traffic, n_launches):
    """(bytes, flops, per-unit statement) of one decode's launches of a kernel class.
    Bytes are the unique operands a launch must read from HBM: weights for a
    projection (its activations are L2-resident), the K/V rows for attention.
    A class's verify calls are its launches over its launches per call (the
    few-row and the tensor-core layers each run in some of a decode's calls);
    K/V bytes, counted over all calls, are shared in proportion."""
    es = 2 if dims.dtype == "bf16" else 4
    d, L, F, V = dims.d_model, dims.n_layers, dims.d_ffn, dims.vocab
    calls, self_b, cross_b, _, rows = (float(x) for x in traffic[:5])
    per_call = CLASS_PER_CALL.get(cls, 1) * L or 1
    c_calls = n_launches / per_call
    share = c_calls / calls if calls else 0.0
    mk = {"qkv": (L * 3 * d * d, "3 d^2 weights per layer"),
          "resid": (L * (2 * d * d + F * d), "d^2 + d^2 + F d weights per layer (self out, cross out, MLP down)"),
          "query": (L * d * d, "d^2 weights per layer"),
          "mlp_up": (L * F * d, "F d weights per layer"),
          "lm_head": (V * d, "V d weights")}
    if cls in mk:
        params, what = mk[cls]
        return (c_calls * params * es, 2.0 * rows * share * params,
                f"{what} x {es} bytes per verify call; 2 x scored rows x those parameters in flops")
    if cls == "self_attn":
        return self_b * share, 0.0, "2 (K, V) x (P_b + n_b) keys x d x 2 bytes per active utterance per layer"
    if cls == "cross_attn":
        return cross_b * share, 0.0, "2 (K, V) x T_b frames x d x 2 bytes per active utterance per layer"
    if cls == "qkv_self":
        params = L * 3 * d * d
        return (c_calls * params * es + self_b * share, 2.0 * rows * share * params,
                "3 d^2 weights per layer x %d bytes per verify call + the self K/V rows read (2 x (P_b + n_b) keys "
                "x d x %d bytes per active utterance per layer); 2 x scored rows x weights in flops" % (es, es))
    if cls == "query_cross":
        params = L * d * d
        return (c_calls * params * es + cross_b * share, 2.0 * rows * share * params,
                "d^2 weights per layer x %d bytes per verify call + the encoder K/V read (2 x T_b frames x d x %d "
                "bytes per active utterance per layer); 2 x scored rows x weights in flops" % (es, es))
    if cls == "layernorm":
        return rows * share * (3 * L + 1) * d * (4 + es), 0.0, "rows x d x (4 read + 2 written) bytes per LayerNorm"
    return 0.0, 0.0, ""


def roofline(wl_name, dims, tl, ms, launches, traffic, pk):
    """The kernel with the largest share of the decode (launch timeline, busy
    time past the wait on the previous kernel) against its roofline.
    achieved = algorithmic work / its CUDA-event time (each launch bracketed by
    events on the library stream, launches one by one: no overlap with the
    neighbours); the in-chain figure divides by the timeline's busy time of
    the same launches in the normal (dependent-launch) chain."""
    from paper_2608_12703_gb300.asrspec import PROF_CLASSES
    ns, kinds = tl
    busy = {}
    count = {}
    for (s, w, m, e), k in zip(ns.astype(np.int64), kinds):
        c = kind_class(int(k))
        if c is None or e == 0:
            continue
        busy[c] = busy.get(c, 0.0) + (e - (w or s)) / 1e9
        count[c] = count.get(c, 0) + 1
    total = sum(busy.values())
    name = max(busy, key=busy.get)
    ci = PROF_CLASSES.index(name)
    t = ms[ci] / 1e3
    n = int(launches[ci])
    nbytes, flops, per_unit = algorithmic_work(dims, name, traffic, n)
    balance = pk["bf16_sus"] * 1e12 / (pk["hbm"] * 1e9)
    if flops > 0 and flops / nbytes > balance:
        bound, unit, peak, work, scale = "tensor", "TFLOP/s", pk["bf16_sus"], flops, 1e12
    else:
        bound, unit, peak, work, scale = "hbm", "GB/s", pk["hbm"], nbytes, 1e9
    achieved = work / t / scale
    chain = work / busy[name] / scale
    from paper_2608_12703_gb300.ncu_traffic import lookup
    ncu = lookup(wl_name, name)   # None unless captured on the kernel's current sources
    return {"kernel": name, "bound": bound, "achieved": round(achieved, 2), "peak": peak, "unit": unit,
            "frac": round(achieved / peak, 4), "traffic": ncu[0] if ncu else None,
            "traffic_source": ncu[1] if ncu else None,
            "algorithmic_bytes_per_launch": round(nbytes / max(n, 1), 1), "launches": n,
            "ms_per_launch": round(ms[ci] / max(n, 1), 5), "per_unit": per_unit,
            "units": "work summed over the decode's launches of the kernel; per launch = that / launches",
            "peak_source": pk["src"],
            "share_of_busy_time": round(busy[name] / total, 4),
            "in_chain": {"achieved": round(chain, 2), "frac": round(chain / peak, 4),
                         "us_per_launch": round(1e6 * busy[name] / max(count[name], 1), 3),
                         "timer": "GPU global timer, first CTA past its wait to last CTA exit"},
            "class_ms": {PROF_CLASSES[i]: round(float(ms[i]), 3) for i in range(len(ms))},
            "busy_share": {k: round(v / total, 4) for k, v in sorted(busy.items(), key=lambda kv: -kv[1])}}


def step_bytes(dims, traffic, calls_override=None):
    """Algorithmic bytes per verify call (weights + LM head + K/V reads)."""
    es = 2 if dims.dtype == "bf16" else 4
    d, L, F, V = dims.d_model, dims.n_layers, dims.d_ffn, dims.vocab
    calls = int(traffic[0]) if calls_override is None else calls_override
    w = L * (6 * d * d + 2 * F * d) * es + V * d * es
    kv = float(traffic[1]) + float(traffic[2]) + float(traffic[3])
    return (calls * w + kv) / max(calls, 1)


def extra_config(wl: W.Workload, pk, gpu_index: int, cpu_seconds: float, steps: int = 2, warmup: int = 3):
    """One more workload: whole-decode tokens/s, per-call verify latency, the
    verify step's HBM fraction, and the oracle on a bounded sample of it (the
    whole decode where it fits the time)."""
    run = DecodeRun(wl)
    res = run.timed(steps, warmup, None, gpu_index=gpu_index)
    _, _, traffic = run.profile()
    bpc = step_bytes(wl.dims, traffic)
    med = res["verify_us"]["median"]
    tokens, dt, rounds, desc = oracle_sample(wl, run.truth, cpu_seconds)
    out = {"value": steps * run.tokens_per_decode / (res["ms"] / 1e3), "unit": "tokens/s",
           "ms_per_step": res["ms"] / steps, "steps": steps, "warmup": warmup,
           "dtype": "bf16" if wl.dims.dtype == "bf16" else "f32", "batch": wl.batch, "k": wl.k,
           "verify_us": res["verify_us"], "verify_rounds_per_step": run.rounds,
           "verify_hbm": {"bytes_per_call": bpc, "frac": bpc / (med * 1e-6) / (pk["hbm"] * 1e9),
                          "frac_nominal_8tbs": bpc / (med * 1e-6) / 8e12},
           "clocks": res["clocks"], "gpu_launches": res["launches"],
           "cpu_baseline": {"value": tokens / dt, "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
                            "seconds_per_verify_round": dt / max(rounds, 1), "sample": desc}}
    run.sess.close()
    del run
    return out


# ----------------------------------------------------------------------------
# CPU oracle arm
# ----------------------------------------------------------------------------
def oracle_sample(wl: W.Workload, truth, seconds: float, utt: int = 0, rounds_cap=None):
    """The oracle on utterance `utt` of the workload: encoder cache, prefill,
    then verify rounds with the workload's drafts until that many seconds are spent.
    Returns (tokens emitted, seconds, rounds, description)."""
    from oracle import Oracle
    dims = wl.dims
    enc = W.make_encoder_states(dims, [wl.enc_lens[utt]], wl.t_max)
    t0 = time.perf_counter()
    orc = Oracle(dims, weights(dims))
    t_setup = time.perf_counter() - t0
    t0 = time.perf_counter()
    orc.encode_cache(enc, [wl.enc_lens[utt]])
    prompt = W.make_prompt(dims, 1)
    orc.prefill(prompt)
    corr = W.make_corruption(wl)
    sub = W.Corruption(corr.repl[utt:utt + 1], corr.shift[utt:utt + 1])
    total = [wl.total_lens[utt]]
    tokens = rounds = 0
    while time.perf_counter() - t0 < seconds and (rounds_cap is None or rounds < rounds_cap):
        draft, lens = W.make_drafts(truth[utt:utt + 1], total, orc.kv_len, wl.k, sub)
        if lens[0] < 0:
            break
        r = orc.verify(draft, lens)
        tokens += int(r.accepted[0]) + 1
        rounds += 1
    dt = time.perf_counter() - t0
    desc = (f"utterance {utt} of {wl.name} (T={wl.enc_lens[utt]} frames): encoder cache + prefill + "
            f"{rounds} verify rounds, {tokens} tokens; weight widening ({t_setup:.1f} s) not timed")
    return tokens, dt, rounds, desc


def cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n and n[0]:
            return int(n[0])
    except Exception:
        pass
    return os.cpu_count() or 1


# ----------------------------------------------------------------------------
def base_line(args, wl, n_gpus):
    return {"metric": METRIC, "unit": "tokens/s", "n_gpus": n_gpus, "steps": args.steps,
            "warmup": args.warmup, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if wl.dims.dtype == "bf16" else "f32",
            "data": "synthetic (seeded random-init weights and encoder states shaped like the paper's workloads)",
            "config": {"workload": wl.name, "batch": wl.batch, "k": wl.k, "layers": wl.dims.n_layers,
                       "d_model": wl.dims.d_model, "vocab": wl.dims.vocab,
                       "tokens_per_step": int(sum(wl.n_out)), "parallelism": f"replicas x{n_gpus}",
                       "l2": "inputs larger than L2 (weights and encoder K/V exceed 129 MB per verify call)"}}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = W.CONFIGS[args.config]
    # the reference transcript for the drafts: the oracle's own greedy decoding
    from oracle import Oracle, greedy_transcript
    dims = wl.dims
    utt = 0
    n_total = min(wl.total_lens[utt], W.PROMPT_LEN + 12)
    enc = W.make_encoder_states(dims, [wl.enc_lens[utt]], wl.t_max)
    orc = Oracle(dims, weights(dims))
    orc.encode_cache(enc, [wl.enc_lens[utt]])
    prompt = W.make_prompt(dims, 1)
    orc.prefill(prompt)
    truth = np.zeros((1, dims.max_pos), dtype=np.int64)
    tr = greedy_transcript(orc, prompt, [n_total])
    truth[0, :tr.shape[1]] = tr[0]
    corr = W.make_corruption(wl)
    sub = W.Corruption(corr.repl[utt:utt + 1], corr.shift[utt:utt + 1])
    times, toks = [], []
    for i in range(args.warmup + args.steps):
        orc.rollback([W.PROMPT_LEN - 1], [prompt[0, -1]])
        t0 = time.perf_counter()
        n = 0
        while True:
            draft, lens = W.make_drafts(truth, [n_total], orc.kv_len, wl.k, sub)
            if lens[0] < 0:
                break
            r = orc.verify(draft, lens)
            n += int(r.accepted[0]) + 1
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
            toks.append(n)
    value = sum(toks) / sum(times)
    line = base_line(args, wl, 1)
    cores = cpu_threads()
    sample = (f"utterance {utt} of {wl.name}: decode of {n_total - W.PROMPT_LEN} tokens by verify rounds "
              f"from a prefilled cache, per step")
    line.update({"impl": "reference", "value": value, "ms_per_step": 1e3 * float(np.mean(times)),
                 "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                                  "sample": sample},
                 "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                         "d2h_bytes_per_step": 0}})
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default=MAIN_CONFIG, choices=sorted(W.CONFIGS))
    ap.add_argument("--batch1-config", default=BATCH1_CONFIG)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-batch1", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-extra", action="store_true", help="skip the draft loops and the other workloads")
    ap.add_argument("--cpu-seconds", type=float, default=20.0)
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)

    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as tdist
        tdist.init_process_group("nccl", device_id=torch.device("cuda", local))
        dist = tdist
    from paper_2608_12703_gb300 import build as B
    if rank == 0:
        B.build()
    if dist is not None:
        dist.barrier()
    B.build()
    pk = peaks()
    wl = W.CONFIGS[args.config]
    run = DecodeRun(wl)
    res = run.timed(args.steps, args.warmup, dist, gpu_index=local)
    ms = max_over_ranks(dist, res["ms"])
    value = whole_job_rate(world, args.steps, run.tokens_per_decode, ms / 1e3)
    prof_ms, prof_launches, prof_traffic = run.profile()
    tl = run.launch_timeline()
    fixed = run.fixed_state()
    enc_ms = run.encode_ms()
    line = base_line(args, wl, world)
    bytes_per_call = step_bytes(wl.dims, prof_traffic)
    line.update({
        "value": value, "ms_per_step": ms / args.steps,
        "verify_us": res["verify_us"],
        "fixed_state_verify_us": fixed,
        "encode_cache_ms": enc_ms,
        "verify_rounds_per_step": run.rounds,
        "transcript_tokens_changed_by_batching": run.changed_tokens,
        "verify_hbm": {"bytes_per_call": bytes_per_call,
                       "frac": bytes_per_call / (res["verify_us"]["median"] * 1e-6) / (pk["hbm"] * 1e9),
                       "frac_nominal_8tbs": bytes_per_call / (res["verify_us"]["median"] * 1e-6) / 8e12},
        "clocks": res["clocks"],
        "gpu_launches": res["launches"] + 0,
        "roofline": roofline(wl.name, wl.dims, tl, prof_ms, prof_launches, prof_traffic, pk),
    })
    if not args.no_e2e:
        e2e_steps = max(1, min(args.steps, 2))
        e2e = run.e2e(e2e_steps, dist)
        e2e["value"] = whole_job_rate(world, e2e_steps, run.tokens_per_decode, max_over_ranks(dist, e2e.pop("seconds")))
        line["e2e"] = e2e
    if rank == 0:
        # CPU oracle on a bounded sample of the same workload
        tokens, dt, rounds, desc = oracle_sample(wl, run.truth, args.cpu_seconds)
        line["cpu_baseline"] = {"value": tokens / dt, "unit": "tokens/s", "cores": cpu_threads(),
                                "kind": "oracle", "sample": desc}
        if not args.no_batch1 and args.batch1_config != args.config:
            del run
            torch.cuda.empty_cache()
            wl1 = W.CONFIGS[args.batch1_config]
            r1 = DecodeRun(wl1)
            b1 = r1.timed(args.steps, args.warmup, None, gpu_index=local)
            pm, pl, pt = r1.profile()
            tl1 = r1.launch_timeline()
            fixed1 = r1.fixed_state()
            enc1 = r1.encode_ms()
            bpc = step_bytes(wl1.dims, pt)
            line["batch1"] = {
                "workload": wl1.name, "value": args.steps * r1.tokens_per_decode / (b1["ms"] / 1e3),
                "unit": "tokens/s", "ms_per_step": b1["ms"] / args.steps, "verify_us": b1["verify_us"],
                "fixed_state_verify_us": fixed1, "encode_cache_ms": enc1,
                "verify_rounds_per_step": r1.rounds,
                "verify_hbm": {"bytes_per_call": bpc,
                               "frac": bpc / (b1["verify_us"]["median"] * 1e-6) / (pk["hbm"] * 1e9),
                               "frac_nominal_8tbs": bpc / (b1["verify_us"]["median"] * 1e-6) / 8e12},
                "clocks": b1["clocks"], "roofline": roofline(wl1.name, wl1.dims, tl1, pm, pl, pt, pk)}
            del r1
        if not args.no_extra:
            line["draft_loop"] = {}
            for name in (BATCH1_CONFIG, args.config):
                torch.cuda.empty_cache()
                dl = DraftLoop(W.CONFIGS[name])
                line["draft_loop"][name] = dl.timed(2, 3)
                dl.sess.close()
                del dl
            line["configs"] = {}
            for name in EXTRA_CONFIGS:
                torch.cuda.empty_cache()
                line["configs"][name] = extra_config(W.CONFIGS[name], pk, local, args.cpu_seconds)
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
