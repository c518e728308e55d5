"""A thin owner of one libasrspec handle plus the device buffers its calls need.

PyTorch supplies device memory and the CUDA stream; every computation runs in
the library's kernels.  ``Session`` mirrors the C ABI one call per method;
``DeviceDrafts`` is the library's synthetic draft source (a reference
transcript plus corruptions) and ``DraftModel`` its one-block draft model;
both hand each round's drafts to ``verify_device`` without leaving the GPU.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np
import torch

from . import asrspec as A


def dims_dict(dims, max_batch: int, max_draft: int) -> dict:
    return dict(n_layers=dims.n_layers, d_model=dims.d_model, n_heads=dims.n_heads, d_ffn=dims.d_ffn,
                vocab=dims.vocab, max_pos=dims.max_pos, max_batch=max_batch, max_draft=max_draft,
                max_enc=dims.max_enc, dtype=1 if dims.dtype == "bf16" else 0,
                anchor_layer=dims.anchor_layer)


@dataclasses.dataclass
class StepOut:
    accepted: np.ndarray
    bonus: np.ndarray
    kv_len: np.ndarray
    anchor: np.ndarray
    restart: np.ndarray


class Session:
    def __init__(self, dims, blob: np.ndarray, max_batch: int, max_draft: int, device: str = "cuda"):
        if not torch.cuda.is_available():
            raise A.AsrSpecError("a CUDA device is required")
        self.dims = dims
        self.dev = torch.device(device)
        # one stream for the library and for the torch copies that feed it
        self.stream = torch.cuda.Stream(self.dev)
        self.h = A.asr_spec_create(dims_dict(dims, max_batch, max_draft), blob, self.stream.cuda_stream)
        self.max_batch, self.max_draft = max_batch, max_draft
        self.B = 0
        with torch.cuda.stream(self.stream):
            self.out = torch.zeros((5, max_batch), dtype=torch.int32, device=self.dev)
        self.host_io = False

    @property
    def storage_dtype(self):
        return torch.bfloat16 if self.dims.dtype == "bf16" else torch.float32

    def close(self):
        if self.h:
            A.asr_spec_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_host_io(self, on: bool):
        A.asr_spec_set_host_io(self.h, on)
        self.host_io = on

    # -- one call each -------------------------------------------------------
    def encode_cache(self, enc_states, enc_lens):
        """enc_states: [B, t_max, d] (numpy fp32 or a device tensor of the model dtype)."""
        with torch.cuda.stream(self.stream):
            self._encode_cache(enc_states, enc_lens)

    def _encode_cache(self, enc_states, enc_lens):
        if isinstance(enc_states, np.ndarray):
            enc_states = torch.from_numpy(enc_states).to(self.dev).to(self.storage_dtype)
        enc_states = enc_states.contiguous()
        self._enc = enc_states          # keep alive until the GEMM has read it
        B, t_max, _ = enc_states.shape
        lens = self._i32(enc_lens)
        A.asr_spec_encode_cache(self.h, B, enc_states, t_max, lens)
        self.B = B

    def prefill(self, prompt):
        with torch.cuda.stream(self.stream):
            prompt = self._i32(prompt)
            A.asr_spec_prefill(self.h, prompt, int(prompt.shape[1]))

    def verify(self, draft, lens, k: Optional[int] = None) -> StepOut:
        draft = np.asarray(draft, dtype=np.int32)
        if draft.size == 0:
            draft = np.zeros((self.B, 0), dtype=np.int32)
        draft = draft.reshape(self.B, -1)
        k = draft.shape[1] if k is None else k
        lens = np.asarray(lens, dtype=np.int32)
        if self.host_io:
            acc, bon, kvl, anc, rst = (np.zeros(self.B, np.int32) for _ in range(5))
            A.asr_spec_verify(self.h, np.ascontiguousarray(draft[:, :k]), lens, k, acc, bon, kvl, anc)
            A.asr_spec_restart(self.h, rst)
            return StepOut(acc, bon, kvl, anc, rst)
        with torch.cuda.stream(self.stream):
            d = torch.from_numpy(np.ascontiguousarray(draft[:, :k])).to(self.dev)
            l = torch.from_numpy(lens).to(self.dev)
            o = self.out[:, :self.B]
            A.asr_spec_verify(self.h, d, l, k, o[0], o[1], o[2], o[3])
            A.asr_spec_restart(self.h, o[4])
            oh = o.cpu().numpy()
        return StepOut(*(oh[i].copy() for i in range(5)))

    def verify_tree(self, tokens, parent, lens):
        """Tree verify: tokens / parent [B][n] (node i + 1's token and parent),
        lens [B] nodes used or -1.  Returns the step outputs and path [B][n]."""
        tokens = np.ascontiguousarray(np.asarray(tokens, dtype=np.int32).reshape(self.B, -1))
        parent = np.ascontiguousarray(np.asarray(parent, dtype=np.int32).reshape(self.B, -1))
        n = tokens.shape[1]
        lens = np.asarray(lens, dtype=np.int32)
        if self.host_io:
            acc, bon, kvl, anc, rst = (np.zeros(self.B, np.int32) for _ in range(5))
            path = np.full((self.B, max(n, 1)), -1, dtype=np.int32)
            A.asr_spec_verify_tree(self.h, tokens, parent, lens, n, acc, bon, kvl, anc, path)
            A.asr_spec_restart(self.h, rst)
            return StepOut(acc, bon, kvl, anc, rst), path[:, :n]
        with torch.cuda.stream(self.stream):
            t = torch.from_numpy(tokens).to(self.dev)
            p = torch.from_numpy(parent).to(self.dev)
            l = torch.from_numpy(lens).to(self.dev)
            path = torch.full((self.B, max(n, 1)), -1, dtype=torch.int32, device=self.dev)
            o = self.out[:, :self.B]
            A.asr_spec_verify_tree(self.h, t, p, l, n, o[0], o[1], o[2], o[3], path)
            A.asr_spec_restart(self.h, o[4])
            oh = o.cpu().numpy()
            ph = path.cpu().numpy()[:, :n]
        return StepOut(*(oh[i].copy() for i in range(5))), ph

    def host(self, t) -> np.ndarray:
        """Copy a device tensor written on this session's stream to the host."""
        self.stream.synchronize()
        return t.cpu().numpy()

    def verify_device(self, draft_d, lens_d, k: int):
        """Device-resident verify: inputs and outputs stay on the GPU (no sync)."""
        o = self.out[:, :self.B]
        A.asr_spec_verify(self.h, draft_d, lens_d, k, o[0], o[1], o[2], o[3])
        return o

    def rollback(self, new_len, new_pending):
        with torch.cuda.stream(self.stream):
            A.asr_spec_rollback(self.h, self._i32(new_len), self._i32(new_pending))

    def state(self):
        if self.host_io:
            kvh, peh = np.zeros(self.B, np.int32), np.zeros(self.B, np.int32)
            A.asr_spec_state(self.h, kvh, peh)
            return kvh, peh
        with torch.cuda.stream(self.stream):
            kv = torch.zeros(self.B, dtype=torch.int32, device=self.dev)
            pe = torch.zeros(self.B, dtype=torch.int32, device=self.dev)
            A.asr_spec_state(self.h, kv, pe)
            return kv.cpu().numpy(), pe.cpu().numpy()

    def debug_logits(self, max_rows: int) -> torch.Tensor:
        with torch.cuda.stream(self.stream):
            out = torch.empty((max_rows, self.dims.vocab), dtype=torch.float32, device=self.dev)
            R = A.asr_spec_debug_logits(self.h, out, max_rows)
        self.stream.synchronize()
        return out[:R]

    def anchor_profile(self) -> np.ndarray:
        """The head-mean attention profiles behind the last verify's anchors, [B][max_enc]."""
        with torch.cuda.stream(self.stream):
            out = torch.empty((self.B, self.dims.max_enc), dtype=torch.float32, device=self.dev)
            A.asr_spec_debug_anchor_profile(self.h, out)
        self.stream.synchronize()
        return out.cpu().numpy()

    def status(self) -> int:
        return A.asr_spec_status(self.h)

    def _i32(self, x):
        a = np.ascontiguousarray(np.asarray(x, dtype=np.int32))
        if self.host_io:
            return a
        return torch.from_numpy(a).to(self.dev)


class DeviceDrafts:
    """Synthetic draft source on the device: a reference transcript plus the
    corruption stream, turned into each round's drafts by a library kernel."""

    def __init__(self, sess: Session, truth: np.ndarray, total_lens, corr, k: int):
        B, P = sess.B, sess.dims.max_pos
        t = np.zeros((B, P), dtype=np.int32)
        t[:, :truth.shape[1]] = np.where(truth >= 0, truth, 0)[:, :P]
        dev = sess.dev
        self.sess, self.k = sess, k
        with torch.cuda.stream(sess.stream):
            self.truth = torch.from_numpy(t).to(dev)
            self.total = torch.tensor(np.asarray(total_lens, dtype=np.int32), device=dev)
            self.repl = torch.from_numpy(np.ascontiguousarray(corr.repl[:B, :P, :], dtype=np.int32)).to(dev)
            self.k_repl = int(corr.repl.shape[2])
            self.shift = torch.from_numpy(np.ascontiguousarray(corr.shift[:B, :P], dtype=np.int32)).to(dev)
            self.draft = torch.zeros((B, k), dtype=torch.int32, device=dev)
            self.lens = torch.zeros(B, dtype=torch.int32, device=dev)
        sess.stream.synchronize()

    def next(self):
        A.asr_spec_synth_drafts(self.sess.h, self.truth, self.total, self.repl, self.k_repl, self.shift, self.k,
                                self.draft, self.lens)
        return self.draft, self.lens


class DraftModel:
    """The one-block draft on the device (App. "Draft architecture"): attach it
    to a session before ``encode_cache``; ``propose`` runs one drafting round
    (catch-up of the last verification, restart, continuations) and leaves
    drafts and lens on the device, ready for ``Session.verify_device``."""

    def __init__(self, sess: Session, blob: np.ndarray, total_lens, k: int, window="anchor", threshold: float = 0.0):
        if sess.B:
            raise A.AsrSpecError("attach the draft before encode_cache")
        A.asr_spec_draft_create(sess.h, blob)
        if threshold > 0.0:
            A.asr_spec_draft_set_threshold(sess.h, threshold)
        self.sess, self.k, self.window = sess, k, A.DRAFT_WIN[window]
        dev = sess.dev
        with torch.cuda.stream(sess.stream):
            self.total = torch.tensor(np.asarray(total_lens, dtype=np.int32), device=dev)
            n = self.total.numel()
            self.centers = torch.zeros(n, dtype=torch.int32, device=dev)
            self.draft = torch.zeros((n, max(k, 1)), dtype=torch.int32, device=dev)
            self.lens = torch.zeros(n, dtype=torch.int32, device=dev)
        sess.stream.synchronize()

    def set_centers(self, centers):
        """Window centres of the random control for the next round (host ints)."""
        with torch.cuda.stream(self.sess.stream):
            self.centers.copy_(torch.from_numpy(np.asarray(centers, dtype=np.int32)))

    def propose(self, k: Optional[int] = None):
        """One round of at most k (default: the k given at creation) proposals."""
        k = self.k if k is None else k
        if k > self.k:
            raise A.AsrSpecError("k above the draft buffer's width")
        A.asr_spec_draft_propose(self.sess.h, k, self.window, self.centers, self.total, self.draft, self.lens)
        n = self.lens.numel()
        return self.draft.view(-1)[:n * k].view(n, k), self.lens   # [B][k], row stride k
