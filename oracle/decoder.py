"""CPU oracle for the speculative draft-verify step (float64, numpy).

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  The CUDA path never
calls it and shares no code with it; both only read inputs drawn by
``workload``.

What it computes, and where the paper fixes it:

* The speculative loop (Sec. 3 "Speculative Loop"): a draft proposes up to K
  tokens; the frozen target checks the whole block in one pass and accepts the
  longest prefix that matches its own greedy output.  Under exact arithmetic
  this returns the target-greedy sequence.
* A round advances by one token more than the accepted drafts (App.
  "Correction and Cost", cost derivation: a round advances 1 + L tokens): the
  target's own prediction after the accepted prefix (the "bonus" token).
* The real cached loop (App. "Decoding and Intervention Protocol"): accepted
  tokens and their cached states feed the next round; the decoder cache is
  reused (Sec. 1 and Sec. 3: the draft reuses the encoded audio and decoder
  cache).
* The target is a Whisper-style encoder-decoder (Sec. 3 "Models and
  Protocol"); the decoder block is the pre-LN Whisper block: LN, causal
  self-attention, LN, cross-attention to the encoder states, LN, GELU MLP,
  then a final LN and an LM head tied to the token embedding.
* The runtime re-anchoring readout (Sec. 5 "Verification-Attention
  Correction" and App. "Runtime anchor construction"): average the target's
  audio attention over heads at one decoder layer and take its peak; the
  scores are recomputed from the existing key cache, with no extra target pass.

Readings where the paper is silent (each is listed with its reason in the
design notes of this repository): no key bias (Whisper), LayerNorm eps 1e-5,
1/sqrt(head_dim) score scale, erf GELU, lowest index wins argmax ties, anchor
layer floor(3L/4), anchor taken from the row whose argmax is the bonus token,
head mean of normalised per-head probabilities with padded frames excluded,
restart flag set when a draft was rejected.

Precision: float64 throughout.  bf16 models store bf16-representable values
in the fp32 blob and are widened here; no intermediate is rounded.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Dict, List, Optional

import numpy as np
from scipy.special import erf

from workload import ModelDims, draft_taps, weight_layout

LN_EPS = 1e-5


def layer_norm(x: np.ndarray, g: np.ndarray, b: np.ndarray) -> np.ndarray:
    """LayerNorm over the last axis: biased variance, eps 1e-5, affine g, b."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS) * g + b


def gelu(x: np.ndarray) -> np.ndarray:
    """Exact (erf) GELU, as in Whisper's MLP."""
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def softmax(s: np.ndarray) -> np.ndarray:
    """Softmax over the last axis (max subtracted first)."""
    e = np.exp(s - s.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, n_heads: int) -> np.ndarray:
    """Multi-head scaled dot-product attention of one query row over n keys.

    q [d]; K, V [n, d] with head h in columns h*hd:(h+1)*hd.  Returns [d].
    """
    n, d = K.shape
    hd = d // n_heads
    qh = q.reshape(n_heads, hd)
    Kh = K.reshape(n, n_heads, hd)
    Vh = V.reshape(n, n_heads, hd)
    s = np.einsum("hc,nhc->hn", qh, Kh) / np.sqrt(hd)
    p = softmax(s)
    return np.einsum("hn,nhc->hc", p, Vh).reshape(d)


def head_mean_attention(q: np.ndarray, K: np.ndarray, n_heads: int) -> np.ndarray:
    """Mean over heads of the per-head softmax attention of one query over n keys.

    This is the audio-attention profile whose peak is the runtime anchor
    (Sec. 5 "Verification-Attention Correction"; the head mean is the same
    one the AnchorDraft objective uses on the draft, Sec. 5 "AnchorDraft
    Training Objective").  Returns [n].
    """
    n, d = K.shape
    hd = d // n_heads
    s = np.einsum("hc,nhc->hn", q.reshape(n_heads, hd), K.reshape(n, n_heads, hd)) / np.sqrt(hd)
    return softmax(s).mean(axis=0)


def visible_keys(pos: int) -> int:
    """Self-attention keys a verification row at position pos sees: the
    committed cache and every row of its own block up to itself (Sec. 3: the
    target checks the whole block in one pass, each row causally)."""
    return pos + 1


def tree_keys(P: int, ancestors: List[int]) -> List[int]:
    """Cache slots a tree node attends to: the committed cache [0, P) and the
    slots P + a of its ancestors a (root first, the node itself last); the
    tree attention mask of the tree decoder control."""
    return list(range(P)) + [P + a for a in ancestors]


def accepted_prefix(draft_b: np.ndarray, g_b: np.ndarray, lens_b: int) -> int:
    """Longest prefix of the block kept by the target (Sec. 3 "Speculative
    Loop"): draft j (0-based) stays while it equals the target's argmax at row
    j, the row that scored the token before it (the pending token for j = 0)."""
    n = 0
    while n < lens_b and draft_b[n] == g_b[n]:
        n += 1
    return n


def bonus_row(n: int) -> int:
    """Row of the block whose argmax is the bonus token after n accepted
    drafts: the row that scored the last accepted token (App. "Correction and
    Cost": a round advances 1 + L tokens).  The anchor is read at this row."""
    return n


class OracleError(ValueError):
    pass


@dataclass
class VerifyResult:
    accepted: np.ndarray      # [B] accepted draft tokens n_b (0 for inactive)
    bonus: np.ndarray         # [B] target token after the accepted prefix (-1 inactive)
    kv_len: np.ndarray        # [B] committed cache length after the step
    anchor: np.ndarray        # [B] re-anchored audio frame (-1 inactive)
    restart: np.ndarray       # [B] 1 if a draft was rejected this round
    rows: List[tuple]         # (b, i) of every scored row, in row order
    logits: np.ndarray        # [R, V] float64
    argmax: np.ndarray        # [R] greedy token of every row
    top2_gap: np.ndarray      # [R] top-1 minus top-2 logit
    anchor_profile: Dict[int, np.ndarray]  # b -> head-mean attention over frames
    path: Optional[np.ndarray] = None       # tree verify: [B][n] accepted nodes by depth (-1 past the path)
    feats: Optional[np.ndarray] = None      # [R, 4, d] the target's outputs at the draft's tap layers


class Oracle:
    """Float64 reference of the Whisper-style target decoder and its verify step.

    State per utterance b: encoder K/V of every layer (built once), the
    self-attention K/V cache, the committed length kv_len[b] and the pending
    token (the last emitted token, whose K/V is not yet cached).
    """

    def __init__(self, dims: ModelDims, blob: np.ndarray):
        self.dims = dims
        lay = weight_layout(dims)
        self._w: Dict[str, np.ndarray] = {}
        for name, (off, shape) in lay.items():
            if name == "__total__":
                continue
            self._w[name] = np.asarray(blob[off:off + int(np.prod(shape))],
                                       dtype=np.float64).reshape(shape)
        self.B = 0
        self.enc_len: Optional[np.ndarray] = None
        self.kv_len: Optional[np.ndarray] = None
        self.pending: Optional[np.ndarray] = None

    def W(self, name: str) -> np.ndarray:
        return self._w[name]

    # -- per-utterance set-up ------------------------------------------------

    def encode_cache(self, enc_states: np.ndarray, enc_lens) -> None:
        """Cross-attention keys and values of every layer, once per utterance.

        Kx_l = E Wck_l^T and Vx_l = E Wcv_l^T + bcv_l over the utterance's
        frames (the encoded audio is reused at every step, Sec. 1 and App.
        "Runtime anchor construction": scores come from the existing key cache).
        """
        d = self.dims
        enc_states = np.asarray(enc_states)
        B, T, dm = enc_states.shape
        if dm != d.d_model or T > d.max_enc:
            raise OracleError("encoder states have the wrong shape")
        enc_lens = np.asarray(enc_lens, dtype=np.int64)
        if np.any(enc_lens < 1) or np.any(enc_lens > T):
            raise OracleError("encoder length out of range")
        self.B = B
        self.enc_len = enc_lens.copy()
        E = enc_states.astype(np.float64)
        self.enc = [E[b, :enc_lens[b]].copy() for b in range(B)]   # the draft reads the encoder states too
        self.Kx, self.Vx = [], []
        for l in range(d.n_layers):
            self.Kx.append([E[b, :enc_lens[b]] @ self.W(f"L{l}.wck").T for b in range(B)])
            self.Vx.append([E[b, :enc_lens[b]] @ self.W(f"L{l}.wcv").T + self.W(f"L{l}.bcv")
                            for b in range(B)])
        self.Ks = [np.zeros((B, d.max_pos, d.d_model)) for _ in range(d.n_layers)]
        self.Vs = [np.zeros((B, d.max_pos, d.d_model)) for _ in range(d.n_layers)]
        self.kv_len = None
        self.pending = None

    def prefill(self, prompt) -> None:
        """Cache the prompt: K/V of prompt[:, :-1] at positions 0..P0-2; the last
        prompt token becomes the pending token (its K/V is written by the first
        verify, which scores it at position P0-1)."""
        if self.enc_len is None:
            raise OracleError("prefill before encode_cache")
        prompt = np.asarray(prompt, dtype=np.int64)
        B, P0 = prompt.shape
        if B != self.B or P0 < 1 or P0 > self.dims.max_pos:
            raise OracleError("bad prompt shape")
        self._check_tokens(prompt)
        rows = [(b, int(prompt[b, i]), i) for b in range(B) for i in range(P0 - 1)]
        self.prefill_feats = np.zeros((B, max(P0 - 1, 0), 4, self.dims.d_model))
        if rows:
            self._forward(rows)
            self.prefill_feats[:] = self.last_feats.reshape(B, P0 - 1, 4, self.dims.d_model)
        self.kv_len = np.full(B, P0 - 1, dtype=np.int64)
        self.pending = prompt[:, P0 - 1].copy()

    # -- decoder forward -----------------------------------------------------

    def _check_tokens(self, t) -> None:
        t = np.asarray(t)
        if np.any(t < 0) or np.any(t >= self.dims.vocab):
            raise OracleError("token id out of range")

    def _forward(self, rows, want_logits: bool = False):
        """Run the decoder on rows (b, token, position), writing each row's
        self-attention K/V at its position first, so that a row attends to the
        committed cache plus every earlier row of its own block and itself:
        the block-causal mask of one verification pass (Sec. 3).  A row may
        also be (b, token, position, slot, keys): its K/V go to cache slot
        `slot` and it attends to the cache slots `keys` (a tree node: the
        committed cache, its ancestors and itself).

        Returns final-LN logits [R, V] (if asked) and each row's cross-attention
        query at the anchor layer.
        """
        d = self.dims
        H = d.n_heads
        tok = np.array([r[1] for r in rows], dtype=np.int64)
        pos = np.array([r[2] for r in rows], dtype=np.int64)
        slot = [r[3] if len(r) > 3 else r[2] for r in rows]
        bidx = [r[0] for r in rows]
        x = self.W("tok_emb")[tok] + self.W("pos_emb")[pos]
        q_anchor = None
        taps = draft_taps(d)
        feats = np.zeros((len(rows), 4, d.d_model))
        for l in range(d.n_layers):
            p = f"L{l}."
            # self-attention block
            h = layer_norm(x, self.W(p + "ln1_g"), self.W(p + "ln1_b"))
            q = h @ self.W(p + "wq").T + self.W(p + "bq")
            k = h @ self.W(p + "wk").T
            v = h @ self.W(p + "wv").T + self.W(p + "bv")
            for r, b in enumerate(bidx):
                self.Ks[l][b, slot[r]] = k[r]
                self.Vs[l][b, slot[r]] = v[r]
            o = np.empty_like(x)
            for r, row in enumerate(rows):
                b = row[0]
                if len(row) > 3:
                    keys = row[4]
                    o[r] = attention(q[r], self.Ks[l][b, keys], self.Vs[l][b, keys], H)
                else:
                    nk = visible_keys(row[2])
                    o[r] = attention(q[r], self.Ks[l][b, :nk], self.Vs[l][b, :nk], H)
            x = x + o @ self.W(p + "wo").T + self.W(p + "bo")
            # cross-attention block over the utterance's encoder frames
            h = layer_norm(x, self.W(p + "ln2_g"), self.W(p + "ln2_b"))
            qc = h @ self.W(p + "wcq").T + self.W(p + "bcq")
            if l == d.anchor:
                q_anchor = qc.copy()
            o = np.empty_like(x)
            for r, b in enumerate(bidx):
                o[r] = attention(qc[r], self.Kx[l][b], self.Vx[l][b], H)
            x = x + o @ self.W(p + "wco").T + self.W(p + "bco")
            # MLP block
            h = layer_norm(x, self.W(p + "ln3_g"), self.W(p + "ln3_b"))
            f = gelu(h @ self.W(p + "w1").T + self.W(p + "b1"))
            x = x + f @ self.W(p + "w2").T + self.W(p + "b2")
            for i, t in enumerate(taps):
                if t == l:
                    feats[:, i] = x
        self.last_feats = feats   # the draft's inputs (layer outputs at its tap layers), row order
        logits = None
        if want_logits:
            xf = layer_norm(x, self.W("lnf_g"), self.W("lnf_b"))
            logits = xf @ self.W("tok_emb").T          # LM head tied to the token embedding
        return logits, q_anchor

    # -- the verify step -----------------------------------------------------

    def verify(self, draft, lens) -> VerifyResult:
        """Score pending + drafts in one pass, accept the longest matching prefix,
        emit the bonus token, commit the cache and re-anchor.

        draft [B, k] int; lens [B] with 0 <= lens[b] <= k valid drafts, or -1 for
        an utterance that takes no part in this step.  Row i of utterance b is
        the pending token (i = 0) or draft i, at position kv_len[b] + i.
        """
        d = self.dims
        if self.kv_len is None:
            raise OracleError("verify before prefill")
        draft = np.asarray(draft, dtype=np.int64).reshape(self.B, -1)
        lens = np.asarray(lens, dtype=np.int64)
        k = draft.shape[1]
        if lens.shape != (self.B,) or np.any(lens < -1) or np.any(lens > k):
            raise OracleError("lens out of range")
        rows, row_ids = [], []
        for b in range(self.B):
            if lens[b] < 0:
                continue
            if self.kv_len[b] + lens[b] + 1 > d.max_pos:
                raise OracleError("decoder context capacity exceeded")
            self._check_tokens(draft[b, :lens[b]])
            P = int(self.kv_len[b])
            for i in range(int(lens[b]) + 1):
                t = int(self.pending[b]) if i == 0 else int(draft[b, i - 1])
                rows.append((b, t, P + i))
                row_ids.append((b, i))
        if rows:
            logits, q_anchor = self._forward(rows, want_logits=True)
        else:
            logits, q_anchor = np.zeros((0, d.vocab)), np.zeros((0, d.d_model))
        g = np.argmax(logits, axis=1) if rows else np.zeros(0, dtype=np.int64)
        srt = np.sort(logits, axis=1)[:, -2:] if rows else np.zeros((0, 2))
        gap = srt[:, 1] - srt[:, 0]

        acc = np.zeros(self.B, dtype=np.int64)
        bonus = np.full(self.B, -1, dtype=np.int64)
        anchor = np.full(self.B, -1, dtype=np.int64)
        restart = np.zeros(self.B, dtype=np.int64)
        prof: Dict[int, np.ndarray] = {}
        r0 = 0
        for b in range(self.B):
            if lens[b] < 0:
                continue
            n = accepted_prefix(draft[b], g[r0:r0 + int(lens[b]) + 1], int(lens[b]))
            acc[b] = n
            br = r0 + bonus_row(n)
            bonus[b] = g[br]
            restart[b] = 1 if n < lens[b] else 0
            # re-anchor from the verification row that produced the bonus token
            pbar = head_mean_attention(q_anchor[br], self.Kx[d.anchor][b], d.n_heads)
            prof[b] = pbar
            anchor[b] = int(np.argmax(pbar))
            self.kv_len[b] = self.kv_len[b] + 1 + n
            self.pending[b] = bonus[b]
            r0 += int(lens[b]) + 1
        res = VerifyResult(acc, bonus, self.kv_len.copy(), anchor, restart, row_ids,
                           logits, g, gap, prof)
        res.feats = self.last_feats if rows else np.zeros((0, 4, d.d_model))
        return res

    def verify_tree(self, tokens, parent, lens) -> VerifyResult:
        """Score a candidate tree per utterance in one pass under a tree mask
        (App. "Alternative draft and verification changes", tree decoder):
        node 0 is the pending token, node i + 1 has token tokens[b][i] and
        parent parent[b][i] in [0, i]; lens[b] nodes are used (-1: sits out).
        Node j is scored at position kv_len + depth(j), its K/V in cache slot
        kv_len + j, attending to the committed cache and to its ancestors
        (itself included).  The accepted path starts at the root and moves to
        the first child (lowest index) whose token is the argmax of the current
        node; the bonus is the argmax of its last node, which is also the
        anchor row.  The path's K/V move to positions kv_len + 1 .. + n in
        depth order.  The result carries `path` [B][n] (-1 past the path)."""
        d = self.dims
        if self.kv_len is None:
            raise OracleError("verify before prefill")
        tokens = np.asarray(tokens, dtype=np.int64).reshape(self.B, -1)
        parent = np.asarray(parent, dtype=np.int64).reshape(self.B, -1)
        lens = np.asarray(lens, dtype=np.int64)
        n_max = tokens.shape[1]
        if lens.shape != (self.B,) or np.any(lens < -1) or np.any(lens > n_max):
            raise OracleError("lens out of range")
        rows, row_ids, kids = [], [], {}
        for b in range(self.B):
            if lens[b] < 0:
                continue
            l = int(lens[b])
            if self.kv_len[b] + l + 1 > d.max_pos:
                raise OracleError("decoder context capacity exceeded")
            self._check_tokens(tokens[b, :l])
            par = [-1] + [int(p) for p in parent[b, :l]]
            if any(par[j] < 0 or par[j] >= j for j in range(1, l + 1)):
                raise OracleError("a parent outside [0, node)")
            P = int(self.kv_len[b])
            depth = [0] * (l + 1)
            anc = [[0]] + [None] * l
            for j in range(1, l + 1):
                depth[j] = depth[par[j]] + 1
                anc[j] = anc[par[j]] + [j]
            kids[b] = [[j for j in range(1, l + 1) if par[j] == c] for c in range(l + 1)]
            for j in range(l + 1):
                t = int(self.pending[b]) if j == 0 else int(tokens[b, j - 1])
                keys = tree_keys(P, anc[j])
                rows.append((b, t, P + depth[j], P + j, keys))
                row_ids.append((b, j))
        if rows:
            logits, q_anchor = self._forward(rows, want_logits=True)
        else:
            logits, q_anchor = np.zeros((0, d.vocab)), np.zeros((0, d.d_model))
        g = np.argmax(logits, axis=1) if rows else np.zeros(0, dtype=np.int64)
        srt = np.sort(logits, axis=1)[:, -2:] if rows else np.zeros((0, 2))
        gap = srt[:, 1] - srt[:, 0]
        acc = np.zeros(self.B, dtype=np.int64)
        bonus = np.full(self.B, -1, dtype=np.int64)
        anchor = np.full(self.B, -1, dtype=np.int64)
        restart = np.zeros(self.B, dtype=np.int64)
        path = np.full((self.B, n_max), -1, dtype=np.int64)
        prof: Dict[int, np.ndarray] = {}
        r0 = 0
        for b in range(self.B):
            if lens[b] < 0:
                continue
            c, n = 0, 0
            while True:
                nxt = [j for j in kids[b][c] if int(tokens[b, j - 1]) == int(g[r0 + c])]
                if not nxt:
                    break
                c = nxt[0]
                path[b, n] = c
                n += 1
            acc[b] = n
            bonus[b] = g[r0 + c]
            restart[b] = 1 if kids[b][c] else 0
            pbar = head_mean_attention(q_anchor[r0 + c], self.Kx[d.anchor][b], d.n_heads)
            prof[b] = pbar
            anchor[b] = int(np.argmax(pbar))
            P = int(self.kv_len[b])
            for j in range(n):   # the accepted path to consecutive positions, in depth order
                for l_ in range(d.n_layers):
                    self.Ks[l_][b, P + j + 1] = self.Ks[l_][b, P + path[b, j]]
                    self.Vs[l_][b, P + j + 1] = self.Vs[l_][b, P + path[b, j]]
            self.kv_len[b] = P + 1 + n
            self.pending[b] = bonus[b]
            r0 += int(lens[b]) + 1
        res = VerifyResult(acc, bonus, self.kv_len.copy(), anchor, restart, row_ids, logits, g, gap, prof)
        res.path = path
        res.feats = self.last_feats if rows else np.zeros((0, 4, d.d_model))
        return res

    def rollback(self, new_len, new_pending) -> None:
        """Truncate the committed cache to new_len[b] <= kv_len[b] and set the
        pending token; cache rows at and beyond new_len are dead."""
        new_len = np.asarray(new_len, dtype=np.int64)
        new_pending = np.asarray(new_pending, dtype=np.int64)
        if self.kv_len is None:
            raise OracleError("rollback before prefill")
        if np.any(new_len < 0) or np.any(new_len > self.kv_len):
            raise OracleError("rollback beyond the committed length")
        self._check_tokens(new_pending)
        self.kv_len = new_len.copy()
        self.pending = new_pending.copy()

    def ar_step(self, active=None) -> np.ndarray:
        """Plain greedy decoding, one token: score the pending token and commit it."""
        lens = np.zeros(self.B, dtype=np.int64)
        if active is not None:
            lens[~np.asarray(active, dtype=bool)] = -1
        return self.verify(np.zeros((self.B, 1), dtype=np.int64), lens).bonus

    def snapshot(self):
        """Copy of the mutable state (cache, lengths, pending) for comparisons."""
        return ([k.copy() for k in self.Ks], [v.copy() for v in self.Vs],
                self.kv_len.copy(), self.pending.copy())

    def restore(self, snap) -> None:
        Ks, Vs, kv, pend = snap
        self.Ks = [k.copy() for k in Ks]
        self.Vs = [v.copy() for v in Vs]
        self.kv_len = kv.copy()
        self.pending = pend.copy()


def greedy_transcript(orc: Oracle, prompt, total_lens) -> np.ndarray:
    """Target-greedy transcripts (prompt included), decoded one token at a time
    from a freshly prefilled oracle: [B, max(total_lens)] int64, -1 past each
    utterance's length.  The oracle is left at the end of each transcript."""
    prompt = np.asarray(prompt, dtype=np.int64)
    B, P0 = prompt.shape
    total_lens = np.asarray(total_lens, dtype=np.int64)
    if np.any(orc.kv_len != P0 - 1):
        raise OracleError("greedy_transcript needs a freshly prefilled oracle")
    out = np.full((B, int(total_lens.max())), -1, dtype=np.int64)
    out[:, :P0] = prompt
    while True:
        active = orc.kv_len + 1 < total_lens
        if not active.any():
            break
        pos = orc.kv_len + 1
        nxt = orc.ar_step(active)
        for b in np.nonzero(active)[0]:
            out[b, pos[b]] = nxt[b]
    return out
