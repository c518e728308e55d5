"""One-block draft and the real cached speculative loop (float64, numpy).

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and the CPU legs of ``bench.py`` may import it.

What it computes, and where the paper fixes it:

* The draft (App. "Draft architecture"; the Whisper check of App. "Whisper
  Cross-Architecture Check" uses matched one-layer drafts with per-step audio
  cross-attention): four frozen target representations are combined with the
  current token's embedding, then one causal block applies self-attention,
  cross-attention to the frozen audio representation and a feed-forward
  layer; the target's LM head (frozen, tied to the token embedding) turns the
  block's output into the proposal.  Audio cross-attention runs at every draft
  step.
* The audio window (App. "Attention conditions", "Window geometry"): the
  restricted arms attend only to the frames around a centre, see
  ``oracle.window``; the deployed centre is the anchor the last verification
  returned (Sec. 5 "Verification-Attention Correction").
* The loop (Sec. 3 "Speculative Loop"; App. "Decoding and Intervention
  Protocol": the real cached loop): the draft proposes up to K tokens from the
  verified state (the first is the restart, the others continuation
  proposals), the target verifies them in one pass, the accepted tokens and
  their cached states feed the next round.

Readings where the paper is silent (each listed in the design notes):
* input at position p: w_in [f_1; ...; f_4] + b_in + tok_emb[t_p] + pos_emb[p],
  where f_i is the target's residual stream after tap layer i (workload's
  draft_taps) at the row that scored t_p (position p - 1; zeros at p = 0);
* continuation proposals have no target row: the draft's own block output at
  p - 1 stands in for all four representations;
* the block is the target's pre-LN block (feed-forward width 2d, erf GELU, no
  key bias) with the draft's own cross K/V projections of the encoder states;
  its final LayerNorm is its own, the embeddings and LM head are the target's;
* the draft cache holds one entry per committed position, each computed from
  the target's representations: after a verification the draft re-processes
  the newly committed positions with the verify rows' representations before
  it proposes again (the restart entry already used them);
* before the first verification there is no anchor: the window is centred on
  frame 0.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np

from oracle.decoder import Oracle, attention, gelu, layer_norm
from oracle.window import window, window_center, windowed_attention
from workload import draft_weight_layout, round_lens


class Draft:
    """The one-block draft beside a target oracle (same batch of utterances)."""

    def __init__(self, target: Oracle, blob: np.ndarray):
        self.t = target
        self.dims = target.dims
        self._w: Dict[str, np.ndarray] = {}
        for name, (off, shape) in draft_weight_layout(self.dims).items():
            if name != "__total__":
                self._w[name] = np.asarray(blob[off:off + int(np.prod(shape))], dtype=np.float64).reshape(shape)

    def W(self, name: str) -> np.ndarray:
        return self._w[name]

    def encode(self) -> None:
        """The draft's cross-attention keys and values of every utterance (its own
        projections of the encoder states the target cached), and an empty cache."""
        t, d = self.t, self.dims
        self.Kd = [E @ self.W("wck").T for E in t.enc]
        self.Vd = [E @ self.W("wcv").T + self.W("bcv") for E in t.enc]
        self.Ks = np.zeros((t.B, d.max_pos, d.d_model))
        self.Vs = np.zeros((t.B, d.max_pos, d.d_model))

    def step(self, b: int, token: int, pos: int, feat: np.ndarray, win=None):
        """One draft position: writes its self-attention K/V at `pos` and returns
        (logits [V], block output [d]).  feat: [4, d] representations (the
        target's, or the draft's own output repeated); win: frames [lo, hi) of
        the cross-attention, None = all frames."""
        d, t = self.dims, self.t
        H = d.n_heads
        x = (self.W("w_in") @ feat.reshape(-1) + self.W("b_in") + t.W("tok_emb")[token] + t.W("pos_emb")[pos])
        h = layer_norm(x, self.W("ln1_g"), self.W("ln1_b"))
        q = self.W("wq") @ h + self.W("bq")
        self.Ks[b, pos] = self.W("wk") @ h
        self.Vs[b, pos] = self.W("wv") @ h + self.W("bv")
        o = attention(q, self.Ks[b, :pos + 1], self.Vs[b, :pos + 1], H)
        x = x + self.W("wo") @ o + self.W("bo")
        h = layer_norm(x, self.W("ln2_g"), self.W("ln2_b"))
        qc = self.W("wcq") @ h + self.W("bcq")
        lo, hi = win if win is not None else (0, len(self.Kd[b]))
        o = windowed_attention(qc, self.Kd[b], self.Vd[b], H, lo, hi)
        x = x + self.W("wco") @ o + self.W("bco")
        h = layer_norm(x, self.W("ln3_g"), self.W("ln3_b"))
        x = x + self.W("w2") @ gelu(self.W("w1") @ h + self.W("b1")) + self.W("b2")
        logits = layer_norm(x, self.W("lnf_g"), self.W("lnf_b")) @ t.W("tok_emb").T
        return logits, x

    def prefill(self, prompt) -> None:
        """Cache the prompt's positions 0..P0-2 from the target's prefill rows
        (the target must have been prefilled with the same prompt)."""
        prompt = np.asarray(prompt, dtype=np.int64)
        B, P0 = prompt.shape
        zero = np.zeros((4, self.dims.d_model))
        for b in range(B):
            for p in range(P0 - 1):
                f = self.t.prefill_feats[b, p - 1] if p > 0 else zero
                self.step(b, int(prompt[b, p]), p, f)

    def catch_up(self, b: int, P_old: int, drafts_b, n: int, feats_b: np.ndarray) -> None:
        """After a verification that accepted n drafts from committed length
        P_old: the entries of positions P_old + 1 .. P_old + n from the verify
        rows' target representations (row i is position P_old + i)."""
        for j in range(1, n + 1):
            self.step(b, int(drafts_b[j - 1]), P_old + j, feats_b[j - 1])

    def propose(self, b: int, pending: int, P: int, feat: np.ndarray, k: int, win=None,
                threshold: float = 0.0) -> List[int]:
        """Up to k proposals from the verified state: the restart at position P
        (the pending token with the target's representations of the row that
        scored it), then continuation proposals fed by the draft's own output.
        A proposal whose draft probability (softmax of its logits) is below
        `threshold` ends the block unproposed (App. "Draft length and
        confidence threshold": the block length varies per utterance)."""
        out, tok, f = [], int(pending), feat
        for i in range(k):
            logits, x = self.step(b, tok, P + i, f, win)
            tok = int(np.argmax(logits))
            if threshold > 0.0:
                e = np.exp(logits - logits.max())
                if 1.0 / e.sum() < threshold:   # the top token's probability
                    break
            out.append(tok)
            f = np.tile(x, (4, 1))
        return out


def speculative_decode(target: Oracle, draft: Draft, prompt, total_lens, k: int, kind: Optional[str] = "anchor",
                       rng: Optional[np.random.Generator] = None, threshold: float = 0.0):
    """The real cached loop until every utterance holds total_lens[b] tokens
    (prompt included).  kind: "anchor" (deployed correction), "shifted",
    "random" (controls) or None (unrestricted audio attention); threshold: the
    draft's confidence threshold (0 = always k proposals).  Returns the token
    sequences and, per round, (lens, accepted) of the utterances (lens -1 for
    those that sat out)."""
    prompt = np.asarray(prompt, dtype=np.int64)
    B = prompt.shape[0]
    target.prefill(prompt)
    draft.encode()
    draft.prefill(prompt)
    rng = rng if rng is not None else np.random.default_rng(0)
    seqs = [list(prompt[b]) for b in range(B)]
    feat = [target.prefill_feats[b, -1] if prompt.shape[1] > 1 else np.zeros((4, target.dims.d_model))
            for b in range(B)]
    anchor = [0] * B
    rounds = []
    while True:
        lens = round_lens(total_lens, target.kv_len, k)
        if np.all(lens < 0):
            break
        drafts = np.zeros((B, max(k, 1)), dtype=np.int64)
        for b in range(B):
            if lens[b] < 0:
                continue
            T = len(target.enc[b])
            win = None if kind is None else window(window_center(kind, anchor[b], T, rng), T)
            if lens[b] > 0:
                props = draft.propose(b, int(target.pending[b]), int(target.kv_len[b]), feat[b], int(lens[b]), win,
                                      threshold)
                drafts[b, :len(props)] = props
                lens[b] = len(props)
            else:   # no proposals: the pending position's entry all the same
                draft.step(b, int(target.pending[b]), int(target.kv_len[b]), feat[b], win)
        P_old = target.kv_len.copy()
        res = target.verify(drafts[:, :k], lens)
        r0 = 0
        for b in range(B):
            if lens[b] < 0:
                continue
            n = int(res.accepted[b])
            rows = res.feats[r0:r0 + int(lens[b]) + 1]
            draft.catch_up(b, int(P_old[b]), drafts[b], n, rows)
            feat[b] = rows[n]                  # the row that scored the bonus token
            anchor[b] = int(res.anchor[b])
            seqs[b] += [int(x) for x in drafts[b, :n]] + [int(res.bonus[b])]
            r0 += int(lens[b]) + 1
        rounds.append((lens.copy(), res.accepted.copy()))
    return seqs, rounds


def acceptance_stats(rounds, k: int) -> Dict[str, float]:
    """The speculative loop's acceptance metrics (Sec. 3 "Speculative Loop"):
    s_j, the probability that the first j proposals are accepted, over the
    rounds that offered at least j proposals (s_0 = 1); restart acceptance
    a_1 = s_1; continuation acceptance a_j^c = s_j / s_{j-1}; L, the mean
    accepted length per round (sum_j s_j when every round offers k)."""
    lens = np.concatenate([np.asarray(l) for l, _ in rounds])
    acc = np.concatenate([np.asarray(a) for _, a in rounds])
    live = lens >= 0
    lens, acc = lens[live], acc[live]
    s = [1.0]
    for j in range(1, k + 1):
        offered = lens >= j
        s.append(float(np.mean(acc[offered] >= j)) if offered.any() else float("nan"))
    out = {f"s_{j}": s[j] for j in range(1, k + 1)}
    out["a_1"] = s[1]
    for j in range(2, k + 1):
        out[f"a_{j}^c"] = s[j] / s[j - 1] if s[j - 1] > 0 else float("nan")
    out["L"] = float(np.mean(acc))
    return out
