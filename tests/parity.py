"""Teacher-forced comparison of the CUDA verify step with the CPU oracle.

Both sides start from the same encoder states, prompt and weights and receive
the same drafts every round.  Per round and utterance the accepted length, the
bonus token and the committed length must be identical, except where the
oracle's own top-2 logit gap at the deciding row is below the near-tie margin
(1e-2); such rows are counted separately and the oracle then adopts the GPU's
committed state so that both continue from the same history.  The anchor must
be identical, or (where the oracle's head-mean attention has near-equal peaks)
a frame whose oracle attention mass is within the stated relative margin of
the peak.  Logits of every scored row must agree within the tolerance.
"""
from __future__ import annotations

import dataclasses

import numpy as np

import workload as W
from oracle import Oracle, greedy_transcript

TIE_GAP = 1e-2


def scale_for(dims, std):
    """Tolerance multiplier for test models whose logit scale exceeds the
    workloads': bf16 rounding error grows with the logit scale (std * sqrt(d));
    the workloads (std 0.02, d >= 768) get exactly the stated tolerances."""
    import math
    return max(1.0, std * math.sqrt(dims.d_model) / (0.02 * math.sqrt(768)))


@dataclasses.dataclass
class ParityStats:
    rounds: int = 0
    rows: int = 0
    emitted: int = 0
    near_ties: int = 0
    anchor_exact: int = 0
    anchor_near: int = 0
    anchors: int = 0
    max_logit_err: float = 0.0


def logit_tol(dims, scale=1.0):
    return (3e-2 if dims.dtype == "bf16" else 1e-4) * scale


def anchor_tol(dims):
    return 2e-2 if dims.dtype == "bf16" else 1e-4


def compare_round(orc, sess, draft, lens, st: ParityStats, check_logits=True, sample=None, scale=1.0):
    """One teacher-forced round; `sample` restricts the checks to some utterances
    (the oracle then holds only those, in order)."""
    dims = orc.dims
    idx = list(range(len(lens))) if sample is None else list(sample)
    ro = orc.verify(draft[idx], lens[idx])
    rg = sess.verify(draft, lens)
    if check_logits and sample is None and len(ro.rows):
        lg = sess.debug_logits(len(ro.rows)).double().cpu().numpy()
        assert lg.shape == ro.logits.shape
        err = float(np.abs(lg - ro.logits).max())
        st.max_logit_err = max(st.max_logit_err, err)
        assert err <= logit_tol(dims, scale), f"logits differ by {err}"
    st.rounds += 1
    r0 = 0
    for j, b in enumerate(idx):
        if lens[b] < 0:
            assert rg.bonus[b] == -1 and rg.anchor[b] == -1 and rg.accepted[b] == 0
            assert rg.kv_len[b] == ro.kv_len[j]
            continue
        nrow = int(lens[b]) + 1
        st.rows += nrow
        go = ro.argmax[r0:r0 + nrow]
        lo = ro.logits[r0:r0 + nrow]
        n_o, n_g = int(ro.accepted[j]), int(rg.accepted[b])
        same = (n_o == n_g and ro.bonus[j] == rg.bonus[b])
        if not same:
            row = min(n_o, n_g)
            choice = int(draft[b, row]) if n_g > row else int(rg.bonus[b])
            gap = float(lo[row, go[row]] - lo[row, choice])
            assert gap < TIE_GAP * scale, (f"utt {b}: accepted {n_g} vs {n_o}, bonus {rg.bonus[b]} vs {ro.bonus[j]}, "
                                   f"oracle margin {gap} at row {row}")
            st.near_ties += 1
            orc.kv_len[j] = rg.kv_len[b]
            orc.pending[j] = rg.bonus[b]
        else:
            assert rg.kv_len[b] == ro.kv_len[j]
            st.anchors += 1
            prof = ro.anchor_profile[j]
            if rg.anchor[b] == ro.anchor[j]:
                st.anchor_exact += 1
            else:
                a = int(rg.anchor[b])
                assert 0 <= a < len(prof), a
                assert prof[a] >= (1.0 - anchor_tol(dims)) * prof.max(), (
                    f"utt {b}: anchor {a} has oracle mass {prof[a]} vs peak {prof.max()} at {ro.anchor[j]}")
                st.anchor_near += 1
        st.emitted += int(rg.accepted[b]) + 1
        r0 += nrow
    return ro, rg


def run_decode(dims, blob, enc, enc_lens, prompt, total, k, corr, sess_factory, max_rounds=None,
               check_logits=True, k_schedule=None, scale=1.0):
    """Full teacher-forced decode; returns stats.  Drafts come from the oracle's
    own greedy transcript through the workload corruption stream."""
    orc = Oracle(dims, blob)
    orc.encode_cache(enc, enc_lens)
    orc.prefill(prompt)
    snap = orc.snapshot()
    truth = greedy_transcript(orc, prompt, total)
    orc.restore(snap)
    sess = sess_factory()
    sess.encode_cache(enc, enc_lens)
    sess.prefill(prompt)
    assert sess.status() == 0
    st = ParityStats()
    while max_rounds is None or st.rounds < max_rounds:
        kk = k if k_schedule is None else k_schedule(st.rounds)
        draft, lens = W.make_drafts(truth, total, orc.kv_len, kk, corr)
        if np.all(lens < 0):
            break
        compare_round(orc, sess, draft, lens, st, check_logits=check_logits, scale=scale)
    assert sess.status() == 0
    sess.close()
    return st, truth
