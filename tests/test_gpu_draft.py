"""The draft side on the GPU against the oracle's one-block draft, round by round.

Each round the library's draft proposes on the device (catch-up of the last
verification, restart, continuations, the round's audio window); the oracle's
draft (oracle/draft.py) scores the same positions in float64, fed the GPU's
proposals (teacher-forced), and every GPU proposal must be the oracle draft's
argmax unless the oracle's own top-2 gap there is below the near-tie margin
(and such flips stay within half of those close calls, plus the target's
near-tie allowance).
Both targets then verify the GPU's drafts (tests/parity.py: accepted length,
bonus, committed length, restart, anchor, logits), the oracle draft catches up
on what the GPU committed, and the next round starts from the same state.
With no near-tie the GPU's emitted tokens are the target's greedy transcript
(the lossless invariant of the speculative loop).

Cases: batch 1 with k = 8 (nine verify rows, the few-row layers), a ragged
batch of five under each window kind (anchor, shifted, random centres, none),
a one-token prompt with k = 0 rounds and utterances that finish at once, the
confidence threshold (blocks of varying length);
and the device loop (propose -> verify, nothing read back between rounds)
against the host-stepped loop, output for output.
"""
import numpy as np
import pytest

import workload as W
from oracle import Oracle, greedy_transcript
from oracle.draft import Draft
from oracle.window import window, window_center
from tests.parity import TIE_GAP, ParityStats, assert_bounded, compare_round, near_tie_bound, scale_for

pytestmark = pytest.mark.gpu

# d_ffn = 4 d so that batch-1 verification runs the few-row layers
DIMS = W.ModelDims(n_layers=4, d_model=256, n_heads=4, d_ffn=1024, vocab=1000, dtype="bf16",
                   max_pos=96, max_enc=300, anchor_layer=2)
STD = 0.05


class DraftStats:
    def __init__(self):
        self.proposals = 0
        self.near_ties = 0
        self.max_gap = 0.0
        self.gaps = []          # oracle top-2 gap of every proposal
        self.flip_gaps = []
        self.thr_decisions = 0  # threshold decisions checked, and those within THR_MARGIN that went the other way
        self.thr_near = 0
        self.cut = 0            # rounds the threshold ended early


THR_MARGIN = 0.05   # relative: the draft's top probability within this of the threshold decides either way


def _forced_round(dro, b, pending, P, feat, lens, props, win, ds, scale, threshold=0.0, lens_max=None):
    """The oracle draft over the GPU's round for utterance b: the restart at P
    and the continuations, each fed the GPU's previous proposal.  With a
    confidence threshold the GPU proposes lens <= lens_max tokens; each
    proposal's oracle probability must reach the threshold, and a block the
    GPU ended early must end at a position the oracle also finds below it
    (both unless the probability is within THR_MARGIN of the threshold)."""
    lens_max = lens if lens_max is None else lens_max
    if lens_max == 0:
        dro.step(b, int(pending), P, feat, win)
        return
    tok, f = int(pending), feat
    steps = lens + 1 if lens < lens_max else lens
    for i in range(steps):
        logits, x = dro.step(b, tok, P + i, f, win)
        if threshold > 0.0:
            e = np.exp(logits - logits.max())
            p_top = 1.0 / e.sum()
            below = p_top < threshold
            if below != (i == lens):
                assert abs(p_top / threshold - 1.0) < THR_MARGIN, (
                    f"utt {b}, position {i + 1}: oracle top probability {p_top} vs threshold {threshold}, "
                    f"GPU {'ended' if i == lens else 'proposed'}")
                ds.thr_near += 1
            ds.thr_decisions += 1
        if i == lens:
            break
        a, g = int(np.argmax(logits)), int(props[i])
        ds.proposals += 1
        top2 = np.partition(logits, -2)[-2:]
        ds.gaps.append(float(top2[1] - top2[0]))
        if a != g:
            gap = float(logits[a] - logits[g])
            ds.max_gap = max(ds.max_gap, gap)
            assert gap < TIE_GAP * scale, f"utt {b}, proposal {i + 1}: GPU {g} vs oracle {a}, oracle margin {gap}"
            ds.near_ties += 1
            ds.flip_gaps.append(gap)
        tok, f = g, np.tile(x, (4, 1))


def run_lockstep(enc_lens, total, k, kind, prompt_len=W.PROMPT_LEN, k_sched=None, seed=0, threshold=0.0):
    from paper_2608_12703_gb300.session import DraftModel, Session
    B = len(enc_lens)
    blob = W.make_weights(DIMS, std=STD)
    dblob = W.make_draft_weights(DIMS, std=STD)
    t_max = max(enc_lens)
    enc = W.make_encoder_states(DIMS, enc_lens, t_max)
    prompt = W.make_prompt(DIMS, B, length=prompt_len)
    P0 = prompt.shape[1]
    orc = Oracle(DIMS, blob)
    orc.encode_cache(enc, enc_lens)
    orc.prefill(prompt)
    snap = orc.snapshot()
    truth = greedy_transcript(orc, prompt, total)
    orc.restore(snap)
    dro = Draft(orc, dblob)
    dro.encode()
    dro.prefill(prompt)
    sess = Session(DIMS, blob, max_batch=B, max_draft=k)
    dm = DraftModel(sess, dblob, total, k, kind, threshold=threshold)
    sess.encode_cache(enc, enc_lens)
    sess.prefill(prompt)
    assert sess.status() == 0
    scale = scale_for(DIMS, STD)
    feat = [orc.prefill_feats[b, -1] if P0 > 1 else np.zeros((4, DIMS.d_model)) for b in range(B)]
    anchor = [0] * B
    rng = np.random.default_rng(seed)
    st, ds = ParityStats(), DraftStats()
    seqs = [list(prompt[b]) for b in range(B)]
    log = []
    while True:
        kk = k if k_sched is None else k_sched(st.rounds)
        lens_o = W.round_lens(total, orc.kv_len, kk)
        if np.all(lens_o < 0):
            break
        centers = [int(rng.integers(0, T)) for T in enc_lens]
        if kind == "random":
            dm.set_centers(centers)
        dg, lg = dm.propose(kk)
        dg, lg = sess.host(dg).copy(), sess.host(lg).copy()
        if threshold > 0.0:
            np.testing.assert_array_equal(lg < 0, lens_o < 0)
            assert np.all(lg <= lens_o)
            ds.cut += int(np.sum((lg >= 0) & (lg < lens_o)))
        else:
            np.testing.assert_array_equal(lg, lens_o)
        for b in range(B):
            if lens_o[b] < 0:
                continue
            T = enc_lens[b]
            if kind is None:
                win = None
            else:
                c = centers[b] if kind == "random" else window_center(kind, anchor[b], T)
                win = window(c, T)
            _forced_round(dro, b, orc.pending[b], int(orc.kv_len[b]), feat[b], int(lg[b]), dg[b], win, ds,
                          scale, threshold, int(lens_o[b]))
        P_old = orc.kv_len.copy()
        draft = dg if kk > 0 else np.zeros((B, 0), dtype=np.int32)
        ro, rg = compare_round(orc, sess, draft, lg, st, scale=scale)
        log.append((dg.copy(), lg.copy(), rg.accepted.copy(), rg.bonus.copy()))
        r0 = 0
        for b in range(B):
            if lg[b] < 0:
                continue
            n = int(rg.accepted[b])
            rows = ro.feats[r0:r0 + int(lg[b]) + 1]
            dro.catch_up(b, int(P_old[b]), dg[b], n, rows)
            feat[b] = rows[n]
            anchor[b] = int(rg.anchor[b])
            seqs[b] += [int(x) for x in dg[b, :n]] + [int(rg.bonus[b])]
            r0 += int(lg[b]) + 1
    assert sess.status() == 0
    sess.close()
    return st, ds, seqs, truth, log


def _check(name, st, ds, seqs, truth, total):
    print(f"\n[{name}] rounds={st.rounds} rows={st.rows} proposals={ds.proposals} draft near-ties={ds.near_ties} "
          f"target near-ties={st.near_ties} anchors exact={st.anchor_exact}/{st.anchors}")
    g = np.asarray(ds.gaps)
    print("  oracle draft top-2 gaps: " + " ".join(f"<{t:g}:{int((g < t).sum())}" for t in (0.002, 0.005, 0.01,
          0.02, 0.05)) + f"  flip gaps: {sorted(round(x, 4) for x in ds.flip_gaps)}")
    assert_bounded(st)
    # A flip needs the GPU's logit errors to close the oracle's top-2 gap, in
    # the one direction of the two that reorders them: for errors symmetric
    # about zero at most about half of the close calls (gap below the margin)
    # flip, whatever their size; a systematic error (a wrong window, row or
    # representation) flips most of them and opens gaps beyond the margin.
    close = int((np.asarray(ds.gaps) < TIE_GAP * scale_for(DIMS, STD)).sum())
    assert ds.near_ties <= near_tie_bound(ds.proposals) + close // 2, (ds.near_ties, close)
    for b, s in enumerate(seqs):
        assert len(s) == total[b]
    if st.near_ties == 0:
        for b, s in enumerate(seqs):
            np.testing.assert_array_equal(np.asarray(s), truth[b, :total[b]])


def test_draft_batch1_fewrow(built_lib, cuda):
    total = [W.PROMPT_LEN + 60]
    st, ds, seqs, truth, _ = run_lockstep([300], total, 8, "anchor")
    _check("b1 k8 anchor", st, ds, seqs, truth, total)
    assert ds.proposals > 40


@pytest.mark.parametrize("kind", ["anchor", "shifted", "random", None])
def test_draft_ragged_batch_windows(built_lib, cuda, kind):
    enc_lens = [300, 57, 1, 181, 29]
    total = [W.PROMPT_LEN + n for n in (40, 23, 31, 12, 35)]
    st, ds, seqs, truth, _ = run_lockstep(enc_lens, total, 6, kind, seed=3)
    _check(f"b5 k6 {kind}", st, ds, seqs, truth, total)
    assert ds.proposals > 60


def test_draft_edges(built_lib, cuda):
    """A one-token prompt (zero representations for the first restart), k = 0
    rounds between full ones, an utterance whose only round offers no draft
    (total = prompt + 1) and one that holds its transcript from the start
    (total = prompt)."""
    enc_lens = [200, 9, 77, 40]
    total = [30, 2, 25, 1]
    sched = lambda r: [5, 0, 2, 5, 1][r % 5]
    st, ds, seqs, truth, _ = run_lockstep(enc_lens, total, 5, "anchor", prompt_len=1, k_sched=sched)
    _check("edges", st, ds, seqs, truth, total)


def test_draft_confidence_threshold(built_lib, cuda):
    """Variable block lengths from the confidence threshold (App. "Draft length
    and confidence threshold"), set between the draft's typical top
    probabilities so that some blocks end early and others run to k."""
    enc_lens = [300, 57, 181]
    total = [W.PROMPT_LEN + n for n in (30, 21, 26)]
    st, ds, seqs, truth, _ = run_lockstep(enc_lens, total, 6, "anchor", threshold=0.009)
    _check("threshold 0.009", st, ds, seqs, truth, total)
    print(f"  threshold decisions {ds.thr_decisions}, near-threshold {ds.thr_near}, blocks cut {ds.cut}")
    assert ds.cut > 3
    assert ds.thr_near <= near_tie_bound(ds.thr_decisions)


def test_device_loop_matches_host_stepped(built_lib, cuda):
    """The device loop (draft -> verify -> next round, no host read in between)
    gives the host-stepped lockstep's drafts, lens, accepted and bonus, round
    for round."""
    import torch
    from paper_2608_12703_gb300.session import DraftModel, Session
    enc_lens = [300, 57, 181]
    total = [W.PROMPT_LEN + n for n in (30, 17, 25)]
    k = 6
    _, _, _, _, log = run_lockstep(enc_lens, total, k, "anchor")
    B = len(enc_lens)
    blob = W.make_weights(DIMS, std=STD)
    dblob = W.make_draft_weights(DIMS, std=STD)
    enc = W.make_encoder_states(DIMS, enc_lens, max(enc_lens))
    prompt = W.make_prompt(DIMS, B)
    sess = Session(DIMS, blob, max_batch=B, max_draft=k)
    dm = DraftModel(sess, dblob, total, k, "anchor")
    sess.encode_cache(enc, enc_lens)
    sess.prefill(prompt)
    n_rounds = len(log)
    with torch.cuda.stream(sess.stream):
        rec_d = torch.zeros((n_rounds, B, k), dtype=torch.int32, device=sess.dev)
        rec_o = torch.zeros((n_rounds, 3, B), dtype=torch.int32, device=sess.dev)
        for r in range(n_rounds):
            d, l = dm.propose()
            o = sess.verify_device(d, l, k)
            rec_d[r].copy_(d)
            rec_o[r, 0].copy_(l)
            rec_o[r, 1:].copy_(o[:2])
    rd, ro = sess.host(rec_d), sess.host(rec_o)
    assert sess.status() == 0
    sess.close()
    for r, (dg, lg, acc, bon) in enumerate(log):
        np.testing.assert_array_equal(ro[r, 0], lg)
        np.testing.assert_array_equal(ro[r, 1], acc)
        np.testing.assert_array_equal(ro[r, 2], bon)
        for b in range(B):
            np.testing.assert_array_equal(rd[r, b, :max(lg[b], 0)], dg[b, :max(lg[b], 0)])
