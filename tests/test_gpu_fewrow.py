"""The few-row verify layers (six launches per layer: per-head clusters for
LayerNorm + QKV + self-attention and LayerNorm + cross query +
cross-attention, GEMVs for the projections) against the CPU oracle, against
the tensor-core chain (ASRSPEC_FEWROW=0), and their launch structure.  A
step takes them when the model is bf16 and batch x (k + 1) <= 9 rows."""
import numpy as np
import pytest

import workload as W
from tests.parity import ParityStats, assert_bounded, run_decode, scale_for

pytestmark = pytest.mark.gpu

TL_QKV_SELF, TL_QUERY_CROSS = 8, 9

_BLOBS = {}


def _blob(dims, std=0.02):
    key = (dims, std)
    if key not in _BLOBS:
        _BLOBS[key] = W.make_weights(dims, std=std)
    return _BLOBS[key]


class _Traced:
    """Session factory whose sessions record the launch timeline; the kinds of
    every session are kept when it closes."""

    def __init__(self, dims, blob, B, k):
        self.args = (dims, blob, B, k)
        self.kinds = []

    def __call__(self):
        from paper_2608_12703_gb300 import asrspec as A
        from paper_2608_12703_gb300.session import Session
        dims, blob, B, k = self.args
        s = Session(dims, blob, max_batch=B, max_draft=k)
        A.asr_spec_timeline(s.h, True)
        close = s.close
        rec = self.kinds

        def traced_close():
            if s.h:
                rec.extend(A.asr_spec_timeline_read(s.h)[1].tolist())
            close()
        s.close = traced_close
        return s


def _report(name, st: ParityStats):
    print(f"\n[{name}] rounds={st.rounds} rows={st.rows} emitted={st.emitted} near_ties={st.near_ties} "
          f"anchor exact={st.anchor_exact}/{st.anchors} near={st.anchor_near} "
          f"max_logit_err={st.max_logit_err:.3g} max_profile_err={st.max_profile_err:.3g}")


@pytest.mark.parametrize("B,k,sched", [(1, 8, None), (3, 2, [2, 0, 2, 1])])
def test_fewrow_small_decoder_against_oracle(built_lib, cuda, B, k, sched):
    """Small bf16 decoder (d 768, 12 heads, 12 layers): batch 1 with 8 drafts
    (9 rows, the most a few-row step has), and 3 ragged utterances with k in
    {0, 1, 2} (an utterance that finishes first sits out)."""
    dims = W.SMALL
    blob = _blob(dims)
    enc_lens = [1500, 250, 1][:B]
    total = [W.PROMPT_LEN + n for n in (22, 9, 13)][:B]
    wl = W.Workload("f", dims, B, k, tuple(t - W.PROMPT_LEN for t in total), tuple(enc_lens),
                    (0.25, 0.5, 0.0)[:B], "half")
    enc = W.make_encoder_states(dims, enc_lens, 1500)
    prompt = W.make_prompt(dims, B)
    fac = _Traced(dims, blob, B, k)
    st, _ = run_decode(dims, blob, enc, enc_lens, prompt, total, k, W.make_corruption(wl), fac,
                       k_schedule=(lambda r: sched[r % len(sched)]) if sched else None,
                       scale=scale_for(dims, 0.02))
    _report(f"few-row small B={B} k={k}", st)
    assert st.emitted == sum(t - W.PROMPT_LEN for t in total)
    assert fac.kinds.count(TL_QKV_SELF) == fac.kinds.count(TL_QUERY_CROSS) == st.rounds * dims.n_layers
    assert_bounded(st)


def test_fewrow_long_contexts(built_lib, cuda):
    """Contexts past two key chunks (a 300-token prompt: more self-attention
    chunks than a cluster has CTAs over three utterances) and a long-form
    encoder memory (5200 frames: several chunks per CTA of the cross-attention
    cluster), 3 utterances at k = 2."""
    import dataclasses
    dims = dataclasses.replace(W.SMALL, max_enc=5200)
    blob = _blob(W.SMALL)
    enc_lens = [5200, 1500, 40]
    total = [300 + n for n in (12, 9, 7)]
    wl = W.Workload("lc", dims, 3, 2, tuple(t - 300 for t in total), tuple(enc_lens), (0.2, 0.4, 0.1), "half",
                    t_max=5200)
    enc = W.make_encoder_states(dims, enc_lens, 5200)
    prompt = W.make_prompt(dims, 3, length=300)
    fac = _Traced(dims, blob, 3, 2)
    st, _ = run_decode(dims, blob, enc, enc_lens, prompt, total, 2, W.make_corruption(wl), fac,
                       scale=scale_for(dims, 0.02))
    _report("few-row long contexts", st)
    assert st.emitted == sum(t - 300 for t in total)
    assert fac.kinds.count(TL_QKV_SELF) == st.rounds * dims.n_layers
    assert_bounded(st)


def test_fewrow_large_batch1_against_oracle(built_lib, cuda):
    """Full-size large decoder, batch 1, k = 8: the first rounds, few-row layers."""
    wl = W.CONFIGS["large-bf16-b1-k8"]
    dims = wl.dims
    blob = _blob(dims)
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, 1)
    fac = _Traced(dims, blob, 1, wl.k)
    st, _ = run_decode(dims, blob, enc, list(wl.enc_lens), prompt, [W.PROMPT_LEN + 24], wl.k,
                       W.make_corruption(wl), fac, max_rounds=4)
    _report("few-row " + wl.name, st)
    assert fac.kinds.count(TL_QKV_SELF) == st.rounds * dims.n_layers > 0


def test_fewrow_matches_kernel_chain(built_lib, cuda, monkeypatch):
    """The same rounds through the few-row layers and through the tensor-core
    chain (two sessions in lockstep): logits within bf16 rounding, identical
    accepted / bonus / kv_len / anchor / restart unless a row's top-2 logit gap
    is a near-tie (< 1e-2), after which the two states may differ and the
    comparison stops."""
    from paper_2608_12703_gb300.session import Session
    dims = W.SMALL
    blob = _blob(dims)
    enc_lens = [1100, 300]
    enc = W.make_encoder_states(dims, enc_lens, 1100)
    prompt = W.make_prompt(dims, 2)
    rng = np.random.default_rng(5)
    lens = [np.array([3, 3]), np.array([2, -1]), np.array([0, 3]), np.array([3, 1]), np.array([1, 2])]
    sess = []
    for few in ("1", "0"):
        monkeypatch.setenv("ASRSPEC_FEWROW", few)
        s = Session(dims, blob, max_batch=2, max_draft=3)
        s.encode_cache(enc, enc_lens)
        s.prefill(prompt)
        sess.append(s)
    compared = 0
    for ln in lens + lens:
        dr = rng.integers(0, dims.vocab, size=(2, 3))
        kv0, pend0 = sess[1].state()
        o = [s.verify(dr, ln) for s in sess]
        lg = [s.debug_logits(8).float().cpu().numpy() for s in sess]
        assert lg[0].shape == lg[1].shape
        diff = float(np.max(np.abs(lg[0] - lg[1])))
        assert diff < 3e-2
        same = [(list(x.accepted), list(x.bonus), list(x.kv_len), list(x.anchor), list(x.restart)) for x in o]
        if same[0] != same[1]:
            # two bf16 paths can order a row's top two tokens differently only
            # where their gap is within twice the paths' logit difference
            top2 = np.sort(lg[1], axis=1)[:, -2:]
            assert np.min(top2[:, 1] - top2[:, 0]) <= 2 * diff, (same, "differ without a near-tie")
            # a near-tie: both back to the round's start, with another pending token
            for s in sess:
                s.rollback(kv0, (pend0 + 1) % dims.vocab)
            continue
        compared += 1
    for s in sess:
        assert s.status() == 0
        s.close()
    assert compared >= 7


def test_fewrow_timeline_and_graph_replay(built_lib, cuda):
    """Per step: row plan, embedding, six launches per layer, final LayerNorm,
    LM head, accept + anchor, recorded in order; graph replay gives the
    direct-launch result; rollback then re-verify is bitwise identical."""
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300.session import Session
    dims = W.SMALL
    blob = _blob(dims)
    enc = W.make_encoder_states(dims, [700], 700)
    prompt = W.make_prompt(dims, 1)
    outs = []
    layer = [TL_QKV_SELF, 16 + 2, TL_QUERY_CROSS, 16 + 2, 16 + 4, 16 + 2]
    step = [1, 2] + layer * dims.n_layers + [3, 16 + 6, 6]
    for mode in ("graph", "direct", "timeline"):
        s = Session(dims, blob, max_batch=1, max_draft=8)
        s.encode_cache(enc, [700])
        s.prefill(prompt)
        if mode == "direct":
            A.asr_spec_set_graphs(s.h, False)
        if mode == "timeline":
            A.asr_spec_timeline(s.h, True)
        res = []
        for r in range(3):
            kv0, pend0 = s.state()
            o = s.verify(np.array([[r + 1, 2, 3, 4, 5, 6, 7, 8]]), np.array([8 - r]))
            first = (list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor), list(o.restart))
            l1 = s.debug_logits(9).float().cpu().numpy() if mode != "timeline" else None
            s.rollback(kv0, pend0)
            o = s.verify(np.array([[r + 1, 2, 3, 4, 5, 6, 7, 8]]), np.array([8 - r]))
            again = (list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor), list(o.restart))
            assert first == again
            if mode != "timeline":   # (the logits recomputation is a launch of its own)
                assert np.array_equal(l1, s.debug_logits(9).float().cpu().numpy())
            res.append(first)
        if mode == "timeline":
            ns, kinds = A.asr_spec_timeline_read(s.h)
            assert list(kinds) == step * 6
            ns = ns.astype(np.int64)
            assert np.all(ns[:, 3] > 0) and np.all(ns[:, 0] <= ns[:, 1]) and np.all(ns[:, 1] <= ns[:, 3])
            few = np.isin(np.array(kinds), [TL_QKV_SELF, TL_QUERY_CROSS])
            assert np.all(ns[few, 2] > 0) and np.all(ns[few, 2] <= ns[few, 3])
        assert s.status() == 0
        s.close()
        outs.append(res)
    assert outs[0] == outs[1] == outs[2]
