"""The fused few-row verify (one persistent kernel for the layers and the LM
head) against the CPU oracle, against the multi-kernel chain, and its launch
structure.  With ASRSPEC_FUSED=1 at create, a step runs fused when
batch x (k + 1) <= 9 rows and the model is bf16 with d_model in
{512, 768, 1024, 1280}."""
import numpy as np
import pytest

import workload as W
from tests.parity import ParityStats, compare_round, run_decode, scale_for

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _fused_on(monkeypatch):
    monkeypatch.setenv("ASRSPEC_FUSED", "1")

_BLOBS = {}


def _blob(dims, std=0.02):
    key = (dims, std)
    if key not in _BLOBS:
        _BLOBS[key] = W.make_weights(dims, std=std)
    return _BLOBS[key]


class _Counted:
    """Session factory that records the per-class launch counts of every
    session it made, read just before the session closes."""

    def __init__(self, dims, blob, B, k):
        self.args = (dims, blob, B, k)
        self.launches = []

    def __call__(self):
        from paper_2608_12703_gb300 import asrspec as A
        from paper_2608_12703_gb300.session import Session
        dims, blob, B, k = self.args
        s = Session(dims, blob, max_batch=B, max_draft=k)
        close = s.close
        rec = self.launches

        def counted_close():
            if s.h:
                rec.append(A.asr_spec_profile_read(s.h)[1].copy())
            close()
        s.close = counted_close
        return s


def _fused_launches(counts):
    from paper_2608_12703_gb300 import asrspec as A
    return int(sum(c[A.PROF_CLASSES.index("fused")] for c in counts))


def _report(name, st: ParityStats):
    print(f"\n[{name}] rounds={st.rounds} rows={st.rows} emitted={st.emitted} near_ties={st.near_ties} "
          f"anchor exact={st.anchor_exact}/{st.anchors} near={st.anchor_near} "
          f"max_logit_err={st.max_logit_err:.3g}")


@pytest.mark.parametrize("B,k,sched", [(1, 8, None), (3, 2, [2, 0, 2, 1])])
def test_fused_small_decoder_against_oracle(built_lib, cuda, B, k, sched):
    """Small bf16 decoder (d 768, 12 layers): batch 1 with 8 drafts (9 rows,
    the most one step may have), and 3 ragged utterances with k in {0, 1, 2}
    (an utterance that finishes first sits out)."""
    dims = W.SMALL
    blob = _blob(dims)
    enc_lens = [1500, 250, 1][:B]
    total = [W.PROMPT_LEN + n for n in (22, 9, 13)][:B]
    wl = W.Workload("f", dims, B, k, tuple(t - W.PROMPT_LEN for t in total), tuple(enc_lens),
                    (0.25, 0.5, 0.0)[:B], "half")
    enc = W.make_encoder_states(dims, enc_lens, 1500)
    prompt = W.make_prompt(dims, B)
    fac = _Counted(dims, blob, B, k)
    st, _ = run_decode(dims, blob, enc, enc_lens, prompt, total, k, W.make_corruption(wl), fac,
                       k_schedule=(lambda r: sched[r % len(sched)]) if sched else None,
                       scale=scale_for(dims, 0.02))
    _report(f"fused small B={B} k={k}", st)
    assert st.emitted == sum(t - W.PROMPT_LEN for t in total)
    assert _fused_launches(fac.launches) == st.rounds


def test_fused_large_batch1_against_oracle(built_lib, cuda):
    """Full-size large decoder, batch 1, k = 8: the first rounds, fused."""
    wl = W.CONFIGS["large-bf16-b1-k8"]
    dims = wl.dims
    blob = _blob(dims)
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, 1)
    fac = _Counted(dims, blob, 1, wl.k)
    st, _ = run_decode(dims, blob, enc, list(wl.enc_lens), prompt, [W.PROMPT_LEN + 24], wl.k,
                       W.make_corruption(wl), fac, max_rounds=4)
    _report("fused " + wl.name, st)
    assert _fused_launches(fac.launches) == st.rounds > 0


def test_fused_matches_kernel_chain(built_lib, cuda, monkeypatch):
    """The same rounds through the fused kernel and through the multi-kernel
    chain (two sessions in lockstep): logits within bf16 rounding, identical
    accepted / bonus / kv_len / anchor unless a row's top-2 logit gap is a
    near-tie (< 1e-2), after which the two states may differ and the
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
    for fused in ("1", "0"):
        monkeypatch.setenv("ASRSPEC_FUSED", fused)
        s = Session(dims, blob, max_batch=2, max_draft=3)
        s.encode_cache(enc, enc_lens)
        s.prefill(prompt)
        sess.append(s)
    compared = 0
    for ln in lens:
        dr = rng.integers(0, dims.vocab, size=(2, 3))
        o = [s.verify(dr, ln) for s in sess]
        lg = [s.debug_logits(8).float().cpu().numpy() for s in sess]
        assert lg[0].shape == lg[1].shape
        assert np.max(np.abs(lg[0] - lg[1])) < 3e-2
        same = [(list(x.accepted), list(x.bonus), list(x.kv_len), list(x.anchor)) for x in o]
        if same[0] != same[1]:
            top2 = np.sort(lg[1], axis=1)[:, -2:]
            assert np.min(top2[:, 1] - top2[:, 0]) < 1e-2, (same, "differ without a near-tie")
            break
        compared += 1
    for s in sess:
        assert s.status() == 0
        s.close()
    assert compared >= 3


def test_fused_timeline_and_graph_replay(built_lib, cuda):
    """Three launches per step (row plan, fused layers + LM head, accept +
    anchor), recorded in order; graph replay gives the direct-launch result;
    rollback then re-verify is bitwise identical."""
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300.session import Session
    dims = W.SMALL
    blob = _blob(dims)
    enc = W.make_encoder_states(dims, [700], 700)
    prompt = W.make_prompt(dims, 1)
    outs = []
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
            first = (list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor))
            l1 = s.debug_logits(9).float().cpu().numpy() if mode != "timeline" else None
            s.rollback(kv0, pend0)
            o = s.verify(np.array([[r + 1, 2, 3, 4, 5, 6, 7, 8]]), np.array([8 - r]))
            again = (list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor))
            assert first == again
            if mode != "timeline":   # (the logits recomputation is a launch of its own)
                assert np.array_equal(l1, s.debug_logits(9).float().cpu().numpy())
            res.append(first)
        if mode == "timeline":
            ns, kinds = A.asr_spec_timeline_read(s.h)
            assert list(kinds) == [1, 7, 6] * 6
            ns = ns.astype(np.int64)
            assert np.all(ns[:, 3] > 0) and np.all(ns[:, 0] <= ns[:, 1]) and np.all(ns[:, 1] <= ns[:, 3])
            fused = np.array(kinds) == 7
            assert np.all(ns[fused, 2] > 0) and np.all(ns[fused, 2] <= ns[fused, 3])
        assert s.status() == 0
        s.close()
        outs.append(res)
    assert outs[0] == outs[1] == outs[2]
