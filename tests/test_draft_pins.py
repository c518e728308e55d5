"""Pins of the draft oracle (oracle/draft.py): its block against torch.nn's
decoder layer with the audio window as a memory mask, the lossless invariant
of the real cached loop with it, the window's isolation of the audio, and the
draft cache against a teacher-forced pass over the committed sequence."""
import dataclasses

import numpy as np
import pytest
import torch
import torch.nn as nn
import torch.nn.functional as F

import workload as W
from oracle import Oracle, greedy_transcript
from oracle.draft import Draft, speculative_decode
from oracle.window import window

TINY = W.ModelDims(n_layers=4, d_model=64, n_heads=2, d_ffn=256, vocab=97, dtype="fp32",
                   max_pos=64, max_enc=80, anchor_layer=2)
ENC_LENS = [80, 33, 9]


def _setup(std=0.3):
    blob = W.make_weights(TINY, std=std)
    enc = W.make_encoder_states(TINY, ENC_LENS, max(ENC_LENS))
    o = Oracle(TINY, blob)
    o.encode_cache(enc, ENC_LENS)
    dr = Draft(o, W.make_draft_weights(TINY, std=std))
    return o, dr, blob, enc


def _t(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float64).copy())


def test_draft_block_matches_torch_decoder_layer():
    """Teacher-forced: given tokens and representations per position, the
    draft's step-by-step cached forward equals a full-sequence
    nn.TransformerDecoderLayer (pre-LN, erf GELU, causal, audio window as a
    key-padding mask) with the same weights."""
    o, dr, blob, enc = _setup()
    dr.encode()
    b, n = 0, 12
    rng = np.random.default_rng(1)
    tokens = rng.integers(0, TINY.vocab, size=n)
    feats = rng.standard_normal((n, 4, TINY.d_model))
    lo, hi = window(40, ENC_LENS[b])
    got = np.stack([dr.step(b, int(tokens[p]), p, feats[p], (lo, hi))[0] for p in range(n)])

    dw = W.make_draft_weights(TINY, std=0.3)
    lay = W.draft_weight_layout(TINY)

    def g(name):
        off, shape = lay[name]
        return _t(dw[off:off + int(np.prod(shape))].reshape(shape))
    d, H = TINY.d_model, TINY.n_heads
    m = nn.TransformerDecoderLayer(d, H, dim_feedforward=W.draft_ffn(TINY), dropout=0.0, activation="gelu",
                                   layer_norm_eps=1e-5, batch_first=True, norm_first=True).double().eval()
    z = torch.zeros(d, dtype=torch.float64)
    with torch.no_grad():
        m.self_attn.in_proj_weight.copy_(torch.cat([g("wq"), g("wk"), g("wv")]))
        m.self_attn.in_proj_bias.copy_(torch.cat([g("bq"), z, g("bv")]))
        m.self_attn.out_proj.weight.copy_(g("wo"))
        m.self_attn.out_proj.bias.copy_(g("bo"))
        m.multihead_attn.in_proj_weight.copy_(torch.cat([g("wcq"), g("wck"), g("wcv")]))
        m.multihead_attn.in_proj_bias.copy_(torch.cat([g("bcq"), z, g("bcv")]))
        m.multihead_attn.out_proj.weight.copy_(g("wco"))
        m.multihead_attn.out_proj.bias.copy_(g("bco"))
        m.linear1.weight.copy_(g("w1"))
        m.linear1.bias.copy_(g("b1"))
        m.linear2.weight.copy_(g("w2"))
        m.linear2.bias.copy_(g("b2"))
        for i in (1, 2, 3):
            getattr(m, f"norm{i}").weight.copy_(g(f"ln{i}_g"))
            getattr(m, f"norm{i}").bias.copy_(g(f"ln{i}_b"))
        lnf = nn.LayerNorm(d, eps=1e-5).double()
        lnf.weight.copy_(g("lnf_g"))
        lnf.bias.copy_(g("lnf_b"))
        tok_emb = _t(W.weight_view(TINY, blob, "tok_emb"))
        pos_emb = _t(W.weight_view(TINY, blob, "pos_emb"))
        x = F.linear(_t(feats.reshape(n, 4 * d)), g("w_in"), g("b_in")) + tok_emb[torch.as_tensor(tokens)] + pos_emb[:n]
        mem = _t(enc[b, :ENC_LENS[b]]).unsqueeze(0)
        pad = torch.ones(1, ENC_LENS[b], dtype=torch.bool)
        pad[0, lo:hi] = False
        causal = nn.Transformer.generate_square_subsequent_mask(n, dtype=torch.float64)
        y = m(x.unsqueeze(0), mem, tgt_mask=causal, memory_key_padding_mask=pad)
        ref = (lnf(y[0]) @ tok_emb.T).numpy()
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-10)


@pytest.mark.parametrize("kind", ["anchor", "shifted", "random", None])
def test_real_cached_loop_is_lossless(kind):
    """Whatever the draft proposes, the loop returns the target's greedy
    transcript (Sec. 3: identical under exact arithmetic)."""
    o, dr, blob, enc = _setup()
    prompt = W.make_prompt(TINY, 3)
    total = [40, 25, 31]
    snap_ready = Oracle(TINY, blob)
    snap_ready.encode_cache(enc, ENC_LENS)
    snap_ready.prefill(prompt)
    truth = greedy_transcript(snap_ready, prompt, total)
    seqs, rounds = speculative_decode(o, dr, prompt, total, 4, kind)
    for b in range(3):
        assert seqs[b] == list(truth[b, :total[b]])
    # every round emits its accepted drafts plus the bonus token (Sec. 3)
    emitted = sum(int(acc[b]) + 1 for lens, acc in rounds for b in range(3) if lens[b] >= 0)
    assert emitted == sum(total) - 3 * prompt.shape[1]


def test_window_isolates_the_audio():
    """Proposals from a restricted window do not change when frames outside
    it change; from the unrestricted arm they do."""
    o, dr, blob, enc = _setup()
    prompt = W.make_prompt(TINY, 3)
    o.prefill(prompt)
    dr.encode()
    dr.prefill(prompt)
    b, P = 0, int(o.kv_len[0])
    feat = o.prefill_feats[b, -1]
    win = window(40, ENC_LENS[b])
    cache = (dr.Ks.copy(), dr.Vs.copy())

    def logits(w):
        dr.Ks, dr.Vs = cache[0].copy(), cache[1].copy()
        return dr.step(b, int(o.pending[b]), P, feat, w)[0]

    a_win, a_all = logits(win), logits(None)
    rng = np.random.default_rng(9)
    out = np.ones(ENC_LENS[b], dtype=bool)
    out[win[0]:win[1]] = False
    dr.Kd[b][out] += rng.standard_normal(dr.Kd[b][out].shape)
    dr.Vd[b][out] += rng.standard_normal(dr.Vd[b][out].shape)
    np.testing.assert_array_equal(logits(win), a_win)
    assert np.abs(logits(None) - a_all).max() > 1e-6


def test_draft_cache_is_teacher_forced_on_the_committed_sequence():
    """After the loop, every committed position's draft entry is what a
    teacher-forced pass over the final sequence writes: token p with the
    target's representations of position p - 1 (the catch-up after each
    verification).  An 8-token vocabulary makes some random-init proposals
    right, so that rounds accept drafts and the catch-up runs."""
    dims = dataclasses.replace(TINY, vocab=8)
    blob = W.make_weights(dims, std=0.3)
    enc = W.make_encoder_states(dims, ENC_LENS, max(ENC_LENS))
    o = Oracle(dims, blob)
    o.encode_cache(enc, ENC_LENS)
    dr = Draft(o, W.make_draft_weights(dims, std=0.3))
    prompt = W.make_prompt(dims, 3)
    total = [40, 32, 37]
    seqs, rounds = speculative_decode(o, dr, prompt, total, 4, "anchor")
    assert sum(int(a) for _, acc in rounds for a in acc) >= 5
    ref_t = Oracle(dims, blob)
    ref_t.encode_cache(enc, ENC_LENS)
    ref_d = Draft(ref_t, W.make_draft_weights(dims, std=0.3))
    ref_d.encode()
    for b in range(3):
        kv = int(o.kv_len[b])
        seq = seqs[b]
        rows = [(b, int(seq[p]), p) for p in range(kv)]
        ref_t._forward(rows)
        feats = ref_t.last_feats
        zero = np.zeros((4, dims.d_model))
        for p in range(kv):
            ref_d.step(b, int(seq[p]), p, feats[p - 1] if p > 0 else zero)
        np.testing.assert_allclose(dr.Ks[b, :kv], ref_d.Ks[b, :kv], rtol=0, atol=1e-10)
        np.testing.assert_allclose(dr.Vs[b, :kv], ref_d.Vs[b, :kv], rtol=0, atol=1e-10)


def _no_catch_up(self, b, P_old, drafts_b, n, feats_b):
    return None                     # keeps the entries the continuation proposals wrote


def _step_without_features(orig):
    def step(self, b, token, pos, feat, win=None):
        return orig(self, b, token, pos, np.zeros_like(feat), win)
    return step


@pytest.mark.parametrize("mistake", ["no_catch_up", "features_dropped"])
def test_pins_catch_planted_draft_mistakes(monkeypatch, mistake):
    """A plausible mistake planted in the draft oracle makes a pin fail."""
    import oracle.draft as D
    if mistake == "no_catch_up":
        monkeypatch.setattr(D.Draft, "catch_up", _no_catch_up)
        with pytest.raises(AssertionError):
            test_draft_cache_is_teacher_forced_on_the_committed_sequence()
    else:
        monkeypatch.setattr(D.Draft, "step", _step_without_features(D.Draft.step))
        with pytest.raises(AssertionError):
            test_draft_block_matches_torch_decoder_layer()


def test_confidence_threshold_varies_the_block_and_stays_lossless():
    """Threshold 0 proposes k every round; threshold 1 proposes nothing (plain
    greedy decoding, one token per round); in between the block length varies
    per utterance and the output is still the target's greedy transcript."""
    from oracle.draft import acceptance_stats
    prompt = W.make_prompt(TINY, 3)
    total = [30, 22, 27]
    out = {}
    for thr in (0.0, 0.4, 1.0):
        o, dr, blob, enc = _setup()
        seqs, rounds = speculative_decode(o, dr, prompt, total, 4, "anchor", threshold=thr)
        out[thr] = (seqs, rounds)
    ref_t = Oracle(TINY, W.make_weights(TINY, std=0.3))
    ref_t.encode_cache(W.make_encoder_states(TINY, ENC_LENS, max(ENC_LENS)), ENC_LENS)
    ref_t.prefill(prompt)
    truth = greedy_transcript(ref_t, prompt, total)
    for thr, (seqs, rounds) in out.items():
        assert all(seqs[b] == list(truth[b, :total[b]]) for b in range(3)), thr
    l0 = np.concatenate([l for l, _ in out[0.0][1]])
    l1 = np.concatenate([l for l, _ in out[1.0][1]])
    lm = np.concatenate([l for l, _ in out[0.4][1]])
    assert np.all(l1[l1 >= 0] == 0)
    assert len(out[1.0][1]) == max(total) - prompt.shape[1]      # one token per round
    full = W.round_lens(total, [prompt.shape[1] - 1] * 3, 4)
    assert np.all(l0[:3] == full)
    assert 0 < np.sum(lm[lm >= 0]) < np.sum(l0[l0 >= 0])         # some blocks cut short
    assert acceptance_stats(out[1.0][1], 4)["L"] == 0.0


def test_acceptance_stats_follow_the_definitions():
    """s_j, a_1, a_j^c and L (Sec. 3) on rounds built by hand, and the closed
    form under independent per-token corruption: s_j = q^j, a_j^c = q."""
    from oracle.draft import acceptance_stats
    rounds = [(np.array([3, 3, -1]), np.array([3, 0, 0])), (np.array([3, 1, 2]), np.array([1, 1, 2]))]
    st = acceptance_stats(rounds, 3)
    assert st["s_1"] == pytest.approx(4 / 5) and st["s_2"] == pytest.approx(2 / 4) and st["s_3"] == pytest.approx(1 / 3)
    assert st["a_1"] == st["s_1"] and st["a_2^c"] == pytest.approx((2 / 4) / (4 / 5))
    assert st["L"] == pytest.approx((3 + 0 + 1 + 1 + 2) / 5)
    rng = np.random.default_rng(0)
    q, K, n = 0.7, 4, 20000
    hits = rng.random((n, K)) < q
    acc = np.where(hits.all(axis=1), K, np.argmin(hits, axis=1))
    st = acceptance_stats([(np.full(n, K), acc)], K)
    for j in range(1, K + 1):
        assert st[f"s_{j}"] == pytest.approx(q ** j, abs=0.02)
    assert st["a_2^c"] == pytest.approx(q, abs=0.02) and st["L"] == pytest.approx(sum(q ** j for j in range(1, K + 1)), abs=0.03)
