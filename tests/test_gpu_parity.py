"""The CUDA draft-verify step against the CPU oracle (teacher-forced, every round).

Sizes: every workload at its full configuration -- the tiny fp32 decoder in
full; the small decoder's batch-16 workload and all sixteen (k, error rate)
points of the batch-32 acceptance/rollback sweep, with the oracle following
sampled utterances through their whole transcripts; the large decoder's
224-token batch-1 decode in full and its batch-64 workload with three sampled
utterances followed to the end.  Also: the small decoder with a batch of
ragged utterances (several GEMM tiles, a ragged encoder tail); edge cases
(k = 0, sitting-out utterances, one encoder frame, a one-token prompt, k = 16,
the context capacity); long-form encoder memories.
"""
import numpy as np
import pytest

import workload as W
from tests.parity import (ParityStats, assert_bounded, compare_round, run_decode, run_sampled_decode,
                          sampled_truth, scale_for)

pytestmark = pytest.mark.gpu


_BLOBS = {}


def _blob(dims, std=0.02):
    key = (dims, std)
    if key not in _BLOBS:
        _BLOBS[key] = W.make_weights(dims, std=std)
    return _BLOBS[key]


def _session(dims, blob, B, k):
    from paper_2608_12703_gb300.session import Session
    return lambda: Session(dims, blob, max_batch=B, max_draft=k)


def _report(name, st: ParityStats):
    print(f"\n[{name}] rounds={st.rounds} rows={st.rows} emitted={st.emitted} near_ties={st.near_ties} "
          f"anchor exact={st.anchor_exact}/{st.anchors} near={st.anchor_near} "
          f"max_logit_err={st.max_logit_err:.3g}")


def test_tiny_fp32_full_workload(built_lib, cuda):
    wl = W.CONFIGS["tiny-fp32-b1-k4"]
    dims = wl.dims
    blob = _blob(dims)
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, wl.batch)
    st, truth = run_decode(dims, blob, enc, list(wl.enc_lens), prompt, list(wl.total_lens), wl.k,
                           W.make_corruption(wl), _session(dims, blob, wl.batch, wl.k))
    _report(wl.name, st)
    assert st.emitted == sum(wl.n_out)
    assert st.near_ties == 0
    assert st.anchor_near == 0


@pytest.mark.parametrize("std,ln_kernel", [(0.02, False), (0.05, False), (0.02, True)])
def test_small_bf16_ragged_batch(built_lib, cuda, monkeypatch, std, ln_kernel):
    """ln_kernel: LayerNorm as its own launch instead of folded into its
    neighbouring GEMMs (read from the environment at create time)."""
    if ln_kernel:
        monkeypatch.setenv("ASRSPEC_LN_FOLD", "0")
    dims = W.SMALL
    blob = _blob(dims, std)
    enc_lens = [1500, 777, 250, 1023, 1]
    total = [W.PROMPT_LEN + n for n in (20, 17, 24, 9, 13)]
    wl = W.Workload("t", dims, 5, 8, tuple(t - W.PROMPT_LEN for t in total), tuple(enc_lens),
                    (0.25, 0.1, 0.5, 0.0, 0.3), "half")
    enc = W.make_encoder_states(dims, enc_lens, 1500)
    prompt = W.make_prompt(dims, 5)
    st, _ = run_decode(dims, blob, enc, enc_lens, prompt, total, 8, W.make_corruption(wl),
                       _session(dims, blob, 5, 8), scale=scale_for(dims, std))
    _report(f"small std={std}{' ln-kernel' if ln_kernel else ''}", st)
    assert st.rows > 50
    assert_bounded(st)


def test_edge_cases_bf16(built_lib, cuda):
    """k = 0 rounds, sitting-out utterances, prompt of one token, k = 16 and a
    decode that runs up to the context capacity of a short positional table."""
    dims = W.ModelDims(n_layers=2, d_model=128, n_heads=2, d_ffn=256, vocab=1000, dtype="bf16",
                       max_pos=40, max_enc=300, anchor_layer=1)
    blob = _blob(dims, 0.1)
    enc_lens = [300, 1, 129]
    enc = W.make_encoder_states(dims, enc_lens, 300)
    prompt = W.make_prompt(dims, 3, length=1)
    total = [40, 30, 12]
    wl = W.Workload("e", dims, 3, 16, tuple(t - 1 for t in total), tuple(enc_lens), (0.2, 0.5, 0.0), "half")
    corr = W.make_corruption(wl)
    sched = lambda r: [16, 0, 3, 16, 1][r % 5]
    st, _ = run_decode(dims, blob, enc, enc_lens, prompt, total, 16, corr, _session(dims, blob, 3, 16),
                       k_schedule=sched, scale=scale_for(dims, 0.1))
    _report("edges", st)
    assert_bounded(st)


def test_edge_cases_fp32(built_lib, cuda):
    dims = W.ModelDims(n_layers=2, d_model=64, n_heads=1, d_ffn=128, vocab=300, dtype="fp32",
                       max_pos=30, max_enc=200, anchor_layer=0)
    blob = _blob(dims, 0.3)
    enc_lens = [200, 3]
    enc = W.make_encoder_states(dims, enc_lens, 200)
    prompt = W.make_prompt(dims, 2)
    total = [30, 25]
    wl = W.Workload("e", dims, 2, 5, tuple(t - 4 for t in total), tuple(enc_lens), (0.3, 0.3), "always")
    st, _ = run_decode(dims, blob, enc, enc_lens, prompt, total, 5, W.make_corruption(wl),
                       _session(dims, blob, 2, 5))
    _report("edges fp32", st)
    assert st.near_ties == 0


@pytest.mark.slow
def test_large_bf16_batch1_full_decode(built_lib, cuda):
    """Full-size large decoder, batch 1, k = 8 with a slip every round: the
    whole 224-token decode, logits of every row checked."""
    wl = W.CONFIGS["large-bf16-b1-k8"]
    dims = wl.dims
    blob = _blob(dims)
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, 1)
    st, _ = run_decode(dims, blob, enc, list(wl.enc_lens), prompt, list(wl.total_lens), wl.k,
                       W.make_corruption(wl), _session(dims, blob, 1, wl.k))
    _report(wl.name, st)
    assert st.emitted == sum(wl.n_out)
    assert_bounded(st)


@pytest.mark.slow
def test_large_bf16_batch64_sampled_full_decode(built_lib, cuda):
    """Full-size batch-64 verify (448 rows, ragged encoder lengths): the oracle
    follows utterances 0, 7 and 63 through their whole transcripts (29, 54 and
    65 tokens); their logits are compared every round while the other 61
    utterances decode alongside."""
    from paper_2608_12703_gb300.session import Session
    wl = W.CONFIGS["large-bf16-b64-k6"]
    dims = wl.dims
    blob = _blob(dims)
    sample = [0, 7, 63]
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, wl.batch)
    orc, snap, truth = sampled_truth(dims, blob, wl, sample, enc, prompt)
    sess = Session(dims, blob, max_batch=wl.batch, max_draft=wl.k)
    st = run_sampled_decode(orc, snap, truth, sess, wl, sample, enc, prompt)
    sess.close()
    _report(wl.name, st)
    assert st.emitted == sum(wl.n_out[b] for b in sample)
    assert_bounded(st)


@pytest.mark.slow
def test_small_bf16_batch16_sampled_full_decode(built_lib, cuda):
    """The small decoder's batch-16 workload (1500 frames each, 128 tokens,
    k = 8, error rate 0.25): the oracle follows four utterances through their
    whole transcripts; 144 rows per round."""
    from paper_2608_12703_gb300.session import Session
    wl = W.CONFIGS["small-bf16-b16-k8"]
    dims = wl.dims
    blob = _blob(dims)
    sample = [0, 5, 10, 15]
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, wl.batch)
    orc, snap, truth = sampled_truth(dims, blob, wl, sample, enc, prompt)
    sess = Session(dims, blob, max_batch=wl.batch, max_draft=wl.k)
    st = run_sampled_decode(orc, snap, truth, sess, wl, sample, enc, prompt)
    sess.close()
    _report(wl.name, st)
    assert st.emitted == sum(wl.n_out[b] for b in sample)
    assert_bounded(st)


_SWEEP = {}


def _sweep_state():
    """One GPU session (batch 32, k up to 16) and one oracle snapshot shared by
    the sixteen sweep configurations: they differ only in k, the error rate
    and the corruption stream."""
    if "sess" not in _SWEEP:
        from paper_2608_12703_gb300.session import Session
        wl = W.CONFIGS["small-bf16-b32-k16-p0.05"]
        dims = wl.dims
        blob = _blob(dims)
        sample = [0, 31]
        enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
        prompt = W.make_prompt(dims, wl.batch)
        orc, snap, truth = sampled_truth(dims, blob, wl, sample, enc, prompt)
        _SWEEP.update(sess=Session(dims, blob, max_batch=wl.batch, max_draft=16), orc=orc, snap=snap,
                      truth=truth, sample=sample, enc=enc, prompt=prompt)
    return _SWEEP


@pytest.mark.slow
@pytest.mark.parametrize("k", [2, 4, 8, 16])
@pytest.mark.parametrize("p", [0.05, 0.2, 0.5, 0.8])
def test_acceptance_rollback_sweep(built_lib, cuda, k, p):
    """The acceptance/rollback sweep (small decoder, batch 32, 1500 frames,
    128 tokens; half the rounds carry a one-token slip that forces a rejection
    and a restart): for every (k, error rate) the oracle follows utterances 0
    and 31 through their whole transcripts, logits checked every round, with
    all 32 utterances scored (up to 544 rows at k = 16)."""
    S = _sweep_state()
    wl = W.CONFIGS[f"small-bf16-b32-k{k}-p{p:g}"]
    st = run_sampled_decode(S["orc"], S["snap"], S["truth"], S["sess"], wl, S["sample"], S["enc"], S["prompt"])
    _report(wl.name, st)
    assert st.emitted == sum(wl.n_out[b] for b in S["sample"])
    assert st.restarts > 0
    assert_bounded(st)


def test_long_form_encoder_memory(built_lib, cuda):
    """Encoder memories past Whisper's 30 s window (the paper's long-audio
    setting, up to about 104 s of concatenated audio = 5200 frames at 20 ms):
    the small bf16 decoder, two utterances of 5200 and 2100 frames, k = 8."""
    import dataclasses
    dims = dataclasses.replace(W.SMALL, max_enc=5200)
    blob = _blob(W.SMALL)   # the same weights (max_enc sizes only the cache)
    enc_lens = [5200, 2100]
    enc = W.make_encoder_states(dims, enc_lens, 5200)
    prompt = W.make_prompt(dims, 2)
    total = [W.PROMPT_LEN + 18, W.PROMPT_LEN + 11]
    wl = W.Workload("long", dims, 2, 8, (18, 11), tuple(enc_lens), (0.2, 0.4), "half", t_max=5200)
    st, _ = run_decode(dims, blob, enc, enc_lens, prompt, total, 8, W.make_corruption(wl),
                       _session(dims, blob, 2, 8), max_rounds=6)
    _report("long-form 5200 + 2100 frames", st)
    assert st.rows > 20
    assert_bounded(st)
