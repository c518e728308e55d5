"""The CUDA draft-verify step against the CPU oracle (teacher-forced, every round).

Sizes: the tiny fp32 workload in full; the small bf16 decoder with a batch of
ragged utterances (several GEMM tiles, a ragged encoder tail); edge cases
(k = 0, sitting-out utterances, one encoder frame, a one-token prompt, k = 16,
the context capacity); and the large decoder at full size on sampled rounds
and sampled utterances of the batch-64 workload.
"""
import numpy as np
import pytest

import workload as W
from tests.parity import ParityStats, compare_round, run_decode, scale_for

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


def test_large_bf16_batch1_sampled_rounds(built_lib, cuda):
    """Full-size large decoder, batch 1, k = 8 with slipped drafts: the first rounds."""
    wl = W.CONFIGS["large-bf16-b1-k8"]
    dims = wl.dims
    blob = _blob(dims)
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, 1)
    total = [W.PROMPT_LEN + 24]
    st, _ = run_decode(dims, blob, enc, list(wl.enc_lens), prompt, total, wl.k, W.make_corruption(wl),
                       _session(dims, blob, 1, wl.k), max_rounds=6)
    _report(wl.name, st)


def test_large_bf16_batch64_sampled_utterances(built_lib, cuda):
    """Full-size batch-64 verify (448 rows, ragged encoder lengths); the oracle
    follows three of the utterances, the others take the workload's drafts."""
    from oracle import Oracle, greedy_transcript
    from paper_2608_12703_gb300.session import Session
    wl = W.CONFIGS["large-bf16-b64-k6"]
    dims = wl.dims
    blob = _blob(dims)
    sample = [0, 7, 63]
    enc = W.make_encoder_states(dims, wl.enc_lens, wl.t_max)
    prompt = W.make_prompt(dims, wl.batch)
    total = np.array(wl.total_lens)
    orc = Oracle(dims, blob)
    orc.encode_cache(enc[sample], [wl.enc_lens[i] for i in sample])
    orc.prefill(prompt[sample])
    snap = orc.snapshot()
    truth_s = greedy_transcript(orc, prompt[sample], np.minimum(total[sample], W.PROMPT_LEN + 16))
    orc.restore(snap)
    truth = np.zeros((wl.batch, dims.max_pos), dtype=np.int64)
    truth[:, :W.PROMPT_LEN] = prompt
    for j, b in enumerate(sample):
        truth[b, :truth_s.shape[1]] = np.where(truth_s[j] >= 0, truth_s[j], 0)
    corr = W.make_corruption(wl)
    sess = Session(dims, blob, max_batch=wl.batch, max_draft=wl.k)
    sess.encode_cache(enc, list(wl.enc_lens))
    sess.prefill(prompt)
    st = ParityStats()
    kv = np.full(wl.batch, W.PROMPT_LEN - 1)
    lim = total.copy()
    lim[sample] = np.minimum(total[sample], W.PROMPT_LEN + 16)
    for _ in range(4):
        kv[sample] = orc.kv_len
        draft, lens = W.make_drafts(truth, lim, kv, wl.k, corr)
        if np.all(lens[sample] < 0):
            break
        ro, rg = compare_round(orc, sess, draft, lens, st, sample=sample)
        kv = rg.kv_len.copy()
    _report(wl.name, st)
    assert sess.status() == 0
    sess.close()


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
