"""The seeded input generators both sides read (weights, encoder states,
prompts, drafts), pinned against a library and their stated definitions."""
import dataclasses

import numpy as np
import pytest
import torch

import workload as W


def test_bf16_round_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * s for s in (1e-3, 1.0, 1e3)])
    # exact ties: the halfway point between two bf16 values rounds to even
    ties = (np.arange(1, 2000, dtype=np.uint32) << 16 | 0x8000).view(np.float32)
    x = np.concatenate([x, ties, -ties, np.float32([0.0, -0.0, 1e-38, 3.0e38])])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    np.testing.assert_array_equal(W.bf16_round(x), ref)


def test_weights_are_seeded_shaped_and_bf16_representable():
    dims = W.ModelDims(n_layers=2, d_model=64, n_heads=1, d_ffn=128, vocab=50, dtype="bf16",
                       max_pos=16, max_enc=8, anchor_layer=1)
    a, b = W.make_weights(dims), W.make_weights(dims)
    assert np.array_equal(a, b) and a.size == W.blob_size(dims)
    assert np.array_equal(W.bf16_round(a), a)
    g = W.weight_view(dims, a, "L0.ln1_g")
    w = W.weight_view(dims, a, "L0.wq")
    assert abs(float(g.mean()) - 1.0) < 0.01 and abs(float(w.std()) - 0.02) < 0.002
    assert not np.array_equal(W.make_weights(dims, seed=1), a)
    f32 = dataclasses.replace(dims, dtype="fp32")
    assert not np.array_equal(W.bf16_round(W.make_weights(f32)), W.make_weights(f32))


def test_encoder_states_per_utterance_and_padding():
    dims = W.ModelDims(n_layers=1, d_model=32, n_heads=1, d_ffn=64, vocab=10, dtype="bf16",
                       max_pos=8, max_enc=20, anchor_layer=0)
    e = W.make_encoder_states(dims, [20, 5, 12], 20)
    assert np.all(e[1, 5:] == 0) and np.all(e[2, 12:] == 0) and np.all(e[0] != 0)
    # utterance b's states do not depend on the rest of the batch
    e2 = W.make_encoder_states(dims, [7, 5], 20)
    np.testing.assert_array_equal(e2[1], e[1])
    np.testing.assert_array_equal(e2[0, :7], e[0, :7])
    assert np.array_equal(W.bf16_round(e), e)


def test_round_lengths_end_exactly_at_the_target():
    """A fully accepted round commits 1 + lens tokens; lens = min(k, N - P - 2)
    makes the last one end with kv_len + pending = N tokens, and an utterance
    with P + 1 >= N sits out."""
    for N in range(6, 30):
        P = 3
        while True:
            lens = int(W.round_lens([N], [P], 6)[0])
            if lens < 0:
                break
            assert 0 <= lens <= 6
            P += 1 + lens                       # everything accepted
        assert P + 1 == N                      # committed + pending = the target length


def test_drafts_slip_and_replacement():
    truth = np.arange(100).reshape(1, 100) + 1000
    wl = W.Workload("t", W.SMALL, 1, 8, (60,), (100,), (0.0,), "always")
    corr = W.make_corruption(wl)
    P = 10
    s = int(corr.shift[0, P])
    d, lens = W.make_drafts(truth, [90], [P], 8, corr)
    assert lens[0] == 8 and 1 <= s <= 8
    for i in range(1, 9):
        assert d[0, i - 1] == truth[0, P + i - (1 if i >= s else 0)]
    # no corruption: the truth continuation
    d0, _ = W.make_drafts(truth, [90], [P], 8, None)
    assert list(d0[0]) == list(truth[0, P + 1:P + 9])
    # replacement rate p per token (no slip)
    wl = W.Workload("t", W.SMALL, 1, 8, (60,), (100,), (0.3,), "none")
    corr = W.make_corruption(wl)
    rate = float((corr.repl[0] >= 0).mean())
    assert abs(rate - 0.3) < 0.02 and not np.any(corr.shift)


def test_configs_match_their_names():
    for name, wl in W.CONFIGS.items():
        assert f"b{wl.batch}" in name and f"k{wl.k}" in name
        assert len(wl.enc_lens) == wl.batch and len(wl.n_out) == wl.batch
        assert max(wl.enc_lens) <= wl.t_max <= wl.dims.max_enc
        assert wl.dims.d_model % wl.dims.n_heads == 0 and wl.dims.head_dim == 64
    c4 = W.CONFIGS["large-bf16-b64-k6"]
    assert min(c4.enc_lens) >= 250 and max(c4.enc_lens) <= 1500
