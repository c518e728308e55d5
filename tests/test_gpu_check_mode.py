"""The bounds-check mode (environment ASRSPEC_CHECK=1 when a handle is
created): kernels re-check the indexes they derive from device data and set
ASR_ST_BOUNDS instead of going out of range.  On valid inputs it must change
nothing: these cases run the tensor-core layers (ragged batch), the few-row
layers (batch 1, k = 8), the fp32 path, a tree verify and the draft side
under it, against the oracle or against the same run without the mode, with a
clean status word throughout."""
import numpy as np
import pytest

import workload as W
from tests.parity import assert_bounded, run_decode, scale_for

pytestmark = pytest.mark.gpu


@pytest.fixture
def check_mode(monkeypatch):
    monkeypatch.setenv("ASRSPEC_CHECK", "1")


def _session(dims, blob, B, k):
    from paper_2608_12703_gb300.session import Session
    return lambda: Session(dims, blob, max_batch=B, max_draft=k)


def test_check_mode_bf16_ragged_and_fewrow(built_lib, cuda, check_mode):
    dims = W.ModelDims(n_layers=2, d_model=256, n_heads=4, d_ffn=1024, vocab=1000, dtype="bf16",
                       max_pos=64, max_enc=300, anchor_layer=1)
    blob = W.make_weights(dims, std=0.05)
    for enc_lens, total, k in (([300, 77, 1], [30, 21, 17], 4), ([300], [44], 8)):
        B = len(enc_lens)
        wl = W.Workload("c", dims, B, k, tuple(t - W.PROMPT_LEN for t in total), tuple(enc_lens), (0.3,) * B, "half")
        st, _ = run_decode(dims, blob, W.make_encoder_states(dims, enc_lens, max(enc_lens)), enc_lens,
                           W.make_prompt(dims, B), total, k, W.make_corruption(wl), _session(dims, blob, B, k),
                           scale=scale_for(dims, 0.05))
        assert st.rows > 20
        assert_bounded(st)


def test_check_mode_fp32(built_lib, cuda, check_mode):
    dims = W.ModelDims(n_layers=2, d_model=64, n_heads=1, d_ffn=128, vocab=300, dtype="fp32",
                       max_pos=30, max_enc=200, anchor_layer=0)
    blob = W.make_weights(dims, std=0.1)
    enc_lens, total = [200, 13], [30, 11]
    wl = W.Workload("f", dims, 2, 3, tuple(t - W.PROMPT_LEN for t in total), tuple(enc_lens), (0.3, 0.3), "half")
    st, _ = run_decode(dims, blob, W.make_encoder_states(dims, enc_lens, 200), enc_lens, W.make_prompt(dims, 2),
                       total, 3, W.make_corruption(wl), _session(dims, blob, 2, 3))
    assert st.near_ties == 0


def _tree_and_draft_run():
    from paper_2608_12703_gb300.session import DraftModel, Session
    dims = W.ModelDims(n_layers=4, d_model=256, n_heads=4, d_ffn=1024, vocab=1000, dtype="bf16",
                       max_pos=64, max_enc=200, anchor_layer=2)
    blob = W.make_weights(dims, std=0.05)
    enc_lens, total = [200, 41], [30, 22]
    out = []
    s = Session(dims, blob, max_batch=2, max_draft=5)
    dm = DraftModel(s, W.make_draft_weights(dims, std=0.05), total, 5)
    s.encode_cache(W.make_encoder_states(dims, enc_lens, 200), enc_lens)
    s.prefill(W.make_prompt(dims, 2))
    for _ in range(4):
        d, l = dm.propose()
        dh, lh = s.host(d).copy(), s.host(l).copy()
        o = s.verify(dh, lh)
        out.append((dh.tolist(), lh.tolist(), o.accepted.tolist(), o.bonus.tolist(), o.anchor.tolist()))
    rng = np.random.default_rng(5)
    o, path = s.verify_tree(rng.integers(0, 1000, size=(2, 5)), np.array([[0, 0, 1, 2, 2], [0, 1, 1, 0, 4]]),
                            np.array([5, 3]))
    out.append((o.accepted.tolist(), o.bonus.tolist(), o.kv_len.tolist(), path.tolist()))
    status = s.status()
    s.close()
    return out, status


def test_check_mode_tree_and_draft_change_nothing(built_lib, cuda, monkeypatch):
    ref, st0 = _tree_and_draft_run()
    monkeypatch.setenv("ASRSPEC_CHECK", "1")
    got, st1 = _tree_and_draft_run()
    assert st0 == 0 and st1 == 0
    assert got == ref
