"""Tree verification on the GPU (the tree decoder control of the paper's
appendix: the target verifies a candidate tree in one pass under a tree
attention mask) against the CPU oracle, teacher-forced: both start every step
from the same committed state and score the same tree.  After each tree step a
linear step scores a block on top of the committed path, which checks the
path's K/V were moved to consecutive positions."""
import numpy as np
import pytest

import workload as W
from oracle import Oracle
from tests.parity import ParityStats, anchor_tol, compare_round, logit_tol

pytestmark = pytest.mark.gpu


def _continuation(orc, n):
    snap = orc.snapshot()
    out = [orc.ar_step() for _ in range(n)]
    orc.restore(snap)
    return np.stack(out, axis=1)


def _tree(rng, truth_b, n, vocab, corrupt):
    """An n-node tree: a main branch of the true continuation (each token
    replaced with probability `corrupt`), side branches of random tokens, and a
    duplicate of a true token under a different parent."""
    parent = np.array([rng.integers(0, i + 1) for i in range(n)])
    tokens = rng.integers(0, vocab, size=n)
    m = min(4, n)
    parent[:m] = np.arange(m)
    tokens[:m] = np.where(rng.random(m) < corrupt, rng.integers(0, vocab, size=m), truth_b[:m])
    if n > 6:
        parent[6] = 0
        tokens[6] = truth_b[0]
    return tokens, parent


def _compare_tree(orc, sess, tokens, parent, lens, st, scale=1.0):
    dims = orc.dims
    ro = orc.verify_tree(tokens, parent, lens)
    rg, path = sess.verify_tree(tokens, parent, lens)
    if len(ro.rows):
        lg = sess.debug_logits(len(ro.rows)).double().cpu().numpy()
        assert lg.shape == ro.logits.shape
        err = float(np.abs(lg - ro.logits).max())
        st.max_logit_err = max(st.max_logit_err, err)
        assert err <= logit_tol(dims, scale), f"logits differ by {err}"
    st.rounds += 1
    r0 = 0
    diverged = False
    for b in range(len(lens)):
        if lens[b] < 0:
            assert rg.bonus[b] == -1 and rg.anchor[b] == -1 and rg.accepted[b] == 0 and rg.restart[b] == 0
            assert rg.kv_len[b] == ro.kv_len[b]
            continue
        nrow = int(lens[b]) + 1
        st.rows += nrow
        same = (ro.accepted[b] == rg.accepted[b] and ro.bonus[b] == rg.bonus[b]
                and list(ro.path[b, :ro.accepted[b]]) == list(path[b, :rg.accepted[b]]))
        if not same:   # only where the oracle's decision was a near-tie
            gaps = ro.top2_gap[r0:r0 + nrow]
            assert gaps.min() < 1e-2 * scale, (b, ro.accepted[b], rg.accepted[b], ro.path[b], path[b])
            st.near_ties += 1
            diverged = True
        else:
            assert rg.kv_len[b] == ro.kv_len[b]
            assert np.all(path[b, rg.accepted[b]:] == -1)
            # the tree's restart flag: the path's last node has children (R16)
            assert rg.restart[b] == ro.restart[b], (b, rg.restart[b], ro.restart[b])
            st.restarts += int(rg.restart[b])
            st.anchors += 1
            prof = ro.anchor_profile[b]
            if rg.anchor[b] == ro.anchor[b]:
                st.anchor_exact += 1
            else:
                a = int(rg.anchor[b])
                assert prof[a] >= (1.0 - anchor_tol(dims)) * prof.max()
                st.anchor_near += 1
        st.emitted += int(rg.accepted[b]) + 1
        r0 += nrow
    return ro, rg, diverged


@pytest.mark.parametrize("n", [11, 5])
def test_tree_against_oracle(built_lib, cuda, n):
    """Small bf16 decoder, 3 utterances (encoder lengths 1500, 600, 1): trees of
    n nodes with a corrupted true branch, side branches and a duplicate, then a
    linear step on top of the committed path; lens 0 and sitting out included."""
    from paper_2608_12703_gb300.session import Session
    dims = W.SMALL
    blob = W.make_weights(dims, std=0.02)
    enc_lens = [1500, 600, 1]
    enc = W.make_encoder_states(dims, enc_lens, 1500)
    prompt = W.make_prompt(dims, 3)
    orc = Oracle(dims, blob)
    orc.encode_cache(enc, enc_lens)
    orc.prefill(prompt)
    sess = Session(dims, blob, max_batch=3, max_draft=max(n, 4))
    sess.encode_cache(enc, enc_lens)
    sess.prefill(prompt)
    rng = np.random.default_rng(21)
    st = ParityStats()
    for step in range(5):
        truth = _continuation(orc, 5)
        tokens = np.zeros((3, n), dtype=np.int64)
        parent = np.zeros((3, n), dtype=np.int64)
        for b in range(3):
            tokens[b], parent[b] = _tree(rng, truth[b], n, dims.vocab, corrupt=[0.0, 0.3, 0.6][b])
        lens = np.array([n, [n, 0, 3, -1, n][step], n - 1])
        _, _, diverged = _compare_tree(orc, sess, tokens, parent, lens, st)
        if diverged:
            break
        truth = _continuation(orc, 3)
        compare_round(orc, sess, truth, np.array([3, 2, 3]), st)   # linear block on the committed path
    print(f"\n[tree n={n}] rounds={st.rounds} rows={st.rows} emitted={st.emitted} near_ties={st.near_ties} "
          f"anchor exact={st.anchor_exact}/{st.anchors} near={st.anchor_near} max_logit_err={st.max_logit_err:.3g}")
    assert st.emitted > 20
    assert sess.status() == 0
    sess.close()


def test_tree_one_branch_is_the_linear_verify(built_lib, cuda):
    """A one-branch tree gives the linear verify's outputs and logits, bit for
    bit, from the same state (rollback in between)."""
    from paper_2608_12703_gb300.session import Session
    dims = W.SMALL
    blob = W.make_weights(dims, std=0.02)
    enc = W.make_encoder_states(dims, [900, 300], 900)
    s = Session(dims, blob, max_batch=2, max_draft=6)
    s.encode_cache(enc, [900, 300])
    s.prefill(W.make_prompt(dims, 2))
    rng = np.random.default_rng(4)
    chain = np.tile(np.arange(6), (2, 1))
    for _ in range(3):
        kv0, pend0 = s.state()
        draft = rng.integers(0, dims.vocab, size=(2, 6))
        lens = np.array([6, 4])
        t, path = s.verify_tree(draft, chain, lens)
        lt = s.debug_logits(16).float().cpu().numpy()
        s.rollback(kv0, pend0)
        o = s.verify(draft, lens)
        ll = s.debug_logits(16).float().cpu().numpy()
        assert np.array_equal(lt, ll)
        for f in ("accepted", "bonus", "kv_len", "anchor"):
            assert np.array_equal(getattr(t, f), getattr(o, f)), f
        for b in range(2):
            assert list(path[b, :t.accepted[b]]) == list(range(1, t.accepted[b] + 1))
    assert s.status() == 0
    s.close()


def test_tree_bad_parent_refuses_the_step(built_lib, cuda):
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300.session import Session
    dims = W.ModelDims(n_layers=2, d_model=128, n_heads=2, d_ffn=256, vocab=500, dtype="bf16",
                       max_pos=24, max_enc=64, anchor_layer=1)
    s = Session(dims, W.make_weights(dims, std=0.1), max_batch=2, max_draft=4)
    s.encode_cache(W.make_encoder_states(dims, [64, 10], 64), [64, 10])
    s.prefill(W.make_prompt(dims, 2))
    kv0, pend0 = s.state()
    out, _ = s.verify_tree(np.ones((2, 3)), np.array([[0, 0, 3], [0, 1, 1]]), np.array([3, 3]))
    assert s.status() & A.ST_BAD_TREE
    kv1, pend1 = s.state()
    assert list(kv1) == list(kv0) and list(pend1) == list(pend0)
    out, path = s.verify_tree(np.ones((2, 3)), np.array([[0, 0, 1], [0, 1, 1]]), np.array([3, 3]))
    assert s.status() == 0 and np.all(out.kv_len > kv0)
    s.close()


def test_tree_host_io_matches_device_io(built_lib, cuda):
    from paper_2608_12703_gb300.session import Session
    dims = W.ModelDims(n_layers=2, d_model=128, n_heads=2, d_ffn=256, vocab=500, dtype="bf16",
                       max_pos=32, max_enc=64, anchor_layer=1)
    blob = W.make_weights(dims, std=0.1)
    rng = np.random.default_rng(8)
    trees = [(rng.integers(0, 500, size=(2, 5)), np.array([[0, 0, 1, 2, 2], [0, 1, 1, 0, 4]])) for _ in range(3)]
    outs = []
    for host in (False, True):
        s = Session(dims, blob, max_batch=2, max_draft=5)
        s.set_host_io(host)
        s.encode_cache(W.make_encoder_states(dims, [64, 20], 64), [64, 20])
        s.prefill(W.make_prompt(dims, 2))
        res = []
        for tok, par in trees:
            o, path = s.verify_tree(tok, par, np.array([5, 3]))
            res.append((list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor), path.tolist()))
        assert s.status() == 0
        s.close()
        outs.append(res)
    assert outs[0] == outs[1]
