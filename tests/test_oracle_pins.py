"""Pins of the CPU oracle against things other than itself.

* torch.nn's Transformer decoder (library) for the decoder forward, the
  block-causal mask of a verification pass, the cross-attention padding mask
  and the cached encoder K/V (Sec. 3 "Speculative Loop": the target checks the
  block in one pass);
* torch.nn.MultiheadAttention's head-averaged weights for the runtime anchor
  (Sec. 5 "Verification-Attention Correction");
* brute-force enumeration of every draft block on a tiny vocabulary for the
  longest-prefix rule (Sec. 3);
* the lossless invariant: speculative output equals plain greedy decoding
  (Sec. 1, Sec. 3: identical under exact arithmetic);
* rollback followed by the same verification reproduces outputs and cache;
* special cases: no drafts is one greedy step, true drafts are all accepted,
  wrong drafts are all rejected.
"""
import itertools

import numpy as np
import pytest

import workload as W
from oracle import Oracle, OracleError, greedy_transcript
from tests.torch_ref import TorchDecoder

TINY = W.ModelDims(n_layers=2, d_model=64, n_heads=2, d_ffn=256, vocab=97, dtype="fp32",
                   max_pos=64, max_enc=40, anchor_layer=1)
ENC_LENS = [23, 40, 7]


def _setup(dims=TINY, enc_lens=ENC_LENS, std=0.3, t_max=None, prompt_len=W.PROMPT_LEN):
    blob = W.make_weights(dims, std=std)
    t_max = t_max or max(enc_lens)
    enc = W.make_encoder_states(dims, enc_lens, t_max)
    o = Oracle(dims, blob)
    o.encode_cache(enc, enc_lens)
    prompt = W.make_prompt(dims, len(enc_lens), prompt_len)
    o.prefill(prompt)
    return o, blob, enc, prompt


@pytest.mark.parametrize("std", [0.02, 0.3])
def test_verify_rows_match_torch_decoder(std):
    """Every verify row equals the library decoder's full-sequence logits at the
    same position: the cache, the block-causal mask and the encoder K/V are right."""
    o, blob, enc, prompt = _setup(std=std)
    ref = TorchDecoder(TINY, blob)
    rng = np.random.default_rng(7)
    hist = [list(prompt[b]) for b in range(3)]
    for step in range(4):
        k = 5
        draft = rng.integers(0, TINY.vocab, size=(3, k))
        lens = np.array([5, 2, 0])
        res = o.verify(draft, lens)
        for b in range(3):
            rows = [r for r, (bb, _) in enumerate(res.rows) if bb == b]
            seq = hist[b] + [int(t) for t in draft[b, :lens[b]]]
            logits, _ = ref.forward(seq, enc[b], ENC_LENS[b])
            start = len(hist[b]) - 1          # position of the pending token
            np.testing.assert_allclose(res.logits[rows], logits[start:start + lens[b] + 1],
                                       rtol=0, atol=1e-10)
            hist[b] = hist[b] + [int(t) for t in draft[b, :res.accepted[b]]] + [int(res.bonus[b])]


def test_anchor_matches_torch_head_mean_weights():
    """The anchor profile is torch's head-averaged cross-attention at the anchor
    layer, read at the row whose argmax is the bonus token; the anchor is its peak."""
    o, blob, enc, prompt = _setup()
    ref = TorchDecoder(TINY, blob)
    rng = np.random.default_rng(3)
    hist = [list(prompt[b]) for b in range(3)]
    for step in range(3):
        draft = rng.integers(0, TINY.vocab, size=(3, 3))
        res = o.verify(draft, np.array([3, 3, 1]))
        for b in range(3):
            seq = hist[b] + [int(t) for t in draft[b, :3]]
            _, w = ref.forward(seq, enc[b], ENC_LENS[b], anchor_layer=TINY.anchor)
            row = len(hist[b]) - 1 + int(res.accepted[b])
            np.testing.assert_allclose(res.anchor_profile[b], w[row], rtol=0, atol=1e-12)
            assert res.anchor[b] == int(np.argmax(w[row]))
            hist[b] = hist[b] + [int(t) for t in draft[b, :res.accepted[b]]] + [int(res.bonus[b])]


def test_anchor_planted_peak():
    """Overwriting one frame's anchor-layer keys with a large multiple of the
    scored row's query (per head) must move the anchor to that frame.  The
    anchor-layer query is computed before that layer's cross-attention, so the
    planted keys do not change it."""
    o, blob, enc, prompt = _setup()
    snap = o.snapshot()
    rows = [(b, int(o.pending[b]), int(o.kv_len[b])) for b in range(3)]
    _, q_anchor = o._forward(rows)
    o.restore(snap)
    hd = TINY.head_dim
    targets = [17, 39, 0]
    for b, jstar in enumerate(targets):
        q = q_anchor[b]
        key = np.concatenate([q[h * hd:(h + 1) * hd] / np.linalg.norm(q[h * hd:(h + 1) * hd])
                              for h in range(TINY.n_heads)])
        o.Kx[TINY.anchor][b][jstar] = 80.0 * key
    res = o.verify(np.zeros((3, 1), dtype=int), np.zeros(3, dtype=int))
    assert list(res.anchor) == targets
    for b, jstar in enumerate(targets):
        assert res.anchor_profile[b][jstar] > 0.99


def _greedy_continuation(o, n):
    snap = o.snapshot()
    out = []
    for _ in range(n):
        out.append(o.ar_step())
    o.restore(snap)
    return np.stack(out, axis=1)      # [B, n]


def test_accept_brute_force_tiny_vocab():
    """Accepted length equals the longest prefix of the block that matches the
    target's greedy continuation, for every draft block over an 8-token vocabulary."""
    dims = W.ModelDims(n_layers=1, d_model=64, n_heads=1, d_ffn=128, vocab=8, dtype="fp32",
                       max_pos=32, max_enc=16, anchor_layer=0)
    o, *_ = _setup(dims, enc_lens=[11, 16], std=0.5, prompt_len=2)
    for _ in range(2):   # two different states
        g = _greedy_continuation(o, 4)           # g[:, j] = greedy token j+1 after pending
        snap = o.snapshot()
        for k in (1, 2, 3):
            for block in itertools.product(range(8), repeat=k):
                for lens_b in range(k + 1):
                    o.restore(snap)
                    draft = np.array([block, block[::-1]])
                    res = o.verify(draft, np.array([lens_b, k]))
                    for b in range(2):
                        L = lens_b if b == 0 else k
                        n = 0
                        while n < L and draft[b, n] == g[b, n]:
                            n += 1
                        assert res.accepted[b] == n
                        assert res.bonus[b] == g[b, n]
                        assert res.kv_len[b] == snap[2][b] + 1 + n
                        assert res.restart[b] == int(n < L)
        o.restore(snap)
        o.ar_step()


def test_lossless_speculative_equals_greedy():
    """Speculative decoding with corrupted and slipped drafts returns exactly the
    plain greedy sequence, which itself equals the library decoder's greedy
    decoding by full recomputation."""
    total = [30, 22, 27]
    o, blob, enc, prompt = _setup()
    snap = o.snapshot()
    truth = greedy_transcript(o, prompt, total)
    ref = TorchDecoder(TINY, blob)
    for b in range(3):
        assert list(truth[b, :total[b]]) == ref.greedy(prompt[b], enc[b], ENC_LENS[b], total[b])
    wl = W.Workload("t", TINY, 3, 5, tuple(t - W.PROMPT_LEN for t in total), tuple(ENC_LENS),
                    (0.4, 0.2, 0.6), "half", t_max=40)
    corr = W.make_corruption(wl)
    o.restore(snap)
    seq = [list(prompt[b]) for b in range(3)]
    steps = 0
    while True:
        draft, lens = W.make_drafts(truth, total, o.kv_len, wl.k, corr)
        if np.all(lens < 0):
            break
        res = o.verify(draft, lens)
        steps += 1
        for b in range(3):
            if lens[b] >= 0:
                seq[b] += [int(t) for t in draft[b, :res.accepted[b]]] + [int(res.bonus[b])]
    for b in range(3):
        assert seq[b] == list(truth[b, :total[b]])
    assert steps < max(total) - W.PROMPT_LEN      # drafts were accepted along the way


def test_rollback_then_reverify_reproduces_cache():
    o, *_ = _setup()
    o.verify(np.array([[1, 2], [3, 4], [5, 6]]), np.array([2, 2, 2]))
    snap = o.snapshot()
    draft = np.array([[11, 12, 13], [14, 15, 16], [17, 18, 19]])
    r1 = o.verify(draft, np.array([3, 1, 2]))
    s1 = o.snapshot()
    o.rollback(snap[2], snap[3])
    r2 = o.verify(draft, np.array([3, 1, 2]))
    s2 = o.snapshot()
    for a, b in zip(r1.__dict__.values(), r2.__dict__.values()):
        if isinstance(a, np.ndarray):
            assert np.array_equal(a, b)
    for l in range(TINY.n_layers):
        assert np.array_equal(s1[0][l], s2[0][l]) and np.array_equal(s1[1][l], s2[1][l])
    assert np.array_equal(s1[2], s2[2]) and np.array_equal(s1[3], s2[3])


def test_special_cases():
    o, *_ = _setup()
    snap = o.snapshot()
    g = _greedy_continuation(o, 5)
    # no drafts == one greedy step
    res = o.verify(np.zeros((3, 4), dtype=int), np.zeros(3, dtype=int))
    assert list(res.bonus) == list(g[:, 0]) and list(res.accepted) == [0, 0, 0]
    # true continuation: everything accepted, bonus is the next greedy token
    o.restore(snap)
    res = o.verify(g[:, :4], np.array([4, 4, 4]))
    assert list(res.accepted) == [4, 4, 4] and list(res.bonus) == list(g[:, 4])
    assert list(res.restart) == [0, 0, 0]
    # every draft wrong at depth 1: nothing accepted
    o.restore(snap)
    wrong = (g[:, :4] + 1) % TINY.vocab
    res = o.verify(wrong, np.array([4, 4, 4]))
    assert list(res.accepted) == [0, 0, 0] and list(res.bonus) == list(g[:, 0])
    assert list(res.restart) == [1, 1, 1]
    # an inactive utterance keeps its state
    o.restore(snap)
    res = o.verify(g[:, :2], np.array([2, -1, 0]))
    assert res.kv_len[1] == snap[2][1] and res.bonus[1] == -1 and res.anchor[1] == -1
    assert res.accepted[0] == 2 and res.kv_len[0] == snap[2][0] + 3
    assert res.kv_len[2] == snap[2][2] + 1


def test_errors():
    o, *_ = _setup()
    with pytest.raises(OracleError):
        o.verify(np.array([[1], [2], [TINY.vocab]]), np.array([1, 1, 1]))
    with pytest.raises(OracleError):
        o.verify(np.array([[1], [2], [3]]), np.array([2, 1, 1]))
    with pytest.raises(OracleError):
        o.rollback(o.kv_len + 1, o.pending)
    o2 = Oracle(TINY, W.make_weights(TINY))
    with pytest.raises(OracleError):
        o2.prefill(np.zeros((1, 2), dtype=int))
    # capacity: P + lens + 1 > max_pos
    o.rollback(o.kv_len, o.pending)
    o.kv_len[:] = TINY.max_pos - 2
    with pytest.raises(OracleError):
        o.verify(np.ones((3, 2), dtype=int), np.array([2, 0, 0]))


def _mut_gelu_tanh(x):
    return 0.5 * x * (1 + np.tanh(np.sqrt(2 / np.pi) * (x + 0.044715 * x ** 3)))


def _mut_ln_unbiased(x, g, b):
    mu = x.mean(axis=-1, keepdims=True)
    var = x.var(axis=-1, ddof=1, keepdims=True)
    return (x - mu) / np.sqrt(var + 1e-5) * g + b


def _mut_attention_scale(q, K, V, n_heads):
    import oracle.decoder as D
    # scores scaled by 1/head_dim instead of 1/sqrt(head_dim)
    return D.__dict__["_orig_attention"](q / np.sqrt(K.shape[1] // n_heads), K, V, n_heads)


def _mut_head_mean_logits(q, K, n_heads):
    import oracle.decoder as D
    n, d = K.shape
    hd = d // n_heads
    s = np.einsum("hc,nhc->hn", q.reshape(n_heads, hd), K.reshape(n, n_heads, hd)) / np.sqrt(hd)
    return D.softmax(s.mean(axis=0))


def _mut_prefix_shifted(draft_b, g_b, lens_b):
    # compares draft j with the argmax of row j + 1 (the row that scored draft j itself)
    n = 0
    while n < lens_b and n + 1 < len(g_b) and draft_b[n] == g_b[n + 1]:
        n += 1
    return n


def _mut_prefix_one_more(draft_b, g_b, lens_b):
    # keeps the first mismatching draft too
    n = 0
    while n < lens_b and draft_b[n] == g_b[n]:
        n += 1
    return min(n + 1, lens_b)


def _mut_keys_exclusive(pos):
    return pos          # a row that cannot see its own key


def _mut_bonus_row_next(n):
    return n + 1        # reads the bonus from the row after the last accepted token


def _mut_tree_keys_block_causal(P, ancestors):
    return list(range(P + ancestors[-1] + 1))   # every earlier node, siblings included


@pytest.mark.parametrize("name,fn,pin", [
    ("gelu", _mut_gelu_tanh, "rows"), ("layer_norm", _mut_ln_unbiased, "rows"),
    ("attention", _mut_attention_scale, "rows"), ("head_mean_attention", _mut_head_mean_logits, "anchor"),
    ("visible_keys", _mut_keys_exclusive, "rows"),
    ("accepted_prefix", _mut_prefix_shifted, "accept"), ("accepted_prefix", _mut_prefix_one_more, "accept"),
    ("bonus_row", _mut_bonus_row_next, "accept"),
    ("tree_keys", _mut_tree_keys_block_causal, "tree")])
def test_pins_catch_planted_mistakes(monkeypatch, name, fn, pin):
    """A plausible mistake planted in the oracle makes a pin fail: the library
    decoder (rows), torch's head-averaged attention (anchor), or brute-force
    enumeration of every draft block (accept)."""
    import oracle.decoder as D
    monkeypatch.setitem(D.__dict__, "_orig_attention", D.attention)
    monkeypatch.setattr(D, name, fn)
    with pytest.raises((AssertionError, IndexError, ValueError)):
        if pin == "anchor":
            test_anchor_matches_torch_head_mean_weights()
        elif pin == "accept":
            test_accept_brute_force_tiny_vocab()
        elif pin == "tree":
            test_tree_nodes_equal_linear_branches()
        else:
            test_verify_rows_match_torch_decoder(0.3)


# ---- tree verification (App. "Alternative draft and verification changes": the
# target verifies a candidate tree in one pass under a tree attention mask) ----

def _random_tree(rng, n, vocab):
    parent = np.array([rng.integers(0, i + 1) for i in range(n)])
    tokens = rng.integers(0, vocab, size=n)
    return tokens, parent


def _branch(parent, j):
    """Nodes on the way from the root to node j (excluded root), root first."""
    out = []
    while j > 0:
        out.append(j)
        j = parent[j - 1]
    return out[::-1]


def test_tree_one_branch_equals_linear_verify():
    """A one-branch tree reproduces the linear verify token for token: outputs,
    logits and the committed cache are identical."""
    o, *_ = _setup()
    rng = np.random.default_rng(11)
    for _ in range(3):
        snap = o.snapshot()
        draft = rng.integers(0, TINY.vocab, size=(3, 4))
        lens = np.array([4, 2, -1])
        lin = o.verify(draft, lens)
        s_lin = o.snapshot()
        o.restore(snap)
        chain = np.tile(np.arange(4), (3, 1))      # parent of node i + 1 is node i
        tr = o.verify_tree(draft, chain, lens)
        s_tr = o.snapshot()
        for f in ("accepted", "bonus", "kv_len", "anchor", "restart"):
            assert np.array_equal(getattr(lin, f), getattr(tr, f)), f
        assert np.array_equal(lin.logits, tr.logits)
        for b in range(3):
            n = int(lin.accepted[b]) if lens[b] >= 0 else 0
            assert list(tr.path[b, :n]) == list(range(1, n + 1))
        for l in range(TINY.n_layers):
            for b in range(3):
                kv = int(s_lin[2][b])
                assert np.array_equal(s_lin[0][l][b, :kv], s_tr[0][l][b, :kv])
                assert np.array_equal(s_lin[1][l][b, :kv], s_tr[1][l][b, :kv])


def test_tree_nodes_equal_linear_branches():
    """Every node's logits are those of the linear verify of its branch (root to
    node) from the same state; the accepted path is as long as the longest
    accepted branch, with its bonus; the committed cache equals the one the
    linear verify of the accepted path leaves."""
    o, *_ = _setup()
    rng = np.random.default_rng(12)
    for step in range(3):
        snap = o.snapshot()
        g = _greedy_continuation(o, 4)             # true continuation, to make paths long
        n = 11
        tokens, parent = np.zeros((3, n), dtype=np.int64), np.zeros((3, n), dtype=np.int64)
        for b in range(3):
            tokens[b], parent[b] = _random_tree(rng, n, TINY.vocab)
            parent[b, :3] = [0, 1, 2]              # a branch along the true continuation
            tokens[b, :3] = g[b, :3]
            if step == 1:
                tokens[b, 5] = tokens[b, 1]        # a duplicate of a true token elsewhere
        lens = np.array([n, 7, n])
        tr = o.verify_tree(tokens, parent, lens)
        s_tr = o.snapshot()
        r0 = 0
        for b in range(3):
            l = int(lens[b])
            best = (-1, None)
            for j in range(l + 1):
                nodes = _branch(parent[b], j)
                o.restore(snap)
                dr = np.zeros((3, max(len(nodes), 1)), dtype=np.int64)
                dr[b, :len(nodes)] = tokens[b, np.array(nodes, dtype=int) - 1] if nodes else []
                ln = np.full(3, -1)
                ln[b] = len(nodes)
                lin = o.verify(dr, ln)
                # (the tree pass multiplies more rows at once: BLAS may sum in another order)
                np.testing.assert_allclose(tr.logits[r0 + j], lin.logits[len(nodes)], rtol=0, atol=1e-12)
                if lin.accepted[b] > best[0]:
                    best = (int(lin.accepted[b]), int(lin.bonus[b]))
            assert tr.accepted[b] == best[0] and tr.bonus[b] == best[1]
            # the cache the tree verify committed is the linear verify's of the accepted path
            path = [int(x) for x in tr.path[b, :tr.accepted[b]]]
            o.restore(snap)
            dr = np.zeros((3, max(len(path), 1)), dtype=np.int64)
            dr[b, :len(path)] = tokens[b, np.array(path, dtype=int) - 1] if path else []
            ln = np.full(3, -1)
            ln[b] = len(path)
            lin = o.verify(dr, ln)
            assert lin.accepted[b] == len(path) and lin.bonus[b] == tr.bonus[b]
            s_lin = o.snapshot()
            kv = int(s_tr[2][b])
            assert kv == int(s_lin[2][b])
            for l_ in range(TINY.n_layers):
                np.testing.assert_allclose(s_lin[0][l_][b, :kv], s_tr[0][l_][b, :kv], rtol=0, atol=1e-12)
                np.testing.assert_allclose(s_lin[1][l_][b, :kv], s_tr[1][l_][b, :kv], rtol=0, atol=1e-12)
            r0 += l + 1
        o.restore(s_tr)


def test_tree_errors():
    o, *_ = _setup()
    with pytest.raises(OracleError):
        o.verify_tree(np.zeros((3, 2), dtype=int), np.array([[0, 2], [0, 0], [0, 0]]), np.array([2, 2, 2]))


def test_mean_accepted_length_matches_the_closed_form():
    """Sec. 3 "Speculative Loop": the mean accepted draft length is
    L = sum_{k=1..K} s_k with s_k the probability that the first k proposals
    are accepted.  Drafts that are the target's own greedy continuation with
    every token replaced independently with probability p by a uniform id
    (R12; the replacement equals the true token with probability 1/V) are kept
    up to the first mismatch, so s_k = q^k with q = 1 - p + p/V.  The oracle's
    accepted lengths over full-width rounds must match that law."""
    dims = W.ModelDims(n_layers=2, d_model=64, n_heads=2, d_ffn=128, vocab=1000, dtype="fp32",
                       max_pos=448, max_enc=20, anchor_layer=1)
    K, p = 4, 0.3
    B = 3
    total = [400] * B
    o, *_ = _setup(dims, enc_lens=[20, 13, 7], std=0.3)
    snap = o.snapshot()
    prompt = W.make_prompt(dims, B)
    truth = greedy_transcript(o, prompt, total)
    o.restore(snap)
    wl = W.Workload("acc", dims, B, K, tuple(t - W.PROMPT_LEN for t in total), (20, 13, 7), (p,) * B, "none",
                    t_max=20)
    corr = W.make_corruption(wl)
    ns = []
    while True:
        draft, lens = W.make_drafts(truth, total, o.kv_len, K, corr)
        if np.all(lens < 0):
            break
        res = o.verify(draft, lens)
        ns += [int(res.accepted[b]) for b in range(B) if lens[b] == K]
    q = 1 - p + p / dims.vocab
    pmf = np.array([q ** j * (1 - q) for j in range(K)] + [q ** K])
    mean = float(np.dot(np.arange(K + 1), pmf))
    var = float(np.dot((np.arange(K + 1) - mean) ** 2, pmf))
    assert mean == pytest.approx(sum(q ** k for k in range(1, K + 1)))
    got = float(np.mean(ns))
    assert len(ns) > 250
    assert abs(got - mean) < 4 * np.sqrt(var / len(ns)), (got, mean, len(ns))
