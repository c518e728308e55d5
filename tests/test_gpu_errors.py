"""Error paths and state handling of the C ABI on the GPU: host-side argument
errors return codes; device-side data errors refuse the whole step, leave the
state unchanged and set the status word.  Rollback followed by the same
verification reproduces outputs and logits bit for bit; the host-I/O path
returns what the device path returns."""
import numpy as np
import pytest

import workload as W

pytestmark = pytest.mark.gpu

DIMS = W.ModelDims(n_layers=2, d_model=128, n_heads=2, d_ffn=256, vocab=500, dtype="bf16",
                   max_pos=24, max_enc=64, anchor_layer=1)


@pytest.fixture
def sess(built_lib, cuda):
    from paper_2608_12703_gb300.session import Session
    blob = W.make_weights(DIMS, std=0.1)
    s = Session(DIMS, blob, max_batch=3, max_draft=4)
    yield s
    s.close()


def _ready(s):
    enc = W.make_encoder_states(DIMS, [64, 10, 33], 64)
    s.encode_cache(enc, [64, 10, 33])
    s.prefill(W.make_prompt(DIMS, 3))


def test_call_order_and_arguments(sess):
    import torch
    from paper_2608_12703_gb300 import asrspec as A
    d = torch.zeros((1, 1), dtype=torch.int32, device="cuda")
    o = torch.zeros((5, 1), dtype=torch.int32, device="cuda")
    with pytest.raises(A.AsrSpecError, match="ASR_E_STATE"):
        A.asr_spec_verify(sess.h, d, o[4], 1, o[0], o[1], o[2], o[3])
    with pytest.raises(A.AsrSpecError, match="ASR_E_STATE"):
        A.asr_spec_prefill(sess.h, d, 1)
    _ready(sess)
    with pytest.raises(A.AsrSpecError, match="ASR_E_INVAL"):
        sess.verify(np.zeros((3, 5)), np.zeros(3))         # k > max_draft
    enc = W.make_encoder_states(DIMS, [64], 64)
    with pytest.raises(A.AsrSpecError, match="ASR_E_CAPACITY"):
        import torch
        big = torch.zeros((1, 65, 128), dtype=torch.bfloat16, device="cuda")
        sess.encode_cache(big, [65])
    assert sess.status() == 0


@pytest.mark.parametrize("case,bit", [("token", 1), ("lens", 2), ("capacity", 4)])
def test_device_errors_refuse_the_step(sess, case, bit):
    _ready(sess)
    kv0, p0 = sess.state()
    draft = np.array([[1, 2, 3, 4]] * 3)
    lens = np.array([4, 2, 0])
    if case == "token":
        draft[1, 1] = DIMS.vocab
    elif case == "lens":
        lens[2] = 5
    else:
        for _ in range(4):
            sess.verify(np.array([[7, 7, 7, 7]] * 3), np.array([4, -1, -1]))
        kv0, p0 = sess.state()
        lens = np.array([4, 0, 0])
        draft[0] = [7, 7, 7, 7]
        assert kv0[0] + 5 > DIMS.max_pos or pytest.skip("did not reach capacity")
    out = sess.verify(draft, lens)
    assert sess.status() & bit
    kv1, p1 = sess.state()
    assert list(kv1) == list(kv0) and list(p1) == list(p0)
    assert list(out.bonus) == [-1, -1, -1]
    assert sess.status() == 0


def test_rollback_then_reverify_is_bitwise_identical(sess):
    _ready(sess)
    sess.verify(np.array([[5, 6, 7, 8]] * 3), np.array([4, 1, 0]))
    kv0, p0 = sess.state()
    draft = np.array([[9, 10, 11, 12], [13, 14, 15, 16], [17, 18, 19, 20]])
    lens = np.array([4, 3, 2])
    a = sess.verify(draft, lens)
    la = sess.debug_logits(15).cpu().numpy().copy()
    sess.rollback(kv0, p0)
    b = sess.verify(draft, lens)
    lb = sess.debug_logits(15).cpu().numpy()
    for f in ("accepted", "bonus", "kv_len", "anchor"):
        assert list(getattr(a, f)) == list(getattr(b, f))
    assert np.array_equal(la, lb)
    # rollback beyond the committed length is refused
    kv, pe = sess.state()
    sess.rollback(kv + 1, pe)
    assert sess.status() & 4
    kv2, _ = sess.state()
    assert list(kv2) == list(kv)
    assert sess.status() == 0


def test_host_io_matches_device_io(built_lib, cuda):
    from paper_2608_12703_gb300.session import Session
    blob = W.make_weights(DIMS, std=0.1)
    outs = []
    for host in (False, True):
        s = Session(DIMS, blob, max_batch=3, max_draft=4)
        s.set_host_io(host)
        _ready(s)
        res = []
        for r in range(4):
            o = s.verify(np.array([[r, 2, 3, 4]] * 3), np.array([4, 2, r % 2 - 1]))
            res.append((list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor)))
        outs.append(res)
        assert s.status() == 0
        s.close()
    assert outs[0] == outs[1]


def test_graph_replay_matches_direct_launch_and_profile(built_lib, cuda):
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300.session import Session
    blob = W.make_weights(DIMS, std=0.1)
    outs = []
    for graphs, prof in ((True, False), (False, False), (True, True)):
        s = Session(DIMS, blob, max_batch=3, max_draft=4)
        A.asr_spec_set_graphs(s.h, graphs)
        A.asr_spec_profile(s.h, prof)
        _ready(s)
        A.asr_spec_profile_read(s.h)
        res = []
        for r in range(5):
            o = s.verify(np.array([[r, 2, 3, 4]] * 3), np.array([4, 2, r % 2 - 1]))
            res.append((list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor)))
        ms, launches, traffic = A.asr_spec_profile_read(s.h)
        assert traffic[0] == 5 and launches.sum() > 0
        if prof:
            assert ms[A.PROF_CLASSES.index("qkv")] > 0 and ms[A.PROF_CLASSES.index("resid")] > 0
        outs.append(res)
        assert s.status() == 0
        s.close()
    assert outs[0] == outs[1] == outs[2]


def test_timeline_records_every_launch_in_order(built_lib, cuda):
    """The launch timeline: one record per kernel of the verify chain, in
    launch order and of the expected kind; every record starts, passes its
    wait on the previous kernel and ends in that order, and no kernel passes
    its wait before the previous kernel has ended (dependent launches really
    wait).  Recording changes no result."""
    from paper_2608_12703_gb300 import asrspec as A
    from paper_2608_12703_gb300.session import Session
    blob = W.make_weights(DIMS, std=0.1)
    outs, records = [], None
    for timeline in (False, True):
        s = Session(DIMS, blob, max_batch=3, max_draft=4)
        _ready(s)
        A.asr_spec_timeline(s.h, timeline)
        res = []
        for r in range(3):
            o = s.verify(np.array([[r, 2, 3, 4]] * 3), np.array([4, 2, r % 2 - 1]))
            res.append((list(o.accepted), list(o.bonus), list(o.kv_len), list(o.anchor)))
        if timeline:
            records = A.asr_spec_timeline_read(s.h)
            ns2, _ = A.asr_spec_timeline_read(s.h)
            assert len(ns2) == 0                       # a read clears the record
        outs.append(res)
        assert s.status() == 0
        s.close()
    assert outs[0] == outs[1]
    ns, kinds = records
    g, f = A.TL_GEMM, A.TL_LN_FUSED   # LayerNorm folded into its neighbours (the default)
    layer = [g + 1 + f, 4, g + 2, g + 3 + f, 5, g + 2, g + 4 + f, g + 2]
    one = [1, 2] + layer * DIMS.n_layers + [g + 6 + f, 6]
    assert list(kinds) == one * 3
    ns = ns.astype(np.int64)
    start, work, mid, end = ns[:, 0], ns[:, 1], ns[:, 2], ns[:, 3]
    assert np.all(end > 0)
    assert np.all(start <= work) and np.all(work <= end)
    has_mid = np.array([k >= g or k in (4, 5) for k in kinds])
    assert np.all(mid[has_mid] > 0) and np.all(mid[~has_mid] == 0)
    assert np.all(mid[has_mid] <= end[has_mid])
    slack = 2000   # ns: the timer is global, CTAs on different SMs read it
    assert np.all(work[1:] >= end[:-1] - slack)
