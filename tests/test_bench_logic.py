"""The host arithmetic behind bench.py's roofline object, on synthetic
timelines and timings (no GPU): which kernel is dominant, which bound applies,
achieved = algorithmic work / time, the in-chain figure, and the per-verify
algorithmic bytes (weights + the K/V traffic the plan kernel counts)."""
import numpy as np
import pytest

import bench
import workload as W


PK = dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="test")


def _timeline(entries):
    """entries: (kind, start_ns, work_ns, end_ns) -> (ns [n][4], kinds [n])."""
    ns = np.array([[s, w, 0, e] for _, s, w, e in entries], dtype=np.uint64)
    kinds = np.array([k for k, *_ in entries], dtype=np.int32)
    return ns, kinds


def _ms(calls, L, **kw):
    """Per-class CUDA-event milliseconds, and launches as a decode of `calls`
    verify calls makes them (bench.CLASS_PER_CALL per layer, the LM head once)."""
    from paper_2608_12703_gb300.asrspec import PROF_CLASSES
    ms = np.zeros(len(PROF_CLASSES))
    launches = np.zeros(len(PROF_CLASSES), dtype=np.int64)
    for name, t in kw.items():
        ms[PROF_CLASSES.index(name)] = t
        launches[PROF_CLASSES.index(name)] = calls * (bench.CLASS_PER_CALL[name] * L or 1)
    return ms, launches


def test_dominant_kernel_and_hbm_bound():
    dims = W.LARGE
    d, L, F = dims.d_model, dims.n_layers, dims.d_ffn
    calls, rows = 10, 90          # 9 rows per call: far below the tensor/HBM balance
    traffic = np.array([calls, 5e8, 2.5e9, 3.8e7, rows, 0, 0, 0])
    # resid (kind 18, and 50 = folded-LN variant counted with it) busiest, then cross-attention (5)
    tl = _timeline([(18, 0, 1000, 8000), (50, 9000, 9500, 16500), (5, 17000, 17200, 20200), (17, 21000, 21100, 22100)])
    ms, launches = _ms(calls, L, resid=2.0, cross_attn=1.0, qkv=0.5)
    r = bench.roofline("x", dims, tl, ms, launches, traffic, PK)
    assert r["kernel"] == "resid" and r["bound"] == "hbm" and r["unit"] == "GB/s"
    nbytes = calls * L * (2 * d * d + F * d) * 2
    assert r["achieved"] == pytest.approx(nbytes / 2.0e-3 / 1e9, rel=1e-3)
    assert r["frac"] == pytest.approx(r["achieved"] / PK["hbm"], rel=1e-3)
    busy = (8000 - 1000 + 16500 - 9500) / 1e9
    assert r["in_chain"]["achieved"] == pytest.approx(nbytes / busy / 1e9, rel=1e-3)
    assert r["share_of_busy_time"] == pytest.approx(14000 / (14000 + 3000 + 1000), rel=1e-3)


def test_tensor_bound_when_rows_exceed_the_balance():
    dims = W.LARGE
    calls, rows = 2, 2 * 448      # 448 rows per call: 448 flop per weight byte pair > 1700 / 6.8
    traffic = np.array([calls, 1e8, 1e9, 1e7, rows, 0, 0, 0])
    tl = _timeline([(20, 0, 100, 10100)])
    ms, launches = _ms(calls, dims.n_layers, mlp_up=1.0)
    r = bench.roofline("x", dims, tl, ms, launches, traffic, PK)
    assert r["kernel"] == "mlp_up" and r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    flops = 2.0 * rows * dims.n_layers * dims.d_ffn * dims.d_model
    assert r["achieved"] == pytest.approx(flops / 1e-3 / 1e12, rel=1e-3)
    assert r["peak"] == PK["bf16_sus"]


def test_attention_work_is_the_counted_kv_bytes(tmp_path, monkeypatch):
    import paper_2608_12703_gb300.ncu_traffic as NT
    monkeypatch.setattr(NT, "TRAFFIC_FILE", str(tmp_path / "traffic.json"))
    csv_path = tmp_path / "raw.csv"
    csv_path.write_text('"ID","Kernel Name","dram__bytes_read.sum","dram__bytes_write.sum"\n'
                        '"","","Mbyte","Kbyte"\n'
                        '"0","attn_tc_kernel<1>","330.5","7200"\n')
    NT.record(str(csv_path), "attn_tc", "large-bf16-b64-k6", "cross_attn", "attn_tc", "profiles/x.md")
    dims = W.LARGE
    traffic = np.array([4, 3e8, 9e9, 1e8, 36, 0, 0, 0])
    tl = _timeline([(5, 0, 0, 50000)])
    ms, launches = _ms(4, dims.n_layers, cross_attn=2.0)
    r = bench.roofline("large-bf16-b64-k6", dims, tl, ms, launches, traffic, PK)
    assert r["kernel"] == "cross_attn" and r["bound"] == "hbm"
    assert r["achieved"] == pytest.approx(9e9 / 2e-3 / 1e9, rel=1e-3)
    assert r["traffic"] == pytest.approx(337.7e6) and r["traffic_source"] == "profiles/x.md"


def test_few_row_classes_carry_their_attention_bytes():
    """Batch 1: every call runs the few-row layers; the QKV + self-attention
    launches carry the QKV weights and all the self K/V bytes counted."""
    dims = W.LARGE
    d, L = dims.d_model, dims.n_layers
    calls, rows = 8, 72
    traffic = np.array([calls, 4e8, 2e9, 3e7, rows, 0, 0, 0])
    tl = _timeline([(8, 0, 100, 9100), (18, 9200, 9300, 12300), (9, 12400, 12500, 15500)])
    ms, launches = _ms(calls, L, qkv_self=3.0, resid=1.0, query_cross=1.0)
    r = bench.roofline("x", dims, tl, ms, launches, traffic, PK)
    assert r["kernel"] == "qkv_self" and r["bound"] == "hbm"
    nbytes = calls * L * 3 * d * d * 2 + 4e8
    assert r["achieved"] == pytest.approx(nbytes / 3e-3 / 1e9, rel=1e-3)
    assert r["launches"] == calls * L


def test_step_bytes():
    dims = W.LARGE
    d, L, F, V = dims.d_model, dims.n_layers, dims.d_ffn, dims.vocab
    traffic = np.array([5, 1e8, 2e9, 4e7, 45, 0, 0, 0])
    w = L * (6 * d * d + 2 * F * d) * 2 + V * d * 2
    assert bench.step_bytes(dims, traffic) == pytest.approx((5 * w + 1e8 + 2e9 + 4e7) / 5)
