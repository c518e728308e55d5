"""The measured-traffic file behind bench.py's roofline.traffic: ncu raw-page
CSV parsing (units, kernel filter, mean per launch), and that an entry is
returned only while its kernel's sources hash as they did at capture."""
import json

import pytest

import paper_2608_12703_gb300.ncu_traffic as NT

CSV = ('"==PROF== Connected to process"\n'
       '"ID","Process ID","Kernel Name","dram__bytes_read.sum","dram__bytes_write.sum"\n'
       '"","","","Mbyte","Kbyte"\n'
       '"0","7","gemm_tc_kernel<64, 2, 1>(...)","6.5","250"\n'
       '"1","7","attn_tc_kernel<0>(...)","100","1,000"\n'
       '"2","7","gemm_tc_kernel<64, 2, 1>(...)","7.5","750"\n')


@pytest.fixture
def traffic(tmp_path, monkeypatch):
    monkeypatch.setattr(NT, "TRAFFIC_FILE", str(tmp_path / "t.json"))
    p = tmp_path / "raw.csv"
    p.write_text(CSV)
    return p


def test_parse_mean_per_launch_with_units(traffic):
    b, n = NT.parse_dram_bytes(str(traffic), r"gemm_tc_kernel")
    assert n == 2 and b == pytest.approx(((6.5e6 + 250e3) + (7.5e6 + 750e3)) / 2)
    b, n = NT.parse_dram_bytes(str(traffic), r"attn_tc")
    assert n == 1 and b == pytest.approx(100e6 + 1e6)
    with pytest.raises(ValueError):
        NT.parse_dram_bytes(str(traffic), r"no_such_kernel")


def test_lookup_current_then_stale(traffic):
    e = NT.record(str(traffic), "gemm_tc", "w", "resid", "gemm_tc", "profiles/s.md", scale=2.0)
    assert e["bytes_per_launch"] == pytest.approx(2 * 7.5e6)
    assert NT.lookup("w", "resid") == (pytest.approx(1.5e7), "profiles/s.md")
    assert NT.lookup("w", "qkv") is None
    data = json.load(open(NT.TRAFFIC_FILE))
    data["entries"][0]["source_hash"] = "0" * 16        # as if the kernel changed since the capture
    json.dump(data, open(NT.TRAFFIC_FILE, "w"))
    assert NT.lookup("w", "resid") is None


def test_record_replaces_the_same_key(traffic):
    NT.record(str(traffic), "gemm_tc", "w", "resid", "gemm_tc", "a.md")
    NT.record(str(traffic), "attn_tc", "w", "resid", "attn_tc", "b.md")
    ents = json.load(open(NT.TRAFFIC_FILE))["entries"]
    assert len(ents) == 1 and ents[0]["summary"] == "b.md"


def test_code_text_ignores_comments_and_layout_only():
    a = 'int f(int x) {  // the input\n  return x + 1; /* one more */\n}\nconst char* s = "// kept";\n'
    b = 'int f(int x) {\n    return x + 1;\n}   // reworded note\nconst char* s = "// kept";'
    c = 'int f(int x) { return x + 2; }\nconst char* s = "// kept";'
    assert NT.code_text(a) == NT.code_text(b)
    assert NT.code_text(a) != NT.code_text(c)
    assert '"// kept"' in NT.code_text(a)
    assert NT.code_text("char q = '\"'; /* x */ int y;") == "char q = '\"'; int y;"
