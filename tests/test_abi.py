"""The C-ABI library loads without a GPU and exports every symbol that
include/asrspec.h declares (no compute calls)."""
import os
import re

from paper_2608_12703_gb300 import asrspec as A
from paper_2608_12703_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            src = open(os.path.join(inc, f)).read()
            names |= set(re.findall(r"\b(asr_spec_\w+)\s*\(", src))
    return names


def test_library_exports_every_declared_symbol():
    B.build()
    L = A.lib()
    decl = declared_symbols()
    assert decl, "no declarations found"
    for n in decl:
        assert hasattr(L, n), n
    assert decl == set(A.EXPORTED)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(A, "_lib", None)
    monkeypatch.setattr(A, "LIB_PATH", str(tmp_path / "missing.so"))
    import pytest
    with pytest.raises(A.AsrSpecError):
        A.lib()
