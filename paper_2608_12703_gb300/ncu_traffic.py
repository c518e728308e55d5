"""Measured DRAM traffic per kernel launch, kept in a machine-readable file.

``profiles/ncu_traffic.json`` holds, per (workload, kernel class), the DRAM
bytes one launch moved (``dram__bytes_read.sum + dram__bytes_write.sum``,
averaged over the captured launches of an ncu ``--page raw --csv`` export)
together with a hash of the kernel's source files at capture time.  ``lookup``
returns an entry only while those sources are unchanged, so a figure never
outlives the code it was measured on.

Record a capture (reads the CSV that ``ncu -i <report> --page raw --csv``
printed):

  python -m paper_2608_12703_gb300.ncu_traffic record --csv <file> \
      --kernel '<regex>' --workload <name> --cls <class> --group <gemm_tc|gemm_wide|fewrow|attn_tc|rows> \
      --summary profiles/<summary>.md [--scale <factor>]
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import json
import os
import re
import sys
from typing import Dict, List, Optional, Tuple

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "ncu_traffic.json")

# the sources a kernel's code comes from (its own file, the headers it includes)
SOURCE_GROUPS: Dict[str, List[str]] = {
    "gemm_tc": ["csrc/gemm_tc.cu", "csrc/kernels.h", "csrc/epilogue.cuh", "csrc/common.cuh"],
    "gemm_wide": ["csrc/gemm_wide.cuh", "csrc/gemm_wide.cu", "csrc/kernels.h", "csrc/epilogue.cuh", "csrc/common.cuh"],
    "fewrow": ["csrc/fewrow.cu", "csrc/rowmma.cuh", "csrc/kernels.h", "csrc/epilogue.cuh", "csrc/common.cuh"],
    "attn_tc": ["csrc/attention_tc.cu", "csrc/kernels.h", "csrc/epilogue.cuh", "csrc/common.cuh"],
    "rows": ["csrc/rows.cu", "csrc/kernels.h", "csrc/epilogue.cuh", "csrc/common.cuh"],
}

UNIT = {"byte": 1.0, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "KB": 1e3, "MB": 1e6, "GB": 1e9,
        "Kibyte": 1024.0, "Mibyte": 1024.0 ** 2, "Gibyte": 1024.0 ** 3}


def code_text(src: str) -> str:
    """The source with its comments removed and every run of whitespace made
    one space: what the compiled code depends on (string and character
    literals are kept as they are)."""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if c in "\"'":                                     # a literal, up to its unescaped end
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        elif src.startswith("//", i):                     # to the end of the line
            j = src.find("\n", i)
            i = n if j < 0 else j
            out.append(" ")
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
            out.append(" ")
        else:
            out.append(c)
            i += 1
    return " ".join("".join(out).split())


def source_hash(group: str) -> str:
    """Hash of the code (comments and layout ignored) of a kernel's sources."""
    h = hashlib.sha256()
    for rel in SOURCE_GROUPS[group]:
        with open(os.path.join(PKG, rel), encoding="utf-8") as f:
            h.update(rel.encode() + b"\0" + code_text(f.read()).encode())
    return h.hexdigest()[:16]


def _load(path: Optional[str] = None) -> dict:
    path = path or TRAFFIC_FILE
    if not os.path.exists(path):
        return {"entries": []}
    with open(path) as f:
        return json.load(f)


def lookup(workload: str, cls: str, path: Optional[str] = None) -> Optional[Tuple[float, str]]:
    """(bytes per launch, summary file) of the entry, or None when there is none
    or its kernel sources changed since the capture."""
    for e in _load(path)["entries"]:
        if e["workload"] == workload and e["cls"] == cls:
            if e["source_hash"] != source_hash(e["group"]):
                return None
            return float(e["bytes_per_launch"]), e["summary"]
    return None


def parse_dram_bytes(csv_path: str, kernel_regex: str) -> Tuple[float, int]:
    """Mean DRAM bytes (read + write) per launch of the kernels whose name
    matches, from an ncu raw-page CSV (header row, unit row, one row per launch)."""
    with open(csv_path, newline="") as f:
        rows = [r for r in csv.reader(f)]
    start = next(i for i, r in enumerate(rows) if "Kernel Name" in r)
    head, units = rows[start], rows[start + 1]
    ki = head.index("Kernel Name")
    cols = [head.index("dram__bytes_read.sum"), head.index("dram__bytes_write.sum")]
    pat = re.compile(kernel_regex)
    vals = []
    for r in rows[start + 2:]:
        if len(r) <= max(cols + [ki]) or not pat.search(r[ki]):
            continue
        vals.append(sum(float(r[c].replace(",", "")) * UNIT.get(units[c], 1.0) for c in cols))
    if not vals:
        raise ValueError(f"no launch of /{kernel_regex}/ with DRAM counters in {csv_path}")
    return sum(vals) / len(vals), len(vals)


def record(csv_path: str, kernel_regex: str, workload: str, cls: str, group: str, summary: str,
           scale: float = 1.0, path: Optional[str] = None) -> dict:
    path = path or TRAFFIC_FILE
    per_launch, n = parse_dram_bytes(csv_path, kernel_regex)
    entry = {"workload": workload, "cls": cls, "group": group, "kernel": kernel_regex,
             "bytes_per_launch": per_launch * scale, "launches": n, "scale": scale,
             "source_hash": source_hash(group), "summary": summary}
    data = _load(path)
    data["entries"] = [e for e in data["entries"] if not (e["workload"] == workload and e["cls"] == cls)]
    data["entries"].append(entry)
    data["entries"].sort(key=lambda e: (e["workload"], e["cls"]))
    with open(path, "w") as f:
        json.dump(data, f, indent=1)
        f.write("\n")
    return entry


def main(argv=None):
    ap = argparse.ArgumentParser()
    sub = ap.add_subparsers(dest="cmd", required=True)
    r = sub.add_parser("record")
    r.add_argument("--csv", required=True)
    r.add_argument("--kernel", required=True)
    r.add_argument("--workload", required=True)
    r.add_argument("--cls", required=True)
    r.add_argument("--group", required=True, choices=sorted(SOURCE_GROUPS))
    r.add_argument("--summary", required=True)
    r.add_argument("--scale", type=float, default=1.0,
                   help="launch-size factor when the capture ran a smaller case of the same kernel")
    sub.add_parser("check")
    a = ap.parse_args(argv)
    if a.cmd == "record":
        print(json.dumps(record(a.csv, a.kernel, a.workload, a.cls, a.group, a.summary, a.scale)))
    else:
        for e in _load()["entries"]:
            ok = e["source_hash"] == source_hash(e["group"])
            print(f"{e['workload']:24s} {e['cls']:12s} {e['bytes_per_launch'] / 1e6:10.2f} MB  "
                  f"{'current' if ok else 'STALE (sources changed)'}")
    return 0


if __name__ == "__main__":
    sys.exit(main())
