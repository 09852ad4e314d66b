"""The draft-depth table shipped with the library: for every measured (batch, context) of a
`bench.py --sweep` run, the committed tokens/s at each draft depth K (K = 0 is greedy
decoding).  metrics.DepthPolicy turns it into the depth choice for any (batch, context), and
fastmtp.choose_depth reads the packaged copy (the paper's S = tau / c trade-off of Sec. 6.4,
measured on the GPU the library runs on instead of assumed).

    python -m paper_2609_03181_gb300.depth_table SWEEP.jsonl [--router uniform] > TABLE.json
"""
from __future__ import annotations

import argparse
import json
import os
import sys
from typing import Iterable

PACKAGED = os.path.join(os.path.dirname(os.path.abspath(__file__)), "depth_table_gb300.json")


def build_table(lines: Iterable[str], router: str = "uniform", source: str = "", experts: str = "bf16") -> dict:
    """The table of one router mode and expert format from the JSON lines of a sweep (other lines
    are skipped; lines without an `experts` field are bf16)."""
    pts = {}
    meta = {}
    for line in lines:
        line = line.strip()
        if not line.startswith("{"):
            continue
        d = json.loads(line)
        if d.get("sweep_clocks") is not None:
            meta["clocks"] = d["sweep_clocks"]
        if not d.get("sweep") or d.get("router") != router or d.get("experts", "bf16") != experts:
            continue
        key = (int(d["batch"]), int(d["ctx"]))
        p = pts.setdefault(key, {"batch": key[0], "ctx": key[1], "tokens_per_s": {}, "steps": {}})
        p["tokens_per_s"][str(int(d["K"]))] = float(d["tokens_per_s"])
        p["steps"][str(int(d["K"]))] = int(d.get("steps", 0))
    return {"router": router, "source": source, **meta, "points": [pts[k] for k in sorted(pts)]}


def load_packaged() -> dict:
    with open(PACKAGED) as f:
        return json.load(f)


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("sweep")
    ap.add_argument("--router", default="uniform")
    ap.add_argument("--source", default="")
    a = ap.parse_args(argv)
    with open(a.sweep) as f:
        t = build_table(f, a.router, a.source or os.path.basename(a.sweep))
    json.dump(t, sys.stdout, indent=1)
    sys.stdout.write("\n")


if __name__ == "__main__":
    main()
