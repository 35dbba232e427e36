"""Host-side helpers of bench.py (CPU)."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_source_hash_ignores_comments_and_layout(tmp_path):
    a = tmp_path / "a.cu"
    b = tmp_path / "b.cu"
    c = tmp_path / "c.cu"
    a.write_text("// header\nint f(int x) {\n  return x + 1;  /* one */\n}\n")
    b.write_text("/* other\n   words */ int f(int x)   { return x + 1; }  // trailing\n")
    c.write_text("int f(int x) { return x + 2; }\n")
    ha, hb, hc = (bench.source_hash([str(p)]) for p in (a, b, c))
    assert ha == hb
    assert ha != hc


def test_traffic_figures_are_tied_to_listed_sources():
    import json

    with open(os.path.join(ROOT, "profiles", "traffic.json")) as fh:
        t = json.load(fh)
    for kernel, e in t.items():
        assert e["sources"] and all(os.path.exists(os.path.join(ROOT, s)) for s in e["sources"])
        got = bench.traffic_for(kernel)
        # either the figure (code unchanged since the capture) or None
        assert got in (None, e["traffic_bytes_per_launch"])
