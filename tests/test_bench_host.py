"""Host-side helpers of bench.py (CPU)."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_source_hash_ignores_comments_and_spacing(tmp_path):
    a = tmp_path / "a.cu"
    b = tmp_path / "b.cu"
    c = tmp_path / "c.cu"
    a.write_text("// header\nint f(int x) {\n  return x + 1;  /* one */\n}\n")
    b.write_text("int f(int x)   {\n\treturn   x + 1;\n\n}  // trailing\n")
    c.write_text("int f(int x) {\n  return x + 2;\n}\n")
    ha, hb, hc = (bench.source_hash([str(p)]) for p in (a, b, c))
    assert ha == hb
    assert ha != hc


def test_source_hash_keeps_line_breaks_and_string_literals(tmp_path):
    files = {
        # a token moved onto a preprocessor line changes the code
        "p1.cu": "#define K 4\nint k = K;\n",
        "p2.cu": "#define K 4 int k = K;\n",
        # text after // inside a string literal is code, not a comment
        "s1.cu": 'const char* s = "a // b";\n',
        "s2.cu": 'const char* s = "a // c";\n',
        "q1.cu": "char c = '\"'; int x = 1; // x\n",
        "q2.cu": "char c = '\"'; int x = 2; // x\n",
    }
    h = {}
    for name, text in files.items():
        f = tmp_path / name
        f.write_text(text)
        h[name] = bench.source_hash([str(f)])
    assert h["p1.cu"] != h["p2.cu"]
    assert h["s1.cu"] != h["s2.cu"]
    assert h["q1.cu"] != h["q2.cu"]
    assert bench.strip_comments('x = "/* no */"; /* yes */ y;') == 'x = "/* no */";   y;'


def test_traffic_figures_are_tied_to_listed_sources():
    import json

    with open(os.path.join(ROOT, "profiles", "traffic.json")) as fh:
        t = json.load(fh)
    for kernel, e in t.items():
        assert e["sources"] and all(os.path.exists(os.path.join(ROOT, s)) for s in e["sources"])
        got = bench.traffic_for(kernel)
        # either the figure (code unchanged since the capture) or None
        assert got in (None, e["traffic_bytes_per_launch"])


def test_pick_peak_follows_the_clock_regime():
    pk = {"bf16_tflops": 1904.5, "bf16_tflops_sustained": 1717.4, "sm_max_mhz": 2070.0}
    # a sub-second region runs at burst clocks whatever the samples say
    assert bench.pick_peak(pk, 0.24, {"sm_mhz": 1400.0, "sm_max_mhz": 2070.0})[:2] == (1904.5, "burst")
    # a long region that held its clock near the maximum is still burst
    assert bench.pick_peak(pk, 3.0, {"sm_mhz": 2000.0, "sm_max_mhz": 2070.0})[:2] == (1904.5, "burst")
    # a long region that settled under the power cap is held to the sustained figure
    assert bench.pick_peak(pk, 3.0, {"sm_mhz": 1460.0, "sm_max_mhz": 2070.0})[:2] == (1717.4, "sustained")
    # no clock samples: the burst figure (the larger denominator)
    assert bench.pick_peak(pk, 3.0, None)[:2] == (1904.5, "burst")
