"""The checked build (libmls_checked.so, -DMLS_CHECKED): the same kernels with
their internal invariants (tile and partial indices inside their problems,
compaction within its count, bisection within its pass bound, a sampling step
found) asserted into the status word, which stands in for a sanitizer on a
pool where compute-sanitizer is closed.  Child processes run every entry point
on small ragged cases with each build; the checked one must end with clean
status words and both must give bit-identical outputs."""
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2608_09703_gb300 import build as mbuild

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run_child(path, checked):
    env = dict(os.environ)
    env["MLS_CHECKED"] = "1" if checked else "0"
    env["PYTHONPATH"] = ROOT + os.pathsep + env.get("PYTHONPATH", "")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "checked_run.py"), path],
                       env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    return dict(np.load(path))


def test_checked_build_is_clean_and_identical(tmp_path):
    mbuild.build()
    mbuild.build(checked=True)
    normal = run_child(str(tmp_path / "normal.npz"), checked=False)
    checked = run_child(str(tmp_path / "checked.npz"), checked=True)
    for k in checked:
        if k.startswith("status"):
            assert int(checked[k]) == 0, f"{k}: {int(checked[k])}"
            assert int(normal[k]) == 0, f"{k}: {int(normal[k])}"
        else:
            assert np.array_equal(checked[k], normal[k]), k
