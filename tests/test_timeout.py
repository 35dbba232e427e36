"""Failure detection without a GPU fault: every pipeline wait in the kernels is
bounded.  With the test hook MLS_TEST_STALL_FIRST_STAGE set, the first CTA pair
of the forward head kernel issues nothing for its first stage, so the MMA
issuer's wait on it runs out (about 2 s); the kernel then drains its copies and
MMAs, frees TMEM and returns, and the call reports MLS_STATUS_TIMEOUT.  The
same process then clears the hook and computes the right loss: the context
stays usable.  It runs in a child process so the hook cannot leak into other
tests."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import os, sys, time
sys.path.insert(0, {root!r})
import torch
from oracle import oracle
from paper_2608_09703_gb300 import binding as B, synth
wl = synth.Workload("stall", T=300, d=(64, 128), V=1000, w_sigma=0.05)
H, W, y = synth.make_inputs(wl, seed=3)
Hd, Wd, yd = [h.cuda() for h in H], [w.cuda() for w in W], y.cuda()
op = B.HeadLoss(wl.d, wl.T, wl.V, device="cuda")
os.environ["MLS_TEST_STALL_FIRST_STAGE"] = "1"
t0 = time.time()
op.forward(Hd, Wd, yd)
torch.cuda.synchronize()
print("STALLED", B.mls_get_status(), round(time.time() - t0, 2))
del os.environ["MLS_TEST_STALL_FIRST_STAGE"]
op.forward(Hd, Wd, yd)
torch.cuda.synchronize()
ref = oracle.forward(synth.as_oracle_arrays(H), synth.as_oracle_arrays(W), y.numpy())
print("CLEAN", B.mls_get_status(), op.loss.item(), ref["loss"])
"""


def test_stalled_stage_reports_timeout_and_context_survives():
    env = dict(os.environ)
    env.pop("MLS_TEST_STALL_FIRST_STAGE", None)
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT)], env=env,
                       capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    out = {l.split()[0]: l.split()[1:] for l in r.stdout.splitlines() if l.split()}
    from paper_2608_09703_gb300 import binding as B

    assert int(out["STALLED"][0]) & B.MLS_STATUS_TIMEOUT
    status, got, want = int(out["CLEAN"][0]), float(out["CLEAN"][1]), float(out["CLEAN"][2])
    assert status == 0
    assert abs(got - want) <= 1e-3 * abs(want)
