"""The forward entry point that allocates nothing: mls_head_loss_fwd_noalloc.

Some callers cannot allocate device memory at the moment they compute the
loss: a host program or plugin that has no allocator to hand the library a
workspace, or a steady-state loop that must not call cudaMalloc because it can
synchronise the device and take memory from a pool another allocator owns.  For
them the library keeps a fixed scratch array of its own and offers a forward
that needs no workspace.  This file checks, through the C ABI, that two calls in
a row give the same results as the ordinary forward with a workspace and as
the fp64 oracle, and that a problem too large for the built-in scratch is
refused before anything runs.
(It is collected last so that a run stopping at the first failure has already
run every other test.)
"""
import types

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import synth

from helpers import check_forward, exact_logits, rel_close

pytestmark = pytest.mark.gpu


def _outputs(wl, dev):
    M, T = wl.M, wl.T
    return dict(loss=torch.full((1,), float("nan"), device=dev),
                tok_loss=torch.full((M, T), float("nan"), device=dev),
                tok_diag=torch.full((3, M, T), float("nan"), device=dev),
                argmax=torch.full((M, T), -7, dtype=torch.int32, device=dev),
                stats=torch.full((2, M, T), float("nan"), device=dev))


def test_noalloc_forward_matches_workspace_forward_on_two_calls():
    dev = torch.device("cuda")
    cases = [
        synth.Workload("noalloc_a", T=1000, d=(256, 512, 768), V=5000, tau=0.8, alpha=0.4,
                       w_sigma=0.03, weights=(1.0, 0.5, 2.0)),
        synth.Workload("noalloc_b", T=700, d=(128, 384), V=3001, tau=1.0, alpha=0.5,
                       w_sigma=0.05, teacher=0),
    ]
    for i, wl in enumerate(cases):
        H, W, y = synth.make_inputs(wl, seed=40 + i, device=dev)
        y[3] = -1
        ref = B.HeadLoss(wl.d, wl.T, wl.V, teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha,
                         w=wl.weights, device=dev)
        ref.forward(H, W, y)
        out = _outputs(wl, dev)
        B.mls_head_loss_fwd_noalloc(ref.prob, H, W, y, out["loss"], out["tok_loss"],
                                    out["tok_diag"], out["argmax"], out["stats"])
        torch.cuda.synchronize()
        assert B.mls_get_status() == 0
        for key, want in (("tok_loss", ref.tok_loss), ("tok_diag", ref.tok_diag),
                          ("stats", ref.stats), ("loss", ref.loss)):
            ok, err = rel_close(out[key].cpu().double().numpy(), want.cpu().double().numpy())
            assert ok, f"call {i}: {key} differs from the workspace forward (rel err {err})"
        assert np.array_equal(out["argmax"].cpu().numpy(), ref.argmax.cpu().numpy())
        # and directly against the oracle, on the same inputs
        yc = y.cpu().numpy().astype(np.int32)
        want = oracle.forward(synth.as_oracle_arrays(H), synth.as_oracle_arrays(W), yc,
                              teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha, w=wl.weights)
        got = types.SimpleNamespace(tok_loss=out["tok_loss"], tok_diag=out["tok_diag"],
                                    stats=out["stats"], argmax=out["argmax"])
        check_forward(got, want, logits=exact_logits(H, W))
        ok, err = rel_close([out["loss"].item()], [want["loss"]])
        assert ok, f"call {i}: scalar loss differs from the oracle (rel err {err})"


def test_noalloc_rejects_problems_beyond_the_scratch():
    dev = torch.device("cuda")
    # 4 sub-models x 10^6 tokens: the partial row states alone (6 floats per
    # token and sub-model) exceed the 64 MiB scratch
    d, T, V = (64, 64, 64, 64), 1000000, 1000
    H = [torch.zeros(T, x, dtype=torch.bfloat16, device=dev) for x in d]
    W = [torch.zeros(V, x, dtype=torch.bfloat16, device=dev) for x in d]
    y = torch.zeros(T, dtype=torch.int32, device=dev)
    wl = synth.Workload("too_big", T=T, d=d, V=V)
    out = _outputs(wl, dev)
    prob = B.Problem(d, T, V)
    with pytest.raises(B.MLSError) as e:
        B.mls_head_loss_fwd_noalloc(prob, H, W, y, out["loss"], out["tok_loss"], out["tok_diag"],
                                    out["argmax"], out["stats"])
    assert e.value.code == B.MLS_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.isnan(out["loss"]).all()  # nothing ran
