"""Shared test helpers: run the CUDA path through the C ABI and compare it with
the fp64 oracle using the tolerances stated for this operation:
  per-token losses and the scalar loss   1e-3 relative
  KL                                      |diff| <= 1e-3 * max(1, Ld)
  gradients                               max|diff| / max|ref| <= 2e-2 per tensor
  argmax                                  exact wherever the top-2 logit gap of
                                          the exact logits exceeds 1e-4 * max(1, |z_max|)
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import synth

LOSS_RTOL = 1e-3
GRAD_TOL = 2e-2


def run_gpu(wl: synth.Workload, H, W, y, grad_scale=1.0, vocab_group=0, backward=True):
    """H, W, y may live on the CPU or the GPU; returns the op with its outputs."""
    dev = torch.device("cuda")
    Hd = [h.to(dev).contiguous() for h in H]
    Wd = [w.to(dev).contiguous() for w in W]
    yd = y.to(dev).to(torch.int32).contiguous()
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    op = B.HeadLoss(wl.d, wl.T, wl.V, teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha,
                    w=wl.weights, dtype=dt, device=dev, vocab_group=vocab_group)
    op.forward(Hd, Wd, yd)
    if backward:
        op.backward(Hd, Wd, yd, grad_scale=grad_scale)
    torch.cuda.synchronize()
    status = B.mls_get_status()
    return op, status


def rel_close(got, want, rtol=LOSS_RTOL, atol=1e-6):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    err = np.abs(got - want)
    bad = err > rtol * np.abs(want) + atol
    return not bad.any(), float((err / (np.abs(want) + atol)).max()) if err.size else 0.0


def check_forward(op, ref, rows=None, logits=None):
    """Compare per-token outputs (optionally only `rows`) with the oracle's."""
    sel = (lambda a: a[:, rows]) if rows is not None else (lambda a: a)
    tl = sel(op.tok_loss.cpu().double().numpy())
    diag = op.tok_diag.cpu().double().numpy()
    st = op.stats.cpu().double().numpy()
    ok, e = rel_close(tl, ref["tok_loss"])
    assert ok, f"tok_loss rel err {e}"
    ok, e = rel_close(sel(diag[0]), ref["ce"])
    assert ok, f"CE rel err {e}"
    ok, e = rel_close(sel(diag[1]), ref["ld"])
    assert ok, f"Ld rel err {e}"
    kl_err = np.abs(sel(diag[2]) - ref["kl"]) / np.maximum(1.0, np.abs(ref["ld"]))
    assert kl_err.max() <= LOSS_RTOL, f"KL err {kl_err.max()}"
    ok, e = rel_close(sel(st[0]), ref["lse"])
    assert ok, f"lse rel err {e}"
    ok, e = rel_close(sel(st[1]), ref["lse_tau"])
    assert ok, f"lse_tau rel err {e}"
    if logits is not None:
        am = sel(op.argmax.cpu().numpy())
        for m, z in enumerate(logits):
            z = z.numpy()
            top = np.sort(z, axis=-1)[:, -2:]
            gap = top[:, 1] - top[:, 0]
            decided = gap > 1e-4 * np.maximum(1.0, np.abs(top[:, 1]))
            want = np.argmax(z, -1)
            assert (am[m][decided] == want[decided]).all(), f"argmax mismatch model {m}"
            # undecided rows: the GPU's pick must still be a maximiser within the gap
            idx = np.nonzero(~decided)[0]
            for r in idx:
                assert z[r, am[m][r]] >= top[r, 1] - 1e-4 * max(1.0, abs(top[r, 1]))


def check_grads(op, dH=None, dW=None, dH_rows=None):
    """dH, dW: full oracle gradients (lists) or None; dH_rows: (rows, [per-model rows])."""
    for m in range(op.M):
        pairs = []
        if dW is not None:
            pairs.append(("dW", op.dW[m], dW[m]))
        if dH is not None:
            pairs.append(("dH", op.dH[m], dH[m]))
        if dH_rows is not None:
            rows, want = dH_rows
            pairs.append(("dH rows", op.dH[m][torch.as_tensor(rows, device=op.dH[m].device)], want[m]))
        for name, got, want in pairs:
            g = got.cpu().double().numpy()
            scale = np.abs(want).max()
            err = np.abs(g - want).max() / max(scale, 1e-30)
            assert err <= GRAD_TOL, f"{name}[{m}] max-norm rel err {err}"


def exact_logits(H, W, rows=None):
    """fp64 logits of the stored inputs (library matmul), for argmax checks."""
    out = []
    for h, w in zip(H, W):
        hh = h.detach().cpu().double()
        if rows is not None:
            hh = hh[torch.as_tensor(rows)]
        out.append(hh @ w.detach().cpu().double().T)
    return out
