"""Pins for the fp64 CPU oracle, against facts that do not come from the oracle.

Each check ties the oracle to something independent of its own code: a
worked example derived by hand, closed forms (zero heads, identical student
and teacher), library routines on special cases (``torch.nn.functional``
cross-entropy, soft-target cross-entropy, KL, logsumexp, numpy argmax),
central finite differences, autograd of the loss written from Eq. 2/3, and
invariants of the gradient (rows of dL/dz sum to zero, linearity).
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import oracle as orc


def normal(shape, seed, scale=1.0, dtype=np.float64):
    return (np.random.default_rng(seed).standard_normal(shape) * scale).astype(dtype)


def problem(T, d, V, seed=0, hs=1.0, ws=0.3, dtype=np.float64):
    H = [normal((T, dm), seed + 10 * m, hs, dtype) for m, dm in enumerate(d)]
    W = [normal((V, dm), seed + 10 * m + 5, ws, dtype) for m, dm in enumerate(d)]
    y = np.random.default_rng(seed + 99).integers(0, V, T).astype(np.int32)
    return H, W, y


def logits(H, W):
    return [torch.from_numpy(h.astype(np.float64)) @ torch.from_numpy(w.astype(np.float64)).T
            for h, w in zip(H, W)]


def sig(x):
    return 1.0 / (1.0 + math.exp(-x))


# ---------------------------------------------------------------- worked example
@pytest.mark.parametrize("tau", [1.0, 2.0])
def test_hand_worked_example(tau):
    """Two sub-models, V = 2, width 1, one token with target 0, derived by hand.

    student logits z_s = (1, 0), teacher logits z_T = (2, -2), alpha = 1/2.
    """
    H = [np.array([[1.0]]), np.array([[2.0]])]
    W = [np.array([[1.0], [0.0]]), np.array([[1.0], [-1.0]])]
    y = np.array([0], np.int32)
    alpha = 0.5
    out = orc.forward(H, W, y, teacher=1, tau=tau, alpha=alpha)
    dH, dW = orc.backward(H, W, y, teacher=1, tau=tau, alpha=alpha)

    ce_s = math.log1p(math.exp(-1.0))                 # log(e + 1) - 1
    ce_t = math.log1p(math.exp(-4.0))                 # log(e^2 + e^-2) - 2
    q0, q1 = sig(4.0 / tau), sig(-4.0 / tau)          # softmax((2, -2) / tau)
    lp0 = -math.log1p(math.exp(-1.0 / tau))           # log softmax((1, 0) / tau)
    lp1 = -1.0 / tau - math.log1p(math.exp(-1.0 / tau))
    ld_s = -(q0 * lp0 + q1 * lp1)
    hq = -(q0 * math.log(q0) + q1 * math.log(q1))
    assert out["ce"][0, 0] == pytest.approx(ce_s, abs=1e-14)
    assert out["ce"][1, 0] == pytest.approx(ce_t, abs=1e-14)
    assert out["ld"][0, 0] == pytest.approx(ld_s, abs=1e-14)
    assert out["kl"][0, 0] == pytest.approx(ld_s - hq, abs=1e-14)
    assert out["tok_loss"][0, 0] == pytest.approx(0.5 * ce_s + 0.5 * ld_s, abs=1e-14)
    assert out["tok_loss"][1, 0] == pytest.approx(ce_t, abs=1e-14)
    assert out["loss"] == pytest.approx(0.5 * ce_s + 0.5 * ld_s + ce_t, abs=1e-14)
    assert list(out["argmax"][:, 0]) == [0, 0]

    # gradients: student G = (1-a)(p - e_y) + (a/tau)(p^tau - q); teacher G = p - e_y
    p0, p1 = sig(1.0), sig(-1.0)
    pt0, pt1 = sig(1.0 / tau), sig(-1.0 / tau)
    gs = [0.5 * (p0 - 1.0) + 0.5 / tau * (pt0 - q0), 0.5 * p1 + 0.5 / tau * (pt1 - q1)]
    gt = [sig(4.0) - 1.0, sig(-4.0)]
    assert dH[0][0, 0] == pytest.approx(gs[0] * 1.0 + gs[1] * 0.0, abs=1e-14)
    assert dW[0][:, 0] == pytest.approx([gs[0] * 1.0, gs[1] * 1.0], abs=1e-14)
    assert dH[1][0, 0] == pytest.approx(gt[0] * 1.0 + gt[1] * -1.0, abs=1e-14)
    assert dW[1][:, 0] == pytest.approx([gt[0] * 2.0, gt[1] * 2.0], abs=1e-14)


# ---------------------------------------------------------------- closed forms
@pytest.mark.parametrize("tau", [0.5, 1.0, 2.0])
def test_zero_heads_give_log_v(tau):
    T, d, V = 7, (8, 16, 12), 37
    H, W, y = problem(T, d, V, seed=1)
    W = [np.zeros_like(w) for w in W]
    w = (0.5, 2.0, 1.5)
    out = orc.forward(H, W, y, tau=tau, alpha=0.3, w=w)
    lv = math.log(V)
    np.testing.assert_allclose(out["ce"], lv, atol=1e-12)
    np.testing.assert_allclose(out["ld"], lv, atol=1e-12)
    np.testing.assert_allclose(out["kl"], 0.0, atol=1e-12)
    np.testing.assert_allclose(out["lse"], lv, atol=1e-12)
    np.testing.assert_allclose(out["lse_tau"], lv, atol=1e-12)
    assert out["loss"] == pytest.approx(sum(w) * lv, rel=1e-13)
    assert (out["argmax"] == 0).all()


@pytest.mark.parametrize("tau", [0.5, 1.0, 3.0])
def test_student_equal_teacher(tau):
    """Identical student and teacher: KL = 0, Ld = H(q) and the distillation
    gradient vanishes, so the student's gradients are (1 - alpha) times the
    teacher's."""
    T, V, dm = 9, 29, 12
    H, W, y = problem(T, (dm,), V, seed=2, ws=0.5)
    H2, W2 = [H[0], H[0].copy()], [W[0], W[0].copy()]
    alpha = 0.35
    out = orc.forward(H2, W2, y, teacher=1, tau=tau, alpha=alpha)
    np.testing.assert_allclose(out["kl"][0], 0.0, atol=1e-13)
    z = logits(H, W)[0]
    q = torch.softmax(z / tau, -1)
    Hq = -(q * torch.log(q)).sum(-1).numpy()
    np.testing.assert_allclose(out["ld"][0], Hq, rtol=1e-12)
    dH, dW = orc.backward(H2, W2, y, teacher=1, tau=tau, alpha=alpha)
    np.testing.assert_allclose(dH[0], (1 - alpha) * dH[1], rtol=1e-10, atol=1e-15)
    np.testing.assert_allclose(dW[0], (1 - alpha) * dW[1], rtol=1e-10, atol=1e-15)


# ---------------------------------------------------------------- library routines
def test_alpha_zero_is_library_cross_entropy():
    T, d, V = 16, (8, 24, 16), 50
    H, W, y = problem(T, d, V, seed=3)
    w = (1.0, 0.25, 3.0)
    out = orc.forward(H, W, y, tau=1.7, alpha=0.0, w=w)
    zs = logits(H, W)
    yt = torch.from_numpy(y.astype(np.int64))
    total = 0.0
    for m, z in enumerate(zs):
        ce = F.cross_entropy(z, yt, reduction="none").numpy()
        np.testing.assert_allclose(out["ce"][m], ce, rtol=1e-12)
        np.testing.assert_allclose(out["tok_loss"][m], ce, rtol=1e-12)
        total += w[m] * ce.mean()
    assert out["loss"] == pytest.approx(total, rel=1e-12)


@pytest.mark.parametrize("tau", [0.5, 1.0, 2.0])
def test_distillation_is_soft_target_cross_entropy(tau):
    T, d, V = 11, (8, 16, 24), 64
    H, W, y = problem(T, d, V, seed=4, ws=0.4)
    out = orc.forward(H, W, y, teacher=2, tau=tau, alpha=0.5)
    zs = logits(H, W)
    q = torch.softmax(zs[2] / tau, -1)
    for m in range(3):
        ld = F.cross_entropy(zs[m] / tau, q, reduction="none").numpy()
        kl = F.kl_div(torch.log_softmax(zs[m] / tau, -1), q, reduction="none").sum(-1).numpy()
        np.testing.assert_allclose(out["ld"][m], ld, rtol=1e-11)
        np.testing.assert_allclose(out["kl"][m], kl, rtol=1e-9, atol=1e-13)
        np.testing.assert_allclose(out["lse"][m], torch.logsumexp(zs[m], -1).numpy(), rtol=1e-13)
        np.testing.assert_allclose(out["lse_tau"][m], torch.logsumexp(zs[m] / tau, -1).numpy(),
                                   rtol=1e-13)
        np.testing.assert_array_equal(out["argmax"][m], np.argmax(zs[m].numpy(), -1))
        ce = F.cross_entropy(zs[m], torch.from_numpy(y.astype(np.int64)), reduction="none").numpy()
        want = ce if m == 2 else 0.5 * ce + 0.5 * ld
        np.testing.assert_allclose(out["tok_loss"][m], want, rtol=1e-11)


def test_integer_exact_argmax_and_ties():
    """One-hot hidden rows and small-integer heads make every logit an exact
    integer; argmax then must equal numpy's (first maximum on ties)."""
    T, V, dm = 24, 40, 16
    rng = np.random.default_rng(5)
    H = np.zeros((T, dm), np.float32)
    H[np.arange(T), rng.integers(0, dm, T)] = 1.0
    W = rng.integers(-3, 4, (V, dm)).astype(np.float32)
    W[7] = W[3]          # duplicate rows -> exact ties between v=3 and v=7
    Hs, Ws = [H, H], [W, np.flip(W, 0).copy()]
    y = rng.integers(0, V, T).astype(np.int32)
    out = orc.forward(Hs, Ws, y)
    for m in range(2):
        z = Hs[m].astype(np.int64) @ Ws[m].astype(np.int64).T
        np.testing.assert_array_equal(out["argmax"][m], np.argmax(z, -1))
        ce = out["lse"][m] - z[np.arange(T), y]
        np.testing.assert_allclose(out["ce"][m], ce, rtol=0, atol=1e-12)


def test_bf16_storage_decodes_exactly():
    T, d, V = 5, (8, 16), 33
    H, W, y = problem(T, d, V, seed=6, dtype=np.float32)
    Hb = [torch.from_numpy(h).to(torch.bfloat16) for h in H]
    Wb = [torch.from_numpy(w).to(torch.bfloat16) for w in W]
    bits = lambda ts: [t.view(torch.int16).numpy().view(np.uint16) for t in ts]
    f32 = lambda ts: [t.float().numpy() for t in ts]
    a = orc.forward(bits(Hb), bits(Wb), y, tau=0.7)
    b = orc.forward(f32(Hb), f32(Wb), y, tau=0.7)
    assert a["loss"] == b["loss"]
    np.testing.assert_array_equal(a["tok_loss"], b["tok_loss"])


# ---------------------------------------------------------------- gradients
def _fd_case():
    T, d, V = 4, (8, 16), 32
    H, W, y = problem(T, d, V, seed=7, ws=0.5)
    y[2] = -1            # one ignored token
    return H, W, y, dict(teacher=1, tau=0.8, alpha=0.4, w=(1.3, 0.7))


def test_finite_differences():
    """Central differences in fp64 of the objective.  Student parameters see
    the whole loss; the teacher's see only its own term, because Eq. 2 stops
    the gradient through the teacher's distribution."""
    H, W, y, kw = _fd_case()
    dH, dW = orc.backward(H, W, y, grad_scale=1.0, **kw)
    eps = 1e-6
    T = H[0].shape[0]
    n = int((y >= 0).sum())
    tmask = y >= 0

    def objective(Hc, Wc, m):
        out = orc.forward(Hc, Wc, y, **kw)
        if m == kw["teacher"]:
            return kw["w"][m] * out["tok_loss"][m][tmask].sum() / n
        return out["loss"]

    for m in range(2):
        for which, grad in (("H", dH[m]), ("W", dW[m])):
            base = H if which == "H" else W
            fd = np.zeros_like(grad)
            for idx in np.ndindex(*grad.shape):
                vals = []
                for sgn in (1, -1):
                    arrs = [a.copy() for a in base]
                    arrs[m][idx] += sgn * eps
                    vals.append(objective(arrs, W, m) if which == "H" else objective(H, arrs, m))
                fd[idx] = (vals[0] - vals[1]) / (2 * eps)
            scale = np.abs(grad).max()
            assert np.abs(fd - grad).max() <= 1e-6 * scale, (m, which)


def test_autograd_of_eq2_eq3():
    """Gradients from torch autograd applied to the objective written from
    Eq. 2/3 with q detached (stop_grad)."""
    T, d, V = 12, (16, 24, 8), 40
    H, W, y = problem(T, d, V, seed=8, ws=0.4)
    y[[3, 9]] = -1
    teacher, tau, alpha, w, g = 1, 0.7, 0.3, (0.5, 1.5, 2.0), 1.3
    dH, dW = orc.backward(H, W, y, teacher=teacher, tau=tau, alpha=alpha, w=w, grad_scale=g)
    Ht = [torch.tensor(h, requires_grad=True) for h in H]
    Wt = [torch.tensor(x, requires_grad=True) for x in W]
    yt = torch.from_numpy(y.astype(np.int64))
    valid = yt >= 0
    n = valid.sum()
    z = [h @ x.T for h, x in zip(Ht, Wt)]
    q = torch.softmax(z[teacher] / tau, -1).detach()
    loss = 0.0
    for m in range(3):
        ce = torch.logsumexp(z[m], -1) - z[m].gather(1, yt.clamp(min=0)[:, None])[:, 0]
        if m == teacher:
            lm = ce
        else:
            ld = -(q * torch.log_softmax(z[m] / tau, -1)).sum(-1)
            lm = (1 - alpha) * ce + alpha * ld
        loss = loss + w[m] * (lm * valid).sum() / n
    (g * loss).backward()
    for m in range(3):
        np.testing.assert_allclose(dH[m], Ht[m].grad.numpy(), rtol=1e-10, atol=1e-14)
        np.testing.assert_allclose(dW[m], Wt[m].grad.numpy(), rtol=1e-10, atol=1e-14)


def test_gradient_invariants_and_linearity():
    T, d, V = 10, (8, 16, 24), 30
    H, W, y = problem(T, d, V, seed=9, ws=0.4)
    y[4] = -1
    kw = dict(teacher=2, tau=1.5, alpha=0.6)
    dH, dW = orc.backward(H, W, y, w=(1.0, 1.0, 1.0), grad_scale=1.0, **kw)
    for m in range(3):
        # every row of dL/dz sums to zero, so the columns of dW do too
        assert np.abs(dW[m].sum(0)).max() <= 1e-13 * max(1.0, np.abs(dW[m]).max()) * V
        assert np.abs(dH[m][4]).max() == 0.0          # ignored token
    dH2, dW2 = orc.backward(H, W, y, w=(2.0, 1.0, 3.0), grad_scale=1.5, **kw)
    for m, f in enumerate((3.0, 1.5, 4.5)):
        np.testing.assert_allclose(dH2[m], f * dH[m], rtol=1e-12, atol=1e-16)
        np.testing.assert_allclose(dW2[m], f * dW[m], rtol=1e-12, atol=1e-16)
    a = orc.forward(H, W, y, w=(1.0, 1.0, 1.0), **kw)["loss"]
    b = orc.forward(H, W, y, w=(2.0, 2.0, 2.0), **kw)["loss"]
    assert b == pytest.approx(2 * a, rel=1e-14)
    # the teacher's gradient depends on neither alpha nor tau
    dH3, dW3 = orc.backward(H, W, y, w=(1.0, 1.0, 1.0), teacher=2, tau=0.4, alpha=0.1)
    np.testing.assert_allclose(dH3[2], dH[2], rtol=1e-12, atol=1e-16)
    np.testing.assert_allclose(dW3[2], dW[2], rtol=1e-12, atol=1e-16)


def test_ignored_tokens_equal_dropping_them():
    T, d, V = 14, (8, 16), 26
    H, W, y = problem(T, d, V, seed=10, ws=0.4)
    drop = np.array([1, 5, 6, 13])
    y2 = y.copy()
    y2[drop] = -1
    keep = np.setdiff1d(np.arange(T), drop)
    kw = dict(tau=0.9, alpha=0.45)
    full = orc.forward(H, W, y2, **kw)
    sub = orc.forward([h[keep] for h in H], W, y[keep], **kw)
    assert full["loss"] == pytest.approx(sub["loss"], rel=1e-13)
    dHf, dWf = orc.backward(H, W, y2, **kw)
    dHs, dWs = orc.backward([h[keep] for h in H], W, y[keep], **kw)
    for m in range(2):
        np.testing.assert_allclose(dWf[m], dWs[m], rtol=1e-11, atol=1e-15)
        np.testing.assert_allclose(dHf[m][keep], dHs[m], rtol=1e-11, atol=1e-15)
        assert np.abs(dHf[m][drop]).max() == 0.0
        assert (full["tok_loss"][m][drop] == 0).all()


def test_rows_match_full_problem():
    T, d, V = 9, (8, 16, 8), 21
    H, W, y = problem(T, d, V, seed=11, ws=0.4)
    y[0] = -1
    kw = dict(teacher=1, tau=1.2, alpha=0.5, w=(1.0, 0.5, 2.0))
    full = orc.forward(H, W, y, **kw)
    dH, _ = orc.backward(H, W, y, grad_scale=0.7, **kw)
    sel = [8, 0, 3]
    r = orc.rows(H, W, y, sel, grad_scale=0.7, **kw)
    for key in ("tok_loss", "ce", "ld", "kl", "lse", "lse_tau"):
        np.testing.assert_allclose(r[key], full[key][:, sel], rtol=1e-13, atol=1e-15)
    np.testing.assert_array_equal(r["argmax"], full["argmax"][:, sel])
    for m in range(3):
        np.testing.assert_allclose(r["dH"][m], dH[m][sel], rtol=1e-12, atol=1e-16)


def test_degenerate_cases():
    T, d, V = 6, (8, 8), 10
    H, W, y = problem(T, d, V, seed=12)
    none = np.full(T, -1, np.int32)
    out = orc.forward(H, W, none)
    assert out["loss"] == 0.0
    dH, dW = orc.backward(H, W, none)
    assert all(np.abs(x).max() == 0 for x in dH + dW)
    bad = y.copy()
    bad[2] = V
    with pytest.raises(RuntimeError):
        orc.forward(H, W, bad)
    # a single sub-model is plain cross-entropy
    one = orc.forward(H[:1], W[:1], y, alpha=0.9)
    ce = F.cross_entropy(logits(H[:1], W[:1])[0], torch.from_numpy(y.astype(np.int64)))
    assert one["loss"] == pytest.approx(float(ce), rel=1e-13)
    # zero tokens
    empty = orc.forward([h[:0] for h in H], W, y[:0])
    assert empty["loss"] == 0.0


def test_golden_regression_fixture():
    """The oracle still reproduces tests/golden/oracle_small.json (written by
    tests/golden/make_golden.py, which calls only the oracle)."""
    import json
    import os

    path = os.path.join(os.path.dirname(__file__), "golden", "oracle_small.json")
    fx = json.load(open(path))
    H = [np.asarray(h, np.float32) for h in fx["H"]]
    W = [np.asarray(x, np.float32) for x in fx["W"]]
    y = np.asarray(fx["y"], np.int32)
    kw = dict(teacher=fx["teacher"], tau=fx["tau"], alpha=fx["alpha"], w=fx["w"])
    f = orc.forward(H, W, y, **kw)
    assert f["loss"] == pytest.approx(fx["loss"], rel=1e-12)
    for k in ("tok_loss", "ce", "ld", "kl", "lse", "lse_tau"):
        np.testing.assert_allclose(f[k], np.asarray(fx[k]), rtol=1e-12, atol=1e-15)
    np.testing.assert_array_equal(f["argmax"], np.asarray(fx["argmax"]))
    dH, dW = orc.backward(H, W, y, **kw)
    for m in range(3):
        np.testing.assert_allclose(dH[m], np.asarray(fx["dH"][m]), rtol=1e-11, atol=1e-15)
        np.testing.assert_allclose(dW[m], np.asarray(fx["dW"][m]), rtol=1e-11, atol=1e-15)


# ---------------------------------------------------------------- evaluation metrics
def test_pairwise_kl_pins():
    """Pairwise KL(p_i || p_j) and top-1 agreement (Sec. 3.2.2): library KL on the
    same logits, zero on the diagonal and for identical sub-models, >= 0, and a
    two-token case by hand."""
    T, d, V = 9, (8, 16, 12), 23
    H, W, y = problem(T, d, V, seed=13, ws=0.5)
    H = H + [H[1].copy()]
    W = W + [W[1].copy()]            # sub-model 3 duplicates sub-model 1
    out = orc.pairwise(H, W)
    zs = logits(H, W)
    lp = [torch.log_softmax(z, -1) for z in zs]
    for i in range(4):
        for j in range(4):
            want = F.kl_div(lp[j], lp[i], reduction="none", log_target=True).sum(-1).numpy()
            np.testing.assert_allclose(out["kl"][i, j], want, rtol=1e-11, atol=1e-14)
            am_i, am_j = np.argmax(zs[i].numpy(), -1), np.argmax(zs[j].numpy(), -1)
            np.testing.assert_array_equal(out["agree"][i, j], (am_i == am_j).astype(np.int32))
    assert (out["kl"] >= -1e-14).all()
    np.testing.assert_allclose(out["kl"][1, 3], 0.0, atol=1e-13)
    np.testing.assert_array_equal(out["agree"][1, 3], 1)
    for i in range(4):
        assert (out["kl"][i, i] == 0).all()
    # by hand: z_0 = (1, 0), z_1 = (0, 0): KL(p0||p1) = log 2 - H(sigmoid(1))
    H2 = [np.array([[1.0]]), np.array([[1.0]])]
    W2 = [np.array([[1.0], [0.0]]), np.array([[0.0], [0.0]])]
    o2 = orc.pairwise(H2, W2)
    s1 = sig(1.0)
    h = -(s1 * math.log(s1) + (1 - s1) * math.log(1 - s1))
    assert o2["kl"][0, 1, 0] == pytest.approx(math.log(2.0) - h, abs=1e-14)
    # KL(p1||p0) = sum 0.5 (log 0.5 - log p0) = -log 2 - 0.5 (log s1 + log(1 - s1))
    assert o2["kl"][1, 0, 0] == pytest.approx(-math.log(2.0) - 0.5 * (math.log(s1) + math.log(1 - s1)),
                                              abs=1e-14)
    assert o2["agree"][0, 1, 0] == 1  # argmax (1, 0) is 0; argmax (0, 0) is 0 (lowest index)


# ---------------------------------------------------------------- junction (Eq. 1)
@pytest.mark.parametrize("embed_first", [False, True])
def test_junction_pins(embed_first):
    """The rescaled part has the fresh embedding's norm and o's direction, the
    embedding is copied unchanged, a hand-worked row, and central finite
    differences of a random linear functional of x."""
    rng = np.random.default_rng(14)
    T, dp_, de = 6, 5, 3
    o = rng.standard_normal((T, dp_)) * 3.0
    e = rng.standard_normal((T, de)) * 0.1
    o[4] = 0.0  # zero row: o~ = 0
    x = orc.junction_fwd(o, e, embed_first)
    ot = x[:, de:] if embed_first else x[:, :dp_]
    ee = x[:, :de] if embed_first else x[:, dp_:]
    np.testing.assert_array_equal(ee, e)
    nrm = np.linalg.norm(ot, axis=1)
    for t in range(T):
        if t == 4:
            assert np.abs(ot[t]).max() == 0.0
            continue
        assert nrm[t] == pytest.approx(np.linalg.norm(e[t]), rel=1e-13)
        np.testing.assert_allclose(ot[t] / nrm[t], o[t] / np.linalg.norm(o[t]), rtol=1e-12)
    # by hand: o = (3, 4) (norm 5), e = (0, 6) (norm 6): o~ = (3.6, 4.8)
    xh = orc.junction_fwd(np.array([[3.0, 4.0]]), np.array([[0.0, 6.0]]), embed_first)
    want = [0.0, 6.0, 3.6, 4.8] if embed_first else [3.6, 4.8, 0.0, 6.0]
    np.testing.assert_allclose(xh[0], want, rtol=1e-15)
    # finite differences of f(o, e) = sum(c * x)
    c = rng.standard_normal((T, dp_ + de))
    d_o, d_e = orc.junction_bwd(o, e, c, embed_first)
    eps = 1e-6
    for arr, grad in ((o, d_o), (e, d_e)):
        fd = np.zeros_like(arr)
        for idx in np.ndindex(*arr.shape):
            if arr is o and idx[0] == 4:
                continue  # the zero row sits on the kink of ||o||
            vals = []
            for sgn in (1, -1):
                a2 = arr.copy()
                a2[idx] += sgn * eps
                xo = orc.junction_fwd(a2, e, embed_first) if arr is o else \
                    orc.junction_fwd(o, a2, embed_first)
                vals.append((c * xo).sum())
            fd[idx] = (vals[0] - vals[1]) / (2 * eps)
        mask = np.ones(arr.shape[0], bool)
        if arr is o:
            mask[4] = False
        np.testing.assert_allclose(grad[mask], fd[mask], rtol=1e-6, atol=1e-8)


# ---------------------------------------------------------------- speculative decoding verify
def _onehot_rows(idx, d):
    H = np.zeros((len(idx), d))
    H[np.arange(len(idx)), idx] = 1.0
    return H


def test_spec_verify_greedy_by_construction():
    """Greedy: one-hot hidden rows pick head columns, so the verifier's argmax at
    every position is known; the draft agrees on the first two positions only."""
    V, d, gamma = 6, 4, 3
    Wv = np.zeros((V, d))
    Wv[[2, 4, 1, 5], [0, 1, 2, 3]] = 1.0          # hidden unit k -> token (2, 4, 1, 5)[k]
    Wd = Wv.copy()
    Hv = _onehot_rows([0, 1, 2, 3], d)              # verifier argmax per position: 2, 4, 1, 5
    Hd = _onehot_rows([0, 1, 2], d)
    u = np.full((1, gamma + 1, 2), 0.5)
    n, nxt = orc.spec_verify(Hd, Wd, Hv, Wv, [[2, 4, 0]], u, greedy=True)
    assert (n[0], nxt[0]) == (2, 1)
    n, nxt = orc.spec_verify(Hd, Wd, Hv, Wv, [[2, 4, 1]], u, greedy=True)
    assert (n[0], nxt[0]) == (3, 5)                   # all accepted: bonus token


def test_spec_verify_identical_models_accept_everything():
    rng = np.random.default_rng(15)
    B, gamma, V, d = 5, 4, 30, 8
    W = rng.standard_normal((V, d))
    Hv = rng.standard_normal((B * (gamma + 1), d))
    Hd = np.concatenate([Hv.reshape(B, gamma + 1, d)[:, :gamma]]).reshape(B * gamma, d)
    draft = rng.integers(0, 3, (B, gamma))
    u = rng.random((B, gamma + 1, 2))
    # a draft token outside the nucleus has q = 0 and is rejected; keep top_p = 1
    n, _ = orc.spec_verify(Hd, W, Hv, W, draft, u, temperature=0.4, top_p=1.0)
    assert (n == gamma).all()


def test_spec_verify_nucleus_limits_and_hand_resample():
    # top_p -> 0 keeps only the most likely token: sampling returns the argmax
    V, d = 5, 5
    Wv = np.eye(V) * np.array([1.0, 3.0, 2.0, 0.5, 2.9])[:, None]
    Hv = np.ones((1, d))
    u = np.array([[[0.3, 0.99]]])
    n, nxt = orc.spec_verify(np.zeros((0, d)), Wv, Hv, Wv, np.zeros((1, 0), np.int32), u,
                             temperature=1.0, top_p=1e-9)
    assert (n[0], nxt[0]) == (0, 1)
    # V = 2 by hand: q = (0.8, 0.2), p = (0.5, 0.5) at temperature 1, top_p = 1.
    # draft x = 0: accept iff u * 0.8 < 0.5, i.e. u < 0.625; residual max(0, p - q) = (0, 0.3)
    lq, lp = np.log([0.8, 0.2]), np.log([0.5, 0.5])
    Wd2, Wv2 = np.diag(lq), np.diag(lp)
    Hd2, Hv2 = np.ones((1, 2)), np.ones((2, 2))
    for uacc, want_n in ((0.6, 1), (0.65, 0)):
        uu = np.array([[[uacc, 0.1], [0.0, 0.7]]])
        n, nxt = orc.spec_verify(Hd2, Wd2, Hv2, Wv2, [[0]], uu, temperature=1.0, top_p=1.0)
        assert n[0] == want_n
        if want_n == 0:
            assert nxt[0] == 1                          # the residual puts all mass on token 1
        else:
            assert nxt[0] == 1                          # bonus from p = (0.5, 0.5) with u = 0.7


def test_spec_verify_output_follows_the_verifier():
    """The defining property of speculative sampling: with the draft token drawn
    from q, the first emitted token is distributed as p (Monte Carlo)."""
    rng = np.random.default_rng(16)
    V, d, N = 6, 6, 20000
    zq = np.array([1.0, 0.2, -0.5, 0.9, 0.0, -1.0])
    zp = np.array([0.1, 1.1, -0.2, 0.6, 0.4, -0.8])
    Wd, Wv = np.diag(zq), np.diag(zp)
    q = np.exp(zq / 0.4) / np.exp(zq / 0.4).sum()
    p = np.exp(zp / 0.4) / np.exp(zp / 0.4).sum()
    draft = rng.choice(V, size=(N, 1), p=q)
    u = rng.random((N, 2, 2))
    Hd, Hv = np.ones((N, d)), np.ones((2 * N, d))
    n, nxt = orc.spec_verify(Hd, Wd, Hv, Wv, draft, u, temperature=0.4, top_p=1.0)
    first = np.where(n == 1, draft[:, 0], nxt)
    freq = np.bincount(first, minlength=V) / N
    assert np.abs(freq - p).max() < 4.5 * np.sqrt(p * (1 - p) / N).max()


def test_spec_verify_nucleus_hand_worked_top_p_09():
    """A nucleus cut strictly inside (0, 1), worked out by hand (V = 4, top_p = 0.9,
    temperature 1, logits = log-probabilities so softmax returns them exactly).
    The two nuclei keep different masses, so each renormalisation shows.

    draft    q = (0.50, 0.30, 0.15, 0.05): cumulative 0.50, 0.80, 0.95 >= 0.9, so
             tokens {0, 1, 2} are kept and q' = (0.50, 0.30, 0.15, 0) / 0.95.
    verifier p = (0.08, 0.22, 0.30, 0.40): sorted 0.40, 0.30, 0.22 -> 0.92, so
             tokens {3, 2, 1} are kept and p' = (0, 0.22, 0.30, 0.40) / 0.92.
    Drafted x = 1: accept iff u q'(1) < p'(1), i.e. u < (0.22 / 0.92) / (0.30 / 0.95)
    = 0.75725.  Without renormalising the cut would be 0.73333; renormalising
    only p gives 0.79710, only q 0.69667.
    Residual max(0, p' - q') = (0, 0, 0.30/0.92 - 0.15/0.95, 0.40/0.92) =
    (0, 0, 0.16819, 0.43478): token 2 iff u < 0.16819 / 0.60297 = 0.27894
    (0.27273 without renormalising).
    Bonus position, verifier p = (0.60, 0.25, 0.10, 0.05): kept {0, 1, 2},
    CDF 0.63158, 0.89474, 1: u = 0.88 gives token 1 (keeping token 3 would give 2)."""
    q = np.array([0.50, 0.30, 0.15, 0.05])
    p0 = np.array([0.08, 0.22, 0.30, 0.40])
    p1 = np.array([0.60, 0.25, 0.10, 0.05])
    Wd = np.log(q)[:, None]
    Wv = np.stack([np.log(p0), np.log(p1)], axis=1)
    Hd, Hv = np.ones((1, 1)), np.eye(2)

    def run(x, u_acc, u_res, u_bonus=0.5):
        u = np.array([[[u_acc, u_res], [0.0, u_bonus]]])
        n, nxt = orc.spec_verify(Hd, Wd, Hv, Wv, [[x]], u, temperature=1.0, top_p=0.9)
        return int(n[0]), int(nxt[0])

    # acceptance threshold 0.75725, between the unrenormalised 0.73333 and the
    # p-only 0.79710
    assert run(1, 0.745, 0.1, u_bonus=0.88) == (1, 1)   # accepted, bonus token 1
    assert run(1, 0.77, 0.1) == (0, 2)                  # rejected, residual token 2
    # the residual's cut between tokens 2 and 3 at 0.27894
    assert run(1, 0.99, 0.276) == (0, 2)
    assert run(1, 0.99, 0.282) == (0, 3)
    # token 0 lies outside the verifier's nucleus (p' = 0): always rejected
    assert run(0, 0.0, 0.276) == (0, 2)
    # token 3 lies outside the draft's nucleus (q' = 0): rejected as well
    assert run(3, 0.0, 0.5) == (0, 3)
    # bonus CDF 0.63158, 0.89474: the nucleus drops token 3 before sampling
    assert run(1, 0.5, 0.0, u_bonus=0.62) == (1, 0)
    assert run(1, 0.5, 0.0, u_bonus=0.90) == (1, 2)


def test_spec_verify_temperature_applies_before_the_nucleus():
    """At temperature 0.5 the draft's q = (0.50, 0.30, 0.15, 0.05) sharpens to
    q^2 / sum q^2 = (0.6849, 0.2466, 0.0616, 0.0068), whose cumulative passes 0.9
    at the second token: only {0, 1} are kept, so a drafted token 2 (inside the
    untempered nucleus) is now rejected."""
    q = np.array([0.50, 0.30, 0.15, 0.05])
    p = np.array([0.25, 0.25, 0.25, 0.25])
    Wd, Wv = np.log(q)[:, None], np.stack([np.log(p), np.log(p)], axis=1)
    Hd, Hv = np.ones((1, 1)), np.eye(2)
    u = np.array([[[0.0, 0.5], [0.0, 0.5]]])
    n, _ = orc.spec_verify(Hd, Wd, Hv, Wv, [[2]], u, temperature=0.5, top_p=0.9)
    assert n[0] == 0
    n, _ = orc.spec_verify(Hd, Wd, Hv, Wv, [[2]], u, temperature=1.0, top_p=0.9)
    assert n[0] == 1
