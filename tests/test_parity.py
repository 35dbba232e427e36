"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on the
same seeded inputs.  Small cases span several token and vocabulary tiles with
ragged tails and are compared element by element; the full-size workloads are
compared on sampled tokens plus properties that hold at any size."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import synth

from helpers import check_forward, check_grads, exact_logits, rel_close, run_gpu

pytestmark = pytest.mark.gpu


def full_parity(wl, H, W, y, grad_scale=1.0, vocab_group=0, argmax=True):
    op, status = run_gpu(wl, H, W, y, grad_scale=grad_scale, vocab_group=vocab_group)
    assert status == 0, B.mls_strerror(status)
    Ho, Wo = synth.as_oracle_arrays(H), synth.as_oracle_arrays(W)
    yo = y.cpu().numpy().astype(np.int32)
    kw = dict(teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha, w=wl.weights)
    ref = oracle.forward(Ho, Wo, yo, **kw)
    check_forward(op, ref, logits=exact_logits(H, W) if argmax else None)
    ok, e = rel_close(op.loss.item(), ref["loss"])
    assert ok, f"loss rel err {e}"
    dH, dW = oracle.backward(Ho, Wo, yo, grad_scale=grad_scale, **kw)
    check_grads(op, dH=dH, dW=dW)
    return op


def test_tiny_workload_fp32():
    wl = synth.WORKLOADS["tiny"]
    H, W, y = synth.make_inputs(wl, seed=0)
    full_parity(wl, H, W, y)


def test_small_ragged_bf16_teacher_not_last():
    wl = synth.Workload("ragged", T=200, d=(64, 128, 192), V=1000, tau=0.7, alpha=0.4,
                        w_sigma=0.05, teacher=1, weights=(0.5, 1.0, 2.0))
    H, W, y = synth.make_inputs(wl, seed=3)
    y[[0, 17, 199]] = -1
    full_parity(wl, H, W, y, grad_scale=1.7)


@pytest.mark.parametrize("name,T", [("suite3", 136), ("suite3_big", 136), ("suite4", 24),
                                    ("stress", 24), ("suite3_paper", 136)])
def test_reduced_tokens_full_vocab(name, T):
    """Each benchmark workload at its full V, widths, tau and value
    distribution, with fewer tokens (ragged last token tile)."""
    wl = synth.reduced(synth.WORKLOADS[name], T)
    H, W, y = synth.make_inputs(wl, seed=11)
    full_parity(wl, H, W, y)


@pytest.mark.parametrize("vocab_group", [256, 768])
def test_vocab_groups_match(vocab_group):
    wl = synth.Workload("groups", T=150, d=(64, 128), V=1800, tau=1.5, alpha=0.5, w_sigma=0.05)
    H, W, y = synth.make_inputs(wl, seed=5)
    full_parity(wl, H, W, y, vocab_group=vocab_group)


@pytest.mark.parametrize("T,V,vocab_group", [(520, 35000, 0), (300, 66000, 33024)])
def test_wide_dh_units(T, V, vocab_group):
    """A vocabulary group of at least 512 k-blocks that writes dH, with an even
    number of column tiles in every sub-model, runs dH in wide units (two
    column tiles sharing each A tile of G): widths of 2 and 4 column tiles (the
    last ragged) over 3 or 2 token tiles (the last ragged).  In the second
    case there are two groups of 33024 and 32976 columns: the first runs wide,
    the second plain, accumulating into dH."""
    wl = synth.Workload("wide", T=T, d=(320, 1008), V=V, tau=1.3, alpha=0.5, w_sigma=0.05)
    H, W, y = synth.make_inputs(wl, seed=13)
    full_parity(wl, H, W, y, vocab_group=vocab_group, argmax=False)


def test_token_bands_full_parity():
    """The suite's widths over 24 token tiles (the last ragged) and a small
    vocabulary: the head kernels' pairs run in bands of token tiles (2 bands of
    12 in the forward, 3 of 8 in the backward), every token and every
    gradient entry compared with the oracle."""
    wl = synth.Workload("bands", T=6000, d=(1024, 2048, 3072), V=700, tau=1.0, alpha=0.5,
                        w_sigma=0.02)
    H, W, y = synth.make_inputs(wl, seed=15)
    y[[0, 3100, 5999]] = -1
    full_parity(wl, H, W, y, argmax=False)


@pytest.mark.parametrize("V", [700, 1800, 9000])
def test_merge_partial_counts(V):
    """1000 tokens (4 token tiles, the last ragged) against 3, 8 and 36
    vocabulary tiles: about 3, 8 and 19 partial states per token, so the merge
    runs with one, two and eight warps per group of 8 tokens."""
    wl = synth.Workload("merge", T=1000, d=(64, 128), V=V, tau=0.9, alpha=0.5, w_sigma=0.05)
    H, W, y = synth.make_inputs(wl, seed=14)
    y[[5, 999]] = -1
    full_parity(wl, H, W, y)


def test_edge_shapes():
    # V below one vocabulary tile, a single token, a single sub-model
    for wl in (synth.Workload("v100", T=130, d=(32, 64), V=100, w_sigma=0.1),
               synth.Workload("t1", T=1, d=(64, 64), V=700, w_sigma=0.1, tau=2.0),
               synth.Workload("m1", T=77, d=(96,), V=513, w_sigma=0.1)):
        H, W, y = synth.make_inputs(wl, seed=2)
        full_parity(wl, H, W, y)


def test_alpha_zero_and_one():
    for alpha in (0.0, 1.0):
        wl = synth.Workload("alpha", T=64, d=(64, 128), V=600, alpha=alpha, tau=0.8, w_sigma=0.05)
        H, W, y = synth.make_inputs(wl, seed=4)
        full_parity(wl, H, W, y)


@pytest.mark.parametrize("alpha,tau", [(0.3, 1.0), (0.7, 1.0), (0.5, 0.1), (0.5, 10.0)])
def test_paper_alphas_and_extreme_temperatures(alpha, tau):
    """The paper's alpha sweep values besides 0, 0.5 and 1, and temperatures far
    from 1 (a nearly one-hot q at 0.1, a nearly uniform one at 10), with the
    normalised per-size weights of App. G (1/3 each) and a 3-level suite."""
    wl = synth.Workload("alpha_tau", T=70, d=(64, 128, 192), V=900, alpha=alpha, tau=tau,
                        w_sigma=0.1, weights=(1 / 3, 1 / 3, 1 / 3))
    H, W, y = synth.make_inputs(wl, seed=6)
    full_parity(wl, H, W, y)


def test_all_targets_ignored():
    wl = synth.Workload("ign", T=96, d=(64, 64), V=300, w_sigma=0.05)
    H, W, y = synth.make_inputs(wl, seed=6)
    y[:] = -1
    op, status = run_gpu(wl, H, W, y)
    assert status == 0
    assert op.loss.item() == 0.0
    assert float(op.tok_loss.abs().max()) == 0.0
    assert all(float(g.abs().max()) == 0.0 for g in op.dH + op.dW)


def test_bad_target_sets_status_and_is_ignored():
    wl = synth.Workload("bad", T=64, d=(64, 64), V=300, w_sigma=0.05)
    H, W, y = synth.make_inputs(wl, seed=8)
    y2 = y.clone()
    y2[3] = wl.V + 5
    op, status = run_gpu(wl, H, W, y2)
    assert status & B.MLS_STATUS_BAD_TARGET
    y3 = y.clone()
    y3[3] = -1
    op2, status2 = run_gpu(wl, H, W, y3)
    assert status2 == 0
    assert op.loss.item() == op2.loss.item()


def test_integer_exact_gathers_and_argmax():
    """One-hot hidden rows and small-integer heads: every logit is an exact
    integer in bf16 x bf16 -> fp32, so the target logit (through CE = lse - z_y)
    and the argmax must match bit for bit."""
    T, V, dm = 160, 700, 64
    g = torch.Generator().manual_seed(9)
    H = torch.zeros(T, dm)
    H[torch.arange(T), torch.randint(0, dm, (T,), generator=g)] = 1.0
    Wt = torch.randint(-6, 7, (V, dm), generator=g).float()
    Ws = torch.randint(-6, 7, (V, dm), generator=g).float()
    Hs = [H.to(torch.bfloat16), H.to(torch.bfloat16)]
    Wl = [Ws.to(torch.bfloat16), Wt.to(torch.bfloat16)]
    y = torch.randint(0, V, (T,), generator=g).to(torch.int32)
    wl = synth.Workload("intexact", T=T, d=(dm, dm), V=V)
    op, status = run_gpu(wl, Hs, Wl, y, backward=False)
    assert status == 0
    z = [(H.double() @ w.double().T) for w in (Ws, Wt)]
    for m in range(2):
        want = torch.argmax(z[m], -1).numpy()  # first maximum
        assert (op.argmax[m].cpu().numpy() == want).all()
        zy = z[m][torch.arange(T), y.long()].numpy()
        lse = op.stats[0, m].cpu().double().numpy()
        ce = op.tok_diag[0, m].cpu().double().numpy()
        # CE = lse - z_y exactly up to the fp32 subtraction
        assert np.abs((lse - ce) - zy).max() <= 1e-5 * np.abs(lse).max()


def test_deterministic():
    wl = synth.Workload("det", T=300, d=(64, 128), V=900, tau=0.9, w_sigma=0.05)
    H, W, y = synth.make_inputs(wl, seed=12)
    a, _ = run_gpu(wl, H, W, y)
    r1 = [a.loss.clone(), a.tok_loss.clone()] + [t.clone() for t in a.dH + a.dW]
    b, _ = run_gpu(wl, H, W, y)
    r2 = [b.loss, b.tok_loss] + b.dH + b.dW
    for x, z in zip(r1, r2):
        assert torch.equal(x, z)


def test_workspace_and_alignment_errors():
    wl = synth.Workload("err", T=64, d=(64, 64), V=300)
    H, W, y = synth.make_inputs(wl, seed=1)
    dev = torch.device("cuda")
    Hd = [h.to(dev) for h in H]
    Wd = [w.to(dev) for w in W]
    op = B.HeadLoss(wl.d, wl.T, wl.V, device=dev)
    small = torch.empty(16, dtype=torch.uint8, device=dev)
    with pytest.raises(B.MLSError) as e:
        B.mls_head_loss_fwd(op.prob, Hd, Wd, y.to(dev), op.loss, op.tok_loss, None, None,
                            op.stats, small)
    assert e.value.code == B.MLS_ERR_WORKSPACE
    raw = torch.empty(64 * 64 * 2 + 2, dtype=torch.uint8, device=dev)
    mis = raw[2:].view(torch.bfloat16).view(64, 64)
    with pytest.raises(B.MLSError) as e:
        B.mls_head_loss_fwd(op.prob, [mis, Hd[1]], Wd, y.to(dev), op.loss, op.tok_loss, None, None,
                            op.stats, op.ws)
    assert e.value.code == B.MLS_ERR_ALIGN


# ------------------------------------------------------------------ full-size workloads
def _full_size(name, nsample, seed=21):
    wl = synth.WORKLOADS[name]
    H, W, y = synth.make_inputs(wl, seed=seed, device="cuda")
    op, status = run_gpu(wl, H, W, y)
    assert status == 0, B.mls_strerror(status)
    rng = np.random.default_rng(seed)
    rows = np.unique(np.concatenate([rng.integers(0, wl.T, nsample - 2), [0, wl.T - 1]]))
    Ho = synth.as_oracle_arrays([h[torch.as_tensor(rows, device=h.device)] for h in H])
    Wo = synth.as_oracle_arrays(W)
    yc = y.cpu().numpy().astype(np.int32)
    kw = dict(teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha, w=wl.weights)
    # rows mode needs N of the whole problem: pass the sampled rows as a
    # problem of their own and rescale dH by N_sample / N_full.
    ref = oracle.rows(Ho, Wo, yc[rows], np.arange(len(rows)), **kw)
    n_full = int((yc >= 0).sum())
    scale = ref["n_valid"] / n_full
    check_forward(op, ref, rows=rows,
                  logits=exact_logits([h[torch.as_tensor(rows, device=h.device)] for h in H], W))
    check_grads(op, dH_rows=(rows, [x * scale for x in ref["dH"]]))
    # every row of dL/dz sums to zero, so do the columns of dW
    for m in range(wl.M):
        dw = op.dW[m].double()
        assert bool((dw.sum(0).abs() <= 1e-2 * dw.abs().sum(0) + 1e-30).all()), m
    # the scalar is the weighted mean of the per-token losses
    w = torch.tensor(wl.weights or [1.0] * wl.M, dtype=torch.float64, device=op.tok_loss.device)
    valid = (y >= 0).double()
    want = float(((op.tok_loss.double() * w[:, None]).sum(0) * valid).sum() / valid.sum())
    assert abs(op.loss.item() - want) <= 1e-5 * abs(want)
    return op


@pytest.mark.parametrize("name", ["suite3", "suite3_big", "suite4", "stress", "suite3_paper"])
def test_full_size_sampled(name):
    """64 sampled tokens (the first and last among them) of each full-size
    workload: per-token losses, statistics, argmax and their dH rows."""
    _full_size(name, nsample=64)


def test_empty_token_batch():
    """T = 0 (null hidden states are allowed then): the loss is 0, dW is
    overwritten with zeros, the pairwise means are 0 and the junction does
    nothing; nothing raises a status bit."""
    dev = torch.device("cuda")
    B.mls_get_status()  # clear bits an earlier test may have left
    d, V = (64, 128), 300
    op = B.HeadLoss(d, 0, V, device=dev)
    H = [torch.empty(0, dm, dtype=torch.bfloat16, device=dev) for dm in d]
    W = [torch.randn(V, dm, device=dev).to(torch.bfloat16) for dm in d]
    y = torch.empty(0, dtype=torch.int32, device=dev)
    op.loss.fill_(float("nan"))
    for t in op.dW:
        t.fill_(float("nan"))
    op.forward(H, W, y)
    op.backward(H, W, y)
    _, _, ps = op.pairwise(H, W)
    o = torch.empty(0, 64, dtype=torch.bfloat16, device=dev)
    e = torch.empty(0, 64, dtype=torch.bfloat16, device=dev)
    x = torch.empty(0, 128, dtype=torch.bfloat16, device=dev)
    B.mls_junction_fwd(o, e, x)
    B.mls_junction_bwd(o, e, x, torch.empty_like(o), torch.empty_like(e))
    torch.cuda.synchronize()
    assert op.loss.item() == 0.0
    assert all(bool((t == 0).all()) for t in op.dW)
    assert bool((ps == 0).all())
    assert B.mls_get_status() == 0
