"""GPU parity of the evaluation metrics between sub-models (mls_head_pairwise)
against the fp64 oracle: per-token KL(p_i || p_j), their means, argmax and top-1
agreement (Sec. 3.2.2)."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import synth

from helpers import exact_logits

pytestmark = pytest.mark.gpu

KL_TOL = 1e-3  # |diff| <= KL_TOL * max(1, |KL|)


def run_pairwise(wl, H, W, y):
    dev = torch.device("cuda")
    Hd = [h.to(dev).contiguous() for h in H]
    Wd = [w.to(dev).contiguous() for w in W]
    yd = None if y is None else y.to(dev).to(torch.int32)
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    op = B.HeadLoss(wl.d, wl.T, wl.V, dtype=dt, device=dev)
    kl, am, stats = op.pairwise(Hd, Wd, yd)
    torch.cuda.synchronize()
    assert B.mls_get_status() == 0
    return kl.cpu().double().numpy(), am.cpu().numpy(), stats.cpu().double().numpy()


def check(wl, H, W, y, rows=None):
    kl, am, stats = run_pairwise(wl, H, W, y)
    sub = (lambda h: h[torch.as_tensor(rows, device=h.device)]) if rows is not None else (lambda h: h)
    Hs = [sub(h) for h in H]
    ref = oracle.pairwise(synth.as_oracle_arrays(Hs), synth.as_oracle_arrays(W))
    klg = kl if rows is None else kl[:, :, rows]
    err = np.abs(klg - ref["kl"]) / np.maximum(1.0, np.abs(ref["kl"]))
    assert err.max() <= KL_TOL, f"KL err {err.max()}"
    # argmax against the exact logits, where the top-2 gap decides it
    z = exact_logits(Hs, W)
    amg = am if rows is None else am[:, rows]
    for m in range(wl.M):
        zz = z[m].numpy()
        top = np.sort(zz, -1)[:, -2:]
        decided = (top[:, 1] - top[:, 0]) > 1e-4 * np.maximum(1.0, np.abs(top[:, 1]))
        assert (amg[m][decided] == np.argmax(zz, -1)[decided]).all()
    # the means are the means of the per-token values over the counted tokens
    valid = np.ones(wl.T, bool) if y is None else ((y.cpu().numpy() >= 0) & (y.cpu().numpy() < wl.V))
    if valid.any():
        np.testing.assert_allclose(stats[0], kl[:, :, valid].mean(-1), rtol=1e-4, atol=1e-6)
        agree = (am[:, None, :] == am[None, :, :])[:, :, valid].mean(-1)
        np.testing.assert_allclose(stats[1], agree, rtol=0, atol=1e-6)
    return kl, am, stats


def test_pairwise_small_ragged_bf16():
    wl = synth.Workload("pw", T=200, d=(64, 128, 192), V=1000, w_sigma=0.08)
    H, W, y = synth.make_inputs(wl, seed=31)
    y[[2, 50]] = -1
    check(wl, H, W, y)


def test_pairwise_tiny_fp32_no_targets():
    wl = synth.WORKLOADS["tiny"]
    H, W, _ = synth.make_inputs(wl, seed=32)
    check(wl, H, W, None)


def test_pairwise_four_models_with_a_duplicate():
    wl = synth.Workload("pw4", T=130, d=(64, 128, 64, 192), V=700, w_sigma=0.1)
    H, W, y = synth.make_inputs(wl, seed=33)
    H[2], W[2] = H[0].clone(), W[0].clone()  # sub-model 2 duplicates sub-model 0
    kl, am, stats = check(wl, H, W, y)
    assert np.abs(kl[0, 2]).max() <= 1e-5 and np.abs(kl[2, 0]).max() <= 1e-5
    assert (am[0] == am[2]).all() and stats[1][0, 2] == 1.0


def test_pairwise_suite3_reduced_tokens():
    wl = synth.reduced(synth.WORKLOADS["suite3"], 136)
    H, W, y = synth.make_inputs(wl, seed=34)
    check(wl, H, W, y)


def test_pairwise_suite3_full_size_sampled():
    wl = synth.WORKLOADS["suite3"]
    H, W, y = synth.make_inputs(wl, seed=35, device="cuda")
    rng = np.random.default_rng(35)
    rows = np.unique(np.concatenate([rng.integers(0, wl.T, 8), [0, wl.T - 1]]))
    check(wl, H, W, y, rows=rows)


@pytest.mark.parametrize("name", ["suite4", "stress"])
def test_pairwise_large_vocab_sampled(name):
    """The 4-level suite (M = 4, V = 128256: four resident 128-column tiles)
    and the stress shape (M = 3, V = 256000, teacher head x8: the slot
    schedule over 1000 vocabulary tiles) at full size; ten sampled tokens (the
    first and last among them) against the oracle, their argmax against fp64
    logits computed on the device."""
    wl = synth.WORKLOADS[name]
    H, W, y = synth.make_inputs(wl, seed=44, device="cuda")
    kl, am, stats = run_pairwise(wl, H, W, y)
    rng = np.random.default_rng(44)
    rows = np.unique(np.concatenate([rng.integers(0, wl.T, 8), [0, wl.T - 1]]))
    ri = torch.as_tensor(rows, device=H[0].device)
    ref = oracle.pairwise(synth.as_oracle_arrays([h[ri] for h in H]), synth.as_oracle_arrays(W))
    err = np.abs(kl[:, :, rows] - ref["kl"]) / np.maximum(1.0, np.abs(ref["kl"]))
    assert err.max() <= KL_TOL, f"KL err {err.max()}"
    for m in range(wl.M):
        zz = (H[m][ri].double() @ W[m].double().T).cpu().numpy()
        top = np.sort(zz, -1)[:, -2:]
        decided = (top[:, 1] - top[:, 0]) > 1e-4 * np.maximum(1.0, np.abs(top[:, 1]))
        assert (am[m][rows][decided] == np.argmax(zz, -1)[decided]).all()
    assert np.isfinite(stats).all()


def test_pairwise_single_model():
    """M = 1: no pairs; the argmax and the (zero) KL matrix still come out."""
    wl = synth.Workload("pw1", T=300, d=(96,), V=777, w_sigma=0.1)
    H, W, y = synth.make_inputs(wl, seed=36)
    kl, _, stats = check(wl, H, W, y)
    assert np.abs(kl).max() == 0.0 and stats[1][0, 0] == 1.0


@pytest.mark.parametrize("M", [2, 3, 4])
def test_pairwise_many_tiles_per_pair(M):
    """16 token tiles and a ragged vocabulary of 4999 columns: each CTA pair
    walks several vocabulary tiles (256, 256 or 128 columns wide for M = 2, 3,
    4), so the epilogue's early release of the widest sub-model's columns, the
    two alternating TMEM slots at M = 3 and the accumulator barriers go through
    several phases."""
    wl = synth.Workload("pwm", T=4096, d=(64, 192, 128, 320)[:M], V=4999, w_sigma=0.08)
    H, W, y = synth.make_inputs(wl, seed=37 + M)
    check(wl, H, W, y)


def test_pairwise_three_models_partial_last_half():
    """M = 3 with V = 4900: the last 256-column tile holds 36 columns, so the
    first column half of its threads is cut inside a 16-column chunk and the
    second half has no valid column at all; three token tiles, the last ragged,
    and a width tie (two sub-models of 128)."""
    wl = synth.Workload("pwh", T=520, d=(128, 64, 128), V=4900, w_sigma=0.08)
    H, W, y = synth.make_inputs(wl, seed=43)
    y[[0, 519]] = -1
    check(wl, H, W, y)


def test_pairwise_fp32_three_models():
    """fp32 inputs (tf32 products) at M = 3: 256-column tiles read with
    32-element k-blocks, over a ragged vocabulary and two token tiles.  The
    heads have the fp32 workload's scale (sigma 0.02): tf32 rounds each
    product to ~2^-11, which the KL tolerance covers at logits of that size
    (with sigma 0.1 the largest KL error reached 1.6e-3)."""
    wl = synth.Workload("pwf", T=300, d=(32, 96, 64), V=1234, dtype="fp32", w_sigma=0.02)
    H, W, y = synth.make_inputs(wl, seed=41)
    check(wl, H, W, y)


def test_pairwise_token_bands():
    """The suite's widths over 24 token tiles: the evaluation kernel's pairs run
    in 2 bands of 12 token tiles; every token compared with the oracle."""
    wl = synth.Workload("pwb", T=6000, d=(1024, 2048, 3072), V=700, w_sigma=0.02)
    H, W, y = synth.make_inputs(wl, seed=42)
    check(wl, H, W, y)
