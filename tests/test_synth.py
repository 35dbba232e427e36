"""The seeded synthetic inputs follow the stated recipe (CPU): shapes, storage
types, value distributions, target structure and seeding of the head-loss
workloads, and the nested draft / verifier structure of the verify-step
inputs.  The benchmark workloads themselves are too large for the CPU, so
small workloads with the same parameters are drawn."""
import numpy as np
import pytest
import torch

from paper_2608_09703_gb300 import synth


def test_benchmark_workload_shapes():
    W = synth.WORKLOADS
    assert (W["suite3"].T, W["suite3"].d, W["suite3"].V) == (8192, (1024, 2048, 3072), 50304)
    assert (W["suite3_big"].T, W["suite3_big"].tau) == (65536, 2.0)
    assert (W["suite4"].d, W["suite4"].V, W["suite4"].w_sigma) == ((2048, 4096, 6144, 8192), 128256, 0.01)
    s = W["stress"]
    assert (s.T, s.V, s.tau, s.teacher_scale, s.targets) == (32768, 256000, 0.5, 8.0, "zipf")
    assert (W["suite3_paper"].d, W["suite3_paper"].V) == ((1024, 2304, 4352), 49152)
    assert W["tiny"].dtype == "fp32"
    for wl in W.values():
        assert wl.teacher_index == len(wl.d) - 1 and wl.alpha == 0.5
        assert all(dm % 16 == 0 for dm in wl.d)
    sp = synth.SPEC_WORKLOADS["spec_suite3"]
    assert (sp.B, sp.gamma, sp.V, sp.d_draft, sp.d_verify) == (102, 6, 50304, 1024, 3072)
    assert (sp.temperature, sp.top_p) == (0.4, 0.9)


def test_head_inputs_follow_the_recipe():
    wl = synth.Workload("r", T=4096, d=(64, 128), V=3000, w_sigma=0.02)
    H, W, y = synth.make_inputs(wl, seed=5)
    assert [tuple(h.shape) for h in H] == [(4096, 64), (4096, 128)]
    assert [tuple(w.shape) for w in W] == [(3000, 64), (3000, 128)]
    assert all(t.dtype == torch.bfloat16 and t.is_contiguous() for t in H + W)
    assert y.dtype == torch.int32 and y.shape == (4096,)
    h = torch.cat([t.float().flatten() for t in H])
    assert abs(h.mean().item()) < 0.01 and abs(h.std().item() - 1.0) < 0.01
    for w in W:
        assert abs(w.float().std().item() - 0.02) < 0.0005
    # uniform targets over [0, V)
    assert int(y.min()) >= 0 and int(y.max()) < wl.V
    counts = np.bincount(y.numpy(), minlength=wl.V)
    assert counts.max() < 12  # 4096 draws over 3000 tokens: no heavy head


def test_teacher_scale_zipf_targets_and_fp32():
    wl = synth.Workload("z", T=20000, d=(32, 64), V=500, w_sigma=0.02, teacher_scale=8.0,
                        targets="zipf")
    _, W, y = synth.make_inputs(wl, seed=9)
    assert abs(W[0].float().std().item() - 0.02) < 0.001
    assert abs(W[1].float().std().item() - 0.16) < 0.005  # the teacher's head x8
    counts = np.bincount(y.numpy(), minlength=wl.V).astype(float)
    # P(v) proportional to (v + 1)^-1.1: token 0 is 2^1.1 times as likely as token 1
    assert counts[0] / counts[1] == pytest.approx(2 ** 1.1, rel=0.1)
    assert counts[0] > counts[9] > counts[99]
    tiny = synth.reduced(synth.WORKLOADS["tiny"], 16)
    H, W, _ = synth.make_inputs(tiny, seed=1)
    assert all(t.dtype == torch.float32 for t in H + W)


def test_seeding():
    wl = synth.Workload("s", T=64, d=(32,), V=100)
    a = synth.make_inputs(wl, seed=3)
    b = synth.make_inputs(wl, seed=3)
    c = synth.make_inputs(wl, seed=4)
    assert torch.equal(a[0][0], b[0][0]) and torch.equal(a[1][0], b[1][0]) and torch.equal(a[2], b[2])
    assert not torch.equal(a[0][0], c[0][0]) and not torch.equal(a[2], c[2])
    # H, W and targets come from their own streams (seed, seed + 1, seed + 2)
    h = torch.randn(64, 32, generator=torch.Generator().manual_seed(3)).to(torch.bfloat16)
    w = (torch.randn(100, 32, generator=torch.Generator().manual_seed(4)) * 0.02).to(torch.bfloat16)
    t = torch.randint(0, 100, (64,), generator=torch.Generator().manual_seed(5)).to(torch.int32)
    assert torch.equal(h, a[0][0]) and torch.equal(w, a[1][0]) and torch.equal(t, a[2])
    red = synth.reduced(synth.WORKLOADS["suite3"], 40)
    assert (red.T, red.V, red.d, red.tau) == (40, 50304, (1024, 2048, 3072), 1.0)


def test_spec_inputs_are_nested_like_the_suite():
    wl = synth.SpecWorkload("n", B=16, gamma=3, V=4000, d_draft=64, d_verify=192)
    Hd, Wd, Hv, Wv = synth.make_spec_inputs(wl, seed=7)
    assert Hd.shape == (16 * 3, 64) and Hv.shape == (16 * 4, 192)
    assert Wd.shape == (4000, 64) and Wv.shape == (4000, 192)
    # the verifier's hidden state at a drafted position extends the draft's, and
    # its head extends the draft's head
    hv = Hv.view(16, 4, 192)
    assert torch.equal(hv[:, :3, :64].reshape(48, 64), Hd)
    assert torch.equal(Wv[:, :64], Wd)
    # draft logits at std z_std; the verifier's extra part at extra * z_std
    zd = Hd.float() @ Wd.float().T
    zx = hv[:, :3, 64:].reshape(48, 128).float() @ Wv[:, 64:].float().T
    assert zd.std().item() == pytest.approx(wl.z_std, rel=0.05)
    assert zx.std().item() == pytest.approx(wl.extra * wl.z_std, rel=0.05)
    u = synth.make_uniforms(16, 3, seed=7)
    assert u.shape == (16, 4, 2) and float(u.min()) >= 0.0 and float(u.max()) < 1.0
    # fp32 workloads hold bf16-representable values
    wl32 = synth.SpecWorkload("n32", B=4, gamma=2, V=300, d_draft=32, d_verify=64, dtype="fp32")
    for t in synth.make_spec_inputs(wl32, seed=1):
        assert t.dtype == torch.float32 and torch.equal(t, t.to(torch.bfloat16).float())


def test_spec_suite_rows_are_peaked():
    """At T = 0.4 the draft's rows are peaked: from one to about a hundred
    tokens above 2^-8 of the maximum, a median of about twenty (a reduced
    batch of 32 rows at the full vocabulary)."""
    wl = synth.SpecWorkload("p", B=16, gamma=2, V=50304, d_draft=1024, d_verify=1024)
    Hd, Wd, _, _ = synth.make_spec_inputs(wl, seed=3)
    z = (Hd.float() @ Wd.float().T).double() / wl.temperature
    e = torch.exp(z - z.max(1, keepdim=True).values)
    above = (e >= 2.0 ** -8).sum(1).float()
    assert float(above.min()) >= 1 and float(above.max()) <= 150, above.tolist()
    assert 10 <= float(above.median()) <= 40, above.tolist()
