"""Child process of tests/test_checked.py: runs every entry point of the
library that the environment selects (MLS_CHECKED=1: the checked build) on
small ragged cases and saves the outputs and the status words to an .npz."""
import sys

import numpy as np
import torch

from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import synth


def main(path):
    dev = torch.device("cuda")
    out = {}
    # forward + backward (two vocabulary groups), pairwise metrics
    wl = synth.Workload("chk", T=300, d=(64, 128, 192), V=1000, tau=1.5, w_sigma=0.08)
    H, W, y = synth.make_inputs(wl, seed=71)
    y[[3, 77]] = -1
    Hd, Wd = [h.to(dev) for h in H], [w.to(dev) for w in W]
    yd = y.to(dev).to(torch.int32)
    op = B.HeadLoss(wl.d, wl.T, wl.V, teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha,
                    device=dev, vocab_group=512)
    op.forward(Hd, Wd, yd)
    op.backward(Hd, Wd, yd)
    kl, am, ps = op.pairwise(Hd, Wd, yd)
    torch.cuda.synchronize()
    out["status_head"] = np.array(B.mls_get_status())
    for name, t in (("loss", op.loss), ("tok_loss", op.tok_loss), ("tok_diag", op.tok_diag),
                    ("argmax", op.argmax), ("stats", op.stats), ("kl", kl), ("eval_argmax", am),
                    ("pair_stats", ps)):
        out[name] = t.cpu().numpy()
    for m in range(wl.M):
        out[f"dH{m}"] = op.dH[m].cpu().numpy()
        out[f"dW{m}"] = op.dW[m].cpu().numpy()
    # the backward GEMM's wide dH units (one group of 516 k-blocks, even
    # column-tile counts), 8 partial states per token (two merge warps per 8
    # tokens), and the pairwise metrics at M = 2 and M = 4 (their own tile
    # widths)
    for tag, wl2 in (("w", synth.Workload("chkw", T=1100, d=(320, 1008), V=33000, w_sigma=0.05)),
                     ("m4", synth.Workload("chk4", T=2048, d=(64, 128, 64, 192), V=2000, w_sigma=0.1))):
        H2, W2, y2 = synth.make_inputs(wl2, seed=75)
        H2, W2, y2 = [h.to(dev) for h in H2], [w.to(dev) for w in W2], y2.to(dev).to(torch.int32)
        op2 = B.HeadLoss(wl2.d, wl2.T, wl2.V, device=dev)
        op2.forward(H2, W2, y2)
        op2.backward(H2, W2, y2)
        kl2, _, ps2 = op2.pairwise(H2, W2, y2)
        torch.cuda.synchronize()
        out[f"status_{tag}"] = np.array(B.mls_get_status())
        out[f"{tag}_tok_loss"], out[f"{tag}_kl"], out[f"{tag}_ps"] = (
            t.cpu().numpy() for t in (op2.tok_loss, kl2, ps2))
        for m in range(wl2.M):
            out[f"{tag}_dH{m}"] = op2.dH[m].cpu().numpy()
            out[f"{tag}_dW{m}"] = op2.dW[m].cpu().numpy()
    # junction
    g = torch.Generator().manual_seed(72)
    o = torch.randn(130, 64, generator=g).to(torch.bfloat16).to(dev)
    e = torch.randn(130, 128, generator=g).to(torch.bfloat16).to(dev)
    gr = torch.randn(130, 192, generator=g).to(torch.bfloat16).to(dev)
    x, d_o, d_e = torch.empty_like(gr), torch.empty_like(o), torch.empty_like(e)
    B.mls_junction_fwd(o, e, x)
    B.mls_junction_bwd(o, e, gr, d_o, d_e)
    torch.cuda.synchronize()
    out["status_junction"] = np.array(B.mls_get_status())
    out["jx"], out["jdo"], out["jde"] = (t.float().cpu().numpy() for t in (x, d_o, d_e))
    # verify step, nucleus and greedy
    sw = synth.SpecWorkload("chk", B=20, gamma=4, V=1500, d_draft=64, d_verify=128)
    sd, swd, sv, swv = (t.to(dev) for t in synth.make_spec_inputs(sw, 73))
    u = synth.make_uniforms(sw.B, sw.gamma, 73).to(dev)
    draft = torch.randint(0, sw.V, (sw.B, sw.gamma), generator=torch.Generator().manual_seed(74),
                          dtype=torch.int32).to(dev)
    for greedy in (False, True):
        sp = B.SpecVerify(sw.B, sw.gamma, sw.V, sw.d_draft, sw.d_verify, greedy=greedy, device=dev)
        n, nx = sp(sd, swd, sv, swv, draft, u)
        torch.cuda.synchronize()
        out[f"status_spec{int(greedy)}"] = np.array(B.mls_get_status())
        out[f"n{int(greedy)}"], out[f"next{int(greedy)}"] = n.cpu().numpy(), nx.cpu().numpy()
    np.savez(path, **out)


if __name__ == "__main__":
    main(sys.argv[1])
