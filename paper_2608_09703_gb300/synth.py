"""Seeded synthetic workloads for the Matryoshka-suite output stage.

This module only draws random inputs: it holds none of the loss arithmetic,
so both the CUDA path's tests and the CPU oracle can take their inputs from
it.  The paper trains on FineWeb-Edu with packed sequences of 2048 tokens
(Sec. 3.1, "Training Setup"); that corpus and the trained checkpoints are not
available, so seeded synthetic hidden states, heads and targets with the
shapes of the paper's suites stand in for them:

  H_m ~ N(0, 1)            hidden states at the exit of sub-model m, [T, d_m]
  W_m ~ N(0, sigma^2)      LM head of sub-model m (Sec. 2), [V, d_m]
  y   ~ Uniform[0, V)      next-token targets, or Zipf(s) by token id

Seeds: H_m from ``seed + 0``, W_m from ``seed + 1``, targets from ``seed + 2``
(one generator per role, models drawn in index order).
"""
from __future__ import annotations

import dataclasses
from typing import Optional, Sequence

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    T: int
    d: tuple
    V: int
    dtype: str = "bf16"          # storage type of H and W: "bf16" or "fp32"
    tau: float = 1.0
    alpha: float = 0.5
    w_sigma: float = 0.02
    teacher_scale: float = 1.0   # multiplies the teacher head (peaked teacher logits)
    targets: str = "uniform"     # "uniform" or "zipf"
    zipf_s: float = 1.1
    teacher: Optional[int] = None  # None = the largest (last) sub-model
    weights: Optional[tuple] = None

    @property
    def M(self) -> int:
        return len(self.d)

    @property
    def teacher_index(self) -> int:
        return self.M - 1 if self.teacher is None else self.teacher

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    def flops_fwd_bwd(self) -> int:
        """Algorithmic FLOPs of one forward+backward: forward logits, the
        backward's logit recompute, dH and dW, each 2*T*V*sum(d)."""
        return 8 * self.T * self.V * sum(self.d)


# The paper's 3B suite is 500M/1.5B/3B (Table 1); these workloads are shaped
# like it and like larger stacks, with the sizes the benchmark names.
WORKLOADS = {
    "tiny": Workload("tiny", T=256, d=(128, 256), V=1024, dtype="fp32"),
    "suite3": Workload("suite3", T=8192, d=(1024, 2048, 3072), V=50304),
    "suite3_big": Workload("suite3_big", T=65536, d=(1024, 2048, 3072), V=50304, tau=2.0),
    "suite4": Workload("suite4", T=16384, d=(2048, 4096, 6144, 8192), V=128256, w_sigma=0.01),
    "stress": Workload("stress", T=32768, d=(1024, 2048, 4096), V=256000, tau=0.5,
                       teacher_scale=8.0, targets="zipf"),
    # The paper's own 3B Matryoshka suite (Sec. 3.1, Table 1): widths
    # 1024 / 2304 / 4352 and the 49,152-token vocabulary, at the same four
    # packed 2048-token sequences as suite3.
    "suite3_paper": Workload("suite3_paper", T=8192, d=(1024, 2304, 4352), V=49152),
}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def make_inputs(wl: Workload, seed: int = 0, device="cpu"):
    """Draw (H list, W list, targets) for a workload.

    H[m]: [T, d_m], W[m]: [V, d_m] in the workload's storage dtype, row-major;
    targets: int32 [T].  On a CUDA device the draws use CUDA generators (fast for
    the multi-GB workloads); the CPU draws are what the small parity cases use.
    """
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    gH, gW, gY = _gen(seed, device), _gen(seed + 1, device), _gen(seed + 2, device)
    H, W = [], []
    for m, dm in enumerate(wl.d):
        H.append(torch.randn(wl.T, dm, generator=gH, device=device, dtype=torch.float32).to(dt))
    for m, dm in enumerate(wl.d):
        sigma = wl.w_sigma * (wl.teacher_scale if m == wl.teacher_index else 1.0)
        w = torch.randn(wl.V, dm, generator=gW, device=device, dtype=torch.float32)
        W.append((w * sigma).to(dt))
    y = make_targets(wl, gY, device)
    return H, W, y


def make_targets(wl: Workload, gen: torch.Generator, device="cpu") -> torch.Tensor:
    if wl.targets == "uniform":
        return torch.randint(0, wl.V, (wl.T,), generator=gen, device=device, dtype=torch.int64).to(torch.int32)
    if wl.targets == "zipf":
        # P(v) proportional to (v + 1)^-s, rank = token id
        ranks = torch.arange(1, wl.V + 1, device=device, dtype=torch.float64)
        p = ranks.pow(-wl.zipf_s)
        return torch.multinomial(p, wl.T, replacement=True, generator=gen).to(torch.int32)
    raise ValueError(wl.targets)


def reduced(wl: Workload, T: int) -> Workload:
    """The same workload (V, widths, tau, distributions) with fewer tokens."""
    return wl.with_(name=f"{wl.name}_T{T}", T=T)


def as_oracle_arrays(ts: Sequence[torch.Tensor]):
    """Tensors -> numpy arrays in the oracle's storage convention (bf16 bits as
    uint16, fp32 as float32), copied to host memory."""
    import numpy as np

    out = []
    for t in ts:
        t = t.detach().contiguous().cpu()
        if t.dtype == torch.bfloat16:
            out.append(t.view(torch.int16).numpy().view(np.uint16))
        elif t.dtype == torch.float32:
            out.append(t.numpy())
        else:
            raise TypeError(t.dtype)
    return out


# Speculative-decoding verify inputs (Sec. 3.2.3: a 500M draft and a 3B
# verifier of one suite, batch up to 102, draft length 6, vocabulary of the
# suite).  Nested like the suite: the verifier's hidden state at a drafted
# position extends the draft's (first d_draft channels shared) and its head
# extends the draft's head, so the verifier's logits are the draft's plus an
# independent part whose spread is `extra` times the draft's.
@dataclasses.dataclass(frozen=True)
class SpecWorkload:
    name: str
    B: int
    gamma: int
    V: int
    d_draft: int
    d_verify: int
    dtype: str = "bf16"
    temperature: float = 0.4
    top_p: float = 0.9
    z_std: float = 2.5       # spread of the draft's logits
    extra: float = 0.2       # spread of the verifier's extra logit part / z_std


SPEC_WORKLOADS = {
    "spec_suite3": SpecWorkload("spec_suite3", B=102, gamma=6, V=50304, d_draft=1024, d_verify=3072),
}


def make_spec_inputs(wl: SpecWorkload, seed: int = 0, device="cpu"):
    """Draw (H_draft [B*gamma, d_d], W_draft [V, d_d], H_verify [B*(gamma+1), d_v],
    W_verify [V, d_v]) in the workload's storage dtype.  fp32 workloads hold
    bf16-representable values.  Seeds: hidden states seed + 0, heads seed + 1."""
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    gH, gW = _gen(seed, device), _gen(seed + 1, device)
    dd, dv, G1 = wl.d_draft, wl.d_verify, wl.gamma + 1
    f32 = dict(device=device, dtype=torch.float32)
    hv = torch.randn(wl.B, G1, dv, generator=gH, **f32)
    wd = torch.randn(wl.V, dd, generator=gW, **f32) * (wl.z_std / dd ** 0.5)
    de = dv - dd
    we = torch.randn(wl.V, de, generator=gW, **f32) * (wl.extra * wl.z_std / max(de, 1) ** 0.5)
    Wv = torch.cat([wd, we], 1)
    Hd = hv[:, :wl.gamma, :dd].reshape(wl.B * wl.gamma, dd)
    Hv = hv.reshape(wl.B * G1, dv)

    def st(t):
        return t.to(torch.bfloat16).to(dt).contiguous()

    return st(Hd), st(wd), st(Hv), st(Wv)


def make_uniforms(B: int, gamma: int, seed: int = 0, device="cpu") -> torch.Tensor:
    """Acceptance and sampling draws u [B, gamma+1, 2] in [0, 1), fp32 (seed + 2)."""
    return torch.rand(B, gamma + 1, 2, generator=_gen(seed + 2, device), device=device,
                      dtype=torch.float32)
