#!/usr/bin/env python
"""Benchmark of the fused Matryoshka-suite output stage on GB300.

One step = one forward + backward of the whole hot path (LM heads of every
sub-model, cross-entropy, distillation from the teacher, dH and dW) over one
batch of T tokens of the 3-level suite shaped like 500M/1.5B/3B:
T = 8192 (4 x 2048), d = (1024, 2048, 3072), V = 50304, bf16, tau = 1,
alpha = 0.5, synthetic seeded inputs (the paper's FineWeb-Edu batches are
not available).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mls|reference]

Under torchrun each rank runs its own batch on its own GPU (no collective on
the data path: the loss of one batch needs nothing from another), so scaling
is weak and `value` is the tokens of all ranks per second of the slowest rank.
`--impl reference` times the fp64 CPU oracle (the reference definition of the
method) on the host cores, on a bounded sample of the same workload.
Rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tokens/s fused head+CE+KL fwd+bwd (3-level suite) and % of dense BF16 tensor peak"
UNIT = "tokens/s"
WORKLOAD = "suite3"
# FLOPs of each tensor kernel per step, in units of 2*T*V*sum(d) (gemm_bwd runs dW and dH together)
KERNELS = {"head_fwd": 1, "head_bwd": 1, "gemm_dw": 1, "gemm_dh": 1, "gemm_bwd": 2}
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            d = json.load(fh)
        return d, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


def pick_peak(pk: dict, region_s: float, clocks: dict | None):
    """The bf16 peak a kernel timed in this region is measured against.

    MEASURED_PEAKS.json holds cuBLAS as a burst (best of a few calls, at the
    maximum clock) and as a seconds-long loop under the power cap.  A region
    shorter than a second, or one whose median SM clock stayed within 5% of the
    maximum, ran at burst clocks: the burst figure is its peak.  Only a region
    of seconds that settled below that clock is held to the sustained figure.
    Returns (peak TFLOP/s, regime, reason)."""
    burst, sus = float(pk["bf16_tflops"]), float(pk["bf16_tflops_sustained"])
    mhz = (clocks or {}).get("sm_mhz")
    mx = (clocks or {}).get("sm_max_mhz") or pk.get("sm_max_mhz")
    if region_s < 1.0:
        return burst, "burst", f"timed region {region_s:.2f} s (< 1 s)"
    if mhz and mx and mhz >= 0.95 * mx:
        return burst, "burst", f"median SM clock {mhz:.0f} of {mx:.0f} MHz"
    if not mhz:
        return burst, "burst", "no clock samples; burst assumed"
    return sus, "sustained", f"timed region {region_s:.1f} s at median {mhz:.0f} of {mx:.0f} MHz"


def strip_comments(text: str) -> str:
    """C/CUDA source without its // and /* */ comments; string and character
    literals are copied as they are (a // inside a string is not a comment).
    A block comment becomes one space, or its newlines if it spans lines."""
    out, i, n = [], 0, len(text)
    while i < n:
        c = text[i]
        if c in "\"'":
            j = i + 1
            while j < n and text[j] != c and text[j] != "\n":
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        elif text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            j = n if j < 0 else j + 2
            out.append("\n" * text.count("\n", i, j) or " ")
            i = j
        else:
            out.append(c)
            i += 1
    return "".join(out)


def source_hash(names) -> str:
    """Hash of the code of C/CUDA source files, blind to comments and to the
    spacing within a line: comments are dropped (strip_comments), runs of
    spaces and tabs collapsed, blank lines dropped.  Line breaks are kept, so a
    change that can change the compiled code (a token moved across the end of a
    preprocessor line, say) changes the hash."""
    h = hashlib.sha256()
    for name in names:
        with open(os.path.join(ROOT, name), encoding="utf-8") as fh:
            text = strip_comments(fh.read())
        lines = (" ".join(l.split()) for l in text.splitlines())
        h.update("\n".join(l for l in lines if l).encode())
        h.update(b"\0")
    return h.hexdigest()[:16]


def traffic_for(kernel: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current code of that kernel (the files it lists); else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as fh:
            e = json.load(fh).get(kernel)
        if e.get("source_hash") != source_hash(e["sources"]):
            return None
    except Exception:
        return None
    return e.get("traffic_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.out = tempfile.NamedTemporaryFile("w+", delete=False, suffix=".csv")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.gpu), "-lms", "100"], stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.out.flush()
        self.out.seek(0)
        rows = [l.strip().split(",") for l in self.out.read().splitlines() if l.strip()]
        self.out.close()
        os.unlink(self.out.name)
        sm, mx, power, reasons = [], None, [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx = float(r[2])
                power.append(float(r[3]))
            except ValueError:
                continue
            for name, val in zip(names, r[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_max": max(power) if power else None}


def dist_setup():
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(ms_local: float, tokens_per_rank: int, world: int):
    """Whole-job throughput: every rank processed its own batch; the job took
    as long as the slowest rank.  Returns (ms of the slowest rank, tokens/s)."""
    ms_max = max_over_ranks(ms_local, world)
    return ms_max, world * tokens_per_rank / (ms_max / 1e3)


# ------------------------------------------------------------------------- oracle timing
def oracle_sample(wl, ntok: int, seed: int = 1234, tensors=None):
    """The first `ntok` tokens of the workload's seeded inputs (or of the given
    (H, W, y) tensors), as oracle arrays."""
    import numpy as np

    from paper_2608_09703_gb300 import synth

    H, W, y = tensors if tensors is not None else synth.make_inputs(wl, seed=seed)
    Hs = synth.as_oracle_arrays([h[:ntok] for h in H])
    Ws = synth.as_oracle_arrays(W)
    return Hs, Ws, y[:ntok].cpu().numpy().astype(np.int32)


def oracle_step(wl, Hs, Ws, ys):
    from oracle import oracle

    kw = dict(teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha, w=wl.weights)
    fwd = oracle.forward(Hs, Ws, ys, **kw)
    oracle.backward(Hs, Ws, ys, **kw)
    return fwd


def oracle_rate(wl, budget_s: float, seed: int = 1234, tensors=None):
    """Calibrates the sample size to ~budget_s of CPU work, then times one
    forward+backward of the oracle on it.  Returns (tokens/s, tokens,
    seconds, the oracle's forward results on the sample)."""
    from oracle import oracle

    oracle.build()
    # the oracle runs one token per thread: calibrate with one token per thread
    ncal = max(2, oracle.threads())
    Hs, Ws, ys = oracle_sample(wl, ncal, seed, tensors)
    t0 = time.perf_counter()
    oracle_step(wl, Hs, Ws, ys)
    per_tok = (time.perf_counter() - t0) / ncal
    ntok = int(max(2, min(wl.T, budget_s / max(per_tok, 1e-6))))
    Hs, Ws, ys = oracle_sample(wl, ntok, seed, tensors)
    t0 = time.perf_counter()
    fwd = oracle_step(wl, Hs, Ws, ys)
    dt = time.perf_counter() - t0
    return ntok / dt, ntok, dt, fwd


def reference_arm(args, rank, world):
    from oracle import oracle
    from paper_2608_09703_gb300 import synth

    if rank != 0:
        return
    wl = workload(args)
    oracle.build()
    # size each step so that warmup + steps fit in about three minutes
    ncal = max(2, oracle.threads())
    Hs, Ws, ys = oracle_sample(wl, ncal)
    t0 = time.perf_counter()
    oracle_step(wl, Hs, Ws, ys)
    per_tok = (time.perf_counter() - t0) / ncal
    per_step_budget = max(1.0, 180.0 / (args.steps + args.warmup))
    ntok = int(max(1, min(wl.T, per_step_budget / max(per_tok, 1e-6))))
    Hs, Ws, ys = oracle_sample(wl, ntok)
    for _ in range(args.warmup):
        oracle_step(wl, Hs, Ws, ys)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_step(wl, Hs, Ws, ys)
        times.append(time.perf_counter() - t0)
    step_s = sum(times) / len(times)
    value = ntok / step_s
    sample = (f"first {ntok} of {wl.T} tokens of {wl.name} per step (full V={wl.V} and widths "
              f"{list(wl.d)}); fp64 forward+backward")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_s * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(wl, world),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def workload(args):
    from paper_2608_09703_gb300 import synth

    wl = synth.WORKLOADS[args.workload]
    if args.tokens or args.vocab:
        T, V = args.tokens or wl.T, args.vocab or wl.V
        wl = wl.with_(name=f"{wl.name}_T{T}_V{V}", T=T, V=V)
    return wl


def workload_config(wl, world):
    elt = 2 if wl.dtype == "bf16" else 4
    w_mb = wl.V * sum(wl.d) * elt / 1e6
    seqs = f"{wl.T // 2048}x2048" if wl.T % 2048 == 0 else f"{wl.T}"
    l2 = (f"inputs larger than L2 (W {w_mb:.0f} MB {wl.dtype}), no flush" if w_mb > 129
          else f"inputs smaller than L2 (W {w_mb:.1f} MB {wl.dtype}), no flush")
    return {"workload": f"{wl.name}: {len(wl.d)}-level Matryoshka suite head+CE+distillation, "
                        f"T={wl.T} tokens ({seqs}), d={list(wl.d)}, V={wl.V}, {wl.dtype}, "
                        f"tau={wl.tau}, alpha={wl.alpha}",
            "T": wl.T, "d": list(wl.d), "V": wl.V, "tau": wl.tau, "alpha": wl.alpha,
            "global_batch": wl.T * world, "seq_len": 2048, "parallelism": f"dp{world}",
            "l2": l2}


# ------------------------------------------------------------------------- GPU arm
def gpu_arm(args, rank, world, local):
    import numpy as np
    import torch

    from paper_2608_09703_gb300 import binding as B
    from paper_2608_09703_gb300 import synth

    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    wl = workload(args)
    H, W, y = synth.make_inputs(wl, seed=1234 + rank, device=dev)
    op = B.HeadLoss(wl.d, wl.T, wl.V, teacher=wl.teacher_index, tau=wl.tau, alpha=wl.alpha,
                    w=wl.weights, dtype=torch.bfloat16, device=dev, vocab_group=args.vocab_group)

    nvtx = torch.cuda.nvtx

    def step():
        nvtx.range_push("mls_head_loss_fwd")
        op.forward(H, W, y)
        nvtx.range_pop()
        nvtx.range_push("mls_head_loss_bwd")
        op.backward(H, W, y)
        nvtx.range_pop()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    status = B.mls_get_status()
    if status:
        raise RuntimeError(f"device status after warm-up: {B.mls_strerror(status)}")

    # ---- timed region
    sampler = ClockSampler(dev.index if dev.index is not None else 0)
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.25)
    B.mls_profile_enable(True)
    nvtx.range_push("timed_steps")
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    nvtx.range_pop()
    torch.cuda.synchronize()
    kern = B.mls_profile_read()
    B.mls_profile_enable(False)
    clocks = sampler.stop()
    barrier(world)
    ms = e0.elapsed_time(e1) / args.steps
    ms_max, value = aggregate(ms, wl.T, world)

    pk, pk_src = peaks()
    step_flops = wl.flops_fwd_bwd()
    per_kernel = {}
    for name, (launches, total_ms) in kern.items():
        entry = {"launches_per_step": launches / args.steps, "ms_per_step": total_ms / args.steps}
        if name in KERNELS:
            flops_launch = KERNELS[name] * (step_flops / 4) / (launches / args.steps)
            entry["tflops"] = flops_launch / (total_ms / launches / 1e3) / 1e12
        per_kernel[name] = entry
    dom = max((k for k in KERNELS if k in kern), key=lambda k: kern[k][1])
    launches, total_ms = kern[dom]
    flops_launch = KERNELS[dom] * (step_flops / 4) / (launches / args.steps)
    achieved = flops_launch / (total_ms / launches / 1e3) / 1e12
    burst, sus = float(pk["bf16_tflops"]), float(pk["bf16_tflops_sustained"])
    peak, regime, why = pick_peak(pk, ms * args.steps / 1e3, clocks)
    roofline = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": peak,
                "unit": "TFLOP/s", "frac": achieved / peak, "peak_regime": regime,
                "peak_why": why,
                "peak_source": (f"{pk_src} dense bf16 {regime} (MEASURED_PEAKS.json: burst {burst}, "
                                f"sustained {sus})" if pk_src == "measured"
                                else f"fallback dense bf16 {regime}"),
                "flops_per_launch": flops_launch,
                "traffic": traffic_for(dom)}
    gpu_launches = sum(v[0] for v in kern.values())

    # ---- the same step looped for seconds: the regime of a training run, in
    # which the clock settles under the power cap
    sustained = None
    if args.sustain_s > 0:
        nvtx.range_push("sustained_steps")
        sustained = sustained_run(args, step, ms, stream, dev, pk, step_flops, wl, world)
        nvtx.range_pop()

    # ---- evaluation metrics between sub-models (forward only), same inputs
    pairwise = None
    if not args.no_pairwise:
        for _ in range(2):
            op.pairwise(H, W, y)
        torch.cuda.synchronize()
        B.mls_profile_enable(True)
        e0.record(stream)
        n_pw = max(3, args.steps // 2)
        for _ in range(n_pw):
            op.pairwise(H, W, y)
        e1.record(stream)
        torch.cuda.synchronize()
        kp = B.mls_profile_read()
        B.mls_profile_enable(False)
        pw_ms = e0.elapsed_time(e1) / n_pw
        k_launches, k_ms = kp["pairwise"]
        k_tflops = (step_flops / 4) / (k_ms / k_launches / 1e3) / 1e12
        pw_peak, pw_regime, _ = pick_peak(pk, pw_ms * n_pw / 1e3, None)
        pairwise = {"ms_per_call": pw_ms, "tokens_per_s": wl.T / (pw_ms / 1e3),
                    "kernel_tflops": k_tflops, "kernel_frac": k_tflops / pw_peak,
                    "peak_tflops": pw_peak, "peak_regime": pw_regime,
                    "flops_per_call": step_flops / 4,
                    "what": "per-token KL(p_i||p_j) for all ordered sub-model pairs, means and "
                            "top-1 agreement (forward only)"}

    # ---- inter-model junctions (Eq. 1) of the suite, forward + backward
    junction = None
    if not args.no_junction:
        nvtx.range_push("junction")
        junction = junction_run(args, wl, dev, float(pk["hbm_gbs"]))
        nvtx.range_pop()

    # ---- speculative-decoding verify step (draft 1024 / verifier 3072 of the suite)
    spec = None
    if not args.no_spec:
        nvtx.range_push("spec_verify")
        spec = spec_run(args, dev, pk)
        nvtx.range_pop()

    # ---- end to end through the C ABI with host buffers (pinned), copies timed
    e2e = None
    if not args.no_e2e:
        nvtx.range_push("end_to_end")
        e2e = e2e_run(args, op, H, W, y, world, stream, wl)
        nvtx.range_pop()
    if rank != 0:
        return
    cpu = None
    parity = None
    if world == 1 and not args.no_cpu_baseline:
        # the oracle on the first tokens of the very inputs the GPU ran
        rate, ntok, secs, ref = oracle_rate(wl, budget_s=15.0, tensors=(H, W, y))
        from oracle import oracle

        cpu = {"value": rate, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
               "sample": f"first {ntok} of {wl.T} tokens of {wl.name} (full V and widths), "
                         f"fp64 forward+backward, {secs:.1f} s"}
        # parity of the timed GPU step's per-token outputs on that sample
        import numpy as np

        got = op.tok_loss[:, :ntok].double().cpu().numpy()
        diag = op.tok_diag[:, :, :ntok].double().cpu().numpy()
        rel = lambda a, b: float(np.max(np.abs(a - b) / np.maximum(np.abs(b), 1e-30)))
        kl_err = float(np.max(np.abs(diag[2] - ref["kl"]) / np.maximum(1.0, ref["ld"])))
        parity = {"tokens": ntok, "max_rel_err_tok_loss": rel(got, ref["tok_loss"]),
                  "max_rel_err_ce": rel(diag[0], ref["ce"]), "max_rel_err_ld": rel(diag[1], ref["ld"]),
                  "max_err_kl_vs_max1_ld": kl_err,
                  "argmax_agree": float(np.mean(op.argmax[:, :ntok].cpu().numpy() == ref["argmax"])),
                  "tolerance": "per-token losses 1e-3 relative; KL 1e-3 * max(1, Ld)"}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "tf32",
        "data": f"synthetic (seeded N(0,1) hidden states, N(0,{wl.w_sigma}^2) heads"
        + (f" with the teacher's x{wl.teacher_scale:g}" if wl.teacher_scale != 1.0 else "")
        + f", {wl.targets} targets; FineWeb-Edu not available)",
        "config": workload_config(wl, world),
        # 8*T*V*sum(d) per step against the peak of the timed region's regime
        "tensor_frac_step": step_flops / (ms_max / 1e3) / 1e12 / peak,
        # the model-FLOPs convention 6*T*V*sum(d), which leaves out the
        # backward's recompute of the logits
        "tensor_frac_step_6tvd": 0.75 * step_flops / (ms_max / 1e3) / 1e12 / peak,
        "peak_regime": {"regime": regime, "tflops": peak, "why": why},
        "roofline": roofline, "kernels": per_kernel, "gpu_launches": gpu_launches,
        "clocks": clocks, "sustained": sustained, "e2e": e2e, "cpu_baseline": cpu,
        "pairwise_eval": pairwise,
        "junction": junction, "spec_verify": spec, "parity_sample": parity,
    }
    print(json.dumps(line), flush=True)


def sustained_run(args, step, ms_short, stream, dev, pk, step_flops, wl, world):
    """Back-to-back steps for about args.sustain_s seconds (after the short
    timed region), clocks sampled throughout.  The fractions are of the
    sustained bf16 peak when the clock settled below its maximum, else of the
    burst peak (pick_peak)."""
    import torch

    from paper_2608_09703_gb300 import binding as B

    n = max(10, int(args.sustain_s * 1e3 / max(ms_short, 1e-3)))
    sampler = ClockSampler(dev.index if dev.index is not None else 0)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.25)
    B.mls_profile_enable(True)
    e0.record(stream)
    for _ in range(n):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    kern = B.mls_profile_read()
    B.mls_profile_enable(False)
    clocks = sampler.stop()
    ms = e0.elapsed_time(e1) / n
    ms_max, value = aggregate(ms, wl.T, world)
    peak, regime, why = pick_peak(pk, ms * n / 1e3, clocks)
    out = {"steps": n, "seconds": ms * n / 1e3, "ms_per_step": ms_max, "value": value,
           "unit": UNIT, "tensor_frac_step": step_flops / (ms_max / 1e3) / 1e12 / peak,
           "tensor_frac_step_of_burst": step_flops / (ms_max / 1e3) / 1e12 / float(pk["bf16_tflops"]),
           "peak_regime": {"regime": regime, "tflops": peak, "why": why}, "clocks": clocks,
           "kernels": {}}
    for name, (launches, total_ms) in kern.items():
        entry = {"ms_per_step": total_ms / n}
        if name in KERNELS:
            f = KERNELS[name] * (step_flops / 4) / (launches / n)
            t = f / (total_ms / launches / 1e3) / 1e12
            entry.update({"tflops": t, "frac": t / peak})
        out["kernels"][name] = entry
    return out


def junction_run(args, wl, dev, hbm_gbs):
    """Forward + backward of every junction m -> m+1 of the suite on T tokens,
    bf16, timed with CUDA events.  Algorithmic bytes per junction: forward
    reads o and e and writes x (2 * T * D_{m+1} elements), backward reads g, o,
    e and writes dL/do, dL/de (3 * T * D_{m+1} elements)."""
    import torch

    from paper_2608_09703_gb300 import binding as B

    g = torch.Generator(device=dev)
    g.manual_seed(99)
    bufs = []
    nbytes = 0
    for m in range(wl.M - 1):
        dp, dn = wl.d[m], wl.d[m + 1]
        mk = lambda *sh: torch.randn(*sh, generator=g, device=dev).to(torch.bfloat16)
        o, e, gr = mk(wl.T, dp), mk(wl.T, dn - dp), mk(wl.T, dn)
        x, d_o, d_e = torch.empty_like(gr), torch.empty_like(o), torch.empty_like(e)
        bufs.append((o, e, gr, x, d_o, d_e))
        nbytes += 5 * wl.T * dn * 2

    def run():
        for o, e, gr, x, d_o, d_e in bufs:
            B.mls_junction_fwd(o, e, x)
            B.mls_junction_bwd(o, e, gr, d_o, d_e)

    for _ in range(3):
        run()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n = max(5, args.steps)
    B.mls_profile_enable(True)
    e0.record(stream)
    for _ in range(n):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    kp = B.mls_profile_read()
    B.mls_profile_enable(False)
    ms = e0.elapsed_time(e1) / n
    kern_ms = sum(v[1] for k, v in kp.items() if k.startswith("junction")) / n
    gbs = nbytes / (kern_ms / 1e3) / 1e9
    return {"junctions": wl.M - 1, "ms_per_fwd_bwd": ms, "kernel_ms": kern_ms,
            "bytes": nbytes, "achieved_gbs": gbs, "peak_gbs": hbm_gbs, "frac": gbs / hbm_gbs,
            "bound": "hbm"}


def e2e_run(args, op, H, W, y, world, stream, wl):
    """The same metric through the C ABI with the inputs in pinned host memory.

    Every step copies its own H, W and targets host->device and reads its loss
    back device->host inside the timed region.  The copies run on a second
    stream into the other of two device buffers while the previous step
    computes (a data pipeline's prefetch), so a step waits only for its own
    inputs."""
    import torch

    from paper_2608_09703_gb300 import binding as B

    dev = H[0].device
    Hh = [h.cpu().pin_memory() for h in H]
    Wh = [w.cpu().pin_memory() for w in W]
    yh = y.cpu().pin_memory()
    srcs = Hh + Wh + [yh]
    bufs = [[torch.empty_like(t, device=dev) for t in srcs] for _ in range(2)]
    n_e2e = max(3, min(args.steps, 10))
    loss_h = torch.empty(n_e2e + 1, dtype=torch.float32).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in srcs)
    d2h = 4
    copy_stream = torch.cuda.Stream(device=dev)
    done = [torch.cuda.Event() for _ in range(2)]      # compute finished with buffer b
    landed = [torch.cuda.Event() for _ in range(2)]    # inputs of buffer b copied
    M = wl.M

    def copy_into(b):
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(done[b])
            for src, dst in zip(srcs, bufs[b]):
                dst.copy_(src, non_blocking=True)
            landed[b].record(copy_stream)

    def compute(i, b):
        stream.wait_event(landed[b])
        Hd, Wd, yd = bufs[b][:M], bufs[b][M:2 * M], bufs[b][2 * M]
        op.forward(Hd, Wd, yd)
        op.backward(Hd, Wd, yd)
        loss_h[i].copy_(op.loss[0], non_blocking=True)
        done[b].record(stream)

    for b in range(2):
        done[b].record(stream)
    torch.cuda.synchronize()
    # warm-up step (not timed)
    copy_into(0)
    compute(n_e2e, 0)
    torch.cuda.synchronize()
    barrier(world)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0 = time.perf_counter()
    e0.record(stream)
    copy_stream.wait_event(e0)
    copy_into(0)
    for i in range(n_e2e):
        if i + 1 < n_e2e:
            copy_into((i + 1) % 2)
        compute(i, i % 2)
    e1.record(stream)
    torch.cuda.synchronize()
    host_ms = (time.perf_counter() - t0) * 1e3
    e2e_ms = max(e0.elapsed_time(e1), host_ms) / n_e2e
    e2e_ms = max_over_ranks(e2e_ms, world)
    assert torch.isfinite(loss_h).all()
    e2e = {"value": world * wl.T / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
           "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
           "note": "inputs copied from pinned host memory every step, prefetched one step ahead "
                   "on a copy stream; loss read back every step"}
    status = B.mls_get_status()
    if status:
        raise RuntimeError(f"device status: {B.mls_strerror(status)}")
    return e2e


def spec_run(args, dev, pk):
    """The speculative-decoding verify step on the suite's draft / verifier pair
    at the paper's batch (102 sequences, draft length 6, V = 50304), bf16,
    nucleus sampling (T = 0.4, p = 0.9) and greedy, timed with CUDA events.
    The logits GEMM is 2 V (B gamma d_draft + B (gamma + 1) d_verify) FLOPs; the
    selection kernels are reported against one read of every logits row."""
    import torch

    from paper_2608_09703_gb300 import binding as B
    from paper_2608_09703_gb300 import synth

    wl = synth.SPEC_WORKLOADS["spec_suite3"]
    Hd, Wd, Hv, Wv = synth.make_spec_inputs(wl, 7, device=dev)
    u = synth.make_uniforms(wl.B, wl.gamma, 7, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(8)
    draft = torch.randint(0, wl.V, (wl.B, wl.gamma), generator=g, device=dev, dtype=torch.int32)
    Pd, Pv = wl.B * wl.gamma, wl.B * (wl.gamma + 1)
    flops = 2 * wl.V * (Pd * wl.d_draft + Pv * wl.d_verify)
    stream = torch.cuda.current_stream()
    out = {"config": {"B": wl.B, "gamma": wl.gamma, "V": wl.V, "d_draft": wl.d_draft,
                      "d_verify": wl.d_verify, "temperature": wl.temperature, "top_p": wl.top_p}}
    for mode, greedy in (("nucleus", False), ("greedy", True)):
        op = B.SpecVerify(wl.B, wl.gamma, wl.V, wl.d_draft, wl.d_verify, wl.temperature,
                          wl.top_p, greedy, dtype=torch.bfloat16, device=dev)
        for _ in range(3):
            op(Hd, Wd, Hv, Wv, draft, u)
        torch.cuda.synchronize()
        n = max(5, args.steps // 2)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        B.mls_profile_enable(True)
        e0.record(stream)
        for _ in range(n):
            op(Hd, Wd, Hv, Wv, draft, u)
        e1.record(stream)
        torch.cuda.synchronize()
        kp = B.mls_profile_read()
        B.mls_profile_enable(False)
        ms = e0.elapsed_time(e1) / n
        gemm_ms = kp["spec_logits"][1] / n
        f = flops if not greedy else 2 * wl.V * Pv * wl.d_verify
        sp_peak, sp_regime, _ = pick_peak(pk, ms * n / 1e3, None)
        out[mode] = {
            "ms_per_call": ms, "positions_per_s": Pv / (ms / 1e3),
            "kernel_ms": {k: v[1] / n for k, v in kp.items()},
            "logits_tflops": f / (gemm_ms / 1e3) / 1e12,
            "logits_frac": f / (gemm_ms / 1e3) / 1e12 / sp_peak,
            "peak_tflops": sp_peak, "peak_regime": sp_regime,
        }
        if not greedy:
            # the selection kernels against one read of every probability row
            sel_ms = (kp["spec_rows"][1] + kp["spec_sample"][1]) / n
            out[mode]["selection_gbs_one_read"] = (Pv + Pd) * wl.V * 4 / (sel_ms / 1e3) / 1e9
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mls", choices=["mls", "reference"])
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-pairwise", action="store_true")
    ap.add_argument("--no-junction", action="store_true")
    ap.add_argument("--no-spec", action="store_true")
    ap.add_argument("--tokens", type=int, default=0, help="override T (profiling captures)")
    ap.add_argument("--vocab", type=int, default=0, help="override V (profiling captures)")
    ap.add_argument("--sustain-s", type=float, default=3.0,
                    help="seconds of back-to-back steps for the sustained sub-record (0: skip)")
    ap.add_argument("--vocab-group", type=int, default=0,
                    help="backward vocabulary group in columns (0 = the library's choice)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        # rank 0 alone times the CPU oracle; other ranks exit without work
        reference_arm(args, int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")))
        return
    rank, world, local = dist_setup()
    try:
        gpu_arm(args, rank, world, local)
    finally:
        if world > 1:
            import torch.distributed as dist

            dist.destroy_process_group()


if __name__ == "__main__":
    main()
