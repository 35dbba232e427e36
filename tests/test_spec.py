"""GPU parity of the speculative-decoding verify step (mls_spec_verify) against
the fp64 oracle (Sec. 2 "Speculative Decoding"; Sec. 3.2.3 samples with
temperature 0.4 and nucleus p = 0.9, or greedily).

The CUDA path computes logits and probabilities in fp32, the oracle in fp64, so
a decision that the exact values leave within rounding of its threshold may go
either way.  Each sequence's decision path is therefore replayed here in fp64
with the margin of every comparison on it (nucleus boundary, acceptance test,
inverse-CDF step, greedy top-2 gap), following every kept set that rounding
could give a nucleus whose boundary is that close; a sequence whose outcome
rounding could change is left out of the comparison (at most a quarter of them
unless a test says otherwise), and every other sequence must match the oracle
exactly (n_accepted and next_token).
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import synth

pytestmark = pytest.mark.gpu

# fp32 logits of bf16 products differ from the exact ones by ~1e-5 and the
# probabilities by ~3e-5 relative; decisions closer than this are not compared.
MARGIN = 3e-4


# ---------------------------------------------------------------- fp64 replay with margins
def nucleus_alternatives(z, T, top_p):
    """nucleus(softmax(z / T)) in fp64, with the other kept sets that rounding
    could produce: the cut one token earlier or later when the cumulative is
    within MARGIN of top_p, and the last kept token swapped with the first
    dropped one when their probabilities are within MARGIN (relative).  Exact
    ties are ordered by index on both sides and produce no alternative.
    Returns a list of renormalised distributions, the exact one first, or None
    when the boundary is too crowded to enumerate."""
    e = np.exp((z - z.max()) / T)
    p = e / e.sum()
    if top_p >= 1.0:
        return [p]
    V = len(p)
    order = np.lexsort((np.arange(V), -p))
    ps = p[order]
    cum = np.cumsum(ps)
    hit = np.nonzero(cum >= top_p)[0]
    k = int(hit[0]) if len(hit) else V - 1
    cuts = [k]
    if cum[k] - top_p < MARGIN and k + 1 < V:
        cuts.append(k + 1)
    if k > 0 and top_p - cum[k - 1] < MARGIN:
        cuts.append(k - 1)
    near = lambda a, b: ps[a] != ps[b] and (ps[a] - ps[b]) / ps[a] < MARGIN
    alts = []
    for c in cuts:
        sets = [order[:c + 1]]
        if c + 1 < V and near(c, c + 1):
            if c + 2 < V and near(c, c + 2):
                return None
            s2 = order[:c + 1].copy()
            s2[-1] = order[c + 1]
            sets.append(s2)
        for kept in sets:
            q = np.zeros_like(p)
            q[kept] = p[kept]
            alts.append(q / q.sum())
    return alts


def sample_with_margin(r, u):
    cum = np.cumsum(r)
    want = u * cum[-1]
    v = min(int(np.searchsorted(cum, want, side="right")), len(r) - 1)
    before = cum[v - 1] if v > 0 else 0.0
    return v, min(want - before, cum[v] - want)


def replay(zd, zv, draft, u, T, top_p, greedy):
    """One sequence in fp64: zd [gamma, V], zv [gamma+1, V] exact logits.
    Every nucleus alternative is followed; returns ((n_accepted, next_token) of
    the exact path, True if every path gives that outcome with all margins of
    its comparisons at least MARGIN)."""
    gamma, V = len(draft), zv.shape[1]
    if greedy:
        margin = np.inf
        for i in range(gamma + 1):
            z = zv[i]
            best = int(np.argmax(z))
            top2 = np.sort(z)[-2:]
            if top2[1] != top2[0]:
                margin = min(margin, (top2[1] - top2[0]) / max(1.0, abs(top2[1])))
            if i == gamma or draft[i] != best:
                return (i, best), margin >= MARGIN
    alts_d = [nucleus_alternatives(zd[i], T, top_p) for i in range(gamma)]
    alts_v = [nucleus_alternatives(zv[i], T, top_p) for i in range(gamma + 1)]
    if any(a is None for a in alts_d + alts_v):
        return None, False
    outcomes, margin = [], [np.inf]

    def walk(i):
        if i == gamma:
            for p in alts_v[gamma]:
                v, ms = sample_with_margin(p, u[gamma, 1])
                margin[0] = min(margin[0], ms)
                outcomes.append((gamma, v))
            return
        for q in alts_d[i]:
            for p in alts_v[i]:
                x = int(draft[i])
                ok = False
                if 0 <= x < V and q[x] > 0:
                    a, b = u[i, 0] * q[x], p[x]
                    if b > 0:
                        margin[0] = min(margin[0], abs(a - b) / max(a, b))
                    ok = a < b
                if ok:
                    walk(i + 1)
                else:
                    r = np.maximum(p - q, 0.0)
                    if r.sum() == 0:
                        r = p
                    v, ms = sample_with_margin(r, u[i, 1])
                    margin[0] = min(margin[0], ms)
                    outcomes.append((i, v))

    walk(0)
    return outcomes[0], len(set(outcomes)) == 1 and margin[0] >= MARGIN


def exact(H, W):
    return H.detach().cpu().double().numpy() @ W.detach().cpu().double().numpy().T


def draw_drafts(zd, gamma, T, top_p, seed, p_random=0.1):
    """Draft tokens as the draft model would emit them: drawn from q (a few
    uniformly random ones exercise q(x) = 0)."""
    rng = np.random.default_rng(seed)
    P, V = zd.shape
    out = np.empty(P, np.int32)
    for r in range(P):
        if rng.random() < p_random:
            out[r] = rng.integers(0, V)
        else:
            out[r] = rng.choice(V, p=nucleus_alternatives(zd[r], T, top_p)[0])
    return out.reshape(-1, gamma)


# ---------------------------------------------------------------- runners
def run_gpu(wl, Hd, Wd, Hv, Wv, draft, u, greedy=False, top_p=None):
    dev = torch.device("cuda")
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    op = B.SpecVerify(wl.B, wl.gamma, wl.V, wl.d_draft, wl.d_verify, wl.temperature,
                      wl.top_p if top_p is None else top_p, greedy, dtype=dt, device=dev)
    to = lambda t: None if t is None else t.to(dev).contiguous()
    n, nxt = op(to(Hd), to(Wd), to(Hv), to(Wv),
                torch.as_tensor(np.asarray(draft, np.int32)).to(dev).contiguous(), to(u))
    torch.cuda.synchronize()
    assert B.mls_get_status() == 0
    return n.cpu().numpy(), nxt.cpu().numpy()


def check(wl, Hd, Wd, Hv, Wv, draft, u, greedy=False, top_p=None, seqs=None, min_checked=0.75):
    """GPU vs oracle on the sequences `seqs` (all by default) whose replayed
    margin clears MARGIN."""
    top_p = wl.top_p if top_p is None else top_p
    n_g, nx_g = run_gpu(wl, Hd, Wd, Hv, Wv, draft, u, greedy, top_p)
    G, G1 = wl.gamma, wl.gamma + 1
    seqs = np.arange(wl.B) if seqs is None else np.asarray(seqs)
    draft = np.asarray(draft, np.int32).reshape(wl.B, G)
    un = u.double().numpy()
    rows_d = (seqs[:, None] * G + np.arange(G)[None]).reshape(-1)
    rows_v = (seqs[:, None] * G1 + np.arange(G1)[None]).reshape(-1)
    Hd_s = Hd[torch.as_tensor(rows_d)] if G else Hd[:0]
    Hv_s = Hv[torch.as_tensor(rows_v)]
    n_o, nx_o = oracle.spec_verify(*synth.as_oracle_arrays([Hd_s, Wd, Hv_s, Wv]), draft[seqs],
                                   un[seqs], temperature=wl.temperature, top_p=top_p,
                                   greedy=greedy)
    zd = exact(Hd_s, Wd).reshape(len(seqs), G, wl.V) if G else np.zeros((len(seqs), 0, wl.V))
    zv = exact(Hv_s, Wv).reshape(len(seqs), G1, wl.V)
    checked = 0
    for j, b in enumerate(seqs):
        got, decided = replay(zd[j], zv[j], draft[b], un[b], wl.temperature, top_p, greedy)
        if not decided:
            continue
        checked += 1
        # the replay is an independent fp64 restatement: it must agree with the oracle
        assert got == (n_o[j], nx_o[j]), f"replay vs oracle, sequence {b}"
        assert (n_g[b], nx_g[b]) == (n_o[j], nx_o[j]), \
            f"sequence {b}: gpu ({n_g[b]}, {nx_g[b]}) oracle ({n_o[j]}, {nx_o[j]})"
    assert checked >= min_checked * len(seqs), f"only {checked} of {len(seqs)} sequences decided"
    # every sequence: outputs in range
    assert ((n_g >= 0) & (n_g <= G)).all() and ((nx_g >= 0) & (nx_g < wl.V)).all()
    return n_g, nx_g, checked


def inputs(wl, seed, greedy=False):
    Hd, Wd, Hv, Wv = synth.make_spec_inputs(wl, seed)
    u = synth.make_uniforms(wl.B, wl.gamma, seed)
    zd = exact(Hd, Wd)
    if greedy:
        draft = zd.argmax(1).astype(np.int32).reshape(wl.B, wl.gamma)
    else:
        draft = draw_drafts(zd, wl.gamma, wl.temperature, wl.top_p, seed)
    return Hd, Wd, Hv, Wv, draft, u


# ---------------------------------------------------------------- tests
def test_spec_small_ragged_bf16():
    wl = synth.SpecWorkload("s", B=40, gamma=4, V=1000, d_draft=64, d_verify=128)
    n, _, _ = check(wl, *inputs(wl, 41))
    assert 0 < n.mean() < wl.gamma  # some accepted, some rejected


def test_spec_fp32_inputs_ragged_vocab():
    wl = synth.SpecWorkload("f", B=12, gamma=3, V=777, d_draft=32, d_verify=96, dtype="fp32")
    check(wl, *inputs(wl, 42))


def test_spec_greedy():
    wl = synth.SpecWorkload("g", B=24, gamma=5, V=1000, d_draft=64, d_verify=128, extra=0.1)
    Hd, Wd, Hv, Wv, draft, u = inputs(wl, 43, greedy=True)
    n, _, _ = check(wl, Hd, Wd, Hv, Wv, draft, u, greedy=True)
    assert 0 < n.mean() < wl.gamma
    # greedy needs neither the draft model nor the draws
    n2, nx2 = run_gpu(wl, None, None, Hv, Wv, draft, None, greedy=True)
    n1, nx1 = run_gpu(wl, Hd, Wd, Hv, Wv, draft, u, greedy=True)
    assert (n1 == n2).all() and (nx1 == nx2).all()


def test_spec_flat_and_peaked_distributions():
    # a flat distribution puts many tokens near the nucleus boundary: fewer decided
    for z_std, seed, frac in ((0.8, 44, 0.5), (6.0, 45, 0.75)):
        wl = synth.SpecWorkload("d", B=16, gamma=3, V=2000, d_draft=64, d_verify=128, z_std=z_std)
        check(wl, *inputs(wl, seed), min_checked=frac)


def test_spec_top_p_one_and_gamma_zero():
    wl = synth.SpecWorkload("p1", B=10, gamma=3, V=500, d_draft=64, d_verify=128, top_p=1.0)
    check(wl, *inputs(wl, 46))
    wl0 = synth.SpecWorkload("g0", B=10, gamma=0, V=500, d_draft=64, d_verify=128)
    Hd, Wd, Hv, Wv = synth.make_spec_inputs(wl0, 47)
    u = synth.make_uniforms(wl0.B, 0, 47)
    n, _, _ = check(wl0, Hd, Wd, Hv, Wv, np.zeros((wl0.B, 0), np.int32), u)
    assert (n == 0).all()


@pytest.mark.parametrize("temperature,top_p", [(1.0, 0.5), (0.7, 0.95), (0.2, 0.99)])
def test_spec_other_temperatures_and_nucleus_sizes(temperature, top_p):
    """Temperatures and nucleus sizes other than the paper's 0.4 / 0.9: a
    small nucleus of a softer distribution, a wide one, and a sharp one."""
    wl = synth.SpecWorkload("tp", B=24, gamma=4, V=1500, d_draft=64, d_verify=128,
                            temperature=temperature, top_p=top_p)
    # a wide nucleus of a soft distribution has more tokens near its cut
    check(wl, *inputs(wl, 60 + int(100 * temperature)), min_checked=0.6)


def test_spec_identical_models_accept_every_draft():
    """Draft == verifier: p == q exactly on both sides, so every drafted token
    inside the nucleus is accepted and the bonus token is sampled from p."""
    wl = synth.SpecWorkload("id", B=12, gamma=4, V=900, d_draft=128, d_verify=128)
    _, _, Hv, Wv = synth.make_spec_inputs(wl, 48)
    Hd = Hv.view(wl.B, wl.gamma + 1, -1)[:, :wl.gamma].reshape(wl.B * wl.gamma, -1).contiguous()
    u = synth.make_uniforms(wl.B, wl.gamma, 48)
    draft = draw_drafts(exact(Hd, Wv), wl.gamma, wl.temperature, wl.top_p, 48, p_random=0.0)
    n, _, _ = check(wl, Hd, Wv, Hv, Wv, draft, u)
    assert (n == wl.gamma).all()


def test_spec_exact_ties_at_the_nucleus_boundary():
    """Crafted logits with ten exactly tied tokens at the nucleus boundary, of
    which the cumulative needs only the lowest-index few (verifier: token 5 at
    z = 2, tokens 10..19 at z = 0.375, T = 0.4, top_p = 0.9 keeps 5 and 10..13).
    Hidden rows are one-hot, so the logits are exact on both sides.  Draft rows
    pick one of two draft heads: A (token 5 at 1.5, ties at 0.375: keeps 5 and
    10..17) or B (token 5 at 3.0: keeps 5 only)."""
    V, d, gamma, nseq = 64, 16, 3, 24
    Wv = torch.zeros(V, d)
    Wv[:, 0] = -8.0
    Wv[5, 0] = 2.0
    Wv[10:20, 0] = 0.375
    Wd = torch.zeros(V, d)
    Wd[:, 0] = -8.0
    Wd[:, 1] = -8.0
    Wd[5, 0], Wd[5, 1] = 1.5, 3.0
    Wd[10:20, 0] = 0.375
    Wd[10:20, 1] = 0.375
    rng = np.random.default_rng(49)
    head = rng.integers(0, 2, nseq * gamma)
    Hd = torch.zeros(nseq * gamma, d)
    Hd[torch.arange(nseq * gamma), torch.as_tensor(head)] = 1.0
    Hv = torch.zeros(nseq * (gamma + 1), d)
    Hv[:, 0] = 1.0
    draft = rng.choice([5, 5, 5, 10, 12, 13, 14, 17, 19], size=(nseq, gamma)).astype(np.int32)
    # draws away from every threshold of this construction
    u = torch.as_tensor(rng.choice([0.05, 0.2, 0.45, 0.65, 0.95, 0.99], size=(nseq, gamma + 1, 2)),
                        dtype=torch.float32)
    wl = synth.SpecWorkload("ties", B=nseq, gamma=gamma, V=V, d_draft=d, d_verify=d)
    bf = lambda t: t.to(torch.bfloat16).contiguous()
    n, nx, checked = check(wl, bf(Hd), bf(Wd), bf(Hv), bf(Wv), draft, u, min_checked=1.0)
    # outcomes reached through the partially kept ties occur
    assert set(nx.tolist()) & {10, 11, 12, 13}


def test_spec_suite_shape_sampled():
    """The benchmark's shape (batch 102, draft length 6, 1024/3072 widths,
    V = 50304): every output in range, two calls identical, and 34 of the 102
    sequences (the first, the last and 32 drawn at random) against the oracle,
    at least three quarters of them decided."""
    wl = synth.SPEC_WORKLOADS["spec_suite3"]
    Hd, Wd, Hv, Wv = synth.make_spec_inputs(wl, 50)
    u = synth.make_uniforms(wl.B, wl.gamma, 50)
    pick = np.random.default_rng(50).choice(np.arange(1, wl.B - 1), 32, replace=False)
    seqs = np.unique(np.concatenate([[0, wl.B - 1], pick]))
    rows = (seqs[:, None] * wl.gamma + np.arange(wl.gamma)[None]).reshape(-1)
    zd = exact(Hd[torch.as_tensor(rows)], Wd)
    draft = np.random.default_rng(50).integers(0, wl.V, (wl.B, wl.gamma)).astype(np.int32)
    draft[seqs] = draw_drafts(zd, wl.gamma, wl.temperature, wl.top_p, 50)
    n1, nx1, _ = check(wl, Hd, Wd, Hv, Wv, draft, u, seqs=seqs, min_checked=0.75)
    n2, nx2 = run_gpu(wl, Hd, Wd, Hv, Wv, draft, u)
    assert (n1 == n2).all() and (nx1 == nx2).all()


def test_spec_argument_errors():
    dev = torch.device("cuda")
    ws = torch.empty(1 << 20, dtype=torch.uint8, device=dev)
    h = torch.zeros(8, 64, dtype=torch.bfloat16, device=dev)
    w = torch.zeros(100, 64, dtype=torch.bfloat16, device=dev)
    t = torch.zeros(4, 1, dtype=torch.int32, device=dev)
    u = torch.zeros(4, 2, 2, dtype=torch.float32, device=dev)
    o = torch.zeros(4, dtype=torch.int32, device=dev)
    for kw, code in ((dict(top_p=0.0), B.MLS_ERR_ARG), (dict(temperature=0.0), B.MLS_ERR_ARG),
                     (dict(d_verify=60), B.MLS_ERR_UNSUPPORTED)):
        args = dict(B=4, gamma=1, V=100, d_draft=64, d_verify=64)
        args.update(kw)
        with pytest.raises(B.MLSError) as ei:
            B.mls_spec_verify(B.spec_problem(**args), h, w, h, w, t, u, o, o, ws)
        assert ei.value.code == code
    p = B.spec_problem(4, 1, 100, 64, 64)
    with pytest.raises(B.MLSError) as ei:
        B.mls_spec_verify(p, h, w, h, w, t, u, o, o, ws[:1024])
    assert ei.value.code == B.MLS_ERR_WORKSPACE


def test_spec_tiny_top_p_is_greedy_at_suite_shape():
    """top_p -> 0 keeps only the most likely token (ties apart), so with drafts
    equal to the draft model's argmax, nucleus verification must reproduce
    greedy verification exactly: accept while the verifier's argmax agrees,
    then emit it (the residual max(0, p - q) is one-hot there).  Checked on
    the benchmark's shape, every sequence, against the greedy path itself."""
    wl = synth.SPEC_WORKLOADS["spec_suite3"]
    Hd, Wd, Hv, Wv = synth.make_spec_inputs(wl, 51, device="cuda")
    u = synth.make_uniforms(wl.B, wl.gamma, 51, device="cuda")
    zd = Hd.float() @ Wd.float().T
    draft = zd.argmax(1).to(torch.int32).reshape(wl.B, wl.gamma).cpu().numpy()
    # the verifier agrees on a prefix of varying length
    n_g, nx_g = run_gpu(wl, Hd, Wd, Hv, Wv, draft, u, greedy=True)
    n_s, nx_s = run_gpu(wl, Hd, Wd, Hv, Wv, draft, u, greedy=False, top_p=1e-6)
    assert (n_s == n_g).all() and (nx_s == nx_g).all()
    assert 0 < n_g.mean() < wl.gamma


def test_spec_long_drafts():
    wl = synth.SpecWorkload("long", B=6, gamma=16, V=1500, d_draft=64, d_verify=128, extra=0.05)
    n, _, _ = check(wl, *inputs(wl, 52))
    assert n.max() > 4
