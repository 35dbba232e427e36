"""GPU parity of the inter-model junction (Eq. 1) against the fp64 oracle."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import synth

pytestmark = pytest.mark.gpu


def run(o, e, g, embed_first):
    dev = torch.device("cuda")
    od, ed, gd = o.to(dev), e.to(dev), g.to(dev)
    x = torch.empty(o.shape[0], o.shape[1] + e.shape[1], dtype=o.dtype, device=dev)
    d_o, d_e = torch.empty_like(od), torch.empty_like(ed)
    B.mls_junction_fwd(od, ed, x, embed_first)
    B.mls_junction_bwd(od, ed, gd, d_o, d_e, embed_first)
    torch.cuda.synchronize()
    return x.cpu().double().numpy(), d_o.cpu().double().numpy(), d_e.cpu().double().numpy()


def compare(o, e, g, embed_first, tol_x, tol_g):
    x, d_o, d_e = run(o, e, g, embed_first)
    oo, ee, gg = synth.as_oracle_arrays([o, e, g])
    xr = oracle.junction_fwd(oo, ee, embed_first)
    d_or, d_er = oracle.junction_bwd(oo, ee, gg, embed_first)
    err = np.abs(x - xr) / (np.abs(xr) + tol_x * np.abs(xr).max(axis=1, keepdims=True) + 1e-30)
    assert err.max() <= tol_x, f"x rel err {err.max()}"
    for got, want, name in ((d_o, d_or, "d_o"), (d_e, d_er, "d_e")):
        e_ = np.abs(got - want).max() / max(np.abs(want).max(), 1e-30)
        assert e_ <= tol_g, f"{name} max-norm rel err {e_}"
    return x, d_o, d_e


@pytest.mark.parametrize("embed_first", [False, True])
def test_junction_bf16(embed_first):
    g = torch.Generator().manual_seed(41)
    T, dp, de = 300, 64, 128
    o = (torch.randn(T, dp, generator=g) * 4).to(torch.bfloat16)
    e = (torch.randn(T, de, generator=g) * 0.05).to(torch.bfloat16)
    gr = torch.randn(T, dp + de, generator=g).to(torch.bfloat16)
    o[7] = 0  # zero row: o~ = 0, dL/do = 0, dL/de = g_e
    x, d_o, d_e = compare(o, e, gr, embed_first, tol_x=4e-3, tol_g=1e-2)
    assert np.abs(d_o[7]).max() == 0.0


@pytest.mark.parametrize("embed_first", [False, True])
def test_junction_fp32(embed_first):
    g = torch.Generator().manual_seed(42)
    T, dp, de = 200, 128, 64
    o = torch.randn(T, dp, generator=g) * 2
    e = torch.randn(T, de, generator=g) * 0.1
    gr = torch.randn(T, dp + de, generator=g)
    compare(o, e, gr, embed_first, tol_x=1e-5, tol_g=1e-5)


@pytest.mark.parametrize("dp,dn", [(1024, 2048), (2048, 3072)])
def test_junction_suite3_shapes_full_size(dp, dn):
    """The two junctions of the 3-level suite at the benchmark's T."""
    g = torch.Generator().manual_seed(43)
    T = 8192
    o = (torch.randn(T, dp, generator=g) * 8).to(torch.bfloat16)
    e = (torch.randn(T, dn - dp, generator=g) * 0.02).to(torch.bfloat16)
    gr = (torch.randn(T, dn, generator=g) * 1e-3).to(torch.bfloat16)
    compare(o, e, gr, False, tol_x=4e-3, tol_g=1e-2)


# Each register-cache size of the kernels (16-byte vectors per lane per row
# segment: 1, 2, 4, 8), the TMA ring for wider rows and the streaming path for
# rows too wide for two ring buffers, with segments that end part-way through
# a vector round and a ragged last block.
@pytest.mark.parametrize("dtype,dp,de", [
    (torch.bfloat16, 72, 40),      # 1 vector
    (torch.bfloat16, 264, 8),      # 2
    (torch.bfloat16, 520, 1000),   # 4
    (torch.bfloat16, 1800, 200),   # 8
    (torch.bfloat16, 3072, 1024),  # 12: TMA ring
    (torch.bfloat16, 3080, 16),    # o past 12: ring
    (torch.bfloat16, 64, 4096),    # e past 12: ring
    (torch.float32, 1536, 512),    # ring
    (torch.float32, 1540, 4),      # ring
    (torch.float32, 28608, 64),    # a 112 KB row: streaming
])
def test_junction_cache_sizes(dtype, dp, de):
    g = torch.Generator().manual_seed(44 + dp + de)
    T = 37
    o = (torch.randn(T, dp, generator=g) * 3).to(dtype)
    e = (torch.randn(T, de, generator=g) * 0.1).to(dtype)
    gr = torch.randn(T, dp + de, generator=g).to(dtype)
    o[5] = 0   # ||o|| = 0: o~ = 0, dL/do = 0, dL/de = g_e
    e[11] = 0  # ||e|| = 0: o~ = 0, dL/do = 0
    bf = dtype == torch.bfloat16
    for embed_first in (False, True):
        x, d_o, d_e = compare(o, e, gr, embed_first, tol_x=4e-3 if bf else 1e-5,
                              tol_g=1e-2 if bf else 1e-5)
        assert np.abs(d_o[5]).max() == 0.0 and np.abs(d_o[11]).max() == 0.0
        np.testing.assert_array_equal(d_e[5], gr[5, (0 if embed_first else dp):][:de].double().numpy())


def test_junction_ring_many_rows_per_warp():
    """The TMA ring at a size where every warp takes many rows, so each of its
    buffers is refilled several times (3072 -> 4096, bf16, T = 16384)."""
    g = torch.Generator().manual_seed(45)
    T, dp, de = 16384, 3072, 1024
    o = (torch.randn(T, dp, generator=g) * 2).to(torch.bfloat16)
    e = (torch.randn(T, de, generator=g) * 0.05).to(torch.bfloat16)
    gr = (torch.randn(T, dp + de, generator=g) * 1e-2).to(torch.bfloat16)
    o[T - 1] = 0
    for embed_first in (False, True):
        compare(o, e, gr, embed_first, tol_x=4e-3, tol_g=1e-2)
