"""CPU checks of the C ABI: the library builds for sm_103a, loads, exports every
entry point that include/mls.h declares, and its host-side validation answers
with the documented error codes without touching a GPU."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2608_09703_gb300 import binding as B
from paper_2608_09703_gb300 import build as mbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mls.h")


@pytest.fixture(scope="module")
def lib():
    mbuild.build()
    return B.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mls_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("mls_workspace_size", "mls_head_loss_fwd", "mls_head_loss_bwd",
                 "mls_get_status", "mls_strerror"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", B.library_path()], capture_output=True,
                         text=True, check=True).stdout
    exported = set(l.split()[-1] for l in out.splitlines() if l.strip())
    for name in declared_functions():
        assert name in exported, name
        assert hasattr(lib, name)


def test_library_is_built_for_sm_103a(lib):
    out = subprocess.run(["cuobjdump", "--list-elf", B.library_path()], capture_output=True,
                         text=True).stdout
    assert "sm_103a" in out


def test_strerror_and_codes(lib):
    assert B.mls_strerror(0) == "success"
    for c in (B.MLS_ERR_ARG, B.MLS_ERR_ALIGN, B.MLS_ERR_UNSUPPORTED, B.MLS_ERR_WORKSPACE,
              B.MLS_ERR_CUDA, B.MLS_ERR_DEVICE, B.MLS_STATUS_BAD_TARGET, B.MLS_STATUS_TIMEOUT):
        assert B.mls_strerror(c) != "unknown code"


def _call_fwd(lib, prob, hptr=0x1000, wptr=0x1000):
    M = prob.M
    H = (ctypes.c_void_p * M)(*([hptr] * M))
    W = (ctypes.c_void_p * M)(*([wptr] * M))
    p = ctypes.c_void_p(0x2000)
    return lib.mls_head_loss_fwd(prob.ref(), H, W, p, p, p, None, None, p, p, 1 << 30, None)


def test_validation_without_gpu(lib):
    # invalid problems are rejected before any CUDA call
    assert _call_fwd(lib, B.Problem([64, 64], 10, 100, tau=0.0)) == B.MLS_ERR_ARG
    assert _call_fwd(lib, B.Problem([64, 64], 10, 100, alpha=1.5)) == B.MLS_ERR_ARG
    assert _call_fwd(lib, B.Problem([64, 64], 10, 100, teacher=2)) == B.MLS_ERR_ARG
    assert _call_fwd(lib, B.Problem([64] * 5, 10, 100)) == B.MLS_ERR_ARG
    assert _call_fwd(lib, B.Problem([64, 60], 10, 100)) == B.MLS_ERR_UNSUPPORTED
    assert _call_fwd(lib, B.Problem([64, 64], 10, 100, vocab_group=100)) == B.MLS_ERR_ARG
    assert _call_fwd(lib, B.Problem([64, 64], 10, 100), hptr=0x1008) == B.MLS_ERR_ALIGN
    assert lib.mls_head_loss_fwd(None, None, None, None, None, None, None, None, None, None, 0,
                                 None) == B.MLS_ERR_ARG


def test_workspace_size(lib):
    small = B.mls_workspace_size(B.Problem([128, 256], 256, 1024, in_dtype=B.MLS_FP32))
    assert small > 0
    big = B.mls_workspace_size(B.Problem([1024, 2048, 3072], 8192, 50304))
    assert big > small
    # the backward's vocabulary group bounds the gradient workspace
    g256 = B.mls_workspace_size(B.Problem([1024, 2048, 3072], 8192, 50304, vocab_group=256))
    assert g256 < big
    assert B.mls_workspace_size(B.Problem([64, 64], 10, 100, tau=-1.0)) == 0


def test_spec_verify_validation_without_gpu(lib):
    """The verify step's host checks: invalid problems and arguments are
    rejected before any CUDA call; the workspace holds the fp32 logits of every
    verify position plus small per-row state."""
    ws = ctypes.c_void_p(0x100000)

    def call(p, h=0x1000, t=0x2000, u=0x3000, size=1 << 40):
        return lib.mls_spec_verify(ctypes.byref(p), h, h, h, h, t, u, t, t, ws, size, None)

    for kw in (dict(top_p=0.0), dict(top_p=1.5), dict(temperature=0.0), dict(temperature=-1.0)):
        args = dict(B=4, gamma=2, V=100, d_draft=64, d_verify=64)
        args.update(kw)
        p = B.spec_problem(**args)
        assert call(p) == B.MLS_ERR_ARG
        assert B.mls_spec_workspace_size(p) == 0
    assert call(B.spec_problem(-1, 2, 100, 64, 64)) == B.MLS_ERR_ARG
    assert call(B.spec_problem(4, -1, 100, 64, 64)) == B.MLS_ERR_ARG
    assert call(B.spec_problem(4, 2, 0, 64, 64)) == B.MLS_ERR_ARG
    assert call(B.spec_problem(4, 2, 100, 60, 64)) == B.MLS_ERR_UNSUPPORTED
    assert call(B.spec_problem(4, 2, 100, 64, 60)) == B.MLS_ERR_UNSUPPORTED
    # greedy ignores the draft model's width, temperature and top_p
    assert B.mls_spec_workspace_size(B.spec_problem(4, 2, 100, 60, 64, 0.0, 0.0, True)) > 0
    assert call(B.spec_problem(4, 2, 100, 64, 64), h=0x1008) == B.MLS_ERR_ALIGN
    assert call(B.spec_problem(4, 2, 100, 64, 64), u=0) == B.MLS_ERR_ARG
    assert call(B.spec_problem(4, 2, 100, 64, 64), size=1024) == B.MLS_ERR_WORKSPACE
    assert call(B.spec_problem(0, 2, 100, 64, 64)) == B.MLS_OK  # nothing to do
    # sizes: sampling keeps a row of fp32 probabilities per verify position
    # (padded to 4 floats); greedy keeps only per-tile maxima
    ldz = 4 * ((101 + 3) // 4)
    samp = B.mls_spec_workspace_size(B.spec_problem(4, 2, 101, 64, 64))
    greedy = B.mls_spec_workspace_size(B.spec_problem(4, 2, 101, 64, 64, greedy=True))
    assert samp - greedy >= 4 * (4 * 3 + 4 * 2) * ldz
    assert 0 < greedy < 4 * 4 * 3 * ldz
    # sampling keeps a per-tile table in shared memory: V <= 4096 tiles of 256
    assert call(B.spec_problem(4, 2, 4096 * 256 + 1, 64, 64)) == B.MLS_ERR_UNSUPPORTED
    assert B.mls_spec_workspace_size(B.spec_problem(4, 2, 4096 * 256 + 1, 64, 64, greedy=True)) > 0


def test_checked_build_compiles():
    """The checked build (invariant checks compiled in) builds and exports the
    same entry points as the normal one."""
    path = mbuild.build(checked=True)
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True,
                         check=True).stdout
    exported = set(l.split()[-1] for l in out.splitlines() if l.strip())
    for name in declared_functions():
        assert name in exported, name
