"""ctypes wrapper around the fp64 CPU oracle (``mls_oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by the tests, by the package's smoke check
and by the CPU-baseline leg of the benchmark.  The product path never imports
it.  The oracle materialises every logit row and follows the paper's
definitions (Eq. 2, Eq. 3 and the sum over sub-models) in double precision.

Inputs are numpy arrays: H[m] of shape [T, d_m], W[m] of shape [V, d_m], stored
either as bf16 bit patterns (``np.uint16``) or as ``np.float32`` (``np.float64`` for finite-difference checks); targets are
``np.int32`` of shape [T] (negative = ignored).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mls_oracle.c")
_LIB = os.path.join(_HERE, "libmls_oracle.so")
_lock = threading.Lock()
_lib = None


class _Problem(ctypes.Structure):
    _fields_ = [
        ("M", ctypes.c_int),
        ("T", ctypes.c_longlong),
        ("V", ctypes.c_longlong),
        ("d", ctypes.POINTER(ctypes.c_int)),
        ("teacher", ctypes.c_int),
        ("tau", ctypes.c_double),
        ("alpha", ctypes.c_double),
        ("w", ctypes.POINTER(ctypes.c_double)),
        ("in_dtype", ctypes.c_int),
    ]


def build(force: bool = False) -> str:
    """Compile the oracle into a shared library next to its source."""
    with _lock:
        if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
            tmp = _LIB + f".tmp{os.getpid()}"
            subprocess.check_call(
                ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
            )
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.POINTER(_Problem)
        vpp = ctypes.POINTER(ctypes.c_void_p)
        dpp = ctypes.POINTER(ctypes.POINTER(ctypes.c_double))
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int)
        lib.mls_oracle_fwd.argtypes = [P, vpp, vpp, ip, dp, dp, dp, ip, dp]
        lib.mls_oracle_fwd.restype = ctypes.c_int
        lib.mls_oracle_bwd.argtypes = [P, vpp, vpp, ip, ctypes.c_double, dpp, dpp]
        lib.mls_oracle_bwd.restype = ctypes.c_int
        lib.mls_oracle_rows.argtypes = [P, vpp, vpp, ip, ctypes.POINTER(ctypes.c_longlong),
                                        ctypes.c_int, ctypes.c_longlong, ctypes.c_double,
                                        dp, dp, ip, dp, dpp]
        lib.mls_oracle_rows.restype = ctypes.c_int
        lib.mls_oracle_pairwise.argtypes = [P, vpp, vpp, dp, ip]
        lib.mls_oracle_pairwise.restype = ctypes.c_int
        lib.mls_oracle_junction_fwd.argtypes = [ctypes.c_longlong, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                                ctypes.c_void_p, dp]
        lib.mls_oracle_junction_fwd.restype = ctypes.c_int
        lib.mls_oracle_junction_bwd.argtypes = [ctypes.c_longlong, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                                ctypes.c_void_p, ctypes.c_void_p, dp, dp]
        lib.mls_oracle_junction_bwd.restype = ctypes.c_int
        lib.mls_oracle_spec_verify.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_longlong,
                                               ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                               ctypes.c_double, ctypes.c_double, ctypes.c_int,
                                               ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                               ctypes.c_void_p, ip, dp, ip, ip]
        lib.mls_oracle_spec_verify.restype = ctypes.c_int
        lib.mls_oracle_threads.argtypes = []
        lib.mls_oracle_threads.restype = ctypes.c_int
        _lib = lib
    return _lib


def threads() -> int:
    return int(_load().mls_oracle_threads())


def _as_input(a: np.ndarray) -> tuple[np.ndarray, int]:
    if a.dtype == np.uint16:
        return np.ascontiguousarray(a), 0
    if a.dtype == np.float32:
        return np.ascontiguousarray(a), 1
    if a.dtype == np.float64:
        return np.ascontiguousarray(a), 2
    raise TypeError(f"oracle inputs must be bf16 bits (uint16), float32 or float64, got {a.dtype}")


class _Args:
    """Marshals one problem; keeps every buffer alive while the call runs."""

    def __init__(self, H, W, y, teacher, tau, alpha, w):
        M = len(H)
        assert len(W) == M and M >= 1
        hs, dts = zip(*[_as_input(h) for h in H])
        ws_, dtw = zip(*[_as_input(x) for x in W])
        dt = set(dts) | set(dtw)
        if len(dt) != 1:
            raise TypeError("H and W must share one storage type")
        self.H, self.W = list(hs), list(ws_)
        self.T = int(self.H[0].shape[0])
        self.V = int(self.W[0].shape[0])
        self.d = [int(h.shape[1]) for h in self.H]
        for m in range(M):
            assert self.H[m].shape == (self.T, self.d[m]), "H[m] must be [T, d_m]"
            assert self.W[m].shape == (self.V, self.d[m]), "W[m] must be [V, d_m]"
        self.y = np.ascontiguousarray(np.asarray(y, dtype=np.int32))
        assert self.y.shape == (self.T,)
        self.d_arr = (ctypes.c_int * M)(*self.d)
        self.w_arr = None if w is None else (ctypes.c_double * M)(*[float(x) for x in w])
        self.prob = _Problem(M, self.T, self.V, self.d_arr, int(teacher), float(tau), float(alpha),
                             self.w_arr, dt.pop())
        self.Hp = (ctypes.c_void_p * M)(*[h.ctypes.data for h in self.H])
        self.Wp = (ctypes.c_void_p * M)(*[x.ctypes.data for x in self.W])
        self.M = M

    def yp(self):
        return self.y.ctypes.data_as(ctypes.POINTER(ctypes.c_int))


def _dp(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _check(rc: int, what: str):
    if rc != 0:
        raise RuntimeError(f"{what} failed with code {rc}")


def forward(H, W, y, teacher=None, tau=1.0, alpha=0.5, w=None) -> dict:
    """Full forward: scalar loss and every per-token output (fp64)."""
    teacher = len(H) - 1 if teacher is None else teacher
    a = _Args(H, W, y, teacher, tau, alpha, w)
    M, T = a.M, a.T
    loss = np.zeros(1, np.float64)
    tok = np.zeros((M, T), np.float64)
    diag = np.zeros((3, M, T), np.float64)
    am = np.zeros((M, T), np.int32)
    st = np.zeros((2, M, T), np.float64)
    rc = _load().mls_oracle_fwd(ctypes.byref(a.prob), a.Hp, a.Wp, a.yp(), _dp(loss), _dp(tok),
                                _dp(diag), am.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), _dp(st))
    _check(rc, "mls_oracle_fwd")
    return {"loss": float(loss[0]), "tok_loss": tok, "ce": diag[0], "ld": diag[1], "kl": diag[2],
            "argmax": am, "lse": st[0], "lse_tau": st[1]}


def backward(H, W, y, teacher=None, tau=1.0, alpha=0.5, w=None, grad_scale=1.0):
    """Full backward: lists dH[m] [T, d_m] and dW[m] [V, d_m] (fp64)."""
    teacher = len(H) - 1 if teacher is None else teacher
    a = _Args(H, W, y, teacher, tau, alpha, w)
    dH = [np.zeros((a.T, d), np.float64) for d in a.d]
    dW = [np.zeros((a.V, d), np.float64) for d in a.d]
    dHp = (ctypes.POINTER(ctypes.c_double) * a.M)(*[_dp(x) for x in dH])
    dWp = (ctypes.POINTER(ctypes.c_double) * a.M)(*[_dp(x) for x in dW])
    rc = _load().mls_oracle_bwd(ctypes.byref(a.prob), a.Hp, a.Wp, a.yp(), float(grad_scale), dHp, dWp)
    _check(rc, "mls_oracle_bwd")
    return dH, dW


def rows(H, W, y, rows_idx, teacher=None, tau=1.0, alpha=0.5, w=None, grad_scale=1.0,
         with_dh=True) -> dict:
    """Per-token outputs (and dH rows) for the selected tokens of a large problem."""
    teacher = len(H) - 1 if teacher is None else teacher
    a = _Args(H, W, y, teacher, tau, alpha, w)
    r = np.ascontiguousarray(np.asarray(rows_idx, dtype=np.int64))
    n = int(r.shape[0])
    M = a.M
    n_valid = int((a.y >= 0).sum())
    tok = np.zeros((M, n), np.float64)
    diag = np.zeros((3, M, n), np.float64)
    am = np.zeros((M, n), np.int32)
    st = np.zeros((2, M, n), np.float64)
    dH = [np.zeros((n, d), np.float64) for d in a.d] if with_dh else None
    dHp = (ctypes.POINTER(ctypes.c_double) * M)(*[_dp(x) for x in dH]) if with_dh else None
    rc = _load().mls_oracle_rows(ctypes.byref(a.prob), a.Hp, a.Wp, a.yp(),
                                 r.ctypes.data_as(ctypes.POINTER(ctypes.c_longlong)), n, n_valid,
                                 float(grad_scale), _dp(tok), _dp(diag),
                                 am.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), _dp(st), dHp)
    _check(rc, "mls_oracle_rows")
    out = {"tok_loss": tok, "ce": diag[0], "ld": diag[1], "kl": diag[2], "argmax": am,
           "lse": st[0], "lse_tau": st[1], "n_valid": n_valid}
    if with_dh:
        out["dH"] = dH
    return out


def pairwise(H, W) -> dict:
    """Per-token KL(p_i || p_j) [M, M, T] and top-1 agreement [M, M, T] (fp64)."""
    T = H[0].shape[0]
    a = _Args(H, W, np.zeros(T, np.int32), len(H) - 1, 1.0, 0.0, None)
    M = a.M
    kl = np.zeros((M, M, T), np.float64)
    agree = np.zeros((M, M, T), np.int32)
    rc = _load().mls_oracle_pairwise(ctypes.byref(a.prob), a.Hp, a.Wp, _dp(kl),
                                     agree.ctypes.data_as(ctypes.POINTER(ctypes.c_int)))
    _check(rc, "mls_oracle_pairwise")
    return {"kl": kl, "agree": agree}


def junction_fwd(o, e, embed_first=False):
    """Eq. 1: x = concat(o * ||e|| / ||o||, e) per row (or concat(e, ...) with
    embed_first); o [T, D_m], e [T, D_{m+1} - D_m] -> x [T, D_{m+1}] fp64."""
    (o, dt), (e, dt2) = _as_input(o), _as_input(e)
    assert dt == dt2
    T, dp_ = o.shape
    de = e.shape[1]
    x = np.zeros((T, dp_ + de), np.float64)
    rc = _load().mls_oracle_junction_fwd(T, dp_, dp_ + de, dt, int(embed_first), o.ctypes.data,
                                         e.ctypes.data, _dp(x))
    _check(rc, "mls_oracle_junction_fwd")
    return x


def junction_bwd(o, e, g, embed_first=False):
    """Gradients (dL/do, dL/de) of the junction for upstream g = dL/dx (fp64)."""
    (o, dt), (e, _), (g, dt3) = _as_input(o), _as_input(e), _as_input(g)
    assert dt == dt3
    T, dp_ = o.shape
    de = e.shape[1]
    d_o = np.zeros((T, dp_), np.float64)
    d_e = np.zeros((T, de), np.float64)
    rc = _load().mls_oracle_junction_bwd(T, dp_, dp_ + de, dt, int(embed_first), o.ctypes.data,
                                         e.ctypes.data, g.ctypes.data, _dp(d_o), _dp(d_e))
    _check(rc, "mls_oracle_junction_bwd")
    return d_o, d_e


def spec_verify(Hd, Wd, Hv, Wv, draft, u, temperature=0.4, top_p=0.9, greedy=False):
    """Speculative-decoding verify step (fp64): Hd [B*gamma, d_d], Hv [B*(gamma+1), d_v],
    heads Wd [V, d_d], Wv [V, d_v], draft tokens [B, gamma], uniforms u [B, gamma+1, 2].
    Returns (n_accepted [B], next_token [B])."""
    (Hd, dt), (Wd, _), (Hv, _), (Wv, _) = (_as_input(a) for a in (Hd, Wd, Hv, Wv))
    draft = np.ascontiguousarray(np.asarray(draft, np.int32))
    B, gamma = draft.shape
    u = np.ascontiguousarray(np.asarray(u, np.float64))
    assert u.shape == (B, gamma + 1, 2)
    V = Wv.shape[0]
    n = np.zeros(B, np.int32)
    nxt = np.zeros(B, np.int32)
    ip_ = ctypes.POINTER(ctypes.c_int)
    rc = _load().mls_oracle_spec_verify(B, gamma, V, Wd.shape[1], Wv.shape[1], dt, float(temperature),
                                        float(top_p), int(bool(greedy)), Hd.ctypes.data,
                                        Wd.ctypes.data, Hv.ctypes.data, Wv.ctypes.data,
                                        draft.ctypes.data_as(ip_), _dp(u), n.ctypes.data_as(ip_),
                                        nxt.ctypes.data_as(ip_))
    _check(rc, "mls_oracle_spec_verify")
    return n, nxt
