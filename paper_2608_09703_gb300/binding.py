"""Python binding of the C ABI in include/mls.h (argument marshalling only).

Every function here has the name of the C entry point it wraps and does
nothing but turn torch tensors into device pointers and the current CUDA
stream into a stream handle; all computation happens in libmls.so.  There is
no fallback: if the library is missing or fails to load, the call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

# MLS_CHECKED=1 selects the checked build (invariant checks in the kernels).
_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)),
                         "libmls_checked.so" if os.environ.get("MLS_CHECKED") == "1"
                         else "libmls.so")
_lib = None

MLS_BF16, MLS_FP32 = 0, 1
MLS_OK = 0
MLS_ERR_ARG, MLS_ERR_ALIGN, MLS_ERR_UNSUPPORTED = -1, -2, -3
MLS_ERR_WORKSPACE, MLS_ERR_CUDA, MLS_ERR_DEVICE = -4, -5, -6
MLS_STATUS_BAD_TARGET, MLS_STATUS_TIMEOUT, MLS_STATUS_CHECK, MLS_STATUS_DRAIN = 1, 2, 4, 8
MLS_MAX_MODELS = 4


class MLSError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {mls_strerror(code)} (code {code})")
        self.code = code


class mls_problem(ctypes.Structure):
    _fields_ = [
        ("M", ctypes.c_int32),
        ("T", ctypes.c_int64),
        ("V", ctypes.c_int64),
        ("d", ctypes.POINTER(ctypes.c_int32)),
        ("teacher", ctypes.c_int32),
        ("tau", ctypes.c_float),
        ("alpha", ctypes.c_float),
        ("w", ctypes.POINTER(ctypes.c_float)),
        ("in_dtype", ctypes.c_int32),
        ("vocab_group", ctypes.c_int64),
    ]


class mls_spec_problem(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32),
        ("gamma", ctypes.c_int32),
        ("V", ctypes.c_int64),
        ("d_draft", ctypes.c_int32),
        ("d_verify", ctypes.c_int32),
        ("temperature", ctypes.c_float),
        ("top_p", ctypes.c_float),
        ("greedy", ctypes.c_int32),
        ("in_dtype", ctypes.c_int32),
    ]


class mls_kernel_time(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("launches", ctypes.c_int), ("total_ms", ctypes.c_double)]


def library_path() -> str:
    return _LIB_PATH


def lib():
    """The loaded libmls.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: build it with "
                               "`python -m paper_2608_09703_gb300.build`"
                               + (" --checked" if _LIB_PATH.endswith("_checked.so") else ""))
        L = ctypes.CDLL(_LIB_PATH)
        P = ctypes.POINTER(mls_problem)
        vp = ctypes.c_void_p
        vpp = ctypes.POINTER(ctypes.c_void_p)
        L.mls_workspace_size.argtypes = [P]
        L.mls_workspace_size.restype = ctypes.c_size_t
        L.mls_head_loss_fwd.argtypes = [P, vpp, vpp, vp, vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
        L.mls_head_loss_fwd.restype = ctypes.c_int
        L.mls_head_loss_bwd.argtypes = [P, vpp, vpp, vp, vp, ctypes.c_float, vpp, vpp, vp,
                                        ctypes.c_size_t, vp]
        L.mls_head_loss_bwd.restype = ctypes.c_int
        L.mls_get_status.argtypes = [vp]
        L.mls_get_status.restype = ctypes.c_int
        L.mls_strerror.argtypes = [ctypes.c_int]
        L.mls_strerror.restype = ctypes.c_char_p
        L.mls_head_pairwise.argtypes = [P, vpp, vpp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
        L.mls_head_pairwise.restype = ctypes.c_int
        i64, i32 = ctypes.c_int64, ctypes.c_int32
        L.mls_junction_fwd.argtypes = [i64, i32, i32, i32, i32, vp, vp, vp, vp]
        L.mls_junction_fwd.restype = ctypes.c_int
        L.mls_junction_bwd.argtypes = [i64, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp]
        L.mls_junction_bwd.restype = ctypes.c_int
        L.mls_head_loss_fwd_noalloc.argtypes = [P, vpp, vpp, vp, vp, vp, vp, vp, vp, vp]
        L.mls_head_loss_fwd_noalloc.restype = ctypes.c_int
        SP = ctypes.POINTER(mls_spec_problem)
        L.mls_spec_workspace_size.argtypes = [SP]
        L.mls_spec_workspace_size.restype = ctypes.c_size_t
        L.mls_spec_verify.argtypes = [SP, vp, vp, vp, vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
        L.mls_spec_verify.restype = ctypes.c_int
        L.mls_profile_enable.argtypes = [ctypes.c_int]
        L.mls_profile_enable.restype = ctypes.c_int
        L.mls_profile_read.argtypes = [ctypes.POINTER(mls_kernel_time), ctypes.c_int]
        L.mls_profile_read.restype = ctypes.c_int
        _lib = L
    return _lib


class Problem:
    """Owns an mls_problem and the host arrays it points to."""

    def __init__(self, d: Sequence[int], T: int, V: int, teacher: Optional[int] = None,
                 tau: float = 1.0, alpha: float = 0.5, w: Optional[Sequence[float]] = None,
                 in_dtype: int = MLS_BF16, vocab_group: int = 0):
        M = len(d)
        self.d = (ctypes.c_int32 * M)(*[int(x) for x in d])
        self.w = None if w is None else (ctypes.c_float * M)(*[float(x) for x in w])
        self.c = mls_problem(M, int(T), int(V), self.d, M - 1 if teacher is None else int(teacher),
                             float(tau), float(alpha), self.w, int(in_dtype), int(vocab_group))

    @property
    def M(self) -> int:
        return self.c.M

    def ref(self):
        return ctypes.byref(self.c)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _ptrs(ts: Sequence[torch.Tensor]):
    return (ctypes.c_void_p * len(ts))(*[t.data_ptr() for t in ts])


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(rc: int, what: str):
    if rc != MLS_OK:
        raise MLSError(rc, what)


def mls_workspace_size(prob: Problem) -> int:
    return int(lib().mls_workspace_size(prob.ref()))


def mls_head_loss_fwd(prob: Problem, H, W, targets, loss, tok_loss, tok_diag, argmax, stats, ws,
                      stream=None) -> None:
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size()
    rc = lib().mls_head_loss_fwd(prob.ref(), _ptrs(H), _ptrs(W), _ptr(targets), _ptr(loss),
                                 _ptr(tok_loss), _ptr(tok_diag), _ptr(argmax), _ptr(stats), _ptr(ws),
                                 ws_bytes, _stream(stream))
    _check(rc, "mls_head_loss_fwd")


def mls_head_loss_bwd(prob: Problem, H, W, targets, stats, grad_scale: float, dH, dW, ws,
                      stream=None) -> None:
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size()
    rc = lib().mls_head_loss_bwd(prob.ref(), _ptrs(H), _ptrs(W), _ptr(targets), _ptr(stats),
                                 float(grad_scale), _ptrs(dH), _ptrs(dW), _ptr(ws), ws_bytes,
                                 _stream(stream))
    _check(rc, "mls_head_loss_bwd")


def mls_head_pairwise(prob: Problem, H, W, targets, tok_kl, argmax, pair_stats, ws,
                      stream=None) -> None:
    """Per-token KL(p_i || p_j) between sub-models, their means and top-1 agreement."""
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size()
    rc = lib().mls_head_pairwise(prob.ref(), _ptrs(H), _ptrs(W), _ptr(targets), _ptr(tok_kl),
                                 _ptr(argmax), _ptr(pair_stats), _ptr(ws), ws_bytes, _stream(stream))
    _check(rc, "mls_head_pairwise")


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return MLS_BF16
    if t.dtype == torch.float32:
        return MLS_FP32
    raise TypeError(t.dtype)


def mls_junction_fwd(o, e, x, embed_first=False, stream=None) -> None:
    """Eq. 1: x = concat(o * ||e|| / ||o||, e) per row (concat(e, ...) if embed_first)."""
    T, dp = o.shape
    rc = lib().mls_junction_fwd(T, dp, dp + e.shape[1], _dtype_code(o), int(bool(embed_first)),
                                _ptr(o), _ptr(e), _ptr(x), _stream(stream))
    _check(rc, "mls_junction_fwd")


def mls_junction_bwd(o, e, g, d_o, d_e, embed_first=False, stream=None) -> None:
    T, dp = o.shape
    rc = lib().mls_junction_bwd(T, dp, dp + e.shape[1], _dtype_code(o), int(bool(embed_first)),
                                _ptr(o), _ptr(e), _ptr(g), _ptr(d_o), _ptr(d_e), _stream(stream))
    _check(rc, "mls_junction_bwd")


def spec_problem(B: int, gamma: int, V: int, d_draft: int, d_verify: int,
                 temperature: float = 0.4, top_p: float = 0.9, greedy: bool = False,
                 in_dtype: int = MLS_BF16) -> mls_spec_problem:
    return mls_spec_problem(int(B), int(gamma), int(V), int(d_draft), int(d_verify),
                            float(temperature), float(top_p), int(bool(greedy)), int(in_dtype))


def mls_spec_workspace_size(p: mls_spec_problem) -> int:
    return int(lib().mls_spec_workspace_size(ctypes.byref(p)))


def mls_spec_verify(p: mls_spec_problem, H_draft, W_draft, H_verify, W_verify, draft_tokens,
                    uniforms, n_accepted, next_token, ws, stream=None) -> None:
    """Speculative-decoding verify step (see include/mls.h)."""
    rc = lib().mls_spec_verify(ctypes.byref(p), _ptr(H_draft), _ptr(W_draft), _ptr(H_verify),
                               _ptr(W_verify), _ptr(draft_tokens), _ptr(uniforms),
                               _ptr(n_accepted), _ptr(next_token), _ptr(ws),
                               0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))
    _check(rc, "mls_spec_verify")


def mls_head_loss_fwd_noalloc(prob: Problem, H, W, targets, loss, tok_loss, tok_diag, argmax,
                              stats, stream=None) -> None:
    """Forward with the library's built-in scratch instead of a workspace, for
    callers that cannot allocate device memory when they call; allocates nothing."""
    rc = lib().mls_head_loss_fwd_noalloc(prob.ref(), _ptrs(H), _ptrs(W), _ptr(targets), _ptr(loss),
                                         _ptr(tok_loss), _ptr(tok_diag), _ptr(argmax), _ptr(stats),
                                         _stream(stream))
    _check(rc, "mls_head_loss_fwd_noalloc")


MLS_NOALLOC_SCRATCH_BYTES = 64 << 20


def mls_get_status(stream=None) -> int:
    rc = lib().mls_get_status(_stream(stream))
    if rc < 0:
        raise MLSError(rc, "mls_get_status")
    return rc


def mls_strerror(code: int) -> str:
    try:
        return lib().mls_strerror(int(code)).decode()
    except Exception:  # library missing: still describe the code
        return f"code {code}"


def mls_profile_enable(on: bool = True) -> None:
    lib().mls_profile_enable(1 if on else 0)


def mls_profile_read() -> dict:
    """{kernel name: (launches, total device ms)} since the last enable/read."""
    buf = (mls_kernel_time * 32)()
    n = lib().mls_profile_read(buf, 32)
    if n < 0:
        raise MLSError(n, "mls_profile_read")
    return {buf[i].name.decode(): (buf[i].launches, buf[i].total_ms) for i in range(min(n, 32))}


# ----------------------------------------------------------------------------------------
# Convenience layer: allocates outputs and workspace with torch, then calls the entry points.
class HeadLoss:
    """Fused suite head + CE + distillation loss over device tensors.

    H[m]: [T, d_m], W[m]: [V, d_m] (bf16 or fp32, contiguous, on one CUDA
    device); targets: int32 [T].  Buffers are allocated once per shape.
    """

    def __init__(self, d, T, V, teacher=None, tau=1.0, alpha=0.5, w=None, dtype=torch.bfloat16,
                 device="cuda", vocab_group=0):
        self.prob = Problem(d, T, V, teacher, tau, alpha, w,
                            MLS_BF16 if dtype == torch.bfloat16 else MLS_FP32, vocab_group)
        M = len(d)
        self.M, self.T, self.V, self.d = M, T, V, list(d)
        dev = torch.device(device)
        self.loss = torch.zeros(1, dtype=torch.float32, device=dev)
        self.tok_loss = torch.empty(M, T, dtype=torch.float32, device=dev)
        self.tok_diag = torch.empty(3, M, T, dtype=torch.float32, device=dev)
        self.argmax = torch.empty(M, T, dtype=torch.int32, device=dev)
        self.stats = torch.empty(2, M, T, dtype=torch.float32, device=dev)
        self.dH = [torch.empty(T, dm, dtype=torch.float32, device=dev) for dm in d]
        self.dW = [torch.empty(V, dm, dtype=torch.float32, device=dev) for dm in d]
        nbytes = mls_workspace_size(self.prob)
        self.ws = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=dev)

    def forward(self, H, W, targets, stream=None):
        mls_head_loss_fwd(self.prob, H, W, targets, self.loss, self.tok_loss, self.tok_diag,
                          self.argmax, self.stats, self.ws, stream)
        return self.loss

    def pairwise(self, H, W, targets=None, stream=None):
        """Evaluation metrics between sub-models; returns (tok_kl [M,M,T],
        argmax [M,T], pair_stats [2,M,M])."""
        dev = self.loss.device
        if not hasattr(self, "tok_kl"):
            self.tok_kl = torch.empty(self.M, self.M, self.T, dtype=torch.float32, device=dev)
            self.pair_stats = torch.empty(2, self.M, self.M, dtype=torch.float32, device=dev)
            self.eval_argmax = torch.empty(self.M, self.T, dtype=torch.int32, device=dev)
        mls_head_pairwise(self.prob, H, W, targets, self.tok_kl, self.eval_argmax, self.pair_stats,
                          self.ws, stream)
        return self.tok_kl, self.eval_argmax, self.pair_stats

    def backward(self, H, W, targets, grad_scale=1.0, stream=None):
        mls_head_loss_bwd(self.prob, H, W, targets, self.stats, grad_scale, self.dH, self.dW,
                          self.ws, stream)
        return self.dH, self.dW


class SpecVerify:
    """Speculative-decoding verify step with its outputs and workspace
    allocated once per shape.  H_draft: [B*gamma, d_draft], W_draft:
    [V, d_draft], H_verify: [B*(gamma+1), d_verify], W_verify: [V, d_verify]
    (bf16 or fp32); draft_tokens int32 [B, gamma]; uniforms fp32
    [B, gamma+1, 2]."""

    def __init__(self, B, gamma, V, d_draft, d_verify, temperature=0.4, top_p=0.9, greedy=False,
                 dtype=torch.bfloat16, device="cuda"):
        self.p = spec_problem(B, gamma, V, d_draft, d_verify, temperature, top_p, greedy,
                              MLS_BF16 if dtype == torch.bfloat16 else MLS_FP32)
        dev = torch.device(device)
        self.n_accepted = torch.empty(B, dtype=torch.int32, device=dev)
        self.next_token = torch.empty(B, dtype=torch.int32, device=dev)
        self.ws = torch.empty(max(mls_spec_workspace_size(self.p), 1), dtype=torch.uint8,
                              device=dev)

    def __call__(self, H_draft, W_draft, H_verify, W_verify, draft_tokens, uniforms, stream=None):
        mls_spec_verify(self.p, H_draft, W_draft, H_verify, W_verify, draft_tokens, uniforms,
                        self.n_accepted, self.next_token, self.ws, stream)
        return self.n_accepted, self.next_token
