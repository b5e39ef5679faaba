"""Thin ctypes binding of the C ABI in ``include/fibattn.h``.

Argument marshalling only: tensors are passed as raw device pointers with the
caller's current CUDA stream; every step of the computation runs in the CUDA
library.  The binding raises ``RuntimeError`` when the library is missing or
a call returns a non-OK status -- there is no fallback.
"""
from __future__ import annotations

import ctypes
import functools
import os
import threading

import numpy as np
import torch

from . import build as _build

FIBATTN_F32 = 0
FIBATTN_BF16 = 1
FIBATTN_ERR_UNSUPPORTED = 2
_STATUS = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "CUDA", 4: "INTERNAL"}

_lock = threading.Lock()
_lib = None


class FibattnError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"fibattn {_STATUS.get(status, status)}: {message}")
        self.status = status


class Opts(ctypes.Structure):
    _fields_ = [("rope_base", ctypes.c_float), ("scale", ctypes.c_float),
                ("Hkv", ctypes.c_int), ("no_dedup", ctypes.c_int), ("fwd_kernel", ctypes.c_int),
                ("bwd_kernel", ctypes.c_int), ("rotated_k", ctypes.c_void_p), ("residuals", ctypes.c_void_p),
                ("round_offsets", ctypes.c_int)]


def library_path() -> str:
    return _build.LIB


def lib():
    """Load the CUDA library (it must have been built: ``__graft_entry__.build()``)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(f"CUDA library not built ({path} missing); run __graft_entry__.build()")
            L = ctypes.CDLL(path)
            vp, sz, ci, cf = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_float
            fp = ctypes.POINTER(ctypes.c_float)
            ip = ctypes.POINTER(ctypes.c_int)
            op = ctypes.POINTER(Opts)
            L.fibattn_fwd_workspace_bytes.argtypes = [ci] * 7 + [op]
            L.fibattn_fwd_workspace_bytes.restype = sz
            L.fibattn_fwd.argtypes = [vp, vp, vp, vp, vp, ci, ci, ci, ci, ci, cf, vp, ci, ci, op, vp, sz, vp]
            L.fibattn_fwd.restype = ci
            L.fibattn_bwd_workspace_bytes.argtypes = [ci] * 7 + [op]
            L.fibattn_bwd_workspace_bytes.restype = sz
            L.fibattn_bwd.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, ci, ci, ci, ci, ci, cf, vp, ci, ci,
                                      op, vp, sz, vp]
            L.fibattn_bwd.restype = ci
            L.fibattn_last_error.argtypes = []
            L.fibattn_last_error.restype = ctypes.c_char_p
            L.fibattn_rung_params.argtypes = [cf, fp, ci, ci, ci, ci, fp, ip, fp, ip]
            L.fibattn_rung_params.restype = ci
            L.fibattn_base.argtypes = [ci, ci, fp]
            L.fibattn_base.restype = ci
            L.fibattn_alpha_schedule.argtypes = [ci, ci, fp, ci, fp]
            L.fibattn_alpha_schedule.restype = ci
            L.fibattn_theta_of_alpha.argtypes = [ci, fp, fp]
            L.fibattn_theta_of_alpha.restype = ci
            L.fibattn_residual_bytes.argtypes = [ci] * 7
            L.fibattn_residual_bytes.restype = sz
            L.fibattn_check_status.argtypes = [vp, ctypes.POINTER(ctypes.c_uint)]
            L.fibattn_check_status.restype = ci
            L.fibattn_test_wait_timeout.argtypes = [ctypes.c_uint, vp]
            L.fibattn_test_wait_timeout.restype = ci
            _lib = L
    return _lib


def _check(rc: int):
    if rc != 0:
        raise FibattnError(rc, lib().fibattn_last_error().decode(errors="replace"))


def _fptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_float))


def _iptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int))


FWD_KERNELS = {"auto": 0, "gather": 1, "mma": 3}
BWD_KERNELS = {"auto": 0, "gather": 1, "mma": 2}


def _opts(rope_base=1e4, scale=None, Hkv=None, dedup=True, fwd_kernel="auto", bwd_kernel="auto",
          rotated_k=None, residuals=None, round_offsets=False) -> Opts:
    return Opts(float(rope_base), float(scale) if scale else 0.0, int(Hkv or 0), 0 if dedup else 1,
                FWD_KERNELS[fwd_kernel], BWD_KERNELS[bwd_kernel],
                rotated_k.data_ptr() if rotated_k is not None else None,
                residuals.data_ptr() if residuals is not None else None, 1 if round_offsets else 0)


@functools.lru_cache(maxsize=256)
def _residual_bytes(B, H, T, W, K, bf16, D) -> int:
    return int(lib().fibattn_residual_bytes(B, H, T, D, W, K, FIBATTN_BF16 if bf16 else FIBATTN_F32))


def residual_bytes(B, H, T, W, K, dtype=torch.bfloat16, D=64) -> int:
    """Size of the forward residuals (``residuals=``); 0 for fp32 I/O."""
    return _residual_bytes(int(B), int(H), int(T), int(W), int(K), dtype == torch.bfloat16, int(D))


def residuals_like(q: torch.Tensor, W: int, K: int) -> torch.Tensor:
    """A buffer for the forward residuals of queries like q (bf16 I/O): the
    forward fills it, the backward of the same inputs reads it."""
    B, H, T, D = q.shape
    n = residual_bytes(B, H, T, W, K, q.dtype, D)
    if n == 0:
        raise ValueError("forward residuals need bf16 I/O")
    return torch.empty(n, dtype=torch.uint8, device=q.device)


def residual_views(res: torch.Tensor, B, H, T, W, K):
    """Views of a residual buffer: rotated q (bf16 [B,H,T,64]), the
    unnormalised softmax weight exp(s - max) per slot (fp32 [B,H,W+1+K,T]),
    far-minus-floor rung scores (fp32 [B,H,K,T]) and 1 / (sum of the weights)
    per query (fp32 [B,H,T]; p = weight * that); the arrays follow one another,
    each from the next multiple of 256 bytes."""
    def up(x):
        return (x + 255) // 256 * 256
    n = B * H * T
    S = W + 1 + K
    o_p = up(n * 64 * 2)
    o_sd = o_p + up(n * S * 4)
    o_il = o_sd + up(n * K * 4)
    qt = res[:n * 128].view(torch.bfloat16).view(B, H, T, 64)
    P = res[o_p:o_p + n * S * 4].view(torch.float32).view(B, H, S, T)
    sd = res[o_sd:o_sd + n * K * 4].view(torch.float32).view(B, H, K, T)
    il = res[o_il:o_il + n * 4].view(torch.float32).view(B, H, T)
    return qt, P, sd, il


def _check_residuals(res, q, W, K):
    if res is None:
        return
    B, H, T, D = q.shape
    if not (res.is_cuda and res.is_contiguous() and res.numel() * res.element_size() >=
            residual_bytes(B, H, T, W, K, q.dtype, D)):
        raise ValueError("residuals must be a contiguous CUDA buffer of residual_bytes(...) bytes")


def rotated_k_like(k: torch.Tensor) -> torch.Tensor:
    """A buffer for the rotated keys (``rotated_k=``): fp16 for bf16 k, fp32 for fp32 k."""
    return torch.empty(k.shape, dtype=torch.float16 if k.dtype == torch.bfloat16 else torch.float32,
                       device=k.device)


def _check_rotated(rk, k):
    if rk is None:
        return
    want = torch.float16 if k.dtype == torch.bfloat16 else torch.float32
    if not (rk.is_cuda and rk.is_contiguous() and rk.dtype == want and rk.shape == k.shape):
        raise ValueError(f"rotated_k must be a contiguous CUDA {want} tensor of k's shape")


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return FIBATTN_F32
    if t.dtype == torch.bfloat16:
        return FIBATTN_BF16
    raise TypeError(f"unsupported dtype {t.dtype}: fp32 or bf16")


def _stream_ptr(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _offsets(offsets) -> np.ndarray:
    if isinstance(offsets, np.ndarray) and offsets.dtype == np.float32 and offsets.flags.c_contiguous:
        return offsets
    return np.ascontiguousarray(np.asarray(offsets, dtype=np.float32))


# ------------------------------------------------------------- host prep ----

def base(kind: str, K: int) -> np.ndarray:
    f = np.zeros(K, dtype=np.float32)
    _check(lib().fibattn_base({"fib": 0, "pow2": 1}[kind], K, _fptr(f)))
    return f


def alpha_schedule(kind: str, L: int = 16, theta=None, stride: int = 7) -> np.ndarray:
    code = {"fixed": 0, "learned": 1, "linear": 2, "coprime": 3}[kind]
    out = np.zeros(L, dtype=np.float32)
    th = np.ascontiguousarray(np.asarray(theta, dtype=np.float32)) if theta is not None else None
    _check(lib().fibattn_alpha_schedule(code, L, _fptr(th) if th is not None else None, stride, _fptr(out)))
    return out


def theta_of_alpha_array(alpha) -> np.ndarray:
    """theta with 0.5 + sigmoid(theta) = alpha, per entry (fibattn_theta_of_alpha)."""
    a = np.ascontiguousarray(np.atleast_1d(np.asarray(alpha, dtype=np.float32)))
    out = np.zeros(len(a), dtype=np.float32)
    _check(lib().fibattn_theta_of_alpha(len(a), _fptr(a), _fptr(out)))
    return out


def coverage(alphas, offsets, W: int, T: int, dedup: bool = True) -> dict:
    """Distinct key distances of a layer stack (see fibattn_coverage)."""
    al = np.ascontiguousarray(np.asarray(alphas, dtype=np.float32))
    f = _offsets(offsets)
    L = lib()
    ip = ctypes.POINTER(ctypes.c_int)
    L.fibattn_coverage.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_float),
                                   ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ip, ip, ip, ip]
    L.fibattn_coverage.restype = ctypes.c_int
    per = np.zeros(len(al), dtype=np.int32)
    u, bw, hop = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(L.fibattn_coverage(len(al), _fptr(al), _fptr(f), len(f), int(W), int(T), 0 if dedup else 1,
                              _iptr(per), ctypes.byref(u), ctypes.byref(bw), ctypes.byref(hop)))
    return dict(per_layer=per, union=u.value, beyond_window=bw.value, two_hop=hop.value)


def staging_layout(kind: str, T: int, W: int, alpha: float, offsets, dedup: bool = True) -> dict:
    """Shared-memory staging layout of the tensor-core kernels (see
    fibattn_staging_layout): kind "query" (forward, backward query pass) or
    "key" (backward key pass).  Returns the merged intervals (start, len,
    smem arrays) and slab_row per rung (-1 when not staged)."""
    f = _offsets(offsets)
    K = len(f)
    L = lib()
    ip = ctypes.POINTER(ctypes.c_int)
    L.fibattn_staging_layout.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_float,
                                         ctypes.POINTER(ctypes.c_float), ctypes.c_int, ctypes.c_int, ip, ip, ip, ip, ip]
    L.fibattn_staging_layout.restype = ctypes.c_int
    n = ctypes.c_int()
    st, ln, sm = (np.zeros(64, np.int32) for _ in range(3))
    slab = np.zeros(max(K, 1), np.int32)
    _check(L.fibattn_staging_layout({"query": 0, "key": 1}[kind], int(T), int(W), float(alpha), _fptr(f), K,
                                    0 if dedup else 1, ctypes.byref(n), _iptr(st), _iptr(ln), _iptr(sm), _iptr(slab)))
    m = n.value
    return dict(start=st[:m].copy(), len=ln[:m].copy(), smem=sm[:m].copy(), slab_row=slab[:K].copy())


def rung_params(alpha: float, offsets, W: int, dedup: bool = True, round_offsets: bool = False):
    f = _offsets(offsets)
    K = len(f)
    d = np.zeros(K, np.float32); w = np.zeros(K, np.float32)
    s0 = np.zeros(K, np.int32); act = np.zeros(K, np.int32)
    _check(lib().fibattn_rung_params(float(alpha), _fptr(f), K, int(W), 0 if dedup else 1, 1 if round_offsets else 0,
                                     _fptr(d), _iptr(s0), _fptr(w), _iptr(act)))
    return dict(d=d, s0=s0, w=w, active=act.astype(bool))


# --------------------------------------------------------------- compute ----

def fwd_workspace_bytes(B, H, T, W, K, dtype, Hkv=None, D=64) -> int:
    o = _opts(Hkv=Hkv)
    code = FIBATTN_BF16 if dtype == torch.bfloat16 else FIBATTN_F32
    return int(lib().fibattn_fwd_workspace_bytes(B, H, T, D, W, K, code, ctypes.byref(o)))


def bwd_workspace_bytes(B, H, T, W, K, dtype, Hkv=None, D=64) -> int:
    o = _opts(Hkv=Hkv)
    code = FIBATTN_BF16 if dtype == torch.bfloat16 else FIBATTN_F32
    return int(lib().fibattn_bwd_workspace_bytes(B, H, T, D, W, K, code, ctypes.byref(o)))


def fwd(q, k, v, alpha: float, offsets, W: int, *, rope_base=1e4, scale=None, dedup=True,
        out=None, lse=None, workspace=None, stream=None, kernel="auto", rotated_k=None, residuals=None,
        round_offsets=False):
    """Forward pass.  q [B,H,T,64]; k, v [B,Hkv,T,64] (fp32 or bf16, CUDA,
    contiguous).  ``kernel``: "auto", "gather" or "mma".  ``round_offsets``:
    the integer-offset variants (rung distances rounded to integers).
    ``rotated_k``: optional buffer (``rotated_k_like(k)``) that receives the
    rotated keys for a later ``bwd(..., rotated_k=...)``.  ``residuals``:
    optional buffer (``residuals_like(q, W, K)``) that receives the rotated
    queries, p of every slot and the rung score differences for a later
    ``bwd(..., residuals=...)`` (tensor-core forward only).  Returns (out, lse)."""
    B, H, T, D = q.shape
    Hkv = k.shape[1]
    f = _offsets(offsets)
    _check_rotated(rotated_k, k)
    _check_residuals(residuals, q, W, len(f))
    o = _opts(rope_base, scale, Hkv, dedup, kernel, rotated_k=rotated_k, residuals=residuals,
              round_offsets=round_offsets)
    code = _dtype_code(q)
    for t in (q, k, v):
        if not (t.is_cuda and t.is_contiguous() and t.dtype == q.dtype):
            raise ValueError("q, k, v must be contiguous CUDA tensors of one dtype")
    if out is None:
        out = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((B, H, T), dtype=torch.float32, device=q.device)
    if workspace is None:                        # (a given workspace's size is checked by the library)
        need = int(lib().fibattn_fwd_workspace_bytes(B, H, T, D, W, len(f), code, ctypes.byref(o)))
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=q.device)
    _check(lib().fibattn_fwd(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), lse.data_ptr(),
                             B, H, T, D, int(W), float(alpha), f.ctypes.data, len(f), code, ctypes.byref(o),
                             workspace.data_ptr(), workspace.numel(), _stream_ptr(stream)))
    return out, lse


def bwd(q, k, v, lse, dout, alpha: float, offsets, W: int, *, out=None, rope_base=1e4, scale=None, dedup=True,
        dq=None, dk=None, dv=None, dtheta=None, dd=None, workspace=None, stream=None, kernel="auto",
        rotated_k=None, rung_grads=True, residuals=None, round_offsets=False):
    """Backward pass.  ``out``: the forward output (optional; enables the
    tensor-core query pass).  ``kernel``: "auto", "gather" or "mma".
    ``rotated_k``: the buffer the forward of the same k filled (skips rotating
    k again).  ``residuals``: the buffer the forward of the same inputs filled
    (the tensor-core passes then read p, the rung score differences and the
    rotated queries instead of recomputing them).  ``rung_grads=False`` skips
    dL/dtheta and dL/dd_k (a fixed schedule; required with ``round_offsets``).
    Returns (dq, dk, dv, dtheta [1], dd [K]) on the device (dtheta, dd None
    without rung_grads)."""
    B, H, T, D = q.shape
    Hkv = k.shape[1]
    f = _offsets(offsets)
    K = len(f)
    _check_rotated(rotated_k, k)
    _check_residuals(residuals, q, W, K)
    o = _opts(rope_base, scale, Hkv, dedup, bwd_kernel=kernel, rotated_k=rotated_k, residuals=residuals,
              round_offsets=round_offsets)
    code = _dtype_code(q)
    for t in (q, k, v, dout) + ((out,) if out is not None else ()):
        if not (t.is_cuda and t.is_contiguous() and t.dtype == q.dtype):
            raise ValueError("q, k, v, dout, out must be contiguous CUDA tensors of one dtype")
    dq = torch.empty_like(q) if dq is None else dq
    dk = torch.empty_like(k) if dk is None else dk
    dv = torch.empty_like(v) if dv is None else dv
    if rung_grads:
        dtheta = torch.empty(4, dtype=torch.float32, device=q.device) if dtheta is None else dtheta
        dd = torch.empty(max(K, 1), dtype=torch.float32, device=q.device) if dd is None else dd
    if workspace is None:                        # (a given workspace's size is checked by the library)
        need = int(lib().fibattn_bwd_workspace_bytes(B, H, T, D, W, K, code, ctypes.byref(o)))
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=q.device)
    _check(lib().fibattn_bwd(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr() if out is not None else None,
                             lse.data_ptr(), dout.data_ptr(),
                             dq.data_ptr(), dk.data_ptr(), dv.data_ptr(),
                             dtheta.data_ptr() if dtheta is not None else None,
                             dd.data_ptr() if dd is not None else None,
                             B, H, T, D, int(W), float(alpha), f.ctypes.data, K, code, ctypes.byref(o),
                             workspace.data_ptr(), workspace.numel(), _stream_ptr(stream)))
    if dtheta is None and dd is None:
        return dq, dk, dv, None, None
    return dq, dk, dv, (dtheta[:1] if dtheta is not None else None), (dd[:K] if dd is not None else None)


# ---------------------------------------------------------- device status ----

def check_status(stream=None):
    """Synchronise ``stream`` and read and clear the device status word
    (fibattn_check_status).  Returns the flags; raises FibattnError when a
    kernel gave up a bounded wait (status 4) or a rotated row overflowed fp16
    (status 5)."""
    flags = ctypes.c_uint(0)
    rc = lib().fibattn_check_status(_stream_ptr(stream), ctypes.byref(flags))
    if rc != 0:
        e = FibattnError(rc, lib().fibattn_last_error().decode(errors="replace"))
        e.flags = flags.value
        raise e
    return flags.value


def test_wait_timeout(timeout_us: int, stream=None):
    """Launch the library's bounded-wait probe (a wait that no copy completes)."""
    _check(lib().fibattn_test_wait_timeout(int(timeout_us), _stream_ptr(stream)))


# ------------------------------------------------------------- profiling ----

def profile_enable(on: bool = True):
    L = lib()
    L.fibattn_profile_enable.argtypes = [ctypes.c_int]
    L.fibattn_profile_enable.restype = ctypes.c_int
    _check(L.fibattn_profile_enable(1 if on else 0))


def profile_summary() -> dict:
    """{kernel name: (total device ms, launches)} for launches since enable."""
    L = lib()
    L.fibattn_profile_summary.argtypes = [ctypes.c_int, ctypes.c_char_p, ctypes.c_int,
                                          ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int)]
    L.fibattn_profile_summary.restype = ctypes.c_int
    n = L.fibattn_profile_summary(-1, None, 0, None, None)
    out = {}
    for i in range(n):
        buf = ctypes.create_string_buffer(64)
        ms = ctypes.c_double()
        cnt = ctypes.c_int()
        _check(L.fibattn_profile_summary(i, buf, 64, ctypes.byref(ms), ctypes.byref(cnt)))
        out[buf.value.decode()] = (ms.value, cnt.value)
    return out
