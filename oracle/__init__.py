"""fp64 CPU oracle for depth-staggered scaled-Fibonacci sparse attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA library (``paper_2606_28560_gb300``) and imports nothing from it.

The arithmetic lives in ``fibattn_oracle.c`` (plain C, fp64, one query at a
time).  This module compiles it with gcc on first use, and adds the paper's
host-side definitions that the C file does not need:

* the Fibonacci base and the reach-matched power-of-2 control base
  (Section 2, "Attended set" and "Control base");
* the four per-layer alpha schedules (Section 2, "The per-layer scalar").

Every function cites the passage it follows; the readings taken where the
paper is silent are listed in the header of ``fibattn_oracle.c``.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fibattn_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libfibattn_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle (gcc, -O2, OpenMP) into ``oracle/_build``."""
    os.makedirs(_BUILD, exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH)
             or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fno-fast-math", "-ffp-contract=off", "-fopenmp",
               "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _bind(lib):
    dp = ctypes.POINTER(ctypes.c_double)
    ip = ctypes.POINTER(ctypes.c_int)
    c_int, c_double = ctypes.c_int, ctypes.c_double
    lib.fibo_offsets_fp32.argtypes = [c_double, dp, c_int, dp]
    lib.fibo_forward.argtypes = [dp, dp, dp, dp, dp] + [c_int] * 6 + [dp, c_int, c_double, c_double, c_int, c_int]
    lib.fibo_forward.restype = c_int
    lib.fibo_backward.argtypes = [dp, dp, dp, dp, dp, dp, dp, dp] + [c_int] * 6 + [dp, c_int, c_double, c_double, c_int, c_int]
    lib.fibo_backward.restype = c_int
    lib.fibo_dtheta.argtypes = [c_double, dp, dp, c_int, dp, dp]
    lib.fibo_query_slots.argtypes = [dp, dp, c_int, c_int, c_int, c_int, dp, c_int, c_double, c_double, c_int,
                                     ip, ip, dp, dp, dp, ip]
    lib.fibo_query_slots.restype = c_int
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
    return _lib


def _swap_library(path):
    """Tests only: point the wrappers at another build of the C file (used to
    show that the pins catch planted mistakes).  Returns the previous handle."""
    global _lib
    _load()
    with _lock:
        prev = _lib
        _lib = _bind(ctypes.CDLL(path)) if isinstance(path, str) else path
    return prev


def _dp(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def _ip(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int))


def _f64(x) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


# --------------------------------------------------------------------------
# Bases and schedules (Section 2)
# --------------------------------------------------------------------------

def fib_base(K: int = 15) -> np.ndarray:
    """Fibonacci base f = 1, 2, 3, 5, ... (Section 2, "Attended set"): the
    recurrence f_{k+1} = f_k + f_{k-1} started from 1, 2.  K=15 ends at 987."""
    f = []
    a, b = 1, 2
    for _ in range(K):
        f.append(a)
        a, b = b, a + b
    return np.array(f, dtype=np.float64)


def pow2_base(K: int = 10) -> np.ndarray:
    """Power-of-2 control base 1, 2, 4, ... (Section 2, "Control base");
    K=10 gives [1 .. 512]."""
    return np.array([2.0 ** k for k in range(K)], dtype=np.float64)


def alpha_from_theta(theta) -> np.ndarray:
    """alpha = 0.5 + sigmoid(theta) (Section 2, "The per-layer scalar")."""
    t = np.asarray(theta, dtype=np.float64)
    return 0.5 + 1.0 / (1.0 + np.exp(-t))


def alpha_schedule(kind: str, L: int = 16, theta=None, stride: int = 7) -> np.ndarray:
    """Per-layer alpha for the four schedules of Section 2:

    fixed    alpha_l = 1
    learned  alpha_l = 0.5 + sigmoid(theta_l)   (theta given per layer)
    linear   alpha_l = 0.5 + l / (L - 1)
    coprime  the linear multiset reassigned by l -> (S l mod L), S = 7
    """
    if kind == "fixed":
        return np.ones(L)
    if kind == "learned":
        if theta is None or len(theta) != L:
            raise ValueError("learned schedule needs one theta per layer")
        return alpha_from_theta(theta)
    lin = np.array([0.5 + l / (L - 1) for l in range(L)]) if L > 1 else np.ones(1)
    if kind == "linear":
        return lin
    if kind == "coprime":
        if math.gcd(stride, L) != 1:
            raise ValueError("coprime stride must be coprime to L")
        return np.array([lin[(stride * l) % L] for l in range(L)])
    raise ValueError(f"unknown schedule {kind!r}")


def offsets_fp32(alpha: float, f) -> np.ndarray:
    """d_k = alpha * f_k (Section 2), rounded once to fp32 and returned as fp64."""
    f = _f64(f)
    out = np.zeros(len(f))
    _load().fibo_offsets_fp32(float(alpha), _dp(f), len(f), _dp(out))
    return out


def offsets_rounded(alpha: float, f) -> np.ndarray:
    """The integer-offset variants evaluated through the paper's fused
    boolean-mask path (Section 2, "Implementation note"): d_k = fl32(alpha f_k)
    rounded to the nearest integer, ties to even, so that every rung reads one
    whole row (interpolation weight 0)."""
    return np.rint(offsets_fp32(alpha, f))


def coverage(alphas, f, W: int, T: int, dedup: bool = True) -> dict:
    """Distinct key distances a query reads in a stack of layers (Section 4.2,
    "Why staggering widens coverage"), as plain sets.  Layer l reads the window
    distances 0..W and, for each rung with d_k <= T-1 (and d_k > W under dedup),
    the floor row's distance floor(d_k) and, if d_k is fractional, the far row's
    floor(d_k)+1.  Returns the per-layer counts, the size of the union over
    layers, the part of it beyond the window, and the size of the union over
    successive layer pairs of the sums a + b < T."""
    sets = []
    for a in alphas:
        s = set(range(min(W, T - 1) + 1))
        for dk in offsets_fp32(float(a), f):
            if dk > T - 1 or (dedup and not dk > W):
                continue
            s0 = math.floor(dk)
            s.add(s0)
            if dk != s0 and s0 + 1 < T:
                s.add(s0 + 1)
        sets.append(s)
    union = set().union(*sets)
    hop = {a + b for l in range(len(sets) - 1) for a in sets[l] for b in sets[l + 1] if a + b < T}
    return dict(per_layer=[len(x) for x in sets], union=len(union), beyond_window=sum(1 for t in union if t > W),
                two_hop=len(hop))


# --------------------------------------------------------------------------
# Forward / backward (Section 2 "Attended set"; chain rule of that definition)
# --------------------------------------------------------------------------

def _shapes(q, k):
    B, H, T, D = q.shape
    Bk, Hkv, Tk, Dk = k.shape
    if (Bk, Tk, Dk) != (B, T, D) or H % Hkv:
        raise ValueError("q is [B,H,T,D]; k, v are [B,Hkv,T,D] with Hkv | H")
    return B, H, Hkv, T, D


def forward(q, k, v, W: int, d, scale=None, rope_base: float = 1e4, dedup: bool = True,
            nthreads: int = 1):
    """Oracle forward.  q [B,H,T,D]; k, v [B,Hkv,T,D]; d = rung distances (fp64,
    normally ``offsets_fp32(alpha, f)``).  Returns (out [B,H,T,D], lse [B,H,T])."""
    q, k, v, d = _f64(q), _f64(k), _f64(v), _f64(d)
    B, H, Hkv, T, D = _shapes(q, k)
    if scale is None:
        scale = 1.0 / math.sqrt(D)
    out = np.zeros((B, H, T, D))
    lse = np.zeros((B, H, T))
    rc = _load().fibo_forward(_dp(q), _dp(k), _dp(v), _dp(out), _dp(lse), B, H, Hkv, T, D, int(W),
                              _dp(d), len(d), float(scale), float(rope_base), int(bool(dedup)), int(nthreads))
    if rc:
        raise ValueError("oracle forward: bad arguments")
    return out, lse


def backward(q, k, v, dout, W: int, d, scale=None, rope_base: float = 1e4, dedup: bool = True,
             nthreads: int = 1):
    """Oracle backward.  Returns (dq, dk, dv, dd) where dd[k] = dL/dd_k."""
    q, k, v, dout, d = _f64(q), _f64(k), _f64(v), _f64(dout), _f64(d)
    B, H, Hkv, T, D = _shapes(q, k)
    if scale is None:
        scale = 1.0 / math.sqrt(D)
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    dd = np.zeros(max(len(d), 1))
    rc = _load().fibo_backward(_dp(q), _dp(k), _dp(v), _dp(dout), _dp(dq), _dp(dk), _dp(dv), _dp(dd),
                               B, H, Hkv, T, D, int(W), _dp(d), len(d), float(scale), float(rope_base),
                               int(bool(dedup)), int(nthreads))
    if rc:
        raise ValueError("oracle backward: bad arguments")
    return dq, dk, dv, dd[:len(d)]


def dtheta(alpha: float, f, dd):
    """dalpha = sum_k f_k dL/dd_k; dtheta = dalpha (alpha-0.5)(1.5-alpha)
    (Section 2, "The per-layer scalar")."""
    f, dd = _f64(f), _f64(dd)
    da = ctypes.c_double()
    dt = ctypes.c_double()
    _load().fibo_dtheta(float(alpha), _dp(f), _dp(dd), len(f), ctypes.byref(da), ctypes.byref(dt))
    return da.value, dt.value


def query_slots(q, k, W: int, i: int, d, scale=None, rope_base: float = 1e4, dedup: bool = True):
    """Attended slots of query i for one head: q [T,D], k [T,D].  Returns a dict
    of arrays rows0, rows1, c0, c1, prob, rung (rung = -1 for window slots)."""
    q, k, d = _f64(q), _f64(k), _f64(d)
    T, D = q.shape
    if scale is None:
        scale = 1.0 / math.sqrt(D)
    S = W + 1 + len(d)
    rows0 = np.zeros(S, dtype=np.int32); rows1 = np.zeros(S, dtype=np.int32)
    c0 = np.zeros(S); c1 = np.zeros(S); prob = np.zeros(S); rung = np.zeros(S, dtype=np.int32)
    n = _load().fibo_query_slots(_dp(q), _dp(k), T, D, int(W), int(i), _dp(d), len(d), float(scale),
                                 float(rope_base), int(bool(dedup)), _ip(rows0), _ip(rows1), _dp(c0), _dp(c1),
                                 _dp(prob), _ip(rung))
    if n < 0:
        raise ValueError("query index out of range")
    return dict(rows0=rows0[:n], rows1=rows1[:n], c0=c0[:n], c1=c1[:n], prob=prob[:n], rung=rung[:n])
