"""fibattn_fwd_noalloc: the forward pass for callers that cannot allocate
device memory (a framework that owns all device memory and passes plugins only
tensors, or a hot path where cudaMalloc's device synchronisation is not
allowed).  Its scratch is a fixed library-owned device array; the result must
match fibattn_fwd, which uses a caller-provided workspace, on two calls in a
row (the second call finds the first call's contents in the shared array).

Collected last on purpose (file name), so a stop-at-first-failure run has
already run every other test."""
from __future__ import annotations

import ctypes

import numpy as np
import pytest
import torch

import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import binding as B
from paper_2606_28560_gb300 import inputs

pytestmark = pytest.mark.gpu

TOL = {torch.float32: 1e-4, torch.bfloat16: 1e-2}


def _noalloc(q, k, v, alpha, f, W, out, lse):
    L = B.lib()
    vp, ci, cf = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    L.fibattn_fwd_noalloc.argtypes = [vp, vp, vp, vp, vp, ci, ci, ci, ci, ci, cf,
                                      ctypes.POINTER(ctypes.c_float), ci, ci, ctypes.POINTER(B.Opts), vp]
    L.fibattn_fwd_noalloc.restype = ci
    f32 = np.ascontiguousarray(np.asarray(f, dtype=np.float32))
    o = B.Opts(1e4, 0.0, k.shape[1], 0, 0, 0)
    Bn, H, T, D = q.shape
    code = 1 if q.dtype == torch.bfloat16 else 0
    return L.fibattn_fwd_noalloc(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), lse.data_ptr(),
                                 Bn, H, T, D, int(W), float(alpha), B._fptr(f32), len(f32), code, ctypes.byref(o),
                                 torch.cuda.current_stream().cuda_stream)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32], ids=["bf16", "f32"])
def test_noalloc_matches_fwd_two_calls(dtype):
    f = fa.base("fib", 15)
    cases = [(2, 4, 2, 700, 8, 0.77, 11), (3, 8, 8, 1024, 12, 1.3, 12)]
    for Bn, H, Hkv, T, W, alpha, seed in cases:
        q, k, v = (x.cuda() for x in inputs.qkv(Bn, H, T, seed=seed, dtype=dtype, Hkv=Hkv))
        ref_out, ref_lse = fa.fwd(q, k, v, alpha, f, W)
        for _ in range(2):                       # second call reuses the shared array
            out = torch.full_like(q, float("nan"))
            lse = torch.full((Bn, H, T), float("nan"), dtype=torch.float32, device=q.device)
            rc = _noalloc(q, k, v, alpha, f, W, out, lse)
            assert rc == 0, B.lib().fibattn_last_error()
            torch.cuda.synchronize()
            err = (out.float() - ref_out.float()).abs().max().item()
            assert err <= TOL[dtype], f"out differs from fibattn_fwd by {err}"
            assert (lse - ref_lse).abs().max().item() <= TOL[dtype]


def test_noalloc_rejects_oversized_call():
    f = fa.base("fib", 15)
    # 2*8*16384 bf16 rows of 128 B = 32 MiB fits; one more batch element does not
    q = torch.zeros((3, 8, 16384, 64), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(q)
    lse = torch.empty((3, 8, 16384), dtype=torch.float32, device="cuda")
    rc = _noalloc(q, q, q, 1.0, f, 8, out, lse)
    assert rc == 1
    assert b"scratch" in B.lib().fibattn_last_error()
