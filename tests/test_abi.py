"""CPU-only checks of the C ABI: the library loads, exports every function
declared in include/fibattn.h, its host-side prep matches the oracle's
definitions, and bad arguments are rejected before anything is launched."""
from __future__ import annotations

import ctypes
import math
import os
import re

import numpy as np
import pytest

import oracle as O
import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import binding as B
from paper_2606_28560_gb300 import build as build_mod

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    build_mod.build()


def _declared():
    names = []
    for h in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if h.endswith(".h"):
            text = open(os.path.join(ROOT, "include", h)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"\b(fibattn_\w+)\s*\(", text)
    return sorted(set(names))


def test_library_exports_every_declared_function():
    lib = ctypes.CDLL(fa.library_path())
    decl = _declared()
    assert "fibattn_fwd" in decl and "fibattn_bwd" in decl
    for name in decl:
        assert hasattr(lib, name), f"{name} declared in include/ but not exported"


def test_base_and_schedules_match_oracle():
    np.testing.assert_array_equal(fa.base("fib", 15), O.fib_base(15).astype(np.float32))
    np.testing.assert_array_equal(fa.base("pow2", 10), O.pow2_base(10).astype(np.float32))
    for kind in ("fixed", "linear", "coprime"):
        np.testing.assert_allclose(fa.alpha_schedule(kind, 16), O.alpha_schedule(kind, 16), rtol=0, atol=1e-7)
    th = [0.3, -0.8, 0.0, 1.7]
    np.testing.assert_allclose(fa.alpha_schedule("learned", 4, theta=th),
                               O.alpha_schedule("learned", 4, theta=th), rtol=0, atol=1e-7)


@pytest.mark.parametrize("alpha", [0.5, 0.5 + 1 / 15, 0.7333333, 1.0, 1.2345, 1.5])
@pytest.mark.parametrize("W", [0, 8, 12])
def test_rung_params_match_oracle(alpha, W):
    f = O.fib_base(15)
    p = fa.rung_params(np.float32(alpha), f, W)
    d = O.offsets_fp32(float(np.float32(alpha)), f)
    np.testing.assert_array_equal(p["d"].astype(np.float64), d)
    np.testing.assert_array_equal(p["s0"], np.floor(d).astype(np.int32))
    np.testing.assert_array_equal(p["w"].astype(np.float64), d - np.floor(d))
    np.testing.assert_array_equal(p["active"], d > W)
    p2 = fa.rung_params(np.float32(alpha), f, W, dedup=False)
    assert p2["active"].all()
    # the integer-offset variants: rounded to the nearest integer, ties to even
    p3 = fa.rung_params(np.float32(alpha), f, W, round_offsets=True)
    dr = O.offsets_rounded(float(np.float32(alpha)), f)
    np.testing.assert_array_equal(p3["d"].astype(np.float64), dr)
    np.testing.assert_array_equal(p3["s0"], dr.astype(np.int32))
    assert not p3["w"].any()
    np.testing.assert_array_equal(p3["active"], dr > W)


def test_rounded_offsets_reject_rung_gradients():
    """Rounded distances do not vary with alpha: the backward refuses dtheta/dd."""
    lib = B.lib()
    o = B._opts(round_offsets=True)
    f = np.array([1, 2, 3], dtype=np.float32)
    rc = lib.fibattn_bwd(16, 16, 16, None, 16, 16, 16, 16, 16, 16, None, 1, 2, 8, 64, 2, 1.0, B._fptr(f), 3, 0,
                         ctypes.byref(o), 16, 1 << 30, None)
    assert rc == 1 and "dtheta" in lib.fibattn_last_error().decode()


def test_theta_alpha_maps_are_stable_and_inverse():
    """alpha = 0.5 + sigmoid(theta) stays finite at extreme theta; the inverse
    map clamps the ends and inverts the interior."""
    a = fa.alpha_schedule("learned", 4, theta=[-1000.0, 1000.0, 0.0, 2.0])
    assert a[0] == 0.5 and a[1] == 1.5 and a[2] == 1.0
    assert abs(a[3] - (0.5 + 1 / (1 + math.exp(-2.0)))) < 1e-6
    assert fa.alpha_of_theta(-1000.0) == 0.5 and fa.alpha_of_theta(1000.0) == 1.5
    t = fa.theta_of_alpha_array([0.5, 1.5, 1.0, 0.8, 1.3])
    assert t[0] == -30.0 and t[1] == 30.0 and t[2] == 0.0
    back = fa.alpha_schedule("learned", 2, theta=t[3:])
    np.testing.assert_allclose(back, [0.8, 1.3], rtol=0, atol=2e-7)


def _call_fwd(**kw):
    lib = B.lib()
    args = dict(q=16, k=16, v=16, out=16, lse=16, B=1, H=2, T=8, D=64, W=2, alpha=1.0,
                K=3, dtype=0, ws=16, wsb=1 << 30, Hkv=0, rope_base=0.0, rk=None, res=None, fk=0)
    args.update(kw)
    f = np.array([1, 2, 3] + [5] * 40, dtype=np.float32)
    o = B.Opts(args["rope_base"], 0.0, args["Hkv"], 0, args["fk"], 0, args["rk"], args["res"], 0)
    rc = lib.fibattn_fwd(args["q"], args["k"], args["v"], args["out"], args["lse"], args["B"], args["H"],
                         args["T"], args["D"], args["W"], args["alpha"], B._fptr(f), args["K"], args["dtype"],
                         ctypes.byref(o), args["ws"], args["wsb"], None)
    return rc, lib.fibattn_last_error().decode()


@pytest.mark.parametrize("kw,code", [
    (dict(alpha=0.49), 1), (dict(alpha=1.51), 1), (dict(alpha=float("nan")), 1),
    (dict(K=33), 1), (dict(K=-1), 1), (dict(W=-1), 1), (dict(W=1025), 1),
    (dict(D=128), 2), (dict(D=32), 2), (dict(T=0), 1), (dict(H=0), 1), (dict(dtype=7), 1),
    (dict(Hkv=3), 1), (dict(q=0), 1), (dict(lse=0), 1), (dict(ws=0), 1),
    (dict(q=17), 1), (dict(out=24), 1), (dict(wsb=10), 1), (dict(rope_base=-2.0), 1),
    (dict(rk=24), 1),
    # forward residuals: 16-byte alignment; only the tensor-core forward (bf16
    # I/O, fwd_kernel 0 or 3, W <= 16) writes them -- refused before any launch
    (dict(res=24), 1), (dict(res=256, dtype=0), 2), (dict(res=256, dtype=1, W=40), 2),
    (dict(res=256, dtype=1, fk=1), 2), (dict(res=256, dtype=1, fk=2), 2),
])
def test_fwd_rejects_bad_arguments(kw, code):
    rc, msg = _call_fwd(**kw)
    assert rc == code, msg
    assert msg


def test_bwd_rejects_bad_arguments():
    lib = B.lib()
    f = np.array([1, 2, 3], dtype=np.float32)
    o = B.Opts(0.0, 0.0, 0, 0, 0, 0)
    ok_ptr = 16
    rc = lib.fibattn_bwd(ok_ptr, ok_ptr, ok_ptr, None, ok_ptr, ok_ptr, ok_ptr, ok_ptr, None, None, None,
                         1, 2, 8, 64, 2, 1.0, B._fptr(f), 3, 1, ctypes.byref(o), ok_ptr, 1 << 30, None)
    assert rc == 1 and "NULL" in lib.fibattn_last_error().decode()       # dv missing
    rc = lib.fibattn_bwd(ok_ptr, ok_ptr, ok_ptr, None, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, 18, None,
                         1, 2, 8, 64, 2, 1.0, B._fptr(f), 3, 1, ctypes.byref(o), ok_ptr, 1 << 30, None)
    assert rc == 1
    rc = lib.fibattn_bwd(ok_ptr, ok_ptr, ok_ptr, None, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, None,
                         1, 2, 8, 64, 2, 1.0, B._fptr(f), 3, 1, ctypes.byref(o), ok_ptr, 8, None)
    assert rc == 1 and "workspace" in lib.fibattn_last_error().decode()
    rc = lib.fibattn_bwd(ok_ptr, ok_ptr, ok_ptr, 24, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, None,
                         1, 2, 8, 64, 2, 1.0, B._fptr(f), 3, 1, ctypes.byref(o), ok_ptr, 1 << 30, None)
    assert rc == 1 and "aligned" in lib.fibattn_last_error().decode()       # misaligned out
    for kern, code in ((3, 1), (-1, 1)):
        o2 = B.Opts(0.0, 0.0, 0, 0, 0, kern)
        rc = lib.fibattn_bwd(ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, None,
                             1, 2, 8, 64, 2, 1.0, B._fptr(f), 3, 1, ctypes.byref(o2), ok_ptr, 1 << 30, None)
        assert rc == code and "bwd_kernel" in lib.fibattn_last_error().decode()
    # the tensor-core query pass needs the forward output and bf16 I/O
    for out_ptr, dt in ((None, 1), (ok_ptr, 0)):
        o2 = B.Opts(0.0, 0.0, 0, 0, 0, 2)
        rc = lib.fibattn_bwd(ok_ptr, ok_ptr, ok_ptr, out_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, ok_ptr, None,
                             1, 2, 8, 64, 2, 1.0, B._fptr(f), 3, dt, ctypes.byref(o2), ok_ptr, 1 << 30, None)
        assert rc == 2, lib.fibattn_last_error().decode()


def test_workspace_queries():
    import torch
    lib = B.lib()
    code = 1
    with_rk = B.Opts(0.0, 0.0, 0, 0, 0, 0, 256)            # any aligned address: only the size is queried
    assert lib.fibattn_fwd_workspace_bytes(16, 8, 1024, 64, 8, 15, code, ctypes.byref(with_rk)) == 0
    plain = lib.fibattn_bwd_workspace_bytes(16, 8, 1024, 64, 8, 15, code, None)
    assert plain - lib.fibattn_bwd_workspace_bytes(16, 8, 1024, 64, 8, 15, code, ctypes.byref(with_rk)) == \
        16 * 8 * 1024 * 64 * 2                               # no rotated-key region of its own
    assert fa.fwd_workspace_bytes(16, 8, 1024, 8, 15, torch.bfloat16) >= 16 * 8 * 1024 * 64 * 2
    assert fa.bwd_workspace_bytes(16, 8, 1024, 8, 15, torch.bfloat16) > fa.fwd_workspace_bytes(16, 8, 1024, 8, 15,
                                                                                                 torch.bfloat16)
    assert B.lib().fibattn_fwd_workspace_bytes(1, 2, 8, 128, 2, 3, 0, None) == 0    # invalid -> 0


def test_residual_bytes():
    """The residual buffer holds rotated q (fp16 [B,H,T,64]), the unnormalised
    weight per slot (fp32 [B,H,W+1+K,T]), rung score differences (fp32
    [B,H,K,T]) and 1 / (weight sum) per query (fp32 [B,H,T]), each array from
    the next multiple of 256 bytes; fp32 I/O and invalid sizes give 0."""
    import torch

    def up(x):
        return (x + 255) // 256 * 256
    for (Bn, H, T, W, K) in ((2, 3, 100, 8, 15), (1, 1, 1, 0, 0), (16, 8, 1024, 8, 15), (1, 2, 77, 3, 7)):
        n = Bn * H * T
        want = up(n * 128) + up(n * (W + 1 + K) * 4) + up(n * K * 4) + up(n * 4)
        assert B.lib().fibattn_residual_bytes(Bn, H, T, 64, W, K, 1) == want
        assert fa.residual_bytes(Bn, H, T, W, K, torch.bfloat16) == want
        assert B.lib().fibattn_residual_bytes(Bn, H, T, 64, W, K, 0) == 0
        buf = torch.zeros(want, dtype=torch.uint8)
        qt, P, sd, il = fa.residual_views(buf, Bn, H, T, W, K)
        assert qt.shape == (Bn, H, T, 64) and P.shape == (Bn, H, W + 1 + K, T) and sd.shape == (Bn, H, K, T)
        assert il.shape == (Bn, H, T)
        # the (non-empty) views tile the buffer in order without overlap
        ends = [(t.data_ptr() - buf.data_ptr(), t.data_ptr() - buf.data_ptr() + t.numel() * t.element_size())
                for t in (qt, P, sd, il) if t.numel()]
        assert ends[0][0] == 0 and ends[-1][1] <= want
        assert all(a[1] <= b[0] for a, b in zip(ends, ends[1:]))
        assert all(a % 256 == 0 for a, _ in ends)
    assert B.lib().fibattn_residual_bytes(1, 2, 8, 128, 2, 3, 1) == 0                # D != 64
    assert B.lib().fibattn_residual_bytes(1, 2, 8, 64, 2, 33, 1) == 0                # K > 32


def test_offsets_marshalling():
    """Offsets reach the C ABI as a contiguous fp32 host array: one that is
    already so is passed as it is, anything else (a list, fp64, a strided
    view) is copied into one with the same values."""
    f = fa.base("fib", 15)
    assert B._offsets(f) is f
    for other in (list(map(float, f)), f.astype(np.float64), np.repeat(f, 2)[::2]):
        g = B._offsets(other)
        assert g.dtype == np.float32 and g.flags.c_contiguous and np.array_equal(g, f)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(build_mod, "LIB", str(tmp_path / "nope.so"))
    monkeypatch.setattr(B, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        B.lib()
