"""The device status word: a bounded wait that runs out, and a rotated row
that leaves fp16's range, are reported by fibattn_check_status without
faulting the GPU or hanging.

The wait case uses the library's test hook: one warp arms a shared-memory
barrier for bytes that no copy delivers (nothing is issued) and waits with a
2 ms bound, so the wait runs out, the kernel returns and raises bit 0.  The
context stays usable: a forward right after it matches the oracle.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle as O
import paper_2606_28560_gb300 as fa
from paper_2606_28560_gb300 import binding as B
from paper_2606_28560_gb300 import inputs
from tests.test_gpu_parity import check_fwd

pytestmark = pytest.mark.gpu


def _clear():
    try:
        fa.check_status()
    except fa.FibattnError:
        pass


def test_wait_timeout_is_reported_and_cleared():
    torch.cuda.synchronize()
    _clear()
    assert fa.check_status() == 0
    B.test_wait_timeout(2000)
    with pytest.raises(fa.FibattnError) as ei:
        fa.check_status()
    assert ei.value.status == 4 and ei.value.flags & 1
    assert "gave up waiting" in str(ei.value)
    assert fa.check_status() == 0                 # read and cleared
    # the context is intact: a forward still meets the oracle
    q, k, v = inputs.qkv(1, 2, 200, seed=7, dtype=torch.bfloat16)
    check_fwd(q, k, v, 0.9, fa.base("fib", 15), 8)
    assert fa.check_status() == 0


def test_rotated_key_beyond_fp16_is_reported():
    torch.cuda.synchronize()
    _clear()
    q, k, v = inputs.qkv(1, 2, 64, seed=8, dtype=torch.bfloat16)
    k[0, 1, 40, 3] = 1.0e5                        # a bf16 value the fp16 rotated keys cannot hold
    fa.fwd(q.cuda(), k.cuda(), v.cuda(), 1.0, fa.base("fib", 15), 8)
    with pytest.raises(fa.FibattnError) as ei:
        fa.check_status()
    assert ei.value.status == 5 and ei.value.flags & 2
    assert fa.check_status() == 0
    # in range: nothing raised
    k[0, 1, 40, 3] = 3.0e4
    fa.fwd(q.cuda(), k.cuda(), v.cuda(), 1.0, fa.base("fib", 15), 8)
    assert fa.check_status() == 0
