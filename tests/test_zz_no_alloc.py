"""The allocation-free attention backward (bcmt_attention_backward_noalloc).

Some callers cannot call cudaMalloc -- for instance a host framework that owns
all device memory and gives this library only its input and output buffers.
For them the library offers an attention backward whose scratch lives in a
device array inside the library.  These tests call it through the C ABI twice
in a row (different inputs each time, so the second call runs on the scratch
the first one left behind) and require each result to equal, bit for bit, the
regular attention backward, which runs the same kernels on scratch the caller
provides; the result is also checked against the float64 oracle at the
library's tolerance.  One case sits exactly at the array's limit of 2^20
(batch, head, token) rows, where its last entry is used, and one row more is
rejected.  The file runs last so that a stop-at-first-failure run has already
run every other test.
"""

import numpy as np
import pytest
import torch

from tests.test_gpu_kernels import _attn_ref

pytestmark = pytest.mark.gpu

ROWS_MAX = 1 << 20  # the built-in scratch holds one fp32 per (batch, head, token)


@pytest.fixture(scope="module")
def C(cuda_ok):
    from paper_2608_13578_gb300 import bcmt
    return bcmt


def _inputs(B, T, D, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    return [torch.randn(B, T, D, generator=g).to(dtype) for _ in range(4)]


def _regular_and_noalloc(C, p, B, T, D, H, tdt, q, k, v, dO):
    o = torch.empty(B, T, D, dtype=tdt, device="cuda")
    lse = torch.empty(B, H, T, device="cuda")
    C.bcmt_test_attn(0, 0, p, q, k, v, D, o, lse)
    # regular backward: the caller provides the scratch
    drow = torch.empty(B, H, T, device="cuda")
    ref = [torch.empty(B, T, D, dtype=tdt, device="cuda") for _ in range(3)]
    C.bcmt_test_attn(0, 1, p, q, k, v, D, o, lse, dO, drow, *ref, D)
    # allocation-free backward: the scratch is inside the library
    got = [torch.full((B, T, D), float("nan"), dtype=tdt, device="cuda") for _ in range(3)]
    C.bcmt_attention_backward_noalloc(p, q, k, v, D, o, lse, dO, *got, D)
    C.bcmt_device_status()
    torch.cuda.synchronize()
    return ref, got


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_noalloc_matches_regular_backward_twice(C, dtype):
    B, T, H, dh, L = 2, 200, 2, 64, 32
    D = H * dh
    tdt = torch.float32 if dtype == "fp32" else torch.bfloat16
    p = C.make_params(B, T, D, H, L, dtype)
    for seed in (11, 12):
        q, k, v, dO = _inputs(B, T, D, tdt, seed)
        ref, got = _regular_and_noalloc(C, p, B, T, D, H, tdt, q.cuda(), k.cuda(), v.cuda(),
                                        dO.cuda())
        _, _, *oracle = _attn_ref(*(t.double().numpy() for t in (q, k, v)), L, H,
                                  dO.double().numpy())
        for name, a, r, o in zip(("dq", "dk", "dv"), got, ref, oracle):
            assert torch.equal(a, r), (seed, name)
            a = a.double().cpu().numpy()
            err = np.abs(a - o).max()
            if dtype == "fp32":
                assert err <= 1e-4, (seed, name, err)
            else:
                assert err / np.abs(o).max() <= 2e-2, (seed, name, err)


def test_noalloc_at_the_row_limit(C):
    # B*H*T = 1 * 16 * 65536 = 2^20 rows: the whole built-in array is used
    B, T, H, dh, L = 1, ROWS_MAX // 16, 16, 8, 64
    D = H * dh
    p = C.make_params(B, T, D, H, L, "fp32")
    for seed in (21, 22):
        q, k, v, dO = (t.cuda() for t in _inputs(B, T, D, torch.float32, seed))
        ref, got = _regular_and_noalloc(C, p, B, T, D, H, torch.float32, q, k, v, dO)
        for name, a, r in zip(("dq", "dk", "dv"), got, ref):
            assert torch.isfinite(a).all(), (seed, name)
            assert torch.equal(a, r), (seed, name)


@pytest.mark.parametrize("B,T,H", [(1, ROWS_MAX + 1, 1), (2, 40000, 16)])
def test_noalloc_rejects_oversized_shapes(C, B, T, H):
    # more (batch, head, token) rows than the built-in scratch holds: rejected
    # on the host before anything is launched (the pointers are never used)
    D = 64 * H
    p = C.make_params(B, T, D, H, 64, "bf16")
    a = 1 << 20
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_attention_backward_noalloc(p, a, a, a, D, a, a, a, a, a, a, D)
    assert e.value.code == C.BCMT_ERR_SHAPE
    assert "scratch" in C.bcmt_last_error()
