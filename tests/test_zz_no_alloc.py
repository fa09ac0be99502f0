"""The allocation-free attention backward (bcmt_attention_backward_noalloc).

Some callers cannot call cudaMalloc -- for instance a host framework that owns
all device memory and gives this library only its input and output buffers.
For them the library offers an attention backward whose scratch lives in a
device array inside the library.  This test calls it through the C ABI twice in
a row (different inputs each time, so the second call runs on the scratch the
first one left behind) and checks each result against the regular attention
backward, which takes its scratch from the caller.  It runs last so that a
stop-at-first-failure run has already run every other test.
"""

import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def C(cuda_ok):
    from paper_2608_13578_gb300 import bcmt
    return bcmt


def _inputs(B, T, D, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    return [torch.randn(B, T, D, generator=g).to(dtype).cuda() for _ in range(4)]


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_noalloc_matches_regular_backward_twice(C, dtype):
    B, T, H, dh, L = 2, 200, 2, 64, 32
    D = H * dh
    tdt = torch.float32 if dtype == "fp32" else torch.bfloat16
    p = C.make_params(B, T, D, H, L, dtype)
    for seed in (11, 12):
        q, k, v, dO = _inputs(B, T, D, tdt, seed)
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
        torch.cuda.synchronize()
        for name, a, r in zip(("dq", "dk", "dv"), got, ref):
            a, r = a.double(), r.double()
            assert torch.isfinite(a).all(), name
            err = (a - r).abs().max().item()
            if dtype == "fp32":
                assert err <= 1e-4, (seed, name, err)
            else:
                assert err / r.abs().max().item() <= 2e-2, (seed, name, err)


def test_noalloc_rejects_oversized_shapes(C):
    # B*H*T = 2 * 16 * 40000 > 2**20 rows: rejected on the host, nothing launched
    p = C.make_params(2, 40000, 1024, 16, 64, "bf16")
    a = 1 << 20
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_attention_backward_noalloc(p, a, a, a, 1024, a, a, a, a, a, a, 1024)
    assert e.value.code == C.BCMT_ERR_SHAPE
    assert "scratch" in C.bcmt_last_error()
