"""Parity of the whole CUDA mixer (forward and backward, through the C ABI)
with the float64 oracle on the same seeded inputs.

Bar: fp32 max abs error <= 1e-4; bf16 max|gpu - oracle| / max|oracle| <= 2e-2,
for Y and every gradient.  Small cases span several tiles and ragged tails;
the named workloads run at their full sizes in the launch configuration the
benchmark times."""

import numpy as np
import pytest
import torch

from paper_2608_13578_gb300.inputs import WORKLOADS, Workload, make_inputs
from tests.helpers import (GRAD_NAMES_QKV, GRAD_NAMES_X, assert_close, gpu_run, oracle_run,
                           to_device)

pytestmark = pytest.mark.gpu


def W(B, T, D, H, L, dtype, **kw):
    return Workload(name=f"b{B}_t{T}_d{D}_h{H}_l{L}_{dtype}", B=B, T=T, D=D, H=H, L=L,
                    dtype=dtype, decay=kw.pop("decay", (0.5, 0.99)), **kw)


SMALL = [
    W(2, 100, 128, 4, 16, "fp32"),
    W(1, 256, 128, 4, 32, "fp32"),
    W(2, 77, 64, 2, 10, "fp32"),
    W(2, 64, 128, 2, 64, "fp32", decay=(0.0, 0.0)),
    W(1, 50, 128, 4, 64, "fp32"),                      # one ragged block: no memory
    W(2, 256, 128, 2, 64, "bf16"),
    W(2, 200, 256, 4, 32, "bf16"),
    W(1, 384, 128, 2, 128, "bf16"),
    W(2, 130, 128, 2, 16, "bf16"),
    W(1, 300, 128, 2, 256, "bf16"),
    W(2, 150, 128, 2, 48, "bf16"),
    W(1, 96, 192, 2, 32, "bf16"),                       # dh = 96 -> SIMT attention
    W(2, 300, 128, 8, 64, "bf16"),                      # dh = 16 (the paper's D128 h8)
    W(1, 700, 128, 4, 256, "bf16"),                     # dh = 32, key-tile walk
    W(2, 600, 256, 4, 512, "bf16"),                     # dh = 64, L = 512
    W(1, 200, 128, 8, 32, "fp32"),
    W(2, 256, 128, 2, 64, "bf16", decay=(0.0, 0.0)),
    # degenerate shapes
    W(1, 1, 128, 4, 16, "fp32"),                         # a single token
    W(2, 1, 64, 1, 64, "bf16"),                          # single token, one 64-wide head
    W(1, 33, 128, 2, 1, "fp32"),                         # L = 1: every token its own block
    W(2, 50, 128, 2, 8, "bf16"),                         # L = 8 (SIMT attention in bf16)
    W(2, 64, 128, 2, 64, "bf16"),                        # T = L: one full block, no memory
    W(1, 40, 128, 1, 8, "fp32"),                         # the widest head, d_h = 128
    W(1, 1100, 64, 1, 1024, "bf16"),                     # the largest block, ragged tail
]
VARIANTS = [
    W(2, 100, 128, 4, 16, "fp32", input_is_x=False),
    W(2, 200, 256, 4, 32, "bf16", input_is_x=False),
    W(2, 100, 128, 4, 16, "fp32", honly=True),
    W(2, 200, 256, 4, 32, "bf16", honly=True),
]


def _check(w: Workload, backward=True, decay_grad=False):
    t = make_inputs(w)
    y, g = gpu_run(w, to_device(t), backward, decay_grad)
    fw, gr = oracle_run(w, t, backward)
    assert_close("Y", y, fw["Y"], w.dtype)
    if backward:
        names = GRAD_NAMES_X if w.input_is_x else GRAD_NAMES_QKV
        for n in names:
            if n == "d_decay" and not decay_grad:
                assert n not in g
                continue
            got = g[n]
            if w.honly and n in ("dw_p", "dw_m", "dw_g", "d_decay"):
                assert torch.count_nonzero(got).item() == 0
                continue
            assert_close(n, got, gr[n], w.dtype)


def _wid(w):
    return w.name + ("_qkv" if not w.input_is_x else "") + ("_honly" if w.honly else "")


@pytest.mark.parametrize("w", SMALL + VARIANTS, ids=_wid)
def test_layer_small(cuda_ok, w):
    _check(w)


@pytest.mark.parametrize("w", SMALL + VARIANTS, ids=_wid)
def test_layer_small_decay_grad(cuda_ok, w):
    """The same layers with the learned-decay gradient requested (the memory
    gradient then takes the separate reverse-scan kernel)."""
    _check(w, decay_grad=True)


def test_tensor_core_and_simt_paths_agree(cuda_ok):
    """The same bf16 layer through the tcgen05 kernels and the SIMT kernels."""
    from paper_2608_13578_gb300 import bcmt as C
    w = W(2, 256, 128, 2, 64, "bf16")
    t = to_device(make_inputs(w))
    try:
        C.bcmt_test_set_tensor_cores(False, False)
        y0, g0 = gpu_run(w, t)
    finally:
        C.bcmt_test_set_tensor_cores(True, True)
    y1, g1 = gpu_run(w, t)
    scale = y0.float().abs().max().item()
    assert (y0.float() - y1.float()).abs().max().item() / scale < 2e-2
    for n in g0:
        s = g0[n].float().abs().max().item()
        assert (g0[n].float() - g1[n].float()).abs().max().item() / s < 2e-2, n


def test_deterministic(cuda_ok):
    w = WORKLOADS["fwdbwd_bf16_b8_t1024_l64_d512_h8"].replace(B=2)
    t = to_device(make_inputs(w))
    y0, g0 = gpu_run(w, t)
    y1, g1 = gpu_run(w, t)
    assert torch.equal(y0, y1)
    for n in g0:
        assert torch.equal(g0[n], g1[n]), n


def test_causality_bitwise(cuda_ok):
    """Sec. 3.6 on the GPU: perturbing token t leaves every output before t
    bitwise unchanged."""
    w = W(1, 256, 128, 2, 64, "bf16")
    t = make_inputs(w)
    y0, _ = gpu_run(w, to_device(t), backward=False)
    for tok in (5, 64, 130, 255):
        t2 = dict(t)
        x = t["x"].clone()
        x[0, tok] += 1.0
        t2["x"] = x
        y1, _ = gpu_run(w, to_device(t2), backward=False)
        assert torch.equal(y0[0, :tok], y1[0, :tok]), tok
        assert not torch.equal(y0[0, tok], y1[0, tok])


# ------------------------------------------------- the named workloads, full size
@pytest.mark.parametrize("decay_grad", [False, True], ids=["fixed_decay", "decay_grad"])
@pytest.mark.parametrize("name", ["fwd_fp32_b1_t256_l32_d128_h4", "fwdbwd_bf16_b8_t1024_l64_d512_h8"])
def test_workload_full(cuda_ok, name, decay_grad):
    w = WORKLOADS[name]
    _check(w, backward=True, decay_grad=decay_grad)


@pytest.mark.parametrize("L", [32, 64, 128, 256])
def test_block_size_sweep(cuda_ok, L):
    _check(WORKLOADS[f"sweep_bf16_b16_t1024_l{L}_d768_h12"], backward=True)


@pytest.mark.parametrize("T", [2048, 4096, 8192, 16384])
def test_sequence_scaling(cuda_ok, T):
    """The sequence-length sweep at its full size (B = 4, D = 1024, L = 128),
    every output and gradient against the oracle: the weight gradients reduce
    over K = B*T up to 65536 tokens with their own split counts, and the
    reverse scan of Sec. 3.5 runs N_b up to 128 dependent steps."""
    _check(WORKLOADS[f"seqscale_bf16_b4_t{T}_l128_d1024_h16"], backward=True,
           decay_grad=T == 16384)


@pytest.mark.parametrize("L", [256, 512])
def test_sequence_scaling_key_walk(cuda_ok, L):
    """The sequence sweep's shape at T = 4096 with blocks of 256 and 512
    tokens, which take the key-tile-walking attention kernels (several key
    tiles per block), every gradient against the oracle."""
    w = WORKLOADS["seqscale_bf16_b4_t4096_l128_d1024_h16"]
    _check(w.replace(name=f"seqscale_bf16_b4_t4096_l{L}_d1024_h16", L=L), backward=True)


@pytest.mark.parametrize("L", [64, 128, 256, 512])
def test_paper_shape(cuda_ok, L):
    """One layer of the paper's model shape (Sec. 4.1: D 128, 8 heads of 16,
    batch 16, context 1024) at the block sizes of its Table 2, full size."""
    _check(WORKLOADS[f"paper_bf16_b16_t1024_l{L}_d128_h8"], backward=True)
