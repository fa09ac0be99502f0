"""Single-kernel checks on the GPU through the test entry points of the C ABI:
the GEMMs (SIMT and tcgen05, every operand layout the layer uses, K splits)
against a float64 product, and the intra-block attention (SIMT and tcgen05,
forward and backward) against the float64 oracle."""

import math

import numpy as np
import pytest
import torch

from oracle import bcmt_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def C(cuda_ok):
    from paper_2608_13578_gb300 import bcmt
    return bcmt


def _operand(rows, cols, major_rows: bool, dtype, gen, pad=8):
    """A logical [rows, cols] matrix stored row-major (major_rows: the second
    index is contiguous) or column-major, with the leading dimension padded to
    a multiple of `pad` elements.  Returns (storage, stride_row, stride_col, logical)."""
    logical = torch.randn(rows, cols, generator=gen).to(dtype)
    if major_rows:
        ld = -(-cols // pad) * pad
        store = torch.zeros(rows, ld, dtype=dtype)
        store[:, :cols] = logical
        return store, ld, 1, logical
    ld = -(-rows // pad) * pad
    store = torch.zeros(cols, ld, dtype=dtype)
    store[:, :rows] = logical.t()
    return store, 1, ld, logical


# the last two shapes have enough 128 x 256 tiles to take the wide-tile kernel
GEMM_SHAPES = [(128, 64, 64), (200, 128, 100), (256, 192, 512), (1000, 512, 320), (77, 256, 1536),
               (4096, 1024, 256), (4000, 768, 200)]
LAYOUTS = [("k", "n"), ("k", "k"), ("m", "n"), ("m", "k")]


@pytest.mark.parametrize("impl", [0, 1], ids=["simt", "tc"])
@pytest.mark.parametrize("la,lb", LAYOUTS)
@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
def test_gemm(C, impl, la, lb, M, N, K):
    if impl == 1 and not (C.bcmt_test_set_tensor_cores(True, True) & 1):
        pytest.fail("tcgen05 GEMM unavailable on this GPU/build")
    gen = torch.Generator().manual_seed(M * 7 + N * 3 + K)
    dt = torch.bfloat16
    A, sam, sak, Al = _operand(M, K, la == "k", dt, gen)
    B, sbk, sbn, Bl = _operand(K, N, lb == "n", dt, gen)
    ref = Al.double() @ Bl.double()
    Ad, Bd = A.cuda(), B.cuda()
    for dto, tol in ((0, 1e-5), (1, 8e-3)):
        Cd = torch.full((M, N), float("nan"), dtype=torch.float32 if dto == 0 else dt, device="cuda")
        C.bcmt_test_gemm(impl, 1, dto, M, N, K, Ad, sam, sak, Bd, sbk, sbn, Cd, N)
        torch.cuda.synchronize()
        err = (Cd.double().cpu() - ref).abs().max().item() / ref.abs().max().item()
        assert err < tol, (dto, err)


@pytest.mark.parametrize("impl", [0, 1], ids=["simt", "tc"])
def test_gemm_split_k(C, impl):
    M, N, K, splits = 256, 128, 4096, 6
    gen = torch.Generator().manual_seed(5)
    A, sam, sak, Al = _operand(M, K, False, torch.bfloat16, gen)
    B, sbk, sbn, Bl = _operand(K, N, True, torch.bfloat16, gen)
    part = torch.full((splits, M, N), float("nan"), dtype=torch.float32, device="cuda")
    n = C.bcmt_test_gemm(impl, 1, 0, M, N, K, A.cuda(), sam, sak, B.cuda(), sbk, sbn, part, N,
                         splits)
    torch.cuda.synchronize()
    assert 1 < n <= splits
    got = part[:n].double().sum(0).cpu()
    ref = Al.double() @ Bl.double()
    assert (got - ref).abs().max().item() / ref.abs().max().item() < 1e-5


# Grouped CTA-pair launch (the backward's dX, K-split dW_QKV and dW_g): the
# layer's own shapes at B*T = 1024, D = 512, then ragged rows, ragged K and
# split counts that leave a short last range; the second case has no third
# product.
GROUP_SHAPES = [
    # (M0, N0, K0), (M1, N1, K1, splits1), (M2, N2, K2, splits2) or None
    ((1024, 512, 1536), (512, 1536, 1024, 7), (512, 512, 1024, 3)),
    ((1000, 256, 768), (256, 768, 1000, 3), None),
    ((300, 768, 320), (768, 512, 4096, 13), (256, 256, 4000, 5)),
]


def _eff_splits(K, s):
    nkb = -(-K // 64)
    kps = -(-nkb // max(1, min(s, nkb)))
    return -(-nkb // kps)


@pytest.mark.parametrize("p0,p1,p2", GROUP_SHAPES)
def test_gemm_group(C, p0, p1, p2):
    if not (C.bcmt_test_set_tensor_cores(True, True) & 1):
        pytest.fail("tcgen05 GEMM unavailable on this GPU/build")
    (M0, N0, K0), (M1, N1, K1, s1) = p0, p1
    gen = torch.Generator().manual_seed(M0 + N1 + K1)
    dt = torch.bfloat16
    A0, lda0, _, A0l = _operand(M0, K0, True, dt, gen)       # K-major
    B0t, _, ldb0t, B0l = _operand(K0, N0, False, dt, gen)    # stored [N0, K0]: K-major
    A1t, _, lda1t, A1l = _operand(M1, K1, False, dt, gen)    # stored [K1, M1]: MN-major
    B1, ldb1, _, B1l = _operand(K1, N1, True, dt, gen)       # stored [K1, N1]: MN-major
    C0 = torch.full((M0, N0), float("nan"), dtype=dt, device="cuda")
    part1 = torch.full((s1, M1, N1), float("nan"), dtype=torch.float32, device="cuda")
    extra = {}
    if p2 is not None:
        M2, N2, K2, s2 = p2
        A2t, _, lda2t, A2l = _operand(M2, K2, False, dt, gen)
        B2, ldb2, _, B2l = _operand(K2, N2, True, dt, gen)
        part2 = torch.full((s2, M2, N2), float("nan"), dtype=torch.float32, device="cuda")
        extra = dict(M2=M2, N2=N2, K2=K2, A2t=A2t.cuda(), lda2t=lda2t, B2=B2.cuda(), ldb2=ldb2,
                     part2=part2, splits2=s2)
    n1 = C.bcmt_test_gemm_group(M0, N0, K0, A0.cuda(), lda0, B0t.cuda(), ldb0t, C0, M1, N1, K1,
                                A1t.cuda(), lda1t, B1.cuda(), ldb1, part1, s1, **extra)
    torch.cuda.synchronize()
    assert n1 == _eff_splits(K1, s1)
    rel = lambda got, ref: (got - ref).abs().max().item() / ref.abs().max().item()
    assert rel(C0.double().cpu(), A0l.double() @ B0l.double()) < 8e-3
    assert rel(part1[:n1].double().sum(0).cpu(), A1l.double() @ B1l.double()) < 1e-5
    if p2 is not None:
        n2 = _eff_splits(K2, s2)
        assert rel(part2[:n2].double().sum(0).cpu(), A2l.double() @ B2l.double()) < 1e-5


def test_gemm_fp32_simt_exact_enough(C):
    M, N, K = 130, 192, 300
    gen = torch.Generator().manual_seed(9)
    A, sam, sak, Al = _operand(M, K, True, torch.float32, gen, pad=4)
    B, sbk, sbn, Bl = _operand(K, N, False, torch.float32, gen, pad=4)
    Cd = torch.empty(M, N, device="cuda")
    C.bcmt_test_gemm(0, 0, 0, M, N, K, A.cuda(), sam, sak, B.cuda(), sbk, sbn, Cd, N)
    torch.cuda.synchronize()
    ref = Al.double() @ Bl.double()
    assert (Cd.double().cpu() - ref).abs().max().item() < 1e-4


# ------------------------------------------------------------------ attention
ATTN_CASES = [
    # B, T, H, dh, L, dtype
    (2, 256, 2, 64, 64, "bf16"),
    (2, 200, 2, 64, 32, "bf16"),
    (1, 384, 3, 64, 128, "bf16"),
    (2, 130, 2, 64, 16, "bf16"),
    # more (tile, head) items than resident CTAs: several rounds per SM
    (4, 1024, 12, 64, 64, "bf16"),
    (3, 1000, 16, 64, 32, "bf16"),
    (2, 1280, 16, 64, 128, "bf16"),
    (1, 300, 2, 64, 256, "bf16"),
    (1, 600, 2, 64, 256, "bf16"),     # ragged last block, 1-3 key tiles per query tile
    (1, 1100, 1, 64, 512, "bf16"),
    (1, 1024, 1, 64, 1024, "bf16"),
    (2, 300, 4, 16, 64, "bf16"),      # the paper's 16-wide heads
    (2, 200, 8, 16, 128, "bf16"),
    (1, 520, 4, 16, 512, "bf16"),
    (2, 130, 4, 16, 16, "bf16"),
    (1, 520, 2, 32, 256, "bf16"),
    (2, 150, 2, 32, 32, "bf16"),
    (2, 256, 4, 32, 128, "bf16"),
    (4, 1024, 8, 16, 64, "bf16"),     # the paper's layer shape, several CTA rounds
    (2, 100, 2, 32, 24, "fp32"),
    (1, 256, 4, 32, 32, "fp32"),
]


def _impl_ok(impl, dh, L, dtype):
    if impl == 0:
        return True
    if dtype != "bf16":
        return False
    if impl == 1:
        return dh in (16, 32, 64) and L in (16, 32, 64, 128)
    return dh in (16, 32, 64) and ((L >= 16 and 128 % L == 0) or (L % 128 == 0 and L <= 1024))


def _attn_ref(q, k, v, L, H, dO):
    """Oracle attention alone: HOnly layer with W_O = I on the Q/K/V entry."""
    B, T, D = q.shape
    eye = np.eye(D)
    fw = O.forward(None, None, eye, np.zeros(D), np.zeros((D, D)), np.zeros((D, D)),
                   np.zeros(D), L, H, honly=True, q=q, k=k, v=v)
    gr = O.backward(fw, dO)
    dh = D // H
    lse = np.zeros((B, H, T))
    for b in range(B):
        for t0, t1 in O.block_ranges(T, L):
            for h in range(H):
                c = slice(h * dh, (h + 1) * dh)
                s = q[b, t0:t1, c] @ k[b, t0:t1, c].T / math.sqrt(dh)
                s = s + np.triu(np.full(s.shape, -np.inf), 1)
                m = s.max(1, keepdims=True)
                lse[b, h, t0:t1] = (m + np.log(np.exp(s - m).sum(1, keepdims=True)))[:, 0]
    return fw["Hhat"], lse, gr["dq"], gr["dk"], gr["dv"]


@pytest.mark.parametrize("impl", [0, 1, 2], ids=["simt", "tc", "tc_walk"])
@pytest.mark.parametrize("B,T,H,dh,L,dtype", ATTN_CASES)
def test_attention_fwd_bwd(C, impl, B, T, H, dh, L, dtype):
    if not _impl_ok(impl, dh, L, dtype):
        pytest.skip("shape outside this attention kernel")
    D = H * dh
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    gen = torch.Generator().manual_seed(B * 1000 + T + L)
    q, k, v, dO = (torch.randn(B, T, D, generator=gen).to(tdt) for _ in range(4))
    ref_o, ref_lse, ref_dq, ref_dk, ref_dv = _attn_ref(*(t.double().numpy() for t in (q, k, v)),
                                                       L, H, dO.double().numpy())
    p = C.make_params(B, T, D, H, L, dtype)
    qd, kd, vd, dOd = q.cuda(), k.cuda(), v.cuda(), dO.cuda()
    o = torch.full((B, T, D), float("nan"), dtype=tdt, device="cuda")
    lse = torch.full((B, H, T), float("nan"), device="cuda")
    C.bcmt_test_attn(impl, 0, p, qd, kd, vd, D, o, lse)
    drow = torch.empty(B, H, T, device="cuda")
    dq, dk, dv = (torch.full((B, T, D), float("nan"), dtype=tdt, device="cuda") for _ in range(3))
    C.bcmt_test_attn(impl, 1, p, qd, kd, vd, D, o, lse, dOd, drow, dq, dk, dv, D)
    C.bcmt_device_status()
    torch.cuda.synchronize()
    tol = 1e-4 if dtype == "fp32" else 2e-2

    def chk(name, got, ref):
        g = got.double().cpu().numpy()
        assert np.all(np.isfinite(g)), name
        err = np.abs(g - ref).max()
        if dtype != "fp32":
            err /= np.abs(ref).max()
        assert err <= tol, (name, err)

    chk("o", o, ref_o)
    chk("lse", lse, ref_lse)
    chk("dq", dq, ref_dq)
    chk("dk", dk, ref_dk)
    chk("dv", dv, ref_dv)


PAIR_SHAPES = [(256, 256, 64), (1000, 512, 320), (4096, 1536, 512), (77, 256, 1536),
               (4000, 768, 200), (520, 256, 64)]


@pytest.mark.parametrize("la,lb", LAYOUTS)
@pytest.mark.parametrize("M,N,K", PAIR_SHAPES)
def test_gemm_cta_pair(C, la, lb, M, N, K):
    """The CTA-pair (cta_group::2) GEMM against a float64 product."""
    gen = torch.Generator().manual_seed(M * 5 + N + K)
    dt = torch.bfloat16
    A, sam, sak, Al = _operand(M, K, la == "k", dt, gen)
    B, sbk, sbn, Bl = _operand(K, N, lb == "n", dt, gen)
    ref = Al.double() @ Bl.double()
    Ad, Bd = A.cuda(), B.cuda()
    for dto, tol in ((0, 1e-5), (1, 8e-3)):
        Cd = torch.full((M, N), float("nan"), dtype=torch.float32 if dto == 0 else dt, device="cuda")
        C.bcmt_test_gemm(2, 1, dto, M, N, K, Ad, sam, sak, Bd, sbk, sbn, Cd, N)
        C.bcmt_device_status()
        torch.cuda.synchronize()
        err = (Cd.double().cpu() - ref).abs().max().item() / ref.abs().max().item()
        assert err < tol, (dto, err)


def test_gemm_cta_pair_split_k(C):
    M, N, K, splits = 512, 256, 4096, 6
    gen = torch.Generator().manual_seed(6)
    A, sam, sak, Al = _operand(M, K, False, torch.bfloat16, gen)
    B, sbk, sbn, Bl = _operand(K, N, True, torch.bfloat16, gen)
    part = torch.full((splits, M, N), float("nan"), dtype=torch.float32, device="cuda")
    n = C.bcmt_test_gemm(2, 1, 0, M, N, K, A.cuda(), sam, sak, B.cuda(), sbk, sbn, part, N, splits)
    torch.cuda.synchronize()
    got = part[:n].double().sum(0).cpu()
    ref = Al.double() @ Bl.double()
    assert (got - ref).abs().max().item() / ref.abs().max().item() < 1e-5
