"""Pins of the float64 oracle to facts outside itself (CPU only).

Each test ties one stage of the BCMT forward (Sec. 3.2-3.8) or the hand-derived
backward to something the oracle does not compute itself: hand-derived worked
examples, a library routine that the method reduces to in a special case, a
closed form, a structural invariant, or central finite differences.  A dropped
term, a wrong sign or index, or a transposed operand in the oracle fails at
least one of them.
"""

import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.special import softmax as scipy_softmax

from oracle import bcmt_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_examples.json")


def rand_problem(B=2, T=10, D=8, H=2, seed=0, decay=None, scale=1.0):
    rng = np.random.default_rng(seed)
    p = dict(
        x=rng.standard_normal((B, T, D)) * scale,
        w_qkv=rng.standard_normal((D, 3 * D)) / math.sqrt(D),
        w_o=rng.standard_normal((D, D)) / math.sqrt(D),
        w_p=rng.standard_normal(D) / math.sqrt(D),
        w_m=rng.standard_normal((D, D)) / math.sqrt(D),
        w_g=rng.standard_normal((D, D)) / math.sqrt(D),
        decay=rng.uniform(0.5, 0.99, D) if decay is None else np.broadcast_to(
            np.asarray(decay, dtype=np.float64), (D,)).copy(),
    )
    return p


def run(p, L, H, **kw):
    return O.forward(p["x"], p["w_qkv"], p["w_o"], p["w_p"], p["w_m"], p["w_g"],
                     p["decay"], L, H, **kw)


# ---------------------------------------------------------------- worked examples
@pytest.mark.parametrize("idx", [0, 1])
def test_worked_examples(idx):
    """Hand-derived values with exact fractions (fixture cites Sec. 3.2-3.8)."""
    g = json.load(open(GOLDEN))
    c, ex = g["common"], g["examples"][idx]
    arr = lambda v: np.asarray(v, dtype=np.float64)
    fw = O.forward(arr(c["x"]), arr(c["w_qkv"]), arr(c["w_o"]), arr(ex["w_p"]),
                   arr(c["w_m"]), arr(ex["w_g"]), arr(c["decay"]), c["L"], c["H"])
    for key, val in ex["expect"].items():
        np.testing.assert_allclose(fw[key], arr(val), rtol=0, atol=1e-13, err_msg=key)


# ----------------------------------------------------------- attention stage pins
def _sdpa_heads(q, k, v, H, mask_bool):
    """torch float64 scaled_dot_product_attention per head, heads re-concatenated."""
    B, T, D = q.shape
    dh = D // H
    tq = torch.from_numpy(q).view(B, T, H, dh).transpose(1, 2)
    tk = torch.from_numpy(k).view(B, T, H, dh).transpose(1, 2)
    tv = torch.from_numpy(v).view(B, T, H, dh).transpose(1, 2)
    o = torch.nn.functional.scaled_dot_product_attention(
        tq, tk, tv, attn_mask=torch.from_numpy(mask_bool))
    return o.transpose(1, 2).reshape(B, T, D).numpy()


@pytest.mark.parametrize("T,L", [(7, 7), (7, 16), (12, 12)])
def test_single_block_is_dense_causal_attention(T, L):
    """One block covering the sequence: no memory is injected (Sec. 3.5: the
    first block's causal memory is 0), so Y = H = dense causal MHA + W_O."""
    p = rand_problem(B=2, T=T, D=8, H=2, seed=1)
    fw = run(p, L, 2)
    D = 8
    q, k, v = (p["x"] @ p["w_qkv"][:, i * D:(i + 1) * D] for i in range(3))
    causal = np.tril(np.ones((T, T), dtype=bool))
    ref = _sdpa_heads(q, k, v, 2, causal) @ p["w_o"]
    np.testing.assert_allclose(fw["H"], ref, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(fw["Y"], fw["H"])
    # with no memory path active the summary/memory/gate weights get no gradient
    gr = O.backward(fw, np.random.default_rng(2).standard_normal((2, T, D)))
    for n in ("dw_g", "dw_m", "dw_p"):
        assert np.all(gr[n] == 0.0), n


@pytest.mark.parametrize("T,L,H", [(10, 4, 2), (16, 4, 4), (9, 3, 1)])
def test_blockwise_attention_is_block_diagonal_sdpa(T, L, H):
    """Sec. 3.3: attention inside blocks only = SDPA under a block-diagonal causal mask."""
    p = rand_problem(B=2, T=T, D=8, H=H, seed=3)
    fw = run(p, L, H)
    D = 8
    q, k, v = (p["x"] @ p["w_qkv"][:, i * D:(i + 1) * D] for i in range(3))
    r = np.arange(T)
    allowed = (r[None, :] <= r[:, None]) & ((r[None, :] // L) == (r[:, None] // L))
    np.testing.assert_allclose(fw["Hhat"], _sdpa_heads(q, k, v, H, allowed), rtol=0, atol=1e-12)


# ------------------------------------------------------------- summary stage pins
def test_pooling_weights_are_block_softmax():
    """Sec. 3.4: alpha = softmax(H w_p) over each block; sums to 1 per block."""
    p = rand_problem(B=2, T=11, D=8, H=2, seed=4)
    L = 4
    fw = run(p, L, 2)
    for b in range(2):
        for i, (t0, t1) in enumerate(O.block_ranges(11, L)):
            s = fw["H"][b, t0:t1] @ p["w_p"]
            np.testing.assert_allclose(fw["alpha"][b, t0:t1], scipy_softmax(s), rtol=0, atol=1e-14)
            assert abs(fw["alpha"][b, t0:t1].sum() - 1.0) < 1e-14
            np.testing.assert_allclose(fw["S"][b, i], np.average(fw["H"][b, t0:t1], axis=0,
                                                                 weights=scipy_softmax(s)),
                                       rtol=0, atol=1e-13)


def test_zero_pooling_weights_give_block_mean():
    """w_p = 0 makes every score equal, so S_i is the plain mean of block i."""
    p = rand_problem(B=1, T=10, D=8, H=2, seed=5)
    p["w_p"][:] = 0.0
    fw = run(p, 4, 2)
    for i, (t0, t1) in enumerate(O.block_ranges(10, 4)):
        np.testing.assert_allclose(fw["S"][0, i], fw["H"][0, t0:t1].mean(axis=0), rtol=0, atol=1e-14)


# -------------------------------------------------------------- memory stage pins
def test_decay_zero_memory_is_previous_summary():
    """a = 0: M_i = S_i, so block i receives S_{i-1} W_m (Sec. 3.5 with 0^0 = 1)."""
    p = rand_problem(B=2, T=13, D=8, H=2, seed=6, decay=0.0)
    fw = run(p, 4, 2)
    np.testing.assert_allclose(fw["M"], fw["S"], rtol=0, atol=0)
    np.testing.assert_allclose(fw["C"][:, 1:], fw["S"][:, :-1] @ p["w_m"], rtol=0, atol=1e-13)
    assert np.all(fw["C"][:, 0] == 0.0)


def test_denominator_closed_form():
    """Sum_{j<=i} a^(i-j) = (1 - a^(i+1)) / (1 - a) (geometric series)."""
    p = rand_problem(B=1, T=40, D=8, H=2, seed=7)
    fw = run(p, 4, 2)
    a = p["decay"]
    for i in range(10):
        np.testing.assert_allclose(fw["Z"][i], (1 - a ** (i + 1)) / (1 - a), rtol=1e-14)


def test_memory_is_convex_combination():
    """Constant input: every block has the same summary c, so M_i = c (Sec. 3.5:
    the normalised weights form a convex combination)."""
    p = rand_problem(B=1, T=11, D=8, H=2, seed=8)
    p["x"][:] = p["x"][:, :1, :]
    fw = run(p, 4, 2)
    for i in range(fw["M"].shape[1]):
        np.testing.assert_allclose(fw["M"][0, i], fw["S"][0, 0], rtol=0, atol=1e-13)


def test_memory_brute_force_token_sum():
    """O(T^2) brute force: the memory row a token of block i receives is the
    sum over every token u of an earlier block of a^(i-1-blk(u)) alpha_u H_u,
    divided by (1-a^i)/(1-a), times W_m (Sec. 3.4-3.7 composed)."""
    T, L = 14, 3
    p = rand_problem(B=2, T=T, D=8, H=2, seed=9)
    p["decay"][0] = 0.0
    fw = run(p, L, 2)
    a = p["decay"]
    for b in range(2):
        for t in range(T):
            i = t // L
            if i == 0:
                assert np.all(fw["C"][b, 0] == 0.0)
                continue
            num = np.zeros(8)
            for u in range(T):
                j = u // L
                if j < i:
                    num += np.power(a, i - 1 - j) * fw["alpha"][b, u] * fw["H"][b, u]
            den = np.where(a == 0.0, 1.0, (1 - np.power(a, i)) / np.where(a == 0.0, 1.0, 1 - a))
            expect = (num / den) @ p["w_m"]
            np.testing.assert_allclose(fw["C"][b, i], expect, rtol=0, atol=1e-12)
            np.testing.assert_allclose(fw["Y"][b, t] - fw["H"][b, t], fw["G"][b, t] * expect,
                                       rtol=0, atol=1e-12)


# -------------------------------------------------------- gate / ablation pins
def test_honly_and_zero_memory_projection():
    """Sec. 4.5 HOnly: Y = H.  W_m = 0 removes the memory path: Y = H too."""
    p = rand_problem(B=2, T=10, D=8, H=2, seed=10)
    fw_h = run(p, 4, 2, honly=True)
    np.testing.assert_array_equal(fw_h["Y"], fw_h["H"])
    p["w_m"][:] = 0.0
    fw = run(p, 4, 2)
    np.testing.assert_array_equal(fw["Y"], fw["H"])
    np.testing.assert_array_equal(fw["H"], fw_h["H"])


def test_zero_gate_weights_give_half_gate():
    """W_g = 0: G = sigmoid(0) = 1/2 exactly, Y = H + C/2."""
    p = rand_problem(B=1, T=10, D=8, H=2, seed=11)
    p["w_g"][:] = 0.0
    fw = run(p, 4, 2)
    assert np.all(fw["G"] == 0.5)
    for t in range(10):
        np.testing.assert_allclose(fw["Y"][0, t], fw["H"][0, t] + 0.5 * fw["C"][0, t // 4],
                                   rtol=0, atol=1e-15)


# ------------------------------------------------------------- structural pins
def test_causality():
    """Sec. 3.6: perturbing token t changes no output before t (bitwise)."""
    p = rand_problem(B=1, T=17, D=8, H=2, seed=12)
    base = run(p, 4, 2)["Y"]
    for t in (0, 3, 4, 9, 16):
        q = {k: v.copy() for k, v in p.items()}
        q["x"][0, t] += 1.0
        y = run(q, 4, 2)["Y"]
        np.testing.assert_array_equal(y[0, :t], base[0, :t])
        assert np.any(y[0, t] != base[0, t])


def test_batch_permutation():
    p = rand_problem(B=3, T=9, D=8, H=2, seed=13)
    fw = run(p, 4, 2)
    perm = [2, 0, 1]
    q = dict(p)
    q["x"] = p["x"][perm]
    np.testing.assert_allclose(run(q, 4, 2)["Y"], fw["Y"][perm], rtol=0, atol=1e-14)


# ---------------------------------------------------------------- backward pins
def _loss(p, dY, L, H, honly=False, qkv=None):
    if qkv is None:
        fw = run(p, L, H, honly=honly)
    else:
        fw = O.forward(None, None, p["w_o"], p["w_p"], p["w_m"], p["w_g"], p["decay"], L, H,
                       honly=honly, q=qkv["q"], k=qkv["k"], v=qkv["v"])
    return float(np.sum(fw["Y"] * dY))


def _fd_check(p, L, H, names, honly=False, qkv=None, eps=1e-6):
    B, T = (p["x"].shape[:2] if qkv is None else qkv["q"].shape[:2])
    D = p["w_o"].shape[0]
    dY = np.random.default_rng(99).standard_normal((B, T, D))
    if qkv is None:
        fw = run(p, L, H, honly=honly)
    else:
        fw = O.forward(None, None, p["w_o"], p["w_p"], p["w_m"], p["w_g"], p["decay"], L, H,
                       honly=honly, q=qkv["q"], k=qkv["k"], v=qkv["v"])
    gr = O.backward(fw, dY)
    for n in names:
        src = qkv if (qkv is not None and n in ("q", "k", "v")) else p
        arr = src[n]
        fd = np.zeros_like(arr)
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            idx = it.multi_index
            old = arr[idx]
            arr[idx] = old + eps
            lp = _loss(p, dY, L, H, honly, qkv)
            arr[idx] = old - eps
            lm = _loss(p, dY, L, H, honly, qkv)
            arr[idx] = old
            fd[idx] = (lp - lm) / (2 * eps)
        g = gr["d_decay" if n == "decay" else "d" + n]
        err = np.max(np.abs(g - fd)) / max(1e-12, np.max(np.abs(fd)))
        assert err < 1e-6, (n, err)


def test_backward_finite_differences():
    """Every gradient of the hand-derived backward against central differences
    (ragged last block, per-channel decay including a = 0, two heads)."""
    p = rand_problem(B=2, T=10, D=8, H=2, seed=14)
    p["decay"][1] = 0.0
    _fd_check(p, 4, 2, ["x", "w_qkv", "w_o", "w_p", "w_m", "w_g", "decay"])


def test_backward_finite_differences_qkv_entry():
    """Layer entered at Q, K, V: gradients dq, dk, dv and the mixer weights."""
    p = rand_problem(B=1, T=7, D=4, H=2, seed=15)
    rng = np.random.default_rng(16)
    qkv = {n: rng.standard_normal((1, 7, 4)) for n in ("q", "k", "v")}
    _fd_check(p, 3, 2, ["q", "k", "v", "w_o", "w_p", "w_m", "w_g"], qkv=qkv)


def test_backward_finite_differences_honly():
    p = rand_problem(B=1, T=6, D=4, H=1, seed=17)
    _fd_check(p, 4, 1, ["x", "w_qkv", "w_o", "decay"], honly=True)


def test_decay_gradient_two_blocks_closed_form():
    """Two blocks: M_1 = (a S_0 + S_1) / (1 + a), so dM_1/da = (S_0 - M_1) / (1 + a)
    and d_decay = sum_b dM_1 * (S_0 - M_1) / (1 + a), with dM_1 = dP_1 W_m^T where
    dP_1 = 0 (the last block's memory feeds no block): the decay gradient of two
    blocks is exactly zero, and with three it is the closed form through M_1."""
    p = rand_problem(B=2, T=8, D=6, H=2, seed=31)
    dY = np.random.default_rng(32).standard_normal((2, 8, 6))
    gr = O.backward(run(p, 4, 2), dY)
    np.testing.assert_array_equal(gr["d_decay"], np.zeros(6))
    # three blocks: only M_1 and M_0 get gradient; M_0 = S_0 has no decay
    fw = run(p, 3, 2)   # T = 8, L = 3: blocks of 3, 3, 2 tokens
    gr = O.backward(fw, dY)
    a = p["decay"]
    expect = np.zeros(6)
    for b in range(2):
        dC2 = np.sum(dY[b, 6:8] * fw["G"][b, 6:8], axis=0)   # dP_1 = dC_2
        dM1 = dC2 @ p["w_m"].T
        expect += dM1 * (fw["S"][b, 0] - fw["M"][b, 1]) / (1.0 + a)
    np.testing.assert_allclose(gr["d_decay"], expect, rtol=1e-12, atol=1e-14)


def test_block_never_sees_its_own_summary():
    """Sec. 3.6: the shift makes block i's memory depend on blocks < i only, so
    perturbing any token of block i leaves the memory rows of blocks <= i
    bitwise unchanged, and changes block i+1's."""
    p = rand_problem(B=1, T=16, D=8, H=2, seed=18)
    L = 4
    base = run(p, L, 2)["C"]
    for t in (1, 5, 10, 15):
        i = t // L
        q = {k: v.copy() for k, v in p.items()}
        q["x"][0, t] += 0.5
        c = run(q, L, 2)["C"]
        np.testing.assert_array_equal(c[0, :i + 1], base[0, :i + 1])
        if i + 1 < c.shape[1]:
            assert np.any(c[0, i + 1] != base[0, i + 1])
