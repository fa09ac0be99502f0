"""Float64 CPU oracle of the BCMT token mixer (test infrastructure only).

This is the plain, slow statement of what the mixer computes, used to check
the CUDA library.  Only the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import it; the product path never does.  It
shares no code with the CUDA path: the only module both sides use is the
seeded input generator, which holds none of the method's arithmetic.

Every step follows the paper's order and notation, with one explicit loop per
batch element, per block and per head.  NumPy matmul is the only library
primitive used for the dense products.

Forward (BCMT, Sec. 3.2-3.8):
  Sec. 3.2  block decomposition: N_b = ceil(T/L) contiguous blocks, last one
            ragged (L_i <= L).
  Sec. 3.3  per block and head: Q_i = X W_Q,i, K_i, V_i likewise;
            H_i = softmax(Q_i K_i^T / sqrt(d_h) + causal mask) V_i;
            H^(b) = Concat(H_1..H_h) W_O; H = the blocks stacked in order.
  Sec. 3.4  s = H^(i) W_p (W_p in R^D), alpha = softmax(s) over the block,
            S^(i) = H^(i)^T alpha.
  Sec. 3.5  M^(i) = sum_{j<=i} a^(i-j) S^(j) / sum_{j<=i} a^(i-j)
            (the direct double sum; a^0 = 1 also when a = 0);
            M_proj = M W_m; M_causal^(1) = 0, M_causal^(i) = M_proj^(i-1).
  Sec. 3.7  M_tokens: block i's memory row repeated for each of its tokens.
  Sec. 3.8  G = sigmoid(H W_g); Y = H + G * M_tokens.
  Sec. 4.5  the "HOnly" ablation: Y = H, no summary and no memory.

Backward: the paper gives none (it trains with autograd, Sec. 4.1), so the
gradients below are derived by hand from the forward above, step by step in
reverse order; the tests pin them with central finite differences.

Readings where the paper is silent (each also listed in the design notes):
  * the decay ``a`` is a per-channel vector a[D] in [0,1); the paper's fixed
    scalar 0.8 (Sec. 3.5) is the broadcast case.  The paper does not learn it;
    its gradient d_decay (for the learned per-channel decay that Sec. 5 names
    as future work) is the derivative of the double sum of Sec. 3.5 itself:
    with num_i = sum_j a^(i-j) S_j and den_i = sum_j a^(i-j),
      dM_i/da = (sum_j (i-j) a^(i-j-1) S_j - M_i sum_j (i-j) a^(i-j-1)) / den_i;
  * no biases anywhere, no scale on the pooling scores s;
  * the pooling and attention softmaxes of a ragged last block run over its
    L_i real tokens; the memory denominator counts blocks, not tokens;
  * head i owns columns i*d_h .. (i+1)*d_h - 1 of Q, K, V and of Concat(.);
  * the decay symbol is written ``a`` here because the paper also uses alpha
    for the pooling weights.

All arrays are float64 numpy; shapes: x [B,T,D], w_qkv [D,3D] = [W_Q|W_K|W_V]
(row-vector convention X W), w_o/w_m/w_g [D,D], w_p [D], decay [D].
"""

from __future__ import annotations

import math
from typing import Dict, Optional

import numpy as np


def _sigmoid(u):
    return 1.0 / (1.0 + np.exp(-u))


def _softmax_rows(z):
    # Row softmax with the row maximum subtracted; -inf entries give 0.
    m = np.max(z, axis=-1, keepdims=True)
    e = np.exp(z - m)
    return e / np.sum(e, axis=-1, keepdims=True)


def block_ranges(T: int, L: int):
    """Sec. 3.2: token ranges [start, end) of the N_b = ceil(T/L) blocks."""
    n_b = -(-T // L)
    return [(i * L, min((i + 1) * L, T)) for i in range(n_b)]


def forward(x: Optional[np.ndarray], w_qkv: Optional[np.ndarray], w_o, w_p, w_m, w_g,
            decay, L: int, H: int, honly: bool = False,
            q: Optional[np.ndarray] = None, k: Optional[np.ndarray] = None,
            v: Optional[np.ndarray] = None) -> Dict[str, np.ndarray]:
    """BCMT mixer forward.  Returns a dict holding Y and every intermediate.

    Either ``x`` and ``w_qkv`` are given (the layer projects Q, K, V itself,
    Sec. 3.3), or ``q``, ``k``, ``v`` [B,T,D] are given directly.
    """
    input_is_x = x is not None
    if input_is_x:
        B, T, D = x.shape
    else:
        B, T, D = q.shape
    d_h = D // H
    blocks = block_ranges(T, L)
    n_b = len(blocks)
    a = np.asarray(decay, dtype=np.float64)

    Q = np.zeros((B, T, D))
    K = np.zeros((B, T, D))
    V = np.zeros((B, T, D))
    A = {}                          # attention probabilities per (b, block, head)
    Hhat = np.zeros((B, T, D))      # Concat of head outputs (before W_O)
    Hloc = np.zeros((B, T, D))      # H = Hhat W_O
    s = np.zeros((B, T))
    alpha = np.zeros((B, T))
    S = np.zeros((B, n_b, D))
    M = np.zeros((B, n_b, D))
    Z = np.zeros((n_b, D))
    P = np.zeros((B, n_b, D))       # M_proj
    C = np.zeros((B, n_b, D))       # M_causal
    G = np.zeros((B, T, D))
    Y = np.zeros((B, T, D))

    if input_is_x:
        W_Q = np.ascontiguousarray(w_qkv[:, 0:D])
        W_K = np.ascontiguousarray(w_qkv[:, D:2 * D])
        W_V = np.ascontiguousarray(w_qkv[:, 2 * D:3 * D])

    for b in range(B):
        # Sec. 3.3: local multi-head causal attention, block by block.
        for i, (t0, t1) in enumerate(blocks):
            Li = t1 - t0
            if input_is_x:
                Xb = x[b, t0:t1]
                Qb = Xb @ W_Q
                Kb = Xb @ W_K
                Vb = Xb @ W_V
            else:
                Qb, Kb, Vb = q[b, t0:t1], k[b, t0:t1], v[b, t0:t1]
            Q[b, t0:t1], K[b, t0:t1], V[b, t0:t1] = Qb, Kb, Vb
            # causal mask: key c is hidden from query r when c > r
            mask = np.triu(np.full((Li, Li), -np.inf), k=1)
            for hd in range(H):
                cols = slice(hd * d_h, (hd + 1) * d_h)
                scores = Qb[:, cols] @ Kb[:, cols].T / math.sqrt(d_h) + mask
                Ab = _softmax_rows(scores)
                A[(b, i, hd)] = Ab
                Hhat[b, t0:t1, cols] = Ab @ Vb[:, cols]
            Hloc[b, t0:t1] = Hhat[b, t0:t1] @ w_o

        if honly:
            Y[b] = Hloc[b]
            continue

        # Sec. 3.4: adaptive block summaries.
        for i, (t0, t1) in enumerate(blocks):
            Hb = Hloc[b, t0:t1]
            sb = Hb @ w_p
            ab = _softmax_rows(sb[None, :])[0]
            s[b, t0:t1] = sb
            alpha[b, t0:t1] = ab
            S[b, i] = Hb.T @ ab

        # Sec. 3.5: normalised exponential causal memory, the direct double sum.
        for i in range(n_b):
            num = np.zeros(D)
            den = np.zeros(D)
            for j in range(i + 1):
                wgt = a ** (i - j)          # numpy: 0.0 ** 0 == 1.0
                num += wgt * S[b, j]
                den += wgt
            M[b, i] = num / den
            Z[i] = den
        P[b] = M[b] @ w_m
        C[b, 0] = 0.0
        for i in range(1, n_b):
            C[b, i] = P[b, i - 1]

        # Sec. 3.7-3.8: broadcast to the block's tokens, gate, inject.
        G[b] = _sigmoid(Hloc[b] @ w_g)
        for i, (t0, t1) in enumerate(blocks):
            # every token of block i receives the same memory row C_i
            Y[b, t0:t1] = Hloc[b, t0:t1] + G[b, t0:t1] * C[b, i][None, :]

    return dict(Y=Y, Q=Q, K=K, V=V, A=A, Hhat=Hhat, H=Hloc, s=s, alpha=alpha,
                S=S, M=M, Z=Z, P=P, C=C, G=G,
                _in=dict(x=x, w_qkv=w_qkv, w_o=w_o, w_p=w_p, w_m=w_m, w_g=w_g,
                         decay=a, L=L, H=H, honly=honly, input_is_x=input_is_x))


def backward(fw: Dict[str, np.ndarray], dY: np.ndarray) -> Dict[str, np.ndarray]:
    """Hand-derived gradients of the forward above, in reverse order.

    Returns dx (or dq, dk, dv when the layer started from Q, K, V) and
    dw_qkv (when it started from x), dw_o, dw_p, dw_m, dw_g, d_decay.
    """
    inp = fw["_in"]
    w_qkv, w_o, w_p, w_m, w_g = (inp[n] for n in ("w_qkv", "w_o", "w_p", "w_m", "w_g"))
    a, L, H, honly = inp["decay"], inp["L"], inp["H"], inp["honly"]
    B, T, D = dY.shape
    d_h = D // H
    blocks = block_ranges(T, L)
    n_b = len(blocks)
    Hloc, Hhat, G, C, M, Z, alpha = (fw[n] for n in ("H", "Hhat", "G", "C", "M", "Z", "alpha"))

    dH = np.zeros((B, T, D))
    dw_g = np.zeros((D, D))
    dw_m = np.zeros((D, D))
    dw_p = np.zeros(D)
    d_decay = np.zeros(D)
    dw_o = np.zeros((D, D))
    dQ = np.zeros((B, T, D))
    dK = np.zeros((B, T, D))
    dV = np.zeros((B, T, D))

    for b in range(B):
        dH[b] = dY[b]
        if not honly:
            # Sec. 3.8 reversed: Y = H + G * C_blk, G = sigmoid(U), U = H W_g.
            dC = np.zeros((n_b, D))
            dU = np.zeros((T, D))
            for i, (t0, t1) in enumerate(blocks):
                dG = dY[b, t0:t1] * C[b, i][None, :]
                dU[t0:t1] = dG * G[b, t0:t1] * (1.0 - G[b, t0:t1])
                dC[i] = np.sum(dY[b, t0:t1] * G[b, t0:t1], axis=0)
            dw_g += Hloc[b].T @ dU
            dH[b] += dU @ w_g.T

            # Sec. 3.5 reversed: C_i = P_{i-1}, P = M W_m.
            dP = np.zeros((n_b, D))
            for i in range(n_b - 1):
                dP[i] = dC[i + 1]
            dw_m += M[b].T @ dP
            dM = dP @ w_m.T
            # M_i = sum_{j<=i} a^(i-j) S_j / Z_i  =>  dS_j = sum_{i>=j} a^(i-j) dM_i / Z_i.
            dS = np.zeros((n_b, D))
            for j in range(n_b):
                for i in range(j, n_b):
                    dS[j] += (a ** (i - j)) * dM[i] / Z[i]
            # d M_i / d a from the same double sum (terms j < i; j = i has a^0)
            for i in range(n_b):
                dnum = np.zeros(D)
                dden = np.zeros(D)
                for j in range(i):
                    w = (i - j) * a ** (i - j - 1)
                    dnum += w * fw["S"][b, j]
                    dden += w
                d_decay += dM[i] * (dnum - M[b, i] * dden) / Z[i]

            # Sec. 3.4 reversed: S_i = sum_t alpha_t H_t, alpha = softmax(s), s = H w_p.
            for i, (t0, t1) in enumerate(blocks):
                Hb = Hloc[b, t0:t1]
                ab = alpha[b, t0:t1]
                g = Hb @ dS[i]                       # d S_i / d alpha_t, dotted with dS_i
                ds = ab * (g - np.dot(ab, g))        # softmax Jacobian
                dH[b, t0:t1] += np.outer(ab, dS[i]) + np.outer(ds, w_p)
                dw_p += Hb.T @ ds

        # Sec. 3.3 reversed: H = Hhat W_O, Hhat = Concat(A_h V_h).
        dw_o += Hhat[b].T @ dH[b]
        dHhat = dH[b] @ w_o.T
        for i, (t0, t1) in enumerate(blocks):
            for hd in range(H):
                cols = slice(hd * d_h, (hd + 1) * d_h)
                Ab = fw["A"][(b, i, hd)]
                Qb = fw["Q"][b, t0:t1, cols]
                Kb = fw["K"][b, t0:t1, cols]
                Vb = fw["V"][b, t0:t1, cols]
                dO = dHhat[t0:t1, cols]
                dA = dO @ Vb.T
                dV[b, t0:t1, cols] = Ab.T @ dO
                dScore = Ab * (dA - np.sum(dA * Ab, axis=1, keepdims=True))
                dQ[b, t0:t1, cols] = dScore @ Kb / math.sqrt(d_h)
                dK[b, t0:t1, cols] = dScore.T @ Qb / math.sqrt(d_h)

    out = dict(dw_o=dw_o, dw_p=dw_p, dw_m=dw_m, dw_g=dw_g, d_decay=d_decay)
    if inp["input_is_x"]:
        x = inp["x"]
        dQKV = np.concatenate([dQ, dK, dV], axis=2)       # [B,T,3D]
        out["dx"] = dQKV @ w_qkv.T
        out["dw_qkv"] = x.reshape(B * T, D).T @ dQKV.reshape(B * T, 3 * D)
    else:
        out["dq"], out["dk"], out["dv"] = dQ, dK, dV
    return out


def forward_from_inputs(inputs: dict, L: int, H: int, honly: bool = False,
                        input_is_x: bool = True):
    """Convenience: run ``forward`` on a dict of float64 arrays."""
    if input_is_x:
        return forward(inputs["x"], inputs["w_qkv"], inputs["w_o"], inputs["w_p"],
                       inputs["w_m"], inputs["w_g"], inputs["decay"], L, H, honly=honly)
    return forward(None, None, inputs["w_o"], inputs["w_p"], inputs["w_m"], inputs["w_g"],
                   inputs["decay"], L, H, honly=honly,
                   q=inputs["q"], k=inputs["k"], v=inputs["v"])
