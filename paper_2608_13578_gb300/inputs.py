"""Seeded synthetic inputs for the BCMT token mixer.

This module draws tensors only; it holds none of the mixer's arithmetic, so the
float64 oracle, the tests and the benchmark can all share it.

Every tensor is drawn in fp32 from one CPU ``torch.Generator`` in a fixed order
(x, W_qkv, W_O, w_p, W_m, W_g, decay, dY) and then rounded to the workload's
storage dtype.  The oracle consumes the rounded values upcast to float64, so the
GPU path and the oracle see bit-identical inputs.

Shapes follow the paper's notation (Sec. 3.1-3.8): B batch, T sequence length,
D model width, h heads of width D/h, L block size.  Weights use the row-vector
convention of Sec. 3.3 (``Q = X W_Q``): a weight is stored ``[D_in, D_out]``
row-major, and the three projections are packed side by side as
``W_qkv = [W_Q | W_K | W_V]`` of shape ``[D, 3D]``.  The decay of the
exponential causal memory (Sec. 3.5) is a per-channel fp32 vector ``a[D]``;
the paper's fixed scalar 0.8 is the broadcast case.
"""

from __future__ import annotations

import dataclasses
from typing import Dict, Optional, Tuple

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic BCMT-layer problem."""

    name: str
    B: int
    T: int
    D: int
    H: int
    L: int
    dtype: str = "bf16"          # "fp32" or "bf16": storage type of every tensor
    backward: bool = True        # forward+backward (True) or forward only
    decay: Tuple[float, float] = (0.8, 0.8)  # uniform range; equal ends = broadcast constant
    seed: int = 0
    input_is_x: bool = True      # the layer starts from x (True) or from Q, K, V (False)
    honly: bool = False          # the paper's "HOnly" ablation (Sec. 4.5): Y = H

    @property
    def dh(self) -> int:
        return self.D // self.H

    @property
    def n_blocks(self) -> int:
        return -(-self.T // self.L)

    @property
    def tokens(self) -> int:
        return self.B * self.T

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def _wl(name, B, T, D, H, L, dtype="bf16", backward=True, decay=(0.8, 0.8)):
    return Workload(name=name, B=B, T=T, D=D, H=H, L=L, dtype=dtype,
                    backward=backward, decay=decay)


# The problem families the benchmark and the parity tests use.  Sizes and
# value distributions mirror the paper's language-modelling runs (context up to
# 1024 tokens, Sec. 4.1) plus longer block-size and sequence-length sweeps.
WORKLOADS: Dict[str, Workload] = {}
for _w in [
    _wl("fwd_fp32_b1_t256_l32_d128_h4", 1, 256, 128, 4, 32, dtype="fp32",
        backward=False, decay=(0.5, 0.99)),
    _wl("fwdbwd_bf16_b8_t1024_l64_d512_h8", 8, 1024, 512, 8, 64),
    *[_wl(f"sweep_bf16_b16_t1024_l{L}_d768_h12", 16, 1024, 768, 12, L)
      for L in (32, 64, 128, 256)],
    *[_wl(f"seqscale_bf16_b4_t{T}_l128_d1024_h16", 4, T, 1024, 16, 128,
          decay=(0.9, 0.999)) for T in (2048, 4096, 8192, 16384)],
    # one layer of the paper's own model shape (Sec. 4.1: D 128, 8 heads of 16,
    # batch 16, context 1024), block sizes of its Table 2
    *[_wl(f"paper_bf16_b16_t1024_l{L}_d128_h8", 16, 1024, 128, 8, L)
      for L in (64, 128, 256, 512)],
]:
    WORKLOADS[_w.name] = _w

# The workload the headline throughput number is quoted on.
HEADLINE = "fwdbwd_bf16_b8_t1024_l64_d512_h8"
# The small fp32 case every oracle finishes in well under a second.
SMALL = "fwd_fp32_b1_t256_l32_d128_h4"


def torch_dtype(name: str) -> torch.dtype:
    return {"fp32": torch.float32, "bf16": torch.bfloat16}[name]


def make_inputs(w: Workload, seed: Optional[int] = None) -> Dict[str, torch.Tensor]:
    """Draw every input of workload ``w`` on the CPU, rounded to ``w.dtype``.

    Returns a dict with keys x [B,T,D], w_qkv [D,3D], w_o [D,D], w_p [D],
    w_m [D,D], w_g [D,D], decay [D] (always fp32), dy [B,T,D].  When the
    workload starts from Q, K, V instead of x, the dict also holds q, k, v
    [B,T,D] (head-major columns: head i owns columns i*dh .. i*dh+dh-1), drawn
    N(0,1) after the other tensors.
    """
    g = torch.Generator(device="cpu").manual_seed(w.seed if seed is None else seed)
    D, dt = w.D, torch_dtype(w.dtype)
    std = 1.0 / (D ** 0.5)

    def normal(*shape, scale=1.0):
        return (torch.randn(*shape, generator=g, dtype=torch.float32) * scale).to(dt)

    out = {
        "x": normal(w.B, w.T, D),
        "w_qkv": normal(D, 3 * D, scale=std),
        "w_o": normal(D, D, scale=std),
        "w_p": normal(D, scale=std),
        "w_m": normal(D, D, scale=std),
        "w_g": normal(D, D, scale=std),
    }
    lo, hi = w.decay
    u = torch.rand(D, generator=g, dtype=torch.float32)
    out["decay"] = (lo + (hi - lo) * u).to(torch.float32)
    out["dy"] = normal(w.B, w.T, D)
    if not w.input_is_x:
        out["q"] = normal(w.B, w.T, D)
        out["k"] = normal(w.B, w.T, D)
        out["v"] = normal(w.B, w.T, D)
    return out


def as_float64(t: torch.Tensor):
    """The exact value of a rounded tensor as a float64 numpy array."""
    return t.detach().to("cpu", torch.float64).numpy()
