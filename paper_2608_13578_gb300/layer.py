"""Torch-facing helpers around the BCMT C ABI: output and workspace allocation,
and an autograd Function, so the mixer can be used as a layer.

Marshalling only: the forward and backward passes are the library's
``bcmt_forward`` / ``bcmt_backward`` kernels on the current CUDA stream.
"""

from __future__ import annotations

from typing import Dict, Optional

import torch

from . import bcmt as C

WEIGHTS = ("w_qkv", "w_o", "w_p", "w_m", "w_g")


def params_for(B, T, D, H, L, dtype="bf16", input_is_x=True, honly=False, flags=0):
    return C.make_params(B, T, D, H, L, dtype, input_is_x,
                         flags | (C.BCMT_FLAG_HONLY if honly else 0))


def _buffer(nbytes: int, device) -> torch.Tensor:
    # 256-byte granules; torch's caching allocator returns 512-byte aligned blocks
    return torch.empty(max(256, nbytes), dtype=torch.uint8, device=device)


def forward(p, t: Dict[str, torch.Tensor], stream=None, workspace: Optional[torch.Tensor] = None):
    """Runs bcmt_forward on the tensors in ``t`` (keys as in ``inputs.make_inputs``).

    Returns (y, workspace)."""
    ref = t["x"] if p.input_is_x else t["q"]
    y = torch.empty_like(ref)
    if workspace is None:
        workspace = _buffer(C.bcmt_workspace_size(p), ref.device)
    C.bcmt_forward(p, t.get("x") if p.input_is_x else None,
                   None if p.input_is_x else t["q"], None if p.input_is_x else t["k"],
                   None if p.input_is_x else t["v"], t.get("w_qkv") if p.input_is_x else None,
                   t["w_o"], t["w_p"], t["w_m"], t["w_g"], t["decay"], y, workspace, stream)
    return y, workspace


def backward(p, t: Dict[str, torch.Tensor], workspace: torch.Tensor, dy: torch.Tensor, stream=None,
             scratch: Optional[torch.Tensor] = None, out: Optional[Dict[str, torch.Tensor]] = None,
             decay_grad: bool = False):
    """Runs bcmt_backward; returns a dict of gradients (dx or dq/dk/dv, dw_*, and
    d_decay when ``decay_grad``)."""
    dev = dy.device
    if scratch is None:
        scratch = _buffer(C.bcmt_scratch_size(p), dev)
    g = out if out is not None else {}
    if p.input_is_x:
        g.setdefault("dx", torch.empty_like(t["x"]))
        g.setdefault("dw_qkv", torch.empty_like(t["w_qkv"]))
    else:
        for n in ("dq", "dk", "dv"):
            g.setdefault(n, torch.empty_like(t[n[1]]))
    for n in ("w_o", "w_p", "w_m", "w_g"):
        g.setdefault("d" + n, torch.empty_like(t[n]))
    if decay_grad:
        g.setdefault("d_decay", torch.empty_like(t["decay"]))
    C.bcmt_backward(p, dy, t["x"] if p.input_is_x else t["q"],
                    None if p.input_is_x else t["k"], None if p.input_is_x else t["v"],
                    t.get("w_qkv") if p.input_is_x else None, t["w_o"], t["w_p"], t["w_m"],
                    t["w_g"], t["decay"], workspace, scratch,
                    g["dx"] if p.input_is_x else g["dq"], None if p.input_is_x else g["dk"],
                    None if p.input_is_x else g["dv"], g.get("dw_qkv"), g["dw_o"], g["dw_p"],
                    g["dw_m"], g["dw_g"], stream, g.get("d_decay"))
    return g


class BCMTMixer(torch.autograd.Function):
    """y = BCMT(x) with the weights as differentiable inputs (x-entry layer).
    The decay gets a gradient only when it requires one (learned decay)."""

    @staticmethod
    def forward(ctx, x, w_qkv, w_o, w_p, w_m, w_g, decay, L: int, H: int, honly: bool = False):
        B, T, D = x.shape
        dt = "bf16" if x.dtype == torch.bfloat16 else "fp32"
        p = params_for(B, T, D, H, L, dt, True, honly)
        t = dict(x=x.contiguous(), w_qkv=w_qkv.contiguous(), w_o=w_o.contiguous(),
                 w_p=w_p.contiguous(), w_m=w_m.contiguous(), w_g=w_g.contiguous(),
                 decay=decay.contiguous())
        y, ws = forward(p, t)
        ctx.p = p
        ctx.save_for_backward(t["x"], t["w_qkv"], t["w_o"], t["w_p"], t["w_m"], t["w_g"],
                              t["decay"], ws)
        return y

    @staticmethod
    def backward(ctx, dy):
        x, w_qkv, w_o, w_p, w_m, w_g, decay, ws = ctx.saved_tensors
        t = dict(x=x, w_qkv=w_qkv, w_o=w_o, w_p=w_p, w_m=w_m, w_g=w_g, decay=decay)
        g = backward(ctx.p, t, ws, dy.contiguous(), decay_grad=ctx.needs_input_grad[6])
        return (g["dx"], g["dw_qkv"], g["dw_o"], g["dw_p"], g["dw_m"], g["dw_g"], g.get("d_decay"),
                None, None, None)


class Decoder:
    """Incremental decoding of B sequences in lockstep through one BCMT layer
    (``bcmt_decode_step``): ``step(x_t)`` takes the next token's input rows
    [B, D] and returns the layer's output rows [B, D]."""

    def __init__(self, weights: Dict[str, torch.Tensor], B: int, H: int, L: int,
                 honly: bool = False):
        D = weights["w_o"].shape[0]
        dt = "bf16" if weights["w_o"].dtype == torch.bfloat16 else "fp32"
        self.p = params_for(B, 1, D, H, L, dt, True, honly)
        self.w = weights
        self.state = _buffer(C.bcmt_decode_state_size(self.p), weights["w_o"].device)
        self.reset()

    def reset(self):
        C.bcmt_decode_reset(self.p, self.state)
        self.pos = 0

    def step(self, x_t: torch.Tensor, stream=None) -> torch.Tensor:
        w = self.w
        x_t = x_t.contiguous()
        y = torch.empty(x_t.shape, dtype=x_t.dtype, device=x_t.device)
        C.bcmt_decode_step(self.p, self.state, self.pos, x_t, w["w_qkv"], w["w_o"],
                           w.get("w_p"), w.get("w_m"), w.get("w_g"), w.get("decay"), y, stream)
        self.pos += 1
        return y
