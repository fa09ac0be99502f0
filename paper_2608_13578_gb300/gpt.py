"""A GPT-style decoder whose token mixer is the BCMT layer (Sec. 3), for
whole-model training steps.

The model follows the setting the paper trains (Sec. 4.1): a decoder-only
language model with learned absolute position embeddings, pre-LayerNorm
residual blocks (mixer, then a GELU MLP), a final LayerNorm, an untied LM head
and next-token cross-entropy, trained with AdamW.  The paper does not print its
block wiring; these are the standard choices, named as readings in the design
notes.  Only the mixer is this library: ``BCMTMixer`` calls the C ABI's forward
and backward kernels.  Embeddings, LayerNorm, MLP, LM head, loss and optimizer
are PyTorch's own CUDA kernels.

``mixer="dense"`` swaps in ordinary dense causal attention of the same shape
(x W_qkv -> PyTorch SDPA with a causal mask -> W_O), the baseline the paper
compares against; ``honly=True`` is the HOnly ablation of Sec. 4.5 (no block
summaries and no memory: Y = H).
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import torch
import torch.nn as nn
import torch.nn.functional as F

from .layer import BCMTMixer


@dataclass(frozen=True)
class GPTConfig:
    vocab: int = 32000
    D: int = 512
    H: int = 8
    layers: int = 6
    mlp: int = 2048
    L: int = 64
    T: int = 1024
    mixer: str = "bcmt"          # "bcmt" or "dense"
    honly: bool = False
    decay: float = 0.8           # broadcast per-channel decay (Sec. 3.5)
    learn_decay: bool = False    # learned per-channel decay (Sec. 5, future work)


class Mixer(nn.Module):
    """The token mixer of one block: BCMT (Sec. 3.3-3.8) or dense causal attention."""

    def __init__(self, c: GPTConfig):
        super().__init__()
        D = c.D
        self.c = c
        std = 1.0 / math.sqrt(D)   # weights ~ N(0, 1/D)
        self.w_qkv = nn.Parameter(torch.randn(D, 3 * D) * std)
        self.w_o = nn.Parameter(torch.randn(D, D) * std)
        if c.mixer == "bcmt":
            self.w_p = nn.Parameter(torch.randn(D) * std)
            self.w_m = nn.Parameter(torch.randn(D, D) * std)
            self.w_g = nn.Parameter(torch.randn(D, D) * std)
            decay = torch.full((D,), c.decay, dtype=torch.float32)
            if c.learn_decay:
                self.decay = nn.Parameter(decay)
            else:
                self.register_buffer("decay", decay)
        elif c.mixer != "dense":
            raise ValueError(f"unknown mixer {c.mixer!r}")

    def _apply(self, fn, *args, **kwargs):
        # the decay stays fp32 whatever dtype the rest of the model takes
        out = super()._apply(fn, *args, **kwargs)
        if self.c.mixer == "bcmt" and self.decay.dtype != torch.float32:
            self.decay.data = self.decay.data.float()
        return out

    def forward(self, x):
        c = self.c
        if c.mixer == "bcmt":
            return BCMTMixer.apply(x, self.w_qkv, self.w_o, self.w_p, self.w_m, self.w_g,
                                   self.decay, c.L, c.H, c.honly)
        B, T, D = x.shape
        q, k, v = (x @ self.w_qkv).view(B, T, 3, c.H, D // c.H).permute(2, 0, 3, 1, 4)
        o = F.scaled_dot_product_attention(q, k, v, is_causal=True)
        return o.transpose(1, 2).reshape(B, T, D) @ self.w_o


class Block(nn.Module):
    def __init__(self, c: GPTConfig):
        super().__init__()
        self.ln1 = nn.LayerNorm(c.D)
        self.mix = Mixer(c)
        self.ln2 = nn.LayerNorm(c.D)
        self.fc1 = nn.Linear(c.D, c.mlp)
        self.fc2 = nn.Linear(c.mlp, c.D)

    def forward(self, x):
        x = x + self.mix(self.ln1(x))
        return x + self.fc2(F.gelu(self.fc1(self.ln2(x))))


class GPT(nn.Module):
    def __init__(self, c: GPTConfig):
        super().__init__()
        self.c = c
        self.tok = nn.Embedding(c.vocab, c.D)
        self.pos = nn.Parameter(torch.randn(c.T, c.D) * 0.02)
        self.blocks = nn.ModuleList(Block(c) for _ in range(c.layers))
        self.ln_f = nn.LayerNorm(c.D)
        self.head = nn.Linear(c.D, c.vocab, bias=False)

    def forward(self, ids):
        x = self.tok(ids) + self.pos[: ids.shape[1]]
        for blk in self.blocks:
            x = blk(x)
        return self.head(self.ln_f(x))


def build(c: GPTConfig, device="cuda", dtype=torch.bfloat16, seed: int = 0) -> GPT:
    torch.manual_seed(seed)
    return GPT(c).to(device=device, dtype=dtype)


def make_optimizer(model: GPT, lr: float = 3e-4):
    return torch.optim.AdamW(model.parameters(), lr=lr, weight_decay=0.1,
                             fused=next(model.parameters()).is_cuda)


def train_step(model: GPT, opt, ids, targets):
    """One optimisation step on next-token cross-entropy; returns the loss tensor."""
    logits = model(ids)
    loss = F.cross_entropy(logits.reshape(-1, logits.shape[-1]), targets.reshape(-1))
    loss.backward()
    opt.step()
    opt.zero_grad(set_to_none=True)
    if model.c.mixer == "bcmt" and model.c.learn_decay:
        with torch.no_grad():
            for blk in model.blocks:
                blk.mix.decay.clamp_(0.0, 0.999)
    return loss


def flops_per_token(c: GPTConfig) -> float:
    """Algorithmic forward+backward flops per token (3x the forward): the
    mixer's 10 D^2 + 2 D (L+1) + 2 D^2 / L (dense: L -> T; HOnly: no W_m, W_g),
    the MLP's 4 D m and the LM head's 2 D V."""
    D, L = c.D, (c.T if c.mixer == "dense" else c.L)
    mix = 8 * D * D + 2 * D * (L + 1)
    if c.mixer == "bcmt" and not c.honly:
        mix += 2 * D * D + 2 * D * D / c.L
    return 3.0 * (c.layers * (mix + 4 * D * c.mlp) + 2 * D * c.vocab)
