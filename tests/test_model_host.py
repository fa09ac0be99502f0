"""Host-side pieces of the whole-model harness (CPU only): the dense-attention
decoder trains on the CPU, and the flop model matches the per-token counts of
the mixer (Sec. 3) plus the MLP and LM head."""

import pytest
import torch

from paper_2608_13578_gb300 import gpt


def test_flops_per_token_config5():
    c = gpt.GPTConfig()   # V 32000, D 512, 8 heads, MLP 2048, L 64, T 1024, 6 layers
    D, L, V = 512, 64, 32000
    mixer_fwd = 10 * D * D + 2 * D * (L + 1) + 2 * D * D / L
    fwd = 6 * (mixer_fwd + 4 * D * 2048) + 2 * D * V
    assert gpt.flops_per_token(c) == pytest.approx(3 * fwd)
    assert gpt.flops_per_token(c) == pytest.approx(222.4e6, rel=2e-3)
    dense = gpt.GPTConfig(mixer="dense")
    # dense: attention over all T keys, no W_g and no W_m
    assert gpt.flops_per_token(dense) == pytest.approx(
        gpt.flops_per_token(c) + 3 * 6 * (2 * D * (1024 - L) - 2 * D * D - 2 * D * D / L))


def test_dense_decoder_trains_on_cpu():
    c = gpt.GPTConfig(vocab=97, D=64, H=2, layers=2, mlp=128, L=16, T=32, mixer="dense")
    model = gpt.build(c, device="cpu", dtype=torch.float32)
    opt = gpt.make_optimizer(model, lr=3e-3)
    ids = torch.randint(0, c.vocab, (2, c.T + 1), generator=torch.Generator().manual_seed(1))
    losses = [gpt.train_step(model, opt, ids[:, :-1], ids[:, 1:]).item() for _ in range(10)]
    assert losses[-1] < losses[0] - 0.5


def test_decay_stays_fp32_under_dtype_casts():
    c = gpt.GPTConfig(vocab=97, D=64, H=2, layers=1, mlp=128, L=16, T=32, learn_decay=True)
    model = gpt.GPT(c).to(dtype=torch.bfloat16)
    assert model.blocks[0].mix.decay.dtype == torch.float32
    assert model.blocks[0].mix.w_qkv.dtype == torch.bfloat16
    assert isinstance(model.blocks[0].mix.decay, torch.nn.Parameter)
