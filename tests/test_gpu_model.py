"""The mixer as a PyTorch autograd layer, and whole-model training steps.

``BCMTMixer`` is checked against the float64 oracle through autograd (output,
every input and weight gradient, and the learned-decay gradient), and the
GPT-style decoder built around it is trained for a few steps on one fixed batch
(BCMT, its HOnly ablation, learned decay, and the dense-attention model of the
same shape): the loss must stay finite and fall.
"""

import pytest
import torch

from paper_2608_13578_gb300.inputs import Workload, make_inputs
from tests.helpers import assert_close, oracle_run

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype,T,L", [("bf16", 200, 64), ("fp32", 130, 32)])
def test_mixer_autograd_matches_oracle(cuda_ok, dtype, T, L):
    from paper_2608_13578_gb300.layer import BCMTMixer
    w = Workload("autograd", 2, T, 128, 2, L, dtype, True, (0.5, 0.99), 7)
    t = make_inputs(w)
    names = ("x", "w_qkv", "w_o", "w_p", "w_m", "w_g", "decay")
    dev = {n: t[n].cuda().requires_grad_(True) for n in names}
    y = BCMTMixer.apply(*(dev[n] for n in names), L, 2)
    y.backward(t["dy"].cuda())
    fw, gr = oracle_run(w, t)
    assert_close("Y", y, fw["Y"], dtype)
    for n in names:
        key = "d_decay" if n == "decay" else "d" + n
        assert_close(key, dev[n].grad, gr[key], dtype)


def _train(cfg, steps=8, B=2, lr=2e-3):
    from paper_2608_13578_gb300 import gpt
    model = gpt.build(cfg)
    opt = gpt.make_optimizer(model, lr=lr)
    g = torch.Generator().manual_seed(3)
    ids = torch.randint(0, cfg.vocab, (B, cfg.T + 1), generator=g).cuda()
    losses = [gpt.train_step(model, opt, ids[:, :-1], ids[:, 1:]).item() for _ in range(steps)]
    torch.cuda.synchronize()
    return model, losses


@pytest.mark.parametrize("mixer,honly,learn", [("bcmt", False, False), ("bcmt", True, False),
                                               ("bcmt", False, True), ("dense", False, False)],
                         ids=["bcmt", "honly", "learned_decay", "dense"])
def test_decoder_training_steps(cuda_ok, mixer, honly, learn):
    from paper_2608_13578_gb300 import gpt
    cfg = gpt.GPTConfig(vocab=512, D=128, H=2, layers=2, mlp=256, L=32, T=128, mixer=mixer,
                        honly=honly, learn_decay=learn)
    model, losses = _train(cfg)
    assert all(torch.isfinite(torch.tensor(losses))), losses
    assert losses[-1] < losses[0] - 0.5, losses
    if learn:
        d = model.blocks[0].mix.decay
        assert d.dtype == torch.float32
        assert not torch.equal(d.detach(), torch.full_like(d, 0.8))  # the decay was trained
        assert bool(((d >= 0) & (d < 1)).all())


def test_decoder_paper_head_width(cuda_ok):
    """The paper's model shape (D 128, 8 heads of 16) trains through the SIMT attention."""
    from paper_2608_13578_gb300 import gpt
    cfg = gpt.GPTConfig(vocab=512, D=128, H=8, layers=2, mlp=512, L=64, T=256)
    _, losses = _train(cfg)
    assert losses[-1] < losses[0] - 0.5, losses
