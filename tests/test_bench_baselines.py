"""The eager-torch BCMT baseline that bench.py times computes the layer the
oracle computes (Sec. 3.3-3.8): float64 on the CPU, ragged last block."""
import os
import sys

import numpy as np
import pytest
import torch

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402
from oracle import bcmt_oracle as O  # noqa: E402


@pytest.mark.parametrize("B,T,D,H,L", [(2, 100, 32, 4, 16), (1, 64, 16, 2, 64), (1, 70, 24, 3, 32)])
def test_torch_baseline_matches_oracle(B, T, D, H, L):
    g = torch.Generator().manual_seed(T + D)
    x = torch.randn(B, T, D, generator=g, dtype=torch.float64)
    w = {n: torch.randn(*s, generator=g, dtype=torch.float64) / D ** 0.5
         for n, s in dict(w_qkv=(D, 3 * D), w_o=(D, D), w_p=(D,), w_m=(D, D), w_g=(D, D)).items()}
    decay = torch.rand(D, generator=g, dtype=torch.float64) * 0.9
    y = bench.torch_bcmt_layer(x, w["w_qkv"], w["w_o"], w["w_p"], w["w_m"], w["w_g"], decay, L, H)
    fw = O.forward(x.numpy(), w["w_qkv"].numpy(), w["w_o"].numpy(), w["w_p"].numpy(),
                   w["w_m"].numpy(), w["w_g"].numpy(), decay.numpy(), L, H)
    # the baseline does the pooling and memory in fp32, as bench.py runs it
    assert np.abs(y.detach().numpy() - fw["Y"]).max() < 1e-4
