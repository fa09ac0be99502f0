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


def test_reference_arm_runs_the_requested_steps():
    """bench.py --impl reference times the oracle (host only) for exactly the
    requested warm-up and timed steps and prints the contract's JSON line."""
    import json
    import subprocess
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference",
                        "--workload", "fwd_fp32_b1_t256_l32_d128_h4", "--steps", "3",
                        "--warmup", "1"], capture_output=True, text=True, timeout=600, cwd=root)
    assert r.returncode == 0, r.stderr[-2000:]
    d = json.loads(r.stdout.strip().splitlines()[-1])
    assert d["impl"] == "reference" and d["steps"] == 3 and d["warmup"] == 1
    assert d["value"] > 0 and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
