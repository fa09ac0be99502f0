"""Incremental decoding through the C ABI (bcmt_decode_step) against the
float64 oracle: decoding tokens 0..T-1 one at a time must give the rows of the
oracle's forward output Y (the layer is causal, Sec. 3.6), within the same
tolerances as the forward; ragged last blocks, HOnly, the paper's 16-wide
heads and a long block are covered."""

import pytest
import torch

from paper_2608_13578_gb300.inputs import Workload, make_inputs
from tests.helpers import assert_close, oracle_run

pytestmark = pytest.mark.gpu

CASES = [
    # B, T, D, H, L, dtype, honly
    (2, 100, 128, 4, 16, "fp32", False),
    (3, 200, 128, 2, 32, "bf16", False),
    (2, 150, 256, 4, 64, "bf16", False),
    (2, 90, 128, 8, 64, "bf16", False),      # dh = 16
    (1, 300, 128, 2, 256, "bf16", False),
    (2, 100, 128, 2, 32, "bf16", True),
    (17, 40, 128, 2, 8, "fp32", False),      # more sequences than one product tile
]


def _decode(w, t, H, L, honly):
    from paper_2608_13578_gb300 import layer
    dev = {k: v.cuda() for k, v in t.items()}
    dec = layer.Decoder(dev, w.B, H, L, honly=honly)
    ys = [dec.step(dev["x"][:, i]) for i in range(w.T)]
    torch.cuda.synchronize()
    return torch.stack(ys, dim=1), dec


@pytest.mark.parametrize("B,T,D,H,L,dtype,honly", CASES)
def test_decode_matches_oracle_forward(cuda_ok, B, T, D, H, L, dtype, honly):
    w = Workload("decode", B, T, D, H, L, dtype, False, (0.5, 0.99), 21, True, honly)
    t = make_inputs(w)
    y, _ = _decode(w, t, H, L, honly)
    fw, _ = oracle_run(w, t, backward=False)
    assert_close("Y", y, fw["Y"], dtype)


def test_decode_reset_restarts_bitwise(cuda_ok):
    w = Workload("decode", 2, 70, 128, 2, 16, "bf16", False, (0.5, 0.99), 22)
    t = make_inputs(w)
    y0, dec = _decode(w, t, 2, 16, False)
    dec.reset()
    x = t["x"].cuda()
    y1 = torch.stack([dec.step(x[:, i]) for i in range(w.T)], dim=1)
    torch.cuda.synchronize()
    assert torch.equal(y0, y1)


def test_decode_rejects_qkv_entry_and_negative_pos(cuda_ok):
    from paper_2608_13578_gb300 import bcmt as C
    p = C.make_params(1, 1, 128, 2, 16, "bf16", input_is_x=False)
    with pytest.raises(C.BCMTError):
        C.bcmt_decode_step(p, 1 << 20, 0, *([1 << 20] * 9))
    p = C.make_params(1, 1, 128, 2, 16, "bf16")
    with pytest.raises(C.BCMTError):
        C.bcmt_decode_step(p, 1 << 20, -1, *([1 << 20] * 9))
