"""Shared helpers of the GPU parity tests: running the CUDA layer through the C
ABI and comparing against the float64 oracle on the same seeded inputs."""

from __future__ import annotations

import numpy as np
import torch

from oracle import bcmt_oracle as O
from paper_2608_13578_gb300.inputs import Workload, as_float64, make_inputs

# Tolerances: fp32 max abs error <= 1e-4; bf16 max|gpu - oracle| / max|oracle| <= 2e-2,
# for the output and every gradient.
FP32_ABS = 1e-4
BF16_REL = 2e-2

GRAD_NAMES_X = ("dx", "dw_qkv", "dw_o", "dw_p", "dw_m", "dw_g", "d_decay")
GRAD_NAMES_QKV = ("dq", "dk", "dv", "dw_o", "dw_p", "dw_m", "dw_g", "d_decay")


def errors(gpu: torch.Tensor, ref: np.ndarray):
    g = gpu.detach().to("cpu", torch.float64).numpy()
    diff = np.max(np.abs(g - ref)) if ref.size else 0.0
    scale = np.max(np.abs(ref)) if ref.size else 0.0
    return float(diff), float(diff / scale) if scale > 0 else float(diff)


def assert_close(name: str, gpu: torch.Tensor, ref: np.ndarray, dtype: str):
    assert tuple(gpu.shape) == tuple(ref.shape), (name, tuple(gpu.shape), ref.shape)
    g = gpu.detach().to("cpu", torch.float64).numpy()
    assert np.all(np.isfinite(g)), f"{name}: non-finite values"
    ab, rel = errors(gpu, ref)
    if dtype == "fp32":
        assert ab <= FP32_ABS, f"{name}: max abs error {ab:.3e} > {FP32_ABS}"
    else:
        assert rel <= BF16_REL, f"{name}: relative error {rel:.3e} > {BF16_REL} (abs {ab:.3e})"
    return ab, rel


def to_device(t: dict, device="cuda"):
    return {k: v.to(device) for k, v in t.items()}


def oracle_run(w: Workload, t_cpu: dict, backward: bool = True, batch=None):
    """Oracle forward (and backward) on the rounded inputs; optionally on a
    subset of batch elements (the layer is independent across the batch)."""
    f = {k: as_float64(v) for k, v in t_cpu.items()}
    if batch is not None:
        for k in ("x", "q", "k", "v", "dy"):
            if k in f:
                f[k] = f[k][batch]
    fw = O.forward_from_inputs(f, w.L, w.H, honly=w.honly, input_is_x=w.input_is_x)
    gr = O.backward(fw, f["dy"]) if backward else None
    return fw, gr


def gpu_run(w: Workload, t_dev: dict, backward: bool = True, decay_grad: bool = False):
    """Forward (and backward) through the C ABI.  Without decay_grad the
    backward runs as in training with the paper's fixed decay (the benchmark's
    launch sequence); with it the decay gradient d_decay is returned too."""
    from paper_2608_13578_gb300 import layer
    p = layer.params_for(w.B, w.T, w.D, w.H, w.L, w.dtype, w.input_is_x, w.honly,
                         flags=layer.C.BCMT_FLAG_CHECK)
    y, ws = layer.forward(p, t_dev)
    g = layer.backward(p, t_dev, ws, t_dev["dy"], decay_grad=decay_grad) if backward else None
    torch.cuda.synchronize()
    return y, g
