"""The layer's forward and backward captured into a CUDA graph.

bcmt_forward / bcmt_backward fork library-owned streams (critical path and
side work) from the caller's stream with events and join them back; a CUDA
graph capture of the caller's stream must capture all of it.  Replaying the
graph must give bitwise the same outputs and gradients as the calls made
directly (the kernels are deterministic), twice in a row, with the inputs
changed in place between replays.
"""

import pytest
import torch

from paper_2608_13578_gb300.inputs import Workload, make_inputs

pytestmark = pytest.mark.gpu


def _run(C, p, t, ws, sc, y, g, stream=None):
    C.bcmt_forward(p, t["x"], None, None, None, t["w_qkv"], t["w_o"], t["w_p"], t["w_m"],
                   t["w_g"], t["decay"], y, ws, stream)
    C.bcmt_backward(p, t["dy"], t["x"], None, None, t["w_qkv"], t["w_o"], t["w_p"], t["w_m"],
                    t["w_g"], t["decay"], ws, sc, g["dx"], None, None, g["dw_qkv"], g["dw_o"],
                    g["dw_p"], g["dw_m"], g["dw_g"], stream, g.get("d_decay"))


@pytest.mark.parametrize("decay_grad", [False, True], ids=["fixed_decay", "decay_grad"])
@pytest.mark.parametrize("L", [64, 256])
def test_graph_replay_matches_direct_calls(cuda_ok, L, decay_grad):
    from paper_2608_13578_gb300 import bcmt as C
    from paper_2608_13578_gb300 import layer
    w = Workload("graph", 2, 512, 256, 4, L, "bf16", True, (0.5, 0.99), 41)
    t = {k: v.cuda() for k, v in make_inputs(w).items()}
    p = layer.params_for(w.B, w.T, w.D, w.H, w.L, w.dtype)
    ws = torch.empty(C.bcmt_workspace_size(p), dtype=torch.uint8, device="cuda")
    sc = torch.empty(C.bcmt_scratch_size(p), dtype=torch.uint8, device="cuda")
    y = torch.empty_like(t["x"])
    g = {"dx": torch.empty_like(t["x"]), "dw_qkv": torch.empty_like(t["w_qkv"])}
    if decay_grad:
        g["d_decay"] = torch.empty_like(t["decay"])
    for n in ("w_o", "w_p", "w_m", "w_g"):
        g["d" + n] = torch.empty_like(t[n])
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        _run(C, p, t, ws, sc, y, g)      # warm-up outside the capture
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=s):
            _run(C, p, t, ws, sc, y, g)
    torch.cuda.synchronize()
    gen = torch.Generator().manual_seed(42)
    for rep in range(2):
        # new inputs in place, then the graph and the direct calls on them
        t["x"].copy_(torch.randn(t["x"].shape, generator=gen).to(t["x"].dtype))
        t["dy"].copy_(torch.randn(t["dy"].shape, generator=gen).to(t["dy"].dtype))
        graph.replay()
        torch.cuda.synchronize()
        got = {"y": y.clone(), **{k: v.clone() for k, v in g.items()}}
        _run(C, p, t, ws, sc, y, g)
        torch.cuda.synchronize()
        C.bcmt_device_status()
        ref = {"y": y, **g}
        for k in ref:
            assert torch.equal(got[k], ref[k]), (rep, k)
