"""Throughput benchmark of the BCMT token mixer (forward + backward) on GB300.

One step = bcmt_forward + bcmt_backward of one BCMT layer over one batch of
synthetic inputs already resident in HBM (workload: B=8, T=1024, L=64,
D=512, 8 heads of 64, bf16 storage with fp32 accumulation).  Prints one JSON
line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (launched by torchrun, one rank per GPU) every rank runs its own
batch (weak scaling, no data-path collective); the time is the maximum over
ranks.  ``--impl reference`` times the float64 CPU oracle on a bounded sample
of the same workload on the host cores.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "BCMT layer fwd+bwd tokens/s on 1 GB300 and % of tensor/HBM roofline vs oracle"
UNIT = "tokens/s"
L2_FLUSH_BYTES = 256 << 20  # > 129 MB L2


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=None)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-dense", action="store_true")
    return ap.parse_args()


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def rank_seed(base_seed: int, rank: int) -> int:
    """Every rank draws its own batch (weak scaling over independent batches)."""
    return base_seed + rank


def max_over_ranks(ms: float, world: int, device=None) -> float:
    """The slowest rank's time: the job's time."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(world: int, tokens_per_rank_step: int, steps: int, max_ms: float) -> float:
    """Whole-job throughput: the tokens all ranks processed over the slowest rank's time."""
    return world * tokens_per_rank_step * steps / (max_ms / 1e3)


# ----------------------------------------------------------------- CPU oracle
ORACLE_SNIPPET = r"""
import json, os, sys, time
sys.path.insert(0, {root!r})
from oracle import bcmt_oracle as O
from paper_2608_13578_gb300.inputs import WORKLOADS, as_float64, make_inputs
w = WORKLOADS[{name!r}].replace(B=1)
t = {{k: as_float64(v) for k, v in make_inputs(w).items()}}
budget, reps, t0 = {budget}, 0, time.perf_counter()
times = []
while True:
    s = time.perf_counter()
    fw = O.forward_from_inputs(t, w.L, w.H)
    O.backward(fw, t["dy"])
    times.append(time.perf_counter() - s)
    reps += 1
    # a budget of 0 runs exactly max_reps repetitions
    if reps >= {max_reps} or (budget > 0 and time.perf_counter() - t0 > budget):
        break
print(json.dumps({{"tokens": w.T, "reps": reps, "seconds": sum(times), "times": times}}))
"""


def run_oracle_sample(name: str, budget_s: float, max_reps: int):
    """Times the oracle's fwd+bwd on one batch element of the workload in a fresh
    process (no CUDA context) with every BLAS thread count pinned to the host's
    core count."""
    cores = os.cpu_count() or 1
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[v] = str(cores)
    code = ORACLE_SNIPPET.format(root=ROOT, name=name, budget=budget_s, max_reps=max_reps)
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                       timeout=600)
    if r.returncode != 0:
        raise RuntimeError("oracle timing failed: " + r.stderr[-2000:])
    d = json.loads(r.stdout.strip().splitlines()[-1])
    d["cores"] = cores
    return d


# ------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, FileNotFoundError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------ roofline model
def kernel_model(w):
    """Algorithmic work per launch of each named kernel: (bound, amount) with
    amount in flops for tensor-core GEMMs and bytes for HBM-bound kernels."""
    n, D, H, Nb, B = w.B * w.T, w.D, w.H, w.n_blocks, w.B
    es = 2 if w.dtype == "bf16" else 4
    npart = D // 32 if w.dtype == "bf16" else D // 4  # score partials per token
    g = lambda m, nn, k: ("tensor", 2.0 * m * nn * k)
    return {
        "gemm_qkv": g(n, 3 * D, D),
        "gemm_wo": g(n, D, D),
        "gemm_gate": g(n, D, D),
        # H and the gate pre-activation in one product: Concat [W_O | W_O W_g]
        "gemm_wo_gate": g(n, 2 * D, D),
        "gemm_wog": g(D, D, D),
        # the Q/K/V projection with the weight product W_O W_g in the same launch
        "gemm_qkv_wog": ("tensor", 2.0 * n * 3 * D * D + 2.0 * D * D * D),
        # Sec. 3.8 injection: read H, G and C; write Y
        "inject": ("hbm", 3 * n * D * es + B * Nb * D * 4),
        "gemm_dh": g(n, D, D),
        # dM^T = W_m dP^T with the reverse scan of Sec. 3.5 in its epilogue
        "gemm_dm_scan": g(D, B * Nb, D),
        "gemm_dhhat": g(n, D, D),
        "gemm_dx": g(n, D, 3 * D),
        "gemm_dw_g": g(D, D, n),
        "gemm_dw_o": g(D, D, n),
        "gemm_dw_qkv": g(D, 3 * D, n),
        # one grouped CTA-pair launch when D is a multiple of 256: dX, dW_QKV, dW_g, dW_O
        "gemm_dx_dw": ("tensor", 2 * 2.0 * n * D * 3 * D + 2 * 2.0 * n * D * D),
        # read Q, K, V; write Concat(heads) and the log-sum-exp
        "attn_fwd_tc": ("hbm", 3 * n * D * es + n * D * es + n * H * 4),
        "attn_fwd_simt": ("hbm", 3 * n * D * es + n * D * es + n * H * 4),
        "attn_fwd_fl": ("hbm", 3 * n * D * es + n * D * es + n * H * 4),
        # read Q, K, V, dO, O and the log-sum-exp; write dQ, dK, dV
        "attn_bwd_tc": ("hbm", 5 * n * D * es + n * H * 4 + 3 * n * D * es),
        "attn_bwd_simt": ("hbm", 5 * n * D * es + n * H * 4 + 3 * n * D * es),
        # two kernels (dQ, then dK/dV); the row dot products Drow are written and re-read
        "attn_bwd_fl": ("hbm", 5 * n * D * es + n * H * 4 + 3 * n * D * es + 2 * n * H * 4),
        # Sec. 3.4 summaries: read H and the score partials, write alpha and S
        "summary_fwd": ("hbm", n * D * es + n * 4 * npart + n * 4 + B * Nb * D * 4),
        # Sec. 3.5 scan with the projection P = M W_m (warp-level mma): read S and
        # W_m, write P, M (fp32 and bf16), Z and 1/Z
        "memory_proj_fwd": ("hbm", B * Nb * D * 4 + D * D * es + B * Nb * D * (4 + 4 + 2)
                            + 2 * Nb * D * 4),
        # Sec. 3.5 scan: read S, write M (fp32 and the bf16 operand copy) and Z
        "memory_scan_fwd": ("hbm", B * Nb * D * (4 + 4 + 2) + Nb * D * 4),
        "gemm_wm": g(B * Nb, D, D),
        # Sec. 3.8 reversed: read dY, G and C; write dU and dP (fp32 + bf16)
        "gate_bwd": ("hbm", 3 * n * D * es + B * Nb * D * (4 + 4 + 2)),
        "gemm_dm": g(B * Nb, D, D),
        # reverse scan: read dM and Z, write dS
        "memory_scan_bwd": ("hbm", 2 * B * Nb * D * 4 + Nb * D * 4),
        # pooling backward: read H, dY, alpha and dS; write ds and the dW_p
        # partials; complete dH in place (read and write)
        "summary_bwd": ("hbm", 4 * n * D * es + 2 * n * 4 + 2 * B * Nb * D * 4),
        "gemm_dwm": g(D, D, B * Nb),
        "reduce_rows": ("hbm", B * Nb * D * 4 + D * es),
    }


# The sources each timed kernel is built from (its translation unit and the
# headers every kernel shares): an ncu figure stays valid while they do.
SHARED_SOURCES = ("common.cuh", "tc.cuh", "tmap.h", "internal.h")
KERNEL_SOURCES = {
    "attn_fwd_tc": ("attn_tc.cu", "attn_common.cuh"),
    "attn_bwd_tc": ("attn_tc.cu", "attn_common.cuh"),
    "attn_fwd_fl": ("attn_flash.cu", "attn_common.cuh"),
    "attn_bwd_fl": ("attn_flash.cu", "attn_common.cuh"),
    "attn_fwd_simt": ("attn_simt.cu",),
    "attn_bwd_simt": ("attn_simt.cu",),
}


def kernel_sources(kernel: str):
    if kernel in KERNEL_SOURCES:
        own = KERNEL_SOURCES[kernel]
    elif kernel.startswith("gemm"):
        own = ("gemm.cu", "epilogues.cuh")
    else:
        own = ("memory.cu",)
    return own + SHARED_SOURCES


def csrc_digest(kernel: str):
    """Hash of the sources `kernel` is compiled from."""
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2608_13578_gb300", "csrc")
    for f in sorted(kernel_sources(kernel)):
        path = os.path.join(d, f)
        if os.path.exists(path):
            with open(path, "rb") as fh:
                h.update(f.encode() + fh.read())
    return h.hexdigest()[:16]


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"], "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "source": "fallback"}


def ncu_traffic(kernel: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if it
    was taken on the current kernel sources."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        e = d.get(kernel)
        if e and e.get("sources_digest") == csrc_digest(kernel):
            return e.get("dram_bytes_per_launch")
    except (OSError, ValueError):
        pass
    return None


# ------------------------------------------------------------- our arm (GPU)
def bench_ours(args):
    import torch
    import torch.distributed as dist

    rank, local_rank, world = dist_env()
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)

    if local_rank == 0:
        from paper_2608_13578_gb300 import build
        build.build()
    if world > 1:
        dist.barrier()
    from paper_2608_13578_gb300 import bcmt as C
    from paper_2608_13578_gb300 import layer
    from paper_2608_13578_gb300.inputs import HEADLINE, WORKLOADS, make_inputs

    name = args.workload or HEADLINE
    w = WORKLOADS[name]
    t_cpu = make_inputs(w, seed=rank_seed(w.seed, rank))
    t = {k: v.to(dev) for k, v in t_cpu.items()}
    p = layer.params_for(w.B, w.T, w.D, w.H, w.L, w.dtype)
    pprof = layer.params_for(w.B, w.T, w.D, w.H, w.L, w.dtype, flags=C.BCMT_FLAG_PROFILE)
    ws = torch.empty(C.bcmt_workspace_size(p), dtype=torch.uint8, device=dev)
    sc = torch.empty(C.bcmt_scratch_size(p), dtype=torch.uint8, device=dev)
    y = torch.empty_like(t["x"])
    grads = {"dx": torch.empty_like(t["x"]), "dw_qkv": torch.empty_like(t["w_qkv"])}
    for n in ("w_o", "w_p", "w_m", "w_g"):
        grads["d" + n] = torch.empty_like(t[n])
    stream = torch.cuda.current_stream()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def step(pp):
        # launches on the current stream (the capture stream while a graph is recorded)
        C.bcmt_forward(pp, t["x"], None, None, None, t["w_qkv"], t["w_o"], t["w_p"], t["w_m"],
                       t["w_g"], t["decay"], y, ws, None)
        C.bcmt_backward(pp, t["dy"], t["x"], None, None, t["w_qkv"], t["w_o"], t["w_p"], t["w_m"],
                        t["w_g"], t["decay"], ws, sc, grads["dx"], None, None, grads["dw_qkv"],
                        grads["dw_o"], grads["dw_p"], grads["dw_m"], grads["dw_g"], None)

    for _ in range(max(3, args.warmup)):
        step(p)
    C.bcmt_device_status(stream)
    torch.cuda.synchronize()
    # One step recorded as a CUDA graph: the same launches, replayed without
    # per-launch host work.
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step(p)
    graph.replay()
    torch.cuda.synchronize()
    C.bcmt_device_status(stream)

    def timed(run):
        """K steps, each bracketed by CUDA events on the launching stream, with
        L2 evicted before each step; returns the summed device time in ms."""
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps)]
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        for i in range(args.steps):
            flush.fill_(i & 0xFF)            # evict L2 between timed steps
            ev[i][0].record(stream)
            run()
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        return sum(a.elapsed_time(b) for a, b in ev)

    # the measured region: graph replays of the step, no per-kernel events
    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    total_ms = timed(graph.replay)
    eager_ms = timed(lambda: step(p))
    clk = clocks.stop()
    C.bcmt_device_status(stream)
    # the same K steps again with CUDA events around every kernel, for the
    # per-kernel breakdown and the roofline of the dominant kernel
    C.bcmt_profile_reset()
    prof_ms = timed(lambda: step(pprof))
    C.bcmt_device_status(stream)
    prof = C.bcmt_profile_read()
    launches = sum(c for c, _ in prof.values())

    total_ms = max_over_ranks(total_ms, world, dev)
    eager_ms = max_over_ranks(eager_ms, world, dev)
    tokens_per_step = w.B * w.T
    value = job_tokens_per_s(world, tokens_per_step, args.steps, total_ms)

    # ---- end to end through the public API: every step copies its inputs in
    # from pinned host memory and its output and every gradient back out.  The
    # copies run on their own streams and overlap the previous/next step's
    # compute (double-buffered device inputs and outputs), as a training loop
    # that streams its batches would; the compute of a step is the two C-ABI
    # calls recorded once per buffer pair as a CUDA graph, as such a loop
    # would record its step.
    # the step's inputs (x, dY) and its outputs (Y and every gradient) each
    # live in one contiguous buffer, host and device side, so that a step moves
    # one copy in and one copy out; the C ABI gets views into them
    def packed(specs, pin, device=None):
        """One flat buffer holding tensors of the given (name, shape, dtype),
        each at a 256-byte aligned offset; returns (flat, {name: view})."""
        offs, total = [], 0
        for _, shape, dtype in specs:
            nbytes = int(torch.Size(shape).numel()) * torch.empty((), dtype=dtype).element_size()
            offs.append(total)
            total += (nbytes + 255) // 256 * 256
        flat = torch.empty(total, dtype=torch.uint8, device=device)
        if pin:
            flat = flat.pin_memory()
        views = {}
        for (name, shape, dtype), off in zip(specs, offs):
            nbytes = int(torch.Size(shape).numel()) * torch.empty((), dtype=dtype).element_size()
            views[name] = flat[off:off + nbytes].view(dtype).view(shape)
        return flat, views

    in_specs = [("x", t_cpu["x"].shape, t_cpu["x"].dtype), ("dy", t_cpu["dy"].shape, t_cpu["dy"].dtype)]
    out_specs = [("y", t_cpu["x"].shape, t_cpu["x"].dtype)] + \
        [(n, g_.shape, g_.dtype) for n, g_ in grads.items()]
    in_h, in_hv = packed(in_specs, pin=True)
    in_hv["x"].copy_(t_cpu["x"])
    in_hv["dy"].copy_(t_cpu["dy"])
    out_h, _ = packed(out_specs, pin=True)
    in_d, out_d = [], []
    for _ in range(2):
        in_d.append(packed(in_specs, pin=False, device=dev))
        out_d.append(packed(out_specs, pin=False, device=dev))
    x_d = [v["x"] for _, v in in_d]
    dy_d = [v["dy"] for _, v in in_d]
    y_d = [v["y"] for _, v in out_d]
    g_d = [{n: v[n] for n in grads} for _, v in out_d]
    h2d = sum(int(torch.Size(sh).numel()) * torch.empty((), dtype=dt).element_size()
              for _, sh, dt in in_specs)
    d2h = sum(int(torch.Size(sh).numel()) * torch.empty((), dtype=dt).element_size()
              for _, sh, dt in out_specs)
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_done = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]

    def e2e_compute(b):
        gb = g_d[b]
        C.bcmt_forward(p, x_d[b], None, None, None, t["w_qkv"], t["w_o"], t["w_p"], t["w_m"],
                       t["w_g"], t["decay"], y_d[b], ws, None)
        C.bcmt_backward(p, dy_d[b], x_d[b], None, None, t["w_qkv"], t["w_o"], t["w_p"],
                        t["w_m"], t["w_g"], t["decay"], ws, sc, gb["dx"], None, None,
                        gb["dw_qkv"], gb["dw_o"], gb["dw_p"], gb["dw_m"], gb["dw_g"], None)

    e2e_graphs = []
    for b in range(2):
        e2e_compute(b)
        torch.cuda.synchronize()
        gr_b = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr_b):
            e2e_compute(b)
        e2e_graphs.append(gr_b)
    torch.cuda.synchronize()

    def e2e_steps(k_steps):
        for i in range(k_steps):
            b = i % 2
            with torch.cuda.stream(s_in):
                if i >= 2:
                    s_in.wait_event(ev_done[b])  # step i-2 has read buffer b
                in_d[b][0].copy_(in_h, non_blocking=True)
                ev_in[b].record(s_in)
            stream.wait_event(ev_in[b])
            if i >= 2:
                stream.wait_event(ev_out[b])  # step i-2's outputs are on the host
            gb = g_d[b]
            e2e_graphs[b].replay()  # on `stream`, the current stream
            ev_done[b].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_done[b])
                out_h.copy_(out_d[b][0], non_blocking=True)
                ev_out[b].record(s_out)

    e2e_steps(3)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_in.wait_event(e0)
    e2e_steps(args.steps)
    e1.record(s_out)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    e2e_ms = max_over_ranks(e2e_ms, world, dev)
    e2e_value = job_tokens_per_s(world, tokens_per_step, args.steps, e2e_ms)

    # ---- roofline of the dominant kernel: the largest total time among the
    # kernels with an algorithmic model (the K-split reductions have none: their
    # bytes depend on the split counts the library picks per shape)
    model = kernel_model(w)
    peaks = load_peaks()
    modelled = [kv for kv in prof.items() if kv[0] in model] or list(prof.items())
    dom = max(modelled, key=lambda kv: kv[1][1])
    dname, (dcount, dms) = dom
    bound, amount = model.get(dname, ("hbm", None))
    roof = None
    if amount is not None:
        per_launch_s = dms / dcount / 1e3
        if bound == "tensor":
            ach = amount / per_launch_s / 1e12
            peak = peaks["bf16_tflops"]
            unit = "TFLOP/s"
        else:
            ach = amount / per_launch_s / 1e9
            peak = peaks["hbm_gbs"]
            unit = "GB/s"
        roof = {"kernel": dname, "bound": bound, "achieved": round(ach, 2), "peak": peak,
                "unit": unit, "frac": round(ach / peak, 4), "traffic": ncu_traffic(dname),
                "algorithmic_per_launch": amount, "avg_launch_us": round(per_launch_s * 1e6, 3),
                "peak_source": peaks["source"] + " (burst)"}
    kernels = {k: {"launches": c, "avg_us": round(ms / c * 1e3, 3),
                   "share": round(ms / sum(v[1] for v in prof.values()), 4)}
               for k, (c, ms) in sorted(prof.items(), key=lambda kv: -kv[1][1])}

    # ---- dense causal attention of the same shape (library SDPA), and the same
    # BCMT layer written with eager torch ops: context only
    dense = eager_bcmt = None
    if not args.no_dense and rank == 0:
        dense = bench_dense(w, t, stream, flush, args)
        eager_bcmt = bench_torch_bcmt(w, t, stream, flush, args)

    out = None
    if rank == 0:
        cpu = None
        if not args.no_cpu_baseline:
            d = run_oracle_sample(name, budget_s=15.0, max_reps=50)
            cpu = {"value": round(d["tokens"] * d["reps"] / d["seconds"], 2), "unit": UNIT,
                   "cores": d["cores"], "kind": "oracle",
                   "sample": f"float64 oracle fwd+bwd on batch element 0 of the workload "
                             f"({d['tokens']} tokens), {d['reps']} repetitions, "
                             f"{d['seconds']:.1f} s"}
        out = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup),
            "ms_per_step": round(total_ms / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
            "data": "synthetic (seeded N(0,1) tokens, N(0,1/D) weights, decay 0.8)",
            "config": {"workload": name, "B": w.B, "T": w.T, "L": w.L, "D": w.D, "H": w.H,
                       "per_rank_batch": w.B, "parallelism": f"batch-sharded x{world}",
                       "launch": "CUDA graph of bcmt_forward + bcmt_backward",
                       "l2": "flushed between timed steps (256 MiB write)"},
            "clocks": clk,
            "e2e": {"value": round(e2e_value, 1), "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "gpu_launches": launches,  # kernels of ours per K steps
            "roofline": roof,
            "cpu_baseline": cpu,
            "kernels": kernels,
            "eager": {"ms_per_step": round(eager_ms / args.steps, 4),
                      "value": round(job_tokens_per_s(world, tokens_per_step, args.steps, eager_ms), 1),
                      "note": "same steps launched call by call instead of as a graph"},
            "profiled_pass": {"ms_per_step_with_kernel_events": round(prof_ms / args.steps, 4),
                              "note": "per-kernel times come from this second pass of the "
                                      "same steps; value comes from the pass without them"},
            "dense_causal_baseline": dense,
            "torch_eager_bcmt_baseline": eager_bcmt,
        }
        print(json.dumps(out))
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return out


def bench_dense(w, t, stream, flush, args):
    """Same projections with torch's dense causal SDPA (flash backend) instead of
    the blockwise mixer: fwd+bwd tokens/s.  A library baseline for context."""
    import torch
    import torch.nn.functional as F
    B, T, D, H = w.B, w.T, w.D, w.H
    params = [t[n].detach().clone().requires_grad_(True) for n in ("w_qkv", "w_o")]
    x = t["x"].detach().clone().requires_grad_(True)
    dy = t["dy"]

    def step():
        qkv = x @ params[0]
        q, k, v = qkv.view(B, T, 3, H, D // H).permute(2, 0, 3, 1, 4)
        o = F.scaled_dot_product_attention(q, k, v, is_causal=True)
        y = o.transpose(1, 2).reshape(B, T, D) @ params[1]
        y.backward(dy)

    for _ in range(3):
        step()
    torch.cuda.synchronize()
    tot = 0.0
    for i in range(args.steps):
        flush.fill_(i & 0xFF)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        step()
        b.record(stream)
        torch.cuda.synchronize()
        tot += a.elapsed_time(b)
    return {"value": round(B * T * args.steps / (tot / 1e3), 1), "unit": UNIT,
            "what": "x W_qkv -> torch SDPA(is_causal) over the full sequence -> W_O, fwd+bwd, bf16"}


def torch_bcmt_layer(x, w_qkv, w_o, w_p, w_m, w_g, decay, L, H):
    """The BCMT layer (Sec. 3.3-3.8) written with eager torch ops, as a
    framework-level implementation would: blocks folded into the batch for
    torch's SDPA (is_causal), the pooling softmax per block, the decayed memory
    as a masked weight matrix over blocks, the shifted projection, the gate.
    A baseline for context, differentiable by autograd."""
    import torch
    import torch.nn.functional as F
    B, T, D = x.shape
    dh = D // H
    Nb = (T + L - 1) // L
    Tp = Nb * L
    qkv = x @ w_qkv
    if Tp != T:
        qkv = F.pad(qkv, (0, 0, 0, Tp - T))
    q, k, v = qkv.view(B, Nb, L, 3, H, dh).permute(3, 0, 1, 4, 2, 5).reshape(3, B * Nb, H, L, dh)
    o = F.scaled_dot_product_attention(q, k, v, is_causal=True)
    hhat = o.view(B, Nb, H, L, dh).permute(0, 1, 3, 2, 4).reshape(B, Tp, D)[:, :T]
    hm = hhat @ w_o
    s = (hm @ w_p.unsqueeze(1)).squeeze(-1).float()
    hp = hm.float()
    if Tp != T:
        s = F.pad(s, (0, Tp - T), value=float("-inf"))
        hp = F.pad(hp, (0, 0, 0, Tp - T))
    alpha = torch.softmax(s.view(B, Nb, L), dim=-1)
    S = torch.einsum("bnl,bnld->bnd", alpha, hp.view(B, Nb, L, D))
    idx = torch.arange(Nb, device=x.device)
    e = (idx[:, None] - idx[None, :]).clamp(min=0).to(torch.float32)
    lower = (idx[:, None] >= idx[None, :]).to(torch.float32)
    wts = decay.float()[None, None, :] ** e[:, :, None] * lower[:, :, None]
    M = torch.einsum("ijd,bjd->bid", wts, S) / wts.sum(1)
    P = M.to(x.dtype) @ w_m
    C = torch.cat([torch.zeros_like(P[:, :1]), P[:, :-1]], dim=1)
    G = torch.sigmoid(hm @ w_g)
    return hm + G * C.repeat_interleave(L, dim=1)[:, :T]


def bench_torch_bcmt(w, t, stream, flush, args):
    """The same layer in eager torch (torch_bcmt_layer), fwd+bwd tokens/s."""
    import torch
    names = ("w_qkv", "w_o", "w_p", "w_m", "w_g")
    params = {n: t[n].detach().clone().requires_grad_(True) for n in names}
    x = t["x"].detach().clone().requires_grad_(True)
    dy, decay = t["dy"], t["decay"]

    def step():
        y = torch_bcmt_layer(x, params["w_qkv"], params["w_o"], params["w_p"], params["w_m"],
                             params["w_g"], decay, w.L, w.H)
        y.backward(dy)

    for _ in range(3):
        step()
    torch.cuda.synchronize()
    tot = 0.0
    for i in range(args.steps):
        flush.fill_(i & 0xFF)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        step()
        b.record(stream)
        torch.cuda.synchronize()
        tot += a.elapsed_time(b)
    return {"value": round(w.B * w.T * args.steps / (tot / 1e3), 1), "unit": UNIT,
            "what": "the BCMT layer in eager torch ops (blocks folded into the batch for SDPA, "
                    "pooling, masked decay weights, shifted W_m, gate), fwd+bwd, autograd"}


# ------------------------------------------------ whole-model training steps
# Config 5 of the benchmark set (a 6-layer GPT-style decoder with the BCMT
# mixer), and the paper's own throughput shape (Tables 1-2: D 128, 8 heads,
# 6 layers, batch 16) for BCMT, its HOnly ablation and dense attention.
MODEL_WORKLOADS = {
    "gpt6_v32000_d512_h8_mlp2048_l64_t1024_b16": dict(
        B=16, vocab=32000, D=512, H=8, layers=6, mlp=2048,
        runs=[("bcmt", 64, 1024), ("bcmt_learned_decay", 64, 1024)]),
    "paper_d128_h8_6l_b16_sweep": dict(
        B=16, vocab=50257, D=128, H=8, layers=6, mlp=512,
        runs=[(m, L, T) for T in (128, 256, 512, 1024) for L in (64, 128, 256, 512) if L <= T
              for m in ("bcmt", "honly")] + [("dense", 0, T) for T in (128, 256, 512, 1024)]),
}


def bench_models(args):
    """Training-step tokens/s of whole models (embedding, 6 blocks, LM head,
    cross-entropy, AdamW) with the BCMT mixer from this library and the rest
    from PyTorch; the dense-attention model of the same shape beside it."""
    import torch
    from paper_2608_13578_gb300 import build
    build.build()
    from paper_2608_13578_gb300 import bcmt as C
    from paper_2608_13578_gb300 import gpt, layer

    rank, local_rank, world = dist_env()
    if world > 1:
        if rank != 0:
            return None  # model steps are measured on one GPU
    torch.cuda.set_device(local_rank)
    name = args.workload
    spec = MODEL_WORKLOADS[name]
    B = spec["B"]
    stream = torch.cuda.current_stream()

    def run(mixer, L, T, steps, warmup):
        c = gpt.GPTConfig(vocab=spec["vocab"], D=spec["D"], H=spec["H"], layers=spec["layers"],
                          mixer="dense" if mixer == "dense" else "bcmt", mlp=spec["mlp"],
                          L=max(L, 1), T=T, honly=mixer == "honly",
                          learn_decay=mixer == "bcmt_learned_decay")
        model = gpt.build(c)
        opt = gpt.make_optimizer(model)
        g = torch.Generator().manual_seed(rank_seed(0, rank))
        ids_h = torch.randint(0, c.vocab, (B, T + 1), generator=g).pin_memory()
        ids = ids_h.cuda()
        inp, tgt = ids[:, :-1].contiguous(), ids[:, 1:].contiguous()
        for _ in range(max(3, warmup)):
            gpt.train_step(model, opt, inp, tgt)
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        for i in range(steps):
            ev[i][0].record(stream)
            gpt.train_step(model, opt, inp, tgt)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        ms = sum(a.elapsed_time(b) for a, b in ev)
        # end to end: the step's token ids copied in from pinned host memory and
        # its loss read back, every step
        d_ids = torch.empty_like(ids)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        losses = []
        for _ in range(steps):
            d_ids.copy_(ids_h, non_blocking=True)
            loss = gpt.train_step(model, opt, d_ids[:, :-1], d_ids[:, 1:])
            losses.append(loss.item())
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = e0.elapsed_time(e1)
        tok = B * T * steps
        r = {"mixer": mixer, "L": L if mixer != "dense" else None, "T": T,
             "flops_per_token": gpt.flops_per_token(c),
             "tokens_per_s": round(tok / (ms / 1e3), 1), "ms_per_step": round(ms / steps, 3),
             "e2e_tokens_per_s": round(tok / (e2e_ms / 1e3), 1),
             "tflops": round(gpt.flops_per_token(c) * tok / (ms / 1e3) / 1e12, 1),
             "loss_first_last": [round(losses[0], 4), round(losses[-1], 4)],
             "h2d_bytes_per_step": ids_h.numel() * ids_h.element_size(), "d2h_bytes_per_step": 4}
        del model, opt
        torch.cuda.empty_cache()
        return r

    def mixer_launches(L, T, honly):
        """Our kernels per mixer forward+backward at this shape (profiled call)."""
        D, H = spec["D"], spec["H"]
        p = layer.params_for(B, T, D, H, L, "bf16", True, honly, flags=C.BCMT_FLAG_PROFILE)
        t = {"x": torch.randn(B, T, D, device="cuda").bfloat16(),
             "w_qkv": torch.randn(D, 3 * D, device="cuda").bfloat16(),
             "decay": torch.full((D,), 0.8, device="cuda")}
        for n in ("w_o", "w_m", "w_g"):
            t[n] = torch.randn(D, D, device="cuda").bfloat16()
        t["w_p"] = torch.randn(D, device="cuda").bfloat16()
        C.bcmt_profile_reset()
        y, ws = layer.forward(p, t)
        layer.backward(p, t, ws, torch.randn_like(y))
        n = sum(c for c, _ in C.bcmt_profile_read().values())
        C.bcmt_profile_reset()
        return n

    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    rows = [run(m, L, T, args.steps, args.warmup) for m, L, T in spec["runs"]]
    clk = clocks.stop()
    head = rows[0]
    dense = None
    if name.startswith("gpt"):
        dense = run("dense", 0, spec["runs"][0][2], args.steps, args.warmup)
    launches = sum(mixer_launches(L, T, m == "honly") * spec["layers"] * args.steps
                   for m, L, T in spec["runs"][:1] if m != "dense")
    out = {"metric": "training-step tokens/s of a 6-layer decoder with the BCMT mixer",
           "value": head["tokens_per_s"], "unit": UNIT, "n_gpus": 1, "steps": args.steps,
           "warmup": max(3, args.warmup), "ms_per_step": head["ms_per_step"],
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
           "data": "synthetic token ids uniform over the vocabulary, random init",
           "config": {"workload": name, "B": B, "T": head["T"], "L": head["L"], "D": spec["D"],
                      "H": spec["H"], "layers": spec["layers"], "mlp": spec["mlp"],
                      "vocab": spec["vocab"], "optimizer": "AdamW (fused, bf16 params)",
                      "l2": "working set (weights, activations, optimizer state) > L2"},
           "clocks": clk,
           "e2e": {"value": head["e2e_tokens_per_s"], "unit": UNIT,
                   "h2d_bytes_per_step": head["h2d_bytes_per_step"],
                   "d2h_bytes_per_step": head["d2h_bytes_per_step"]},
           "gpu_launches": launches, "model_tflops": head["tflops"], "runs": rows,
           "dense_model": dense}
    print(json.dumps(out))
    return out


# ------------------------------------------------------------- decoding
# Incremental decoding through one layer: B sequences decoded in lockstep, one
# token per call (bcmt_decode_step).  The L steps of a block are captured
# once as a CUDA graph (a block's slots 0..L-1 repeat in every block; the
# state carries the memory across blocks) and replayed block after block.
DECODE_WORKLOADS = {
    "decode_bf16_b16_t1024_l64_d512_h8": dict(B=16, T=1024, D=512, H=8, L=64, dtype="bf16"),
    "decode_bf16_b1_t1024_l64_d512_h8": dict(B=1, T=1024, D=512, H=8, L=64, dtype="bf16"),
}


def bench_decode(args):
    import torch
    from paper_2608_13578_gb300 import build
    build.build()
    from paper_2608_13578_gb300 import bcmt as C
    from paper_2608_13578_gb300 import layer
    from paper_2608_13578_gb300.inputs import Workload, make_inputs

    rank, local_rank, world = dist_env()
    if rank != 0:
        return None
    torch.cuda.set_device(local_rank)
    name = args.workload
    sp = DECODE_WORKLOADS[name]
    B, T, D, H, L = sp["B"], sp["T"], sp["D"], sp["H"], sp["L"]
    w = Workload(name, B, T, D, H, L, sp["dtype"], False, (0.8, 0.8), rank_seed(0, rank))
    t = {k: v.cuda() for k, v in make_inputs(w).items()}
    x_all = t["x"].transpose(0, 1).contiguous()          # [T, B, D]: token i of every sequence
    xin = torch.empty(L, B, D, dtype=x_all.dtype, device="cuda")  # the graph's input rows
    yout = torch.empty(T, B, D, dtype=x_all.dtype, device="cuda")
    ybuf = torch.empty(L, B, D, dtype=x_all.dtype, device="cuda")
    dec = layer.Decoder(t, B, H, L)
    stream = torch.cuda.current_stream()

    def block(pos0):
        for j in range(L):
            C.bcmt_decode_step(dec.p, dec.state, pos0 + j, xin[j], t["w_qkv"], t["w_o"], t["w_p"],
                               t["w_m"], t["w_g"], t["decay"], ybuf[j], None)

    xin.copy_(x_all[:L])
    for _ in range(2):  # warm-up: two blocks
        block(0)
    torch.cuda.synchronize()
    C.bcmt_decode_reset(dec.p, dec.state)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        block(0)
    C.bcmt_decode_reset(dec.p, dec.state)
    torch.cuda.synchronize()

    def run_all():
        for k in range(T // L):
            xin.copy_(x_all[k * L:(k + 1) * L])
            graph.replay()
            yout[k * L:(k + 1) * L].copy_(ybuf)

    run_all()  # warm the graph
    torch.cuda.synchronize()
    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    reps = max(1, args.steps // 4)
    ms = []
    for _ in range(reps):
        C.bcmt_decode_reset(dec.p, dec.state)
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        run_all()
        b_.record(stream)
        torch.cuda.synchronize()
        ms.append(a.elapsed_time(b_))
    clk = clocks.stop()
    C.bcmt_device_status(stream)
    tot = statistics.median(ms)
    tok_s = B * T / (tot / 1e3)
    # our launches per token step: widen, Q/K/V, attention, W_O, W_g, post (+ W_m per block)
    launches = T * 6 + T // L
    out = {"metric": "incremental decoding tokens/s through one BCMT layer", "value": round(tok_s, 1),
           "unit": UNIT, "n_gpus": 1, "steps": reps, "warmup": 2,
           "ms_per_step": round(tot / T, 5), "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": sp["dtype"], "data": "synthetic (seeded N(0,1) tokens, N(0,1/D) weights, decay 0.8)",
           "config": {"workload": name, "B": B, "T": T, "D": D, "H": H, "L": L,
                      "launch": f"CUDA graph of one block's {L} decode steps, replayed per block",
                      "note": "ms_per_step is per decoded position (B tokens)"},
           "clocks": clk, "gpu_launches": launches * reps,
           "e2e": None}
    print(json.dumps(out))
    return out


# ------------------------------------------------------ reference arm (oracle)
def bench_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return None
    from paper_2608_13578_gb300.inputs import HEADLINE, WORKLOADS
    name = args.workload or HEADLINE
    if name in MODEL_WORKLOADS or name in DECODE_WORKLOADS:
        out = {"impl": "reference", "unavailable": "the reference arm times the layer's forward "
                                                   "and backward only"}
        print(json.dumps(out))
        return out
    w = WORKLOADS[name]
    # each step: the oracle's fwd+bwd on one batch element of the workload
    d = run_oracle_sample(name, budget_s=0.0, max_reps=args.warmup + args.steps)
    times = d["times"][args.warmup:] or d["times"]
    secs = sum(times)
    value = d["tokens"] * len(times) / secs
    cpu = {"value": round(value, 2), "unit": UNIT, "cores": d["cores"], "kind": "oracle",
           "sample": f"float64 oracle fwd+bwd on batch element 0 of {name} ({d['tokens']} tokens) "
                     f"per step"}
    out = {"impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": UNIT,
           "n_gpus": world, "steps": len(times), "warmup": args.warmup,
           "ms_per_step": round(secs / len(times) * 1e3, 2), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic (seeded), one batch element per step",
           "config": {"workload": name, "B": w.B, "T": w.T, "L": w.L, "D": w.D, "H": w.H},
           "cpu_baseline": cpu,
           "e2e": {"value": round(value, 2), "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out))
    return out


def main():
    args = parse()
    if args.impl == "reference":
        bench_reference(args)
    elif args.workload in MODEL_WORKLOADS:
        bench_models(args)
    elif args.workload in DECODE_WORKLOADS:
        bench_decode(args)
    else:
        bench_ours(args)


if __name__ == "__main__":
    main()
