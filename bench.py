"""Benchmark: sparse dReLU FFN decode throughput on the 32-layer Mistral-shaped stack.

One step = one decode token (batch 1) through all 32 FFN layers of the
pre-norm residual stack (d=4096, m=14336, bf16 weights, ~10% combined dReLU
activation), replayed from one CUDA graph. Weights (11.3 GB) exceed L2, so no
flush is needed between steps. The K timed steps form one region; the region
is repeated (at least 3 times, enough to cover half a second) and the median
region is reported. Prints one JSON line (rank 0). By default that line also
carries, under "other_configs", the fp32 single FFN, the predictor-driven mode
on the same 32 layers, the Mixtral-shaped MoE stack at batch 1 and 8, and the
batch x activation sweep next to dense cuBLAS (--headline-only skips them).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload stack|predictor|moe|sweep] [--batch B]

``--workload moe`` times the 32-layer Mixtral-shaped MoE stack (8 experts,
top-2, ~90 GB of weights) at ``--batch``; ``--workload sweep`` prints one line
per (activation, batch) point of the Mistral-shaped stack next to dense
cuBLAS on the same weights. The default line is the batch-1 dense stack.

``--impl reference`` times the fp64 CPU oracle on a bounded sample of the
same workload (host cores only). Under torchrun with N > 1 every rank runs an
independent replica on its own GPU (the path has no cross-GPU exchange) and
``value`` counts the tokens of all ranks over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "sparse-FFN decode tokens/s and achieved HBM GB/s vs needed-bytes roofline"
UNIT = "tokens/s"
NOMINAL_HBM_GBS = 7900.0


# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of one gate+up
# launch on one full-size layer of the batch-1 stacks (bf16 rows: k_gate_up_rows;
# INT4 rows: k_gate_up_q4w), from one ncu capture each, and the SHA-256 of the
# kernel sources they were taken on: once those change, the figures no longer
# describe the kernels and are reported as null.
KERNEL_SOURCES = ("paper_2406_05955_gb300/csrc/ts_gate_up.cu", "paper_2406_05955_gb300/csrc/ts_kernels.cuh")
NCU_TRAFFIC = {"bytes": {"bf16": 164.46e6, "int4": 45.69e6},
               "sources": KERNEL_SOURCES,
               "sha256": "1dffd86c23421f56c66f947e8e8ada4f087e60ca9d85d582a0f1422c09050c43"}


def kernel_sources_sha256(paths) -> str:
    h = hashlib.sha256()
    for rel in paths:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def ncu_traffic(kind: str) -> float | None:
    try:
        ok = kernel_sources_sha256(NCU_TRAFFIC["sources"]) == NCU_TRAFFIC["sha256"]
    except OSError:
        ok = False
    return NCU_TRAFFIC["bytes"][kind] if ok else None


def load_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return {"hbm_gbs": float(j["hbm_gbs"]), "source": "measured"}
    return {"hbm_gbs": 6800.0, "source": "fallback"}


# ---------------------------------------------------------------------------
# distributed plumbing (replicas only)
# ---------------------------------------------------------------------------
class Dist:
    def __init__(self, n_gpus: int):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist

            backend = "nccl" if torch.cuda.is_available() else "gloo"
            dist.init_process_group(backend=backend)
            self.pg = dist
        if n_gpus != self.world and self.world > 1 and self.rank == 0:
            print(f"warning: --gpus {n_gpus} but WORLD_SIZE {self.world}", file=sys.stderr)

    def barrier(self):
        if self.pg is not None:
            if torch.cuda.is_available():
                self.pg.barrier(device_ids=[self.local])
            else:
                self.pg.barrier()

    def max(self, v: float) -> float:
        if self.pg is None:
            return v
        dev = torch.device("cuda", self.local) if torch.cuda.is_available() else torch.device("cpu")
        t = torch.tensor([v], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg is not None:
            self.pg.destroy_process_group()


def whole_job_value(batch: int, steps: int, world: int, t_max: float) -> float:
    """Tokens of every replica over the slowest replica's time (replicas run the same work)."""
    return batch * steps * world / t_max


# ---------------------------------------------------------------------------
# clock sampling during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.lines: list[str] = []
        self.t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (FileNotFoundError, OSError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# workload set-up
# ---------------------------------------------------------------------------
def stack_workload(args) -> str:
    if args.workload == "predictor":
        return "mistral7b-ffn-stack-bf16-predictor"
    if args.workload == "int4":
        return "mistral7b-ffn-stack-int4-b1-act10"
    return "mistral7b-ffn-stack-bf16-b1-act10"


def make_stack(ts, wl, dev, batch: int, predictor: bool, n_layers: int | None = None, name: str | None = None):
    cfg = dict(wl.WORKLOADS[name or ("mistral7b-ffn-stack-bf16-predictor" if predictor
                                     else "mistral7b-ffn-stack-bf16-b1-act10")])
    if n_layers:
        cfg["layers"] = n_layers
    d, m, n_layers = cfg["d"], cfg["m"], cfg["layers"]
    int4 = cfg["dtype"] == "int4"
    layers, ffns, lists = [], [], []
    for l in range(n_layers):
        if int4:
            L = wl.ffn_layer_int4(d, m, activation=cfg["activation"], seed=wl.layer_seed(cfg["seed"], l),
                                  device=dev)
        else:
            L = wl.ffn_layer(d, m, activation=cfg["activation"], dtype=torch.bfloat16,
                             seed=wl.layer_seed(cfg["seed"], l), device=dev)
        layers.append(L)
        ffns.append(ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=batch))
        if predictor:
            lists.append(wl.predictor_list(L.offsets, cfg["list_len"], zipf_s=cfg["zipf_s"],
                                           seed=wl.layer_seed(cfg["seed"], l) + 7).to(dev))
    return cfg, layers, ffns, (lists if predictor else None)


def row_bytes(f) -> int:
    """Bytes of one weight row of an Ffn handle (bf16, fp32 or INT4 rows)."""
    if f.wcode == 2:
        return f.d // 2 + f.d // 16
    return f.d * (2 if f.dtype == torch.bfloat16 else 4)


def needed_bytes_stack(ffns, lists) -> dict:
    """Per-layer algorithmic bytes from the last forward's active sets (union over the batch)."""
    tot_gate_up, tot_down, per = 0, 0, []
    for l, f in enumerate(ffns):
        g, b = f.get_active(-1)
        n_rows = f.m if lists is None else int(lists[l].numel())
        rb = row_bytes(f)
        gate_kernel = (n_rows + len(g)) * rb  # gate rows + gathered up rows
        down_kernel = len(b) * rb
        tot_gate_up += gate_kernel
        tot_down += down_kernel
        per.append((len(g), len(b)))
    return {"gate_up": tot_gate_up, "down": tot_down, "per_layer_counts": per}


def time_graph(graph, stream, steps: int) -> float:
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record(stream)
    for _ in range(steps):
        graph.launch(stream)
    e.record(stream)
    e.synchronize()
    return s.elapsed_time(e) / 1e3


MIN_TIMED_S = 0.5  # the repeats of a timed region cover at least this long, so the clock sampler sees the load


def time_repeats(graph, stream, steps: int, dist, min_total_s: float = MIN_TIMED_S):
    """Time ``steps`` replays R >= 3 times, each region bracketed by a barrier and a
    synchronize, R large enough that the regions cover ``min_total_s``.
    Returns (per-region seconds, max over ranks; clocks sampled meanwhile)."""
    dist.barrier()
    torch.cuda.synchronize()
    probe = time_graph(graph, stream, steps)
    reps = int(max(3, min(500, math.ceil(min_total_s / max(probe, 1e-6)))))
    reps = int(dist.max(float(reps)))
    clocks = ClockSampler(dist.local)
    clocks.start()
    time.sleep(0.3)
    times = []
    for _ in range(reps):
        dist.barrier()
        torch.cuda.synchronize()
        el = time_graph(graph, stream, steps)
        torch.cuda.synchronize()
        dist.barrier()
        times.append(dist.max(el))
    return times, clocks.stop()


def time_kernel_gate_up(ts, ffns, x, stream, lists, reps: int = 20) -> float:
    """Average duration of one gate+up launch (the dominant kernel) launched
    back to back, one per layer, the way the stack runs it (programmatic
    dependent launch between consecutive launches): CUDA events on its stream
    around ``reps`` passes over the layers, divided by the launches. The host
    enqueues a launch in a few microseconds, well ahead of the ~35 us kernels."""
    def body():
        for f_i, f in enumerate(ffns):
            f.gate_up(x, active_idx=None if lists is None else lists[f_i], stream=stream)

    for _ in range(2):
        body()
    torch.cuda.synchronize()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record(stream)
    for _ in range(reps):
        body()
    e.record(stream)
    e.synchronize()
    return s.elapsed_time(e) / 1e3 / (reps * len(ffns))


def dense_cublas_tokens_per_s(layers, batch, dev, steps=10) -> float:
    """The same 32-layer stack as a dense ReLU-gated FFN on cuBLAS (torch.matmul), graph-replayed."""
    d = layers[0].d
    h = torch.randn(batch, d, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def body():
        hh = h
        for L in layers:
            x = (hh * torch.rsqrt(hh.pow(2).mean(-1, keepdim=True) + 1e-5)).to(torch.bfloat16)
            g = x @ L.w_gate.t()
            u = x @ L.w_up.t()
            c = torch.relu(g) * torch.relu(u)
            hh = hh + (c @ L.w_down).float()  # W_down is neuron-major [m][d]
        return hh

    with torch.cuda.stream(stream):
        for _ in range(3):
            body()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        body()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record()
    for _ in range(steps):
        g.replay()
    e.record()
    e.synchronize()
    return batch * steps / (s.elapsed_time(e) / 1e3)


def cpu_baseline(layers, lists, batch, n_layers_total, budget_s=12.0, budget_1t_s=6.0) -> dict:
    """The oracle as it stands, on the host cores, over a bounded sample of
    layers: with every core (OpenMP over independent outputs), then with one
    thread (reported beside it)."""
    import oracle

    host = [(oracle.as_array(L.w_gate), oracle.as_array(L.w_up), oracle.as_array(L.w_down))
            for L in layers[:2]]
    hl = None if lists is None else [x.cpu().numpy() for x in lists[:2]]
    cores = oracle.max_threads()

    def sample(threads: int, budget: float):
        rng = np.random.default_rng(0)
        h = rng.standard_normal((batch, layers[0].d)).astype(np.float32)
        done = 0
        t0 = time.perf_counter()
        while True:
            i = done % len(host)
            x = oracle.rmsnorm(h, oracle.BF16)
            r = oracle.ffn(x, *host[i], rows=None if hl is None else hl[i], threads=threads)
            h = (h + r["y"]).astype(np.float32)
            done += 1
            el = time.perf_counter() - t0
            if el >= budget or done >= 400:
                return done, el

    done, el = sample(cores, budget_s)
    done1, el1 = sample(1, budget_1t_s)
    oracle.ffn(*([np.zeros((1, 1), np.float32)] * 4), threads=cores)  # restore the thread count
    value = batch * done / n_layers_total / el
    return {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{done} layer evaluations (cycling over 2 of the {n_layers_total} layers, batch {batch}) "
                      f"in {el:.1f} s, scaled to full {n_layers_total}-layer tokens",
            "single_thread": {"value": batch * done1 / n_layers_total / el1, "unit": UNIT, "cores": 1,
                              "sample": f"{done1} layer evaluations in {el1:.1f} s, one OpenMP thread"}}


# ---------------------------------------------------------------------------
# arms
# ---------------------------------------------------------------------------
def predictor_line(ts, wl, ffns, layers, h0, stream, args, dist) -> dict:
    """Predictor-driven mode (Sec. 7) on the given 32 layers at batch 1: per
    layer a sorted list of 1434 neurons drawn with Zipf(1.1) weights over
    hotness; gate, up and down touch only listed rows."""
    name = "mistral7b-ffn-stack-bf16-predictor"
    cfg = wl.WORKLOADS[name]
    dev = h0.device
    lists = [wl.predictor_list(L.offsets, cfg["list_len"], zipf_s=cfg["zipf_s"],
                               seed=wl.layer_seed(cfg["seed"], l) + 7).to(dev) for l, L in enumerate(layers)]
    h = h0.clone()
    graph = ts.Graph.stack(ffns, h, active_idx=lists)
    for _ in range(args.warmup):
        graph.launch(stream)
    torch.cuda.synchronize()
    times, clk = time_repeats(graph, stream, args.steps, dist)
    t = statistics.median(times)
    nb = needed_bytes_stack(ffns, lists)
    peaks = load_peaks()
    step_s = t / args.steps
    graph.close()
    return {"workload": name, "value": whole_job_value(1, args.steps, dist.world, t), "unit": UNIT,
            "ms_per_step": step_s * 1e3, "timed_regions": len(times),
            "list_len": cfg["list_len"],
            "needed_bytes_roofline": {"bytes_per_token": nb["gate_up"] + nb["down"],
                                      "achieved_gbs": (nb["gate_up"] + nb["down"]) / step_s / 1e9,
                                      "frac_of_measured": (nb["gate_up"] + nb["down"]) / step_s / 1e9 / peaks["hbm_gbs"]},
            "clocks": clk}


def fp32_small_line(ts, wl, dev, args, dist) -> dict:
    """The fp32 single-FFN configuration (d=512, m=1408): 16 decode tokens one
    at a time through one FFN, replayed from a graph. Its 4 MB of weights sit
    in L2, so it is reported for speed only, not against the HBM roofline."""
    name = "drelu-ffn-fp32-d512-m1408"
    cfg = wl.WORKLOADS[name]
    d, m, n_tok = cfg["d"], cfg["m"], cfg["n_tokens"]
    L = wl.ffn_layer(d, m, mu=cfg["mu"], dtype=torch.float32, seed=cfg["seed"], device=dev)
    f = ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=1)
    xs = wl.tokens(n_tok, d, dtype=torch.float32, seed=cfg["seed"] + 1, device=dev)
    ys = torch.empty(n_tok, d, dtype=torch.float32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def body():
        for t in range(n_tok):
            f.forward(xs[t:t + 1], y=ys[t:t + 1], stream=stream)

    with torch.cuda.stream(stream):
        body()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        body()
    calls = _Calls(lambda st: g.replay())
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g.replay()
        torch.cuda.synchronize()
        times, clk = time_repeats(calls, stream, args.steps, dist)
    t = statistics.median(times)
    del g
    f.close()
    return {"workload": name, "value": whole_job_value(n_tok, args.steps, dist.world, t), "unit": UNIT,
            "us_per_token": t / (args.steps * n_tok) * 1e6, "timed_regions": len(times),
            "note": "L2-resident (4 MB of weights): a correctness configuration, no HBM roofline", "clocks": clk}


def moe_lines(ts, wl, dev, args, dist, batches, int4: bool = False) -> list:
    """32-layer Mixtral-shaped MoE stack (router + top-2 of 8 sparse experts
    per layer), one timed line per batch size; the weights are drawn once."""
    name = "mixtral47b-moe-stack-int4-top2" if int4 else "mixtral47b-moe-stack-bf16-top2"
    cfg = wl.WORKLOADS[name]
    d, m, E, k = cfg["d"], cfg["m"], cfg["experts"], cfg["top_k"]
    n_layers = args.layers or cfg["layers"]
    max_b = max(batches)
    experts, moes = [], []
    for l in range(n_layers):
        if int4:
            ex = [wl.ffn_layer_int4(d, m, activation=cfg["activation"], seed=wl.layer_seed(cfg["seed"], l, e),
                                    device=dev) for e in range(E)]
        else:
            ex = [wl.ffn_layer(d, m, activation=cfg["activation"], dtype=torch.bfloat16,
                               seed=wl.layer_seed(cfg["seed"], l, e), device=dev) for e in range(E)]
        ffns = [ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=max_b) for L in ex]
        wr = wl.router(E, d, seed=wl.layer_seed(cfg["seed"], l) + 99, device=dev)
        experts.append((ex, ffns, wr))
        moes.append(ts.Moe(wr, ffns, top_k=k, max_batch=max_b))
    peaks = load_peaks()
    out = []
    for B in batches:
        h0 = wl.residual(B, d, seed=cfg["seed"] - 1, device=dev)
        h = h0.clone()
        stream = torch.cuda.Stream(device=dev)
        graph = ts.Graph.moe_stack(moes, h)
        for _ in range(args.warmup):
            graph.launch(stream)
        torch.cuda.synchronize()
        times, clk = time_repeats(graph, stream, args.steps, dist)
        t = statistics.median(times)
        # needed bytes of the last replay: per layer, every expert a token was routed to
        graph.launch(stream)
        torch.cuda.synchronize()
        need = 0
        for mo in moes:
            sel, _ = mo.get_routing(B)
            for e in sorted(set(sel.ravel().tolist())):
                g, b = mo.get_active(e, -1)
                need += (m + len(g) + len(b)) * row_bytes(mo.experts[e])
        step_s = t / args.steps
        out.append({"workload": name, "batch": B, "value": whole_job_value(B, args.steps, dist.world, t),
                    "unit": UNIT, "ms_per_step": step_s * 1e3, "timed_regions": len(times),
                    "config": {"d": d, "m": m, "experts": E, "top_k": k, "layers": n_layers,
                               "activation": cfg["activation"],
                               "weights_gb": round(E * 3 * m * row_bytes(experts[0][1][0]) * n_layers / 1e9, 1)},
                    "needed_bytes_roofline": {"bytes_per_step": need, "achieved_gbs": need / step_s / 1e9,
                                              "frac_of_measured": need / step_s / 1e9 / peaks["hbm_gbs"]},
                    "gpu_launches": 3 * n_layers * args.steps * ((B + 7) // 8),
                    "clocks": clk})
        graph.close()
    for mo in moes:
        mo.close()
    for _, ffns, _ in experts:
        for f in ffns:
            f.close()
    del experts, moes
    torch.cuda.empty_cache()
    return out


def _sweep_summary(r: dict) -> dict:
    return {"batch": r["config"]["batch"], "activation": r["config"]["activation"], "value": r["value"],
            "unit": r["unit"], "ms_per_step": r["ms_per_step"],
            "frac_of_measured": r["needed_bytes_roofline"]["frac_of_measured"],
            "dense_cublas": r["dense_cublas"]["value"], "speedup_vs_dense": r["speedup_vs_dense"]}


def run_ours(args, dist: Dist) -> dict | None:
    import paper_2406_05955_gb300 as ts
    from paper_2406_05955_gb300 import workload as wl

    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    B = args.batch
    predictor = args.workload == "predictor"
    int4 = args.workload == "int4"
    cfg, layers, ffns, lists = make_stack(ts, wl, dev, B, predictor, args.layers, name=stack_workload(args))
    n_layers = cfg["layers"]
    h0 = wl.residual(B, cfg["d"], seed=cfg["seed"] - 1, device=dev)
    h = h0.clone()
    stream = torch.cuda.Stream(device=dev)
    graph = ts.Graph.stack(ffns, h, active_idx=lists)
    for _ in range(args.warmup):
        graph.launch(stream)
    torch.cuda.synchronize()

    # timed region: K graph replays, barrier + sync on both sides, clocks
    # sampled; repeated (>= 3 regions) and the median region taken
    times, clk = time_repeats(graph, stream, args.steps, dist)
    t_max = statistics.median(times)
    value = whole_job_value(B, args.steps, dist.world, t_max)

    # end-to-end through the public API with host buffers (pinned), copies
    # inside the timed region; as many regions as above, median
    h_host = torch.empty_like(h0, device="cpu").pin_memory()
    h_host.copy_(h0.cpu())
    out_host = torch.empty_like(h_host).pin_memory()
    with_copies = _Calls(lambda st: (h.copy_(h_host, non_blocking=True), graph.launch(st),
                                     out_host.copy_(h, non_blocking=True)))
    e2e_times = []
    with torch.cuda.stream(stream):
        for _ in range(len(times)):
            dist.barrier()
            torch.cuda.synchronize()
            e2e_times.append(dist.max(time_graph(with_copies, stream, args.steps)))
    e2e_t = statistics.median(e2e_times)
    e2e = {"value": B * args.steps * dist.world / e2e_t, "unit": UNIT,
           "h2d_bytes_per_step": h_host.numel() * 4, "d2h_bytes_per_step": out_host.numel() * 4}

    # dominant kernel: gate+up, one launch per layer replayed from a graph
    x = wl.tokens(B, cfg["d"], dtype=torch.bfloat16, seed=5, device=dev)  # bf16 activations (INT4 too)
    graph.launch(stream)
    torch.cuda.synchronize()
    nb = needed_bytes_stack(ffns, lists)
    wide = B > 8  # one wide pass per layer (gate, up, down, reduction kernels)
    peaks = load_peaks()
    step_s = t_max / args.steps
    if not wide:
        t_gate_up = time_kernel_gate_up(ts, ffns, x, stream, lists)
        nb_x = needed_bytes_stack(ffns, lists)  # active sets of the x used in the kernel timing
        # passes of 1-2 tokens: the gate+up kernel also gathers the W_down rows
        # (each CTA's share of the down projection)
        gate_up_bytes = (nb_x["gate_up"] + (nb_x["down"] if B <= 2 else 0)) / n_layers
    else:
        # the wide pass's kernels depend on one another; the layer is the unit
        t_gate_up = step_s / n_layers
        gate_up_bytes = (nb["gate_up"] + nb["down"]) / n_layers
    achieved = gate_up_bytes / t_gate_up / 1e9
    needed_per_token = (nb["gate_up"] + nb["down"]) / B
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int4 weights, bf16 activations, fp32 accumulate" if int4 else "bf16",
        "data": "synthetic",
        "timing": {"timed_regions": len(times), "statistic": "median over regions",
                   "ms_per_step_min": min(times) / args.steps * 1e3,
                   "ms_per_step_max": max(times) / args.steps * 1e3},
        "config": {"workload": stack_workload(args),
                   "d": cfg["d"], "m": cfg["m"], "layers": n_layers, "batch": B,
                   "activation": cfg["activation"], "weights_gb": round(3 * cfg["m"] * row_bytes(ffns[0]) * n_layers / 1e9, 2),
                   "l2": f"no flush: the {3 * cfg['m'] * row_bytes(ffns[0]) * n_layers / 1e9:.2f} GB of weights "
                         "streamed per step exceed the 129 MB L2",
                   "parallelism": f"replicas x{dist.world}"},
        "layers_per_s": value * n_layers / B,
        "needed_bytes_roofline": {
            "bytes_per_token": needed_per_token,
            "achieved_gbs": needed_per_token * B / step_s / 1e9,
            "frac_of_measured": needed_per_token * B / step_s / 1e9 / peaks["hbm_gbs"],
            "frac_of_nominal": needed_per_token * B / step_s / 1e9 / NOMINAL_HBM_GBS,
            "gate_active_per_layer": statistics.mean(c[0] for c in nb["per_layer_counts"]),
            "both_active_per_layer": statistics.mean(c[1] for c in nb["per_layer_counts"]),
        },
        "roofline": {"bound": "hbm",
                     "kernel": (("k_gate_up_q4w" if int4 else "k_gate_up_rows") +
                                " (gate GEMV, gathered up projection, this CTA's share of the down projection)"
                                if B <= 2 else ("k_gate_up_mma (gate GEMM + gathered up projection)" if not wide
                                                else "wide pass: k_wide_gate + k_wide_up + down + reduction, per layer")),
                     "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / peaks["hbm_gbs"], "peak_source": peaks["source"],
                     "traffic": None if predictor or B != 1 else ncu_traffic("int4" if int4 else "bf16"),
                     "bytes_per_launch": gate_up_bytes,
                     "avg_launch_us": t_gate_up * 1e6,
                     "timed_as": (f"{n_layers} gate+up launches (one per layer) back to back, 20 passes, "
                                  "CUDA events on the launching stream") if not wide
                                 else "the stack's graph replays, per layer"},
        "e2e": e2e,
        "gpu_launches": (5 if wide else 2) * n_layers * args.steps * (1 if wide else (B + 7) // 8),
        "clocks": clk,
    }
    if not args.no_dense and not int4:
        result["dense_cublas"] = {"value": dense_cublas_tokens_per_s(layers, B, dev), "unit": UNIT,
                                  "what": "same weights, dense ReLU-gated FFN via torch.matmul (cuBLAS), graph-replayed"}
    if dist.rank == 0 and not args.no_cpu_baseline and not int4:
        result["cpu_baseline"] = cpu_baseline(layers, lists, B, n_layers)
    if args.workload == "stack" and B == 1 and not args.headline_only:
        # the predictor-driven mode on the same 32 layers (its lists favour hot neurons)
        graph.close()
        result["other_configs"] = {"predictor_mode": predictor_line(ts, wl, ffns, layers, h0, stream, args, dist)}
    for f in ffns:
        f.close()
    graph.close()
    del layers, ffns
    torch.cuda.empty_cache()
    if args.workload == "stack" and B == 1 and not args.headline_only:
        oc = result["other_configs"]
        oc["fp32_single_ffn"] = fp32_small_line(ts, wl, dev, args, dist)
        oc["moe_top2"] = moe_lines(ts, wl, dev, args, dist, batches=(1, 8))
        oc["sweep"] = [_sweep_summary(r) for r in run_sweep(args, dist)]
    return result


def _clocked_time(graph, stream, steps, dist):
    """Median over >= 3 timed regions of K replays (time_repeats): (seconds, clocks)."""
    times, clk = time_repeats(graph, stream, steps, dist)
    return statistics.median(times), clk


class _Calls:
    """A list of launches that time_graph can replay like a graph."""

    def __init__(self, fn):
        self.fn = fn

    def launch(self, stream):
        self.fn(stream)


def run_topk(args, dist: Dist) -> dict:
    """Top-k magnitude mask (Eq. 3-4) on 32 full-size layers at batch 1: per
    layer one ts_ffn_forward_topk on the token's normalised activations
    (the same x for every layer: the mask, not the stack glue, is measured)."""
    import paper_2406_05955_gb300 as ts
    from paper_2406_05955_gb300 import workload as wl

    name = "mistral7b-ffn-topk5-b1"
    cfg = wl.WORKLOADS[name]
    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    d, m, B, keep = cfg["d"], cfg["m"], cfg["batch"], cfg["keep"]
    n_layers = args.layers or cfg["layers"]
    layers = [wl.ffn_layer(d, m, activation=cfg["activation"], dtype=torch.bfloat16,
                           seed=wl.layer_seed(cfg["seed"], l), device=dev) for l in range(n_layers)]
    ffns = [ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=B) for L in layers]
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=cfg["seed"] + 7, device=dev)
    y = torch.empty(B, d, dtype=torch.float32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step_topk(s):
        for f in ffns:
            f.forward_topk(x, keep, y=y, stream=s)

    def step_plain(s):
        for f in ffns:
            f.forward(x, y=y, stream=s)

    calls = _Calls(step_topk)
    for _ in range(args.warmup):
        calls.launch(stream)
    torch.cuda.synchronize()
    t_max, clk = _clocked_time(calls, stream, args.steps, dist)
    value = whole_job_value(B, args.steps, dist.world, t_max)
    kept = statistics.mean(len(f.get_active(0)[1]) for f in ffns)
    plain = _Calls(step_plain)
    for _ in range(args.warmup):
        plain.launch(stream)
    torch.cuda.synchronize()
    t_plain = time_graph(plain, stream, args.steps)
    step_s = t_max / args.steps
    nb = needed_bytes_stack(ffns, None)  # gate rows + gate-active up rows + kept down rows
    peaks = load_peaks()
    return {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": name, "d": d, "m": m, "layers": n_layers, "batch": B, "keep": keep,
                   "activation": cfg["activation"],
                   "l2": "no flush: the 11.3 GB of weights streamed per step exceed the 129 MB L2",
                   "parallelism": f"replicas x{dist.world}"},
        "kept_per_layer": kept,
        "needed_bytes_roofline": {
            "bytes_per_token": (nb["gate_up"] + nb["down"]) / B,
            "achieved_gbs": (nb["gate_up"] + nb["down"]) / step_s / 1e9,
            "frac_of_measured": (nb["gate_up"] + nb["down"]) / step_s / 1e9 / peaks["hbm_gbs"]},
        "plain_forward_same_layers": {"value": B * args.steps / t_plain, "unit": UNIT},
        "gpu_launches": 4 * n_layers * args.steps,
        "clocks": clk,
    }


def run_prednet(args, dist: Dist) -> dict:
    """Predictor network + predictor mode on the 32-layer Mistral-shaped stack
    at batch 1: per layer, a rank-512 two-layer ReLU MLP scores the 14336
    neurons from rmsnorm(h), the 1434 best form the list, and the FFN runs
    over the listed rows only; the whole step is one CUDA graph."""
    import paper_2406_05955_gb300 as ts
    from paper_2406_05955_gb300 import workload as wl

    name = "mistral7b-ffn-stack-bf16-b1-prednet"
    cfg = dict(wl.WORKLOADS[name])
    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    d, m, r, K, B = cfg["d"], cfg["m"], cfg["rank"], cfg["k"], cfg["batch"]
    n_layers = args.layers or cfg["layers"]
    layers, ffns, preds, pw = [], [], [], []
    for l in range(n_layers):
        L = wl.ffn_layer(d, m, activation=cfg["activation"], dtype=torch.bfloat16,
                         seed=wl.layer_seed(cfg["seed"], l), device=dev)
        P = wl.predictor_weights(d, r, m, L.offsets, dtype=torch.bfloat16,
                                 seed=wl.layer_seed(cfg["seed"], l) + 11, device=dev)
        layers.append(L)
        pw.append(P)
        ffns.append(ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=B))
        preds.append(ts.Predictor(P.w1, P.w2, max_batch=B))
    lists = [torch.empty(K, dtype=torch.int32, device=dev) for _ in range(n_layers)]
    h0 = wl.residual(B, d, seed=cfg["seed"] - 1, device=dev)
    h = h0.clone()
    stream = torch.cuda.Stream(device=dev)
    graph = ts.Graph.stack_predicted(ffns, preds, h, [K] * n_layers, lists)
    for _ in range(args.warmup):
        graph.launch(stream)
    torch.cuda.synchronize()
    t_max, clk = _clocked_time(graph, stream, args.steps, dist)
    value = whole_job_value(B, args.steps, dist.world, t_max)
    step_s = t_max / args.steps
    # algorithmic bytes: both predictor matrices, then the FFN over the lists
    nb = needed_bytes_stack(ffns, lists)
    pred_bytes = n_layers * (r * d + m * r) * 2
    total = nb["gate_up"] + nb["down"] + pred_bytes
    peaks = load_peaks()

    # the prediction alone (3 launches per layer), CUDA events on its stream
    x = wl.tokens(B, d, dtype=torch.bfloat16, seed=cfg["seed"] + 5, device=dev)
    for p_, buf in zip(preds, lists):
        p_.predict(x, K, out=buf, stream=stream)
    torch.cuda.synchronize()
    s_ev, e_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 5
    s_ev.record(stream)
    for _ in range(reps):
        for p_, buf in zip(preds, lists):
            p_.predict(x, K, out=buf, stream=stream)
    e_ev.record(stream)
    e_ev.synchronize()
    t_pred = s_ev.elapsed_time(e_ev) / 1e3 / (reps * n_layers)
    pred_layer_bytes = (r * d + m * r) * 2
    res = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": name, "d": d, "m": m, "rank": r, "k": K, "layers": n_layers, "batch": B,
                   "activation": cfg["activation"],
                   "l2": "no flush: the 12 GB of FFN and predictor weights touched per step exceed the 129 MB L2",
                   "parallelism": f"replicas x{dist.world}"},
        "needed_bytes_roofline": {
            "bytes_per_token": total / B, "predictor_bytes_per_token": pred_bytes / B,
            "achieved_gbs": total / step_s / 1e9,
            "frac_of_measured": total / step_s / 1e9 / peaks["hbm_gbs"]},
        "prediction_only": {"us_per_layer": t_pred * 1e6,
                            "achieved_gbs": pred_layer_bytes / t_pred / 1e9,
                            "frac_of_measured": pred_layer_bytes / t_pred / 1e9 / peaks["hbm_gbs"]},
        # per layer: hidden, score, select, gate+up, down reduction
        "gpu_launches": 5 * n_layers * args.steps,
        "clocks": clk,
    }
    return res


def run_moe(args, dist: Dist) -> dict:
    """32-layer Mixtral-shaped MoE stack (router + top-2 of 8 sparse experts per layer) at --batch."""
    import paper_2406_05955_gb300 as ts
    from paper_2406_05955_gb300 import workload as wl

    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    r = moe_lines(ts, wl, dev, args, dist, batches=(args.batch,), int4=args.workload == "moe-int4")[0]
    int4 = args.workload == "moe-int4"
    return {"metric": METRIC, "value": r["value"], "unit": UNIT, "n_gpus": dist.world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": r["ms_per_step"], "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None,
            "dtype": "int4 weights, bf16 activations, fp32 accumulate" if int4 else "bf16", "data": "synthetic",
            "config": dict(workload=r["workload"], batch=args.batch, **r["config"],
                           l2="no flush: the experts streamed per step exceed the 129 MB L2",
                           parallelism=f"replicas x{dist.world}"),
            "needed_bytes_roofline": r["needed_bytes_roofline"], "gpu_launches": r["gpu_launches"],
            "clocks": r["clocks"]}


def run_sweep(args, dist: Dist) -> list:
    """Batch x activation sweep of the 32-layer Mistral-shaped stack next to dense cuBLAS."""
    import paper_2406_05955_gb300 as ts
    from paper_2406_05955_gb300 import workload as wl

    name = "mistral7b-ffn-stack-bf16-sweep"
    cfg = wl.WORKLOADS[name]
    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    d, m = cfg["d"], cfg["m"]
    n_layers = args.layers or cfg["layers"]
    peaks = load_peaks()
    out = []
    for act in cfg["activations"]:
        layers = [wl.ffn_layer(d, m, activation=act, dtype=torch.bfloat16,
                               seed=wl.layer_seed(cfg["seed"], l), device=dev) for l in range(n_layers)]
        ffns = [ts.Ffn(L.w_gate, L.w_up, L.w_down, max_batch=max(cfg["batches"])) for L in layers]
        for B in cfg["batches"]:
            h = wl.residual(B, d, seed=cfg["seed"] - 1, device=dev)
            stream = torch.cuda.Stream(device=dev)
            graph = ts.Graph.stack(ffns, h)
            for _ in range(args.warmup):
                graph.launch(stream)
            torch.cuda.synchronize()
            steps = max(3, args.steps // max(1, B // 4))
            times, clk = time_repeats(graph, stream, steps, dist, min_total_s=0.2)
            t_max = statistics.median(times)
            value = whole_job_value(B, steps, dist.world, t_max)
            nb = needed_bytes_stack(ffns, None)
            step_s = t_max / steps
            dense = dense_cublas_tokens_per_s(layers, B, dev) * dist.world
            out.append({
                "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": steps,
                "warmup": args.warmup, "ms_per_step": step_s * 1e3, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": name, "d": d, "m": m, "layers": n_layers, "batch": B, "activation": act,
                           "parallelism": f"replicas x{dist.world}"},
                "needed_bytes_roofline": {
                    "bytes_per_step": nb["gate_up"] + nb["down"],
                    "achieved_gbs": (nb["gate_up"] + nb["down"]) / step_s / 1e9,
                    "frac_of_measured": (nb["gate_up"] + nb["down"]) / step_s / 1e9 / peaks["hbm_gbs"]},
                "dense_cublas": {"value": dense, "unit": UNIT},
                "speedup_vs_dense": value / dense,
                "clocks": clk,
            })
            graph.close()
        for f in ffns:
            f.close()
        del layers, ffns
        torch.cuda.empty_cache()
    return out


def run_reference(args, dist: Dist) -> dict | None:
    """The oracle (fp64, host cores) on a bounded sample per step, same metric and config."""
    if dist.rank != 0:
        return None
    import oracle
    from paper_2406_05955_gb300 import workload as wl

    oracle.build()
    predictor = args.workload == "predictor"
    name = "mistral7b-ffn-stack-bf16-predictor" if predictor else "mistral7b-ffn-stack-bf16-b1-act10"
    cfg = wl.WORKLOADS[name]
    B = args.batch
    L = wl.ffn_layer(cfg["d"], cfg["m"], activation=cfg["activation"], dtype=torch.bfloat16,
                     seed=wl.layer_seed(cfg["seed"], 0))
    w = (oracle.as_array(L.w_gate), oracle.as_array(L.w_up), oracle.as_array(L.w_down))
    rows = wl.predictor_list(L.offsets, cfg["list_len"]).numpy() if predictor else None
    h = wl.residual(B, cfg["d"], seed=cfg["seed"] - 1).numpy()

    def step():
        x = oracle.rmsnorm(h, oracle.BF16)
        return oracle.ffn(x, *w, rows=rows)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t0
    # one step = one layer of the 32-layer stack for B tokens: tokens/s = B / (32 * t_layer)
    value = B * args.steps / (el * cfg["layers"])
    return {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
        "config": {"workload": name, "d": cfg["d"], "m": cfg["m"], "layers": cfg["layers"], "batch": B},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
                         "sample": f"each step: one of the {cfg['layers']} layers (batch {B}), scaled to the full stack"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=["stack", "predictor", "moe", "sweep", "int4", "moe-int4", "topk",
                                           "prednet"],
                    default="stack")
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--layers", type=int, default=0,
                    help="fewer layers than the workload's 32 (profiling cases only; not a bench line)")
    ap.add_argument("--no-dense", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--headline-only", action="store_true",
                    help="default workload: skip the other configurations (fp32 FFN, predictor mode, MoE, sweep)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.impl == "reference" and args.workload not in ("stack", "predictor"):
        ap.error("the reference arm times the oracle on the stack and predictor workloads")
    dist = Dist(args.gpus)
    try:
        if args.impl == "reference":
            res = run_reference(args, dist)
        else:
            from __graft_entry__ import build

            if dist.rank == 0:
                build()
            dist.barrier()
            if args.workload in ("moe", "moe-int4"):
                res = run_moe(args, dist)
            elif args.workload == "sweep":
                res = run_sweep(args, dist)
            elif args.workload == "topk":
                res = run_topk(args, dist)
            elif args.workload == "prednet":
                res = run_prednet(args, dist)
            else:
                res = run_ours(args, dist)
        if res is not None and dist.rank == 0:
            for line in res if isinstance(res, list) else [res]:
                print(json.dumps(line), flush=True)
    finally:
        dist.close()


if __name__ == "__main__":
    main()
