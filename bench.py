#!/usr/bin/env python3
"""Benchmark of the dMoE MoE-layer forward (one block-diffusion decoding step's MoE layer).

Workload (one GPU): d=2048, 256 routed experts, top-8, expert SwiGLU intermediate 512, one
shared expert of intermediate 512, one sequence x one diffusion block of 32 tokens, router
bias 0.5*ln(1/rank), block routing with the coreset floor (p=0, "block top-k"); token
routing and p=0.6 are measured beside it. A step is one full layer forward (router,
Algorithm 1, dispatch, expert GEMMs, combine) through the C ABI.

L2 honesty: the steps rotate over --sets independently seeded copies of the layer (weights,
router and input), so consecutive steps never find their ~60 MB of expert weights in the
129 MB L2. Steps are replayed from CUDA graphs (launch-bound otherwise).

Prints one JSON line (rank 0). --impl reference times the CPU oracle instead. --suite
measures the other workloads instead (one JSON line each): 8 sequences x 32 tokens, the
block-size x batch x bias-scale grid, and the 20-layer stack of 64 x 32 tokens.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

_CORES = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(_CORES))

import numpy as np  # noqa: E402

METRIC = "MoE-layer tokens/s (block routing, block size 32)"
UNIT = "tokens/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def workload_shape(mode: str, top_p: float):
    from dmoe_synth import LAYER, ROUTE_BLOCK, ROUTE_TOKEN
    return LAYER.with_(mode=ROUTE_BLOCK if mode == "block" else ROUTE_TOKEN, top_p=top_p)


def workload_name(shape) -> str:
    mode = "block" if shape.mode == 1 else "token"
    tail = f"_p{shape.top_p:g}" if shape.mode == 1 else ""
    if shape.mode == 1 and getattr(shape, "block_top_k", 0):
        tail += f"_mask{shape.block_top_k}"
    return (f"moe_layer_d{shape.d_model}_E{shape.n_experts}_k{shape.top_k}_I{shape.d_ff}"
            f"_shared{shape.d_ff_shared}_B{shape.block_size}x{shape.n_blocks}_{mode}{tail}")


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


# ----------------------------------------------------------------------------- byte model
def layer_bytes(shape, U: float) -> float:
    """Algorithmic HBM bytes of one layer forward: the unique experts' and the shared
    expert's bf16 weights once, the fp32 router weight and bias, x read and y written."""
    d, E, I, Is, T = shape.d_model, shape.n_experts, shape.d_ff, shape.d_ff_shared, shape.T
    return (U * 3 * d * I * 2 + 3 * d * Is * 2 + d * E * 4 + E * 4 + T * d * 2 * 2)


def experts_bytes(shape, U: float) -> float:
    """Algorithmic bytes of one expert-kernel launch: the gate, up and down weights of the
    unique and shared experts once, the token rows read once and the output rows written
    once (bf16)."""
    d, I, Is, T = shape.d_model, shape.d_ff, shape.d_ff_shared, shape.T
    return U * 3 * d * I * 2 + 3 * d * Is * 2 + T * d * 2 * 2


def layer_flops(shape) -> float:
    d, E, I, Is, T, k = (shape.d_model, shape.n_experts, shape.d_ff, shape.d_ff_shared, shape.T,
                         shape.top_k)
    return 2 * T * (k * 3 * d * I + 3 * d * Is) + 2 * T * d * E


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_uuid: str | None):
        self.uuid = gpu_uuid
        self.proc = None
        self.lines = []

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu=uuid,{self.FIELDS}", "--format=csv,noheader,nounits",
               "-lms", "50"]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"],
                    "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            if self.uuid and parts[0] != self.uuid:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": float(max(smax)) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def gpu_uuid(torch):
    try:
        u = str(torch.cuda.get_device_properties(torch.cuda.current_device()).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return None


# ----------------------------------------------------------------------------- our arm
class Arm:
    """n_sets resident copies of the layer, CUDA graphs of one rotation each."""

    def __init__(self, shape, n_sets, seed0, torch, dm, MoELayer, layer_inputs, host_io=False):
        self.shape, self.torch, self.dm = shape, torch, dm
        self.layers, self.x = [], []
        for s in range(n_sets):
            inp = layer_inputs(shape, seed=seed0 + s, device="cuda")
            if s == 0:
                self.inputs0 = inp
            self.layers.append(MoELayer.from_shape(shape, inp))
            self.x.append(inp["x"])
        self.set_host_io(host_io)

    def set_host_io(self, on: bool):
        self.host_io = on
        if on and not hasattr(self, "x_host"):
            self.x_host = [x.cpu().pin_memory() for x in self.x]
            self.y_host = [self.torch.empty_like(x, device="cpu").pin_memory() for x in self.x]
            self.s_in, self.s_out = self.torch.cuda.Stream(), self.torch.cuda.Stream()

    def step(self, i):
        L = self.layers[i % len(self.layers)]
        if self.host_io:
            x = self.x[i % len(self.x)]
            x.copy_(self.x_host[i % len(self.x)], non_blocking=True)
            y = L.forward(x)
            self.y_host[i % len(self.x)].copy_(y, non_blocking=True)
        else:
            L.forward(self.x[i % len(self.x)])

    def check(self):
        for L in self.layers:
            st, info = self.dm.dmoe_get_device_error(L.ws)
            if st != 0:
                raise RuntimeError(f"device fault {info}")

    def unique_counts(self):
        return [int(L.n_unique.item()) for L in self.layers]

    def capture(self, n_steps, first):
        """A CUDA graph of n_steps consecutive steps starting at index `first`."""
        torch = self.torch
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            if self.host_io:
                self.capture_host_io(n_steps, first)
            else:
                for i in range(n_steps):
                    self.step(first + i)
        return g

    def capture_host_io(self, n_steps, first):
        """Steps with x copied in from pinned host memory and y copied back, pipelined one
        step deep as a double-buffered serving loop would run them: the copy of step j+1's x
        (on its own stream) starts once step j-1's forward has ended and overlaps step j's
        forward; the copy of y_j back overlaps step j+1's forward. Every step's two copies
        are inside the captured steps."""
        torch = self.torch
        main = torch.cuda.current_stream()
        n = len(self.layers)
        self.s_in.wait_stream(main)
        self.s_out.wait_stream(main)
        ev_x = [torch.cuda.Event() for _ in range(n_steps)]
        ev_y = [torch.cuda.Event() for _ in range(n_steps)]

        def copy_in(j):
            idx = (first + j) % n
            with torch.cuda.stream(self.s_in):
                if j >= 2:
                    self.s_in.wait_event(ev_y[j - 2])
                self.x[idx].copy_(self.x_host[idx], non_blocking=True)
                ev_x[j].record(self.s_in)

        if n_steps > 0:
            copy_in(0)
        for j in range(n_steps):
            if j + 1 < n_steps:
                copy_in(j + 1)
            idx = (first + j) % n
            main.wait_event(ev_x[j])
            y = self.layers[idx].forward(self.x[idx])
            ev_y[j].record(main)
            with torch.cuda.stream(self.s_out):
                self.s_out.wait_event(ev_y[j])
                self.y_host[idx].copy_(y, non_blocking=True)
        main.wait_stream(self.s_in)
        main.wait_stream(self.s_out)


def max_over_ranks(secs: float, dist, world: int, device: str = "cuda") -> float:
    """The timed region's length for the whole job: the slowest rank's seconds (every rank
    gets the same value). One scalar all-reduce, outside any timed region."""
    if dist is None or world <= 1:
        return secs
    import torch
    t = torch.tensor([secs], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_step: int, steps: int, world: int, secs_max: float) -> float:
    """Whole-job tokens/s of N independent replicas (weak scaling): the tokens all ranks
    processed over the slowest rank's time."""
    return tokens_per_step * steps * world / secs_max


def timed_region(arm, K, W, torch, dist, world, sampler=None):
    """W warm-up steps, then exactly K steps from graph replays; returns (seconds over the
    timed region, max over ranks; the clock samples)."""
    n_sets = len(arm.layers)
    for i in range(W):
        arm.step(i)
    torch.cuda.synchronize()
    arm.check()
    # graphs of up to 64 steps (whole rotations of the weight sets when K allows): a short
    # timed region is then one or two graph launches, not one per rotation
    M = min(K, max(n_sets, (64 // n_sets) * n_sets))
    R, tail = divmod(K, M)
    NG = 3
    graphs = [arm.capture(M, 0) for _ in range(NG)]
    tail_g = arm.capture(tail, 0) if tail else None
    for g in graphs:       # graph upload
        g.replay()
    if tail_g is not None:
        tail_g.replay()
    torch.cuda.synchronize()
    arm.check()

    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    if sampler is not None:
        sampler.start()
        time.sleep(0.2)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # the device spins ~0.5 ms before the start event while the host enqueues the first graph
    # launches, so that the host's launch latency is not inside the device-timed region
    torch.cuda._sleep(1_000_000)
    start.record()
    for r in range(R):
        graphs[r % NG].replay()
    if tail_g is not None:
        tail_g.replay()
    end.record()
    torch.cuda.synchronize()
    clocks = sampler.stop() if sampler is not None else None
    if dist is not None:
        dist.barrier()
    secs = max_over_ranks(start.elapsed_time(end) / 1e3, dist, world)
    arm.check()
    return secs, clocks


def expert_launch_seconds(arm, n_steps, torch, dm):
    """Mean duration of the expert launch over n_steps steps: CUDA events recorded just
    before and after it on its stream (the library then makes it without programmatic
    overlap, so that they bracket its own execution). The steps are launched eagerly: inside
    a CUDA graph each event-record node adds ~6 us between the kernels it separates."""
    P = 64                                  # event pairs in flight
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(P)]
    for b, e in evs:                        # torch creates the CUDA event on its first record
        b.record()
        e.record()
    ms = []
    for i in range(n_steps + P):
        b, e = evs[i % P]
        if i >= P:                          # the pair's previous use has ended
            e.synchronize()
            ms.append(b.elapsed_time(e))
        if i < n_steps:
            dm.dmoe_set_profile_events("experts", b, e)
            arm.step(i)
    dm.dmoe_set_profile_events("experts", None, None)
    torch.cuda.synchronize()
    arm.check()
    return float(np.mean(ms[8:] if len(ms) > 16 else ms)) / 1e3


def traffic_from_profile(kernel: str, source: str):
    """dram bytes per launch from the committed ncu summary, if it was taken on the current
    source of the kernel (matching source hash); else None."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"{kernel}_layer_block.txt")
    src = os.path.join(ROOT, "paper_2605_30876_gb300", "csrc", source)
    try:
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        vals = {}
        for ln in open(path):
            if ":" in ln:
                k, v = ln.split(":", 1)
                v = v.split()
                vals[k.strip()] = v[0] if v else ""   # the value's first word
        if vals.get("source_sha256_16") != h:
            return None
        return float(vals["dram_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


def host_inputs(shape, seed: int):
    """Host copies of the workload's inputs (drawn on the GPU when there is one: the CPU
    generator needs minutes for the 1.6 GB of weights)."""
    import torch
    from dmoe_synth import layer_inputs, to_numpy
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    return to_numpy(layer_inputs(shape, seed=seed, device=dev))


def cpu_baseline(shape, budget_s: float, host):
    """The oracle as it stands, timed on the host cores on a bounded sample: full layer
    forwards of the same workload until `budget_s` is used (at least one)."""
    import oracle as O
    n, t0 = 0, time.perf_counter()
    while True:
        O.layer_forward(host, shape.top_k, shape.mode, shape.block_size, shape.top_p)
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            break
    return {"value": n * shape.T / el, "unit": UNIT, "cores": _CORES, "kind": "oracle",
            "sample": f"{n} full layer forward(s) of the benchmark workload ({n * shape.T} tokens)"
                      f" in {el:.1f} s; float64 NumPy, BLAS threads = {_CORES}"}


# ----------------------------------------------------------------------------- reference arm
def run_reference(args, shape, rank):
    """The CPU oracle as the reference implementation: K timed steps, each a bounded sample
    of the layer forward. The oracle evaluates a forward expert by expert (one SwiGLU over
    the rows routed to that expert, the shared expert over all tokens); a step runs the next
    m of those expert groups, and re-routes the block (router + Algorithm 1) each time the
    forward wraps around. m is sized so that the whole run takes minutes."""
    if rank != 0:
        return
    import oracle as O
    host = host_inputs(shape, args.seed)
    k, T = shape.top_k, shape.T
    rows_per_token = k + (1 if shape.d_ff_shared else 0)
    x64 = O.bf16_bits_to_f64(host["x"])

    def route():
        r = O.route(host["x"], host["w_r"], host["bias"], k, shape.mode, shape.block_size,
                    shape.top_p)
        groups = []
        for e in sorted(set(int(v) for v in r.idx.ravel())):
            tt, jj = np.nonzero(r.idx == e)
            groups.append((e, tt, r.gate[tt, jj]))
        if shape.d_ff_shared:
            groups.append((-1, np.arange(T), np.ones(T)))
        return groups

    def run_group(grp):
        e, tt, g = grp
        if e >= 0:
            wg, wu, wd = host["w_gate"][e], host["w_up"][e], host["w_down"][e]
        else:
            wg, wu, wd = host["ws_gate"], host["ws_up"], host["ws_down"]
        y = O.swiglu_ffn(x64[tt], O.bf16_bits_to_f64(wg), O.bf16_bits_to_f64(wu),
                         O.bf16_bits_to_f64(wd))
        return g[:, None] * y, len(tt)

    # calibration (untimed)
    t0 = time.perf_counter()
    groups = route()
    c_route = time.perf_counter() - t0
    t0 = time.perf_counter()
    run_group(groups[0])
    c_group = time.perf_counter() - t0
    budget = max(20.0, min(150.0, args.ref_budget)) / max(1, args.steps + args.warmup)
    m = int(max(1, min(len(groups), budget / max(c_group, 1e-6))))
    state = {"groups": groups, "pos": 0}

    def step():
        rows = 0
        for _ in range(m):
            if state["pos"] == len(state["groups"]):
                state["groups"] = route()
                state["pos"] = 0
            rows += run_group(state["groups"][state["pos"]])[1]
            state["pos"] += 1
        return rows

    for _ in range(args.warmup):
        step()
    rows = 0
    t0 = time.perf_counter()
    for _ in range(args.steps):
        rows += step()
    el = time.perf_counter() - t0
    value = rows / rows_per_token / el
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": workload_name(shape), "tokens_per_forward": T,
                   "l2": "n/a (CPU)"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": _CORES, "kind": "oracle",
                         "sample": f"each step: {m} of the {len(groups)} expert groups of one "
                                   f"forward (one fp64 SwiGLU over the rows routed to an "
                                   f"expert), plus the block's routing each time the forward "
                                   f"wraps (routing {c_route * 1e3:.1f} ms, "
                                   f"{c_group * 1e3:.1f} ms per group); tokens counted as "
                                   f"rows / (k + shared)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- suite
def graph_time(torch, calls, target_s: float = 0.25) -> float:
    """Device seconds per call of the `calls` (zero-argument functions), replayed from one
    CUDA graph that runs them once each in order, after warm-up, over about target_s."""
    for _ in range(2):
        for f in calls:
            f()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for f in calls:
            f()
    st, en = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g.replay()
    st.record()
    g.replay()
    en.record()
    torch.cuda.synchronize()
    reps = int(max(3, min(5000, target_s / max(st.elapsed_time(en) * 1e-3, 1e-7))))
    for _ in range(2):
        g.replay()
    st.record()
    for _ in range(reps):
        g.replay()
    en.record()
    torch.cuda.synchronize()
    return st.elapsed_time(en) * 1e-3 / reps / len(calls)


def run_suite(args, torch, dm, MoELayer, hbm: float, bf16_peak: float):
    """The other workloads, one JSON line per point: 8 sequences x 32 tokens (block p = 0,
    block p = 0.6, token routing), a sweep of the coreset threshold p with a line fitted to
    latency against unique experts, fewer experts per token inside the coreset and the Top-4
    token baseline, the block-size x batch x bias-scale grid (block p = 0 and
    token routing), and the 20-layer residual stack of 64 x 32 tokens (block p = 0 and token
    routing; each layer fed the RMS-normalised stream, u_l = bf16(x_l / rms(x_l)), and
    x_{l+1} = bf16(x_l + y_l), both by torch). The single-layer points rotate over --sets
    seeded copies of the layer's weights, as the headline does."""
    from dmoe_synth import (LAYER, LAYER_B8, ROUTE_BLOCK, ROUTE_TOKEN, STACK20, STACK20_LAYERS,
                            layer_inputs, router_bias, sweep_shapes)

    def emit(line):
        print(json.dumps(line), flush=True)

    def stats(shape, sec, U):
        lb = layer_bytes(shape, U)
        fl = layer_flops(shape)
        return {"us_per_forward": sec * 1e6, "tokens_per_s": shape.T / sec,
                "unique_experts_mean": U, "bytes_per_forward": lb,
                "achieved_gbs": lb / sec / 1e9, "hbm_roofline_frac": lb / sec / 1e9 / hbm,
                "flops_per_forward": fl, "tensor_frac": fl / sec / 1e12 / bf16_peak}

    def label(shape):
        base = "token" if shape.mode == ROUTE_TOKEN else f"block_p{shape.top_p:g}"
        if shape.top_k != LAYER.top_k:
            base += f"_k{shape.top_k}"
        if shape.mode == ROUTE_BLOCK and shape.block_top_k:
            base += f"_of{shape.block_top_k}"
        return base

    sets = [layer_inputs(LAYER, seed=args.seed + s, device="cuda") for s in range(args.sets)]

    def point(suite, shape):
        layers, xs = [], []
        for s, w0 in enumerate(sets):
            w = dict(w0)
            w["bias"] = torch.from_numpy(router_bias(shape.n_experts, shape.bias_scale,
                                                     args.seed + s)).to("cuda")
            layers.append(MoELayer.from_shape(shape, w))
            xs.append(layer_inputs(shape, seed=args.seed + s, device="cuda",
                                   with_weights=False)["x"])
        sec = graph_time(torch, [lambda L=L, x=x: L.forward(x) for L, x in zip(layers, xs)],
                         args.suite_time)
        for L in layers:
            st, info = dm.dmoe_get_device_error(L.ws)
            if st != 0:
                raise RuntimeError(f"device fault {info}")
        U = float(np.mean([int(L.n_unique.item()) for L in layers]))
        emit({"suite": suite, "workload": workload_name(shape), "routing": label(shape),
              "block_size": shape.block_size, "batch": shape.n_blocks,
              "bias_scale": shape.bias_scale, "T": shape.T, **stats(shape, sec, U)})
        return sec, U

    if args.suite_point:
        # one point only: "<block size>x<batch>:<block_p<p> | token>", e.g. 32x64:block_p0
        size, routing = args.suite_point.split(":")
        bsz, nb = (int(v) for v in size.split("x"))
        mode, p = ((ROUTE_TOKEN, 0.0) if routing == "token"
                   else (ROUTE_BLOCK, float(routing.replace("block_p", ""))))
        point("point", LAYER.with_(block_size=bsz, n_blocks=nb, mode=mode, top_p=p))
        return
    for mode, p in ((ROUTE_BLOCK, 0.0), (ROUTE_BLOCK, 0.6), (ROUTE_TOKEN, 0.0)):
        point("8x32", LAYER_B8.with_(mode=mode, top_p=p))
    # the coreset threshold as a performance axis: p over the paper's sweep values at block
    # size 32 and four batch sizes, with block top-k and token routing as the two ends; per
    # batch, a least-squares line of latency against the unique-expert count
    for nb in (1, 4, 16, 32):
        pts = []
        shapes = ([LAYER.with_(n_blocks=nb, top_p=p) for p in (0.0, 0.4, 0.5, 0.6, 0.7, 0.8)]
                  + [LAYER.with_(n_blocks=nb, mode=ROUTE_TOKEN)])
        for shape in shapes:
            pts.append(point("top_p_sweep", shape))
        sec_, U_ = np.array([q[0] for q in pts]) * 1e6, np.array([q[1] for q in pts])
        slope, icpt = np.polyfit(U_, sec_, 1)
        fit = slope * U_ + icpt
        r2 = 1.0 - float(np.sum((sec_ - fit) ** 2) / max(np.sum((sec_ - sec_.mean()) ** 2), 1e-30))
        emit({"suite": "top_p_sweep_fit", "batch": nb, "T": 32 * nb, "points": len(pts),
              "us_per_unique_expert": float(slope), "us_at_zero_experts": float(icpt),
              "r2": r2, "hbm_us_per_expert": LAYER.expert_bytes() / hbm / 1e3})
    # fewer experts per token inside the block's coreset (App. A) and the Top-4 token
    # baseline, at 1 and 8 sequences of 32 tokens
    for nb in (1, 8):
        for kw in (dict(top_k=4, block_top_k=8), dict(top_k=2, block_top_k=8),
                   dict(top_k=4, block_top_k=8, top_p=0.6), dict(top_k=4, mode=ROUTE_TOKEN)):
            point("fewer_experts", LAYER.with_(n_blocks=nb, **kw))
    for mode in (ROUTE_BLOCK, ROUTE_TOKEN):
        for shape in sweep_shapes(mode=mode):
            point("grid", shape)
    del sets
    torch.cuda.empty_cache()

    # the stack: separate seeded weights per layer, shared by the two routings
    weights = [layer_inputs(STACK20, seed=args.seed + 1000 + l, device="cuda", layer=l)
               for l in range(STACK20_LAYERS)]
    x0 = layer_inputs(STACK20, seed=args.seed + 999, device="cuda", with_weights=False)["x"]
    for mode in (ROUTE_BLOCK, ROUTE_TOKEN):
        shape = STACK20.with_(mode=mode, top_p=0.0)
        layers = [MoELayer.from_shape(shape, w) for w in weights]
        xs = [x0] + [torch.empty_like(x0) for _ in range(STACK20_LAYERS)]
        us = [torch.empty_like(x0) for _ in range(STACK20_LAYERS)]

        def step():
            for l, L in enumerate(layers):
                xf = xs[l].float()
                us[l].copy_(xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True)))
                y = L.forward(us[l])
                torch.add(xs[l], y, out=xs[l + 1])

        sec = graph_time(torch, [step]) / STACK20_LAYERS
        for L in layers:
            st, info = dm.dmoe_get_device_error(L.ws)
            if st != 0:
                raise RuntimeError(f"device fault {info}")
        per_layer = [int(L.n_unique.item()) for L in layers]
        U = float(np.mean(per_layer))
        line = {"suite": "stack20", "workload": workload_name(shape), "routing": label(shape),
                "layers": STACK20_LAYERS, "T": shape.T, "us_per_step": sec * STACK20_LAYERS * 1e6,
                "step_tokens_per_s": shape.T / (sec * STACK20_LAYERS), **stats(shape, sec, U),
                "unique_experts_per_layer": per_layer,
                "note": "per-layer figures include the torch RMS norm and residual add"}
        emit(line)
        del layers
    del weights


# ----------------------------------------------------------------------------- decode sim
def decode_sim(torch, dm, MoELayer, shape_base, n_layers, n_blocks, vocab, ctx, head_dim,
               seed, modes, on_step=None, conf_target=0.95):
    """A synthetic block-diffusion decoding loop around the MoE stack; returns one record per
    routing mode: step latencies, the MoE and attention shares of a step, and the
    unique-expert count U of every layer at every step (the statistic of the paper's Table 1
    is U's coefficient of variation across steps).

    Model stand-in (random weights; only the costs and the data flow are real): one
    sequence, a block of shape_base.block_size positions decoded at a time; per step every
    position of the block passes n_layers layers, each an attention stand-in (RMS norm,
    q/k/v/o projections, d / head_dim heads over a ctx-token cached context plus the block,
    by torch SDPA) and an MoE layer of shape_base's shape (this library; RMS-normalised input,
    residual add), then a tied embedding / LM head of `vocab` rows; the block's positions carry
    position embeddings. The stand-ins are plain torch, not tuned: their share is an upper
    bound of what a tuned attention would take. Unmasking: every masked position whose top
    softmax probability reaches conf_target takes its argmax token, at least the most
    confident one per step; the logit scale is fixed once so that about two of the masked
    positions of the first step pass. A block ends when all its positions are unmasked; the
    next block starts fully masked over the same context.

    Each step is one CUDA graph replay (its device time is the step latency); the MoE and
    attention shares come from graphs of the MoE layers alone and the attention stand-ins
    alone, replayed on the same step's inputs. `on_step(name, step, layers)` is called after
    every step's replay (the layers' routing outputs then hold that step's routing)."""
    from dmoe_synth import layer_inputs
    NL, B, V, CTX, HD = n_layers, shape_base.block_size, vocab, ctx, head_dim
    d = shape_base.d_model
    H = d // HD
    g = torch.Generator(device="cuda")
    g.manual_seed(seed + 77)

    def rnd(*shape, std=1.0):
        return (torch.randn(*shape, generator=g, device="cuda") * std).to(torch.bfloat16)

    w_head = rnd(V, d, std=0.02)              # tied embedding and LM head
    e_mask = rnd(d, std=0.02)
    pos = rnd(B, d, std=0.02)                 # position embeddings of the block
    # per layer: q|k|v projection [d, 3d], o projection [d, d]; K and V of the cached context
    # followed by the block's own rows (written in place every step)
    attn_w = [(rnd(d, 3 * d, std=d ** -0.5), rnd(d, d, std=d ** -0.5)) for _ in range(NL)]
    kv = [(rnd(1, H, CTX + B, HD), rnd(1, H, CTX + B, HD)) for _ in range(NL)]
    moe_w = [layer_inputs(shape_base, seed=seed + 2000 + l, device="cuda", layer=l)
             for l in range(NL)]
    x_in = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    xs = [torch.empty(B, d, dtype=torch.bfloat16, device="cuda") for _ in range(2 * NL + 1)]
    us = [torch.empty(B, d, dtype=torch.bfloat16, device="cuda") for _ in range(NL)]
    conf = torch.empty(B, dtype=torch.float32, device="cuda")
    arg = torch.empty(B, dtype=torch.int64, device="cuda")
    scale = torch.ones(1, dtype=torch.float32, device="cuda")

    def rms(x):
        return torch.nn.functional.rms_norm(x, (d,), eps=1e-6)

    def attn(l, x, out):
        wqkv, wo = attn_w[l]
        qkv = (rms(x) @ wqkv).view(B, 3, H, HD)
        k, v = kv[l]
        k[0, :, CTX:].copy_(qkv[:, 1].transpose(0, 1))
        v[0, :, CTX:].copy_(qkv[:, 2].transpose(0, 1))
        o = torch.nn.functional.scaled_dot_product_attention(qkv[:, 0].transpose(0, 1)[None], k, v)
        torch.add(x, o[0].transpose(0, 1).reshape(B, d) @ wo, out=out)

    def moe(l, L, x, out):
        us[l].copy_(rms(x))
        torch.add(x, L.forward(us[l]), out=out)

    def head(x):
        logits = (rms(x) @ w_head.t()).float() * scale
        p = torch.softmax(logits, dim=-1)
        c, a = p.max(dim=-1)
        conf.copy_(c)
        arg.copy_(a)

    def capture(fn):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr):
            fn()
        return gr

    def timed(gr, reps=3):
        st, en = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        best = None
        for _ in range(reps):
            st.record()
            gr.replay()
            en.record()
            torch.cuda.synchronize()
            t = st.elapsed_time(en) * 1e-3
            best = t if best is None else min(best, t)
        return best

    records = []
    for name, shape in modes:
        layers = [MoELayer.from_shape(shape, moe_w[l]) for l in range(NL)]

        def step_fn():
            x = x_in
            for l in range(NL):
                attn(l, x, xs[2 * l])
                moe(l, layers[l], xs[2 * l], xs[2 * l + 1])
                x = xs[2 * l + 1]
            head(x)

        def moe_fn():
            for l in range(NL):
                moe(l, layers[l], xs[2 * l], xs[2 * l + 1])

        def attn_fn():
            x = x_in
            for l in range(NL):
                attn(l, x, xs[2 * l])
                x = xs[2 * l + 1]

        tokens = torch.zeros(B, dtype=torch.int64, device="cuda")
        masked = torch.ones(B, dtype=torch.bool, device="cuda")

        def embed():
            x_in.copy_(torch.where(masked[:, None], e_mask[None, :], w_head[tokens]) + pos)

        embed()
        g_step, g_moe, g_attn = capture(step_fn), capture(moe_fn), capture(attn_fn)
        # logit scale: about two of the first step's masked positions reach conf_target
        g_step.replay()
        torch.cuda.synchronize()
        lo, hi = 1.0, 1e4
        for _ in range(40):
            mid = (lo * hi) ** 0.5
            scale.fill_(mid)
            head(xs[2 * NL - 1])
            n_pass = int((conf >= conf_target).sum().item())
            lo, hi = (mid, hi) if n_pass < 2 else (lo, mid)
        scale.fill_(hi)
        t_step, t_moe, t_attn, U, per_step = [], [], [], [], []
        blocks_done = 0
        while blocks_done < n_blocks:
            embed()
            t_step.append(timed(g_step, 1))
            U.append([int(L.n_unique.item()) for L in layers])
            if on_step is not None:
                on_step(name, len(t_step) - 1, layers)
            if len(t_step) % 4 == 1:      # component graphs on this step's inputs
                t_moe.append(timed(g_moe))
                t_attn.append(timed(g_attn))
                g_step.replay()           # the state the unmasking below reads
                torch.cuda.synchronize()
            c = torch.where(masked, conf, torch.full_like(conf, -1.0))
            take = masked & (c >= conf_target)
            if not bool(take.any()):
                take = torch.zeros_like(masked)
                take[int(c.argmax().item())] = True
            tokens = torch.where(take, arg, tokens)
            masked = masked & ~take
            per_step.append(int(take.sum().item()))
            if not bool(masked.any()):
                blocks_done += 1
                masked = torch.ones_like(masked)
        for L in layers:
            st_, info = dm.dmoe_get_device_error(L.ws)
            if st_ != 0:
                raise RuntimeError(f"device fault {info}")
        Ua = np.array(U, dtype=np.float64)
        records.append(dict(routing=name, U=Ua, t_step=np.array(t_step), t_moe=np.array(t_moe),
                            t_attn=np.array(t_attn), tokens_per_step=np.array(per_step)))
        del layers, g_step, g_moe, g_attn
        torch.cuda.empty_cache()
    return records


def unique_count_cv(U):
    """Coefficient of variation (sigma / mu over the steps, population sigma) of each layer's
    unique-expert count; U is [steps, layers]."""
    U = np.asarray(U, np.float64)
    return U.std(0) / np.maximum(U.mean(0), 1e-9)


def run_decode_sim(args, torch, dm, MoELayer):
    """The decoding-step harness at the benchmark shape (20 MoE layers of d=2048, 256
    experts, top-8, block of 32; 128k vocabulary, 1024-token context, heads of 128): one JSON
    line per routing (block top-k, block routing with p = 0.6, token routing)."""
    from dmoe_synth import LAYER, ROUTE_TOKEN, STACK20_LAYERS
    NL = STACK20_LAYERS
    modes = [("block_p0", LAYER), ("block_p0.6", LAYER.with_(top_p=0.6)),
             ("token", LAYER.with_(mode=ROUTE_TOKEN))]
    recs = decode_sim(torch, dm, MoELayer, LAYER, NL, args.sim_blocks, 128000, 1024, 128,
                      args.seed, modes)
    mid = NL // 2
    for r in recs:
        Ua = r["U"]
        cv = unique_count_cv(Ua)
        step_us = float(np.mean(r["t_step"])) * 1e6
        moe_us, attn_us = float(np.mean(r["t_moe"])) * 1e6, float(np.mean(r["t_attn"])) * 1e6
        print(json.dumps({
            "suite": "decode_sim", "routing": r["routing"], "layers": NL, "block_size": LAYER.block_size,
            "vocab": 128000, "context": 1024, "blocks": args.sim_blocks, "steps": len(r["t_step"]),
            "tokens_per_step_mean": float(np.mean(r["tokens_per_step"])),
            "step_us_mean": step_us, "moe_us": moe_us, "attention_us": attn_us,
            "other_us": max(step_us - moe_us - attn_us, 0.0), "moe_share": moe_us / step_us,
            "attention_share": attn_us / step_us,
            f"U_layer{mid}_mean": float(Ua[:, mid].mean()),
            f"U_layer{mid}_cv": float(cv[mid]),
            "U_mean_all_layers": float(Ua.mean()),
            "U_cv_per_layer_mean": float(np.mean(cv)),
            "note": "synthetic stand-ins for attention, embeddings and LM head; MoE by this "
                    "library; shares from graphs of each component replayed on the step's "
                    "inputs"}), flush=True)


# ----------------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=16)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--sets", type=int, default=8, help="weight sets rotated between steps")
    ap.add_argument("--seed", type=int, default=1000)
    ap.add_argument("--side-steps", type=int, default=4000,
                    help="steps of each side-by-side configuration (token routing, p=0.6)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--ref-budget", type=float, default=90.0)
    ap.add_argument("--only-headline", action="store_true",
                    help="skip the e2e and side-by-side arms (small profiling runs)")
    ap.add_argument("--suite", action="store_true",
                    help="measure the other workloads instead of the headline (one JSON line "
                         "per point; one GPU)")
    ap.add_argument("--suite-point", default=None,
                    help="with --suite: measure one point only, '<block size>x<batch>:<routing>' "
                         "with routing block_p<p> or token (e.g. 32x64:block_p0)")
    ap.add_argument("--suite-time", type=float, default=0.25,
                    help="with --suite: seconds of graph replays per point")
    ap.add_argument("--decode-sim", action="store_true",
                    help="the synthetic block-diffusion decoding loop around the MoE stack "
                         "(MoE share of a step, CV of U across steps; one GPU)")
    ap.add_argument("--sim-blocks", type=int, default=4)
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    shape = workload_shape("block", 0.0)

    if args.impl == "reference":
        run_reference(args, shape, rank)
        return

    import torch
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    import paper_2605_30876_gb300 as dm
    from dmoe_synth import layer_inputs
    from paper_2605_30876_gb300.layer import MoELayer

    peaks, peak_src = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    if args.suite:
        run_suite(args, torch, dm, MoELayer, hbm,
                  float(peaks.get("bf16_tflops_sustained", 1700.0)))
        return
    if args.decode_sim:
        run_decode_sim(args, torch, dm, MoELayer)
        return
    sampler = ClockSampler(gpu_uuid(torch)) if rank == 0 else None

    # headline: block routing, p = 0
    arm = Arm(shape, args.sets, args.seed + 97 * rank, torch, dm, MoELayer, layer_inputs)
    # the headline pass records no events; the expert kernel's launch duration is timed by
    # CUDA events in a second pass over the same steps, launched eagerly (while the events
    # are set, the library makes that launch without programmatic overlap, so that they
    # bracket its own execution rather than an early start spent waiting for the routing)
    secs, clocks = timed_region(arm, args.steps, args.warmup, torch, dist, world,
                                sampler=sampler)
    kern_s = expert_launch_seconds(arm, min(args.steps, 4000), torch, dm)
    U = arm.unique_counts()
    U_mean = float(np.mean(U))
    T = shape.T
    tokens_total = T * args.steps * world
    value = job_throughput(T, args.steps, world, secs)
    ms_per_step = secs / args.steps * 1e3

    # end to end: x from pinned host memory in, y back to pinned host memory, every step
    secs_e2e = None
    if not args.only_headline:
        arm.set_host_io(True)
        secs_e2e, _ = timed_region(arm, args.steps, args.warmup, torch, dist, world)
        arm.set_host_io(False)

    # side by side: token routing and the paper's p = 0.6
    side = {}
    side_cfgs = () if args.only_headline else (("token", workload_shape("token", 0.0)),
                                               ("block_p0.6", workload_shape("block", 0.6)))
    for name, sh in side_cfgs:
        a2 = Arm(sh, args.sets, args.seed + 97 * rank, torch, dm, MoELayer, layer_inputs)
        s2, _ = timed_region(a2, args.side_steps, args.warmup, torch, dist, world)
        k2 = expert_launch_seconds(a2, min(args.side_steps, 2000), torch, dm)
        u2 = float(np.mean(a2.unique_counts()))
        us = s2 / args.side_steps * 1e6
        side[name] = {"us_per_forward": us,
                      "tokens_per_s": job_throughput(T, args.side_steps, world, s2),
                      "unique_experts_mean": u2,
                      "hbm_roofline_frac": layer_bytes(sh, u2) / (us * 1e-6) / 1e9 / hbm,
                      "experts_us": k2 * 1e6 if k2 else None}
        del a2

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    lbytes = layer_bytes(shape, U_mean)
    gbytes = experts_bytes(shape, U_mean)
    achieved = gbytes / kern_s / 1e9 if kern_s else None
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": workload_name(shape), "tokens_per_forward": T,
                   "weight_sets_rotated": args.sets,
                   "l2": f"inputs larger than L2: {args.sets} rotated layer copies, "
                         f"~{lbytes / 1e6:.0f} MB of weights touched per step",
                   "graph_steps": args.sets, "parallelism": f"replicas{world}"},
        "us_per_forward": ms_per_step * 1e3,
        "unique_experts": {"per_set": U, "mean": U_mean},
        "layer_roofline": {"bytes_per_forward": lbytes,
                           "achieved_gbs": lbytes / (ms_per_step * 1e-3) / 1e9,
                           "frac_measured_hbm": lbytes / (ms_per_step * 1e-3) / 1e9 / hbm,
                           "frac_nominal_8tbs": lbytes / (ms_per_step * 1e-3) / 1e9 / NOMINAL_HBM_GBS,
                           "peak_source": peak_src},
        "roofline": {"kernel": "moe_decode_kernel", "bound": "hbm", "achieved": achieved,
                     "peak": hbm, "unit": "GB/s", "frac": (achieved / hbm) if achieved else None,
                     "traffic": traffic_from_profile("moe_decode", "expert_decode.cu"),
                     "algorithmic_bytes_per_launch": gbytes,
                     "launch_us": kern_s * 1e6 if kern_s else None,
                     "peak_source": f"{peak_src} hbm_gbs"},
        "side_by_side": side,
        "e2e": None if secs_e2e is None else {"value": job_throughput(T, args.steps, world, secs_e2e),
                "unit": UNIT,
                "h2d_bytes_per_step": T * shape.d_model * 2,
                "d2h_bytes_per_step": T * shape.d_model * 2},
        "gpu_launches": args.steps * dm.dmoe_layer_forward_launches(arm.layers[0].desc),
        "flops_per_forward": layer_flops(shape),
        "clocks": clocks,
    }
    if not args.no_cpu_baseline and world == 1:
        from dmoe_synth import to_numpy
        line["cpu_baseline"] = cpu_baseline(shape, args.cpu_budget, to_numpy(arm.inputs0))
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
