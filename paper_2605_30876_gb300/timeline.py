"""Debug timeline of the decode-size layer forward (a measurement aid, not part of the method).

    python -m paper_2605_30876_gb300.timeline [block | p06 | token]

builds a second copy of the library with -DDMOE_TRACE (in `_build_trace/` beside this file;
the kernels then stamp %globaltimer / clock64 at fixed points) and runs, in a child process
that loads that copy, CUDA-graph replays of eight back-to-back forwards of the benchmark
layer (d=2048, E=256, k=8, I=512, shared 512, one block of 32 tokens; block top-k, block
routing with p = 0.6, or token routing) over eight seeded weight sets. It prints, for the
last replay:
  * every launch's first entry / last exit (after its dependency wait) from the routing
    launch's first entry, averaged over forwards 2..8, and the forward spacing;
  * the routing launch's stages in its continuing cluster (clock64, median over its CTAs);
  * the expert launch's stamps (unit list known, first stage landed, ... exit) over its CTAs.
The stamps cost about 1 us per forward; the release library's timing is `bench.py`'s.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

PKG = os.path.dirname(os.path.abspath(__file__))
TRACE_DIR = os.path.join(PKG, "_build_trace")
TRACE_LIB = os.path.join(TRACE_DIR, "libdmoe_trace.so")

# routing-launch stages (the order they are reached in the continuing cluster)
ROUTER_STAGES = [(1, "W_r / x slices landed"), (2, "partial logits"), (3, "logits reduced"),
                 (4, "ticket"), (10, "softmax"), (11, "token top-k"),
                 (5, "TopKMask rows in place"), (25, "block coreset known"),
                 (26, "coreset at the scoring warps"), (27, "restricted top-k"),
                 (13, "MaskOutside + gates"), (6, "Algorithm 1 done"), (7, "dispatch done")]
# expert-launch stamps (slot: meaning)
EXPERT_SLOTS = [(0, "entry"), (1, "unit list known"), (2, "first gate/up stage landed"),
                (3, "gate/up MMAs committed"), (4, "gate/up tile published"),
                (5, "down weights issued"), (6, "H of the group seen"),
                (12, "first down stage landed"), (13, "last down stage landed"),
                (7, "down MMAs committed"), (8, "down rows stored"), (9, "exit")]


def build_trace_lib() -> str:
    import importlib.util
    spec = importlib.util.spec_from_file_location("_dmoe_build", os.path.join(PKG, "_build.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod.build(extra_flags=["-DDMOE_TRACE"], build_dir=TRACE_DIR, lib_path=TRACE_LIB)


def _run(mode: str) -> None:
    import torch

    import paper_2605_30876_gb300 as dm
    from dmoe_synth import LAYER, layer_inputs
    from paper_2605_30876_gb300.layer import MoELayer

    if os.path.abspath(dm.LIB_PATH) != os.path.abspath(TRACE_LIB):
        raise RuntimeError("the timeline needs the -DDMOE_TRACE library (DMOE_LIB)")
    lib = dm._lib
    shape = {"block": LAYER, "p06": LAYER.with_(top_p=0.6),
             "token": LAYER.with_(mode=0)}[mode]
    NS = 8
    layers, xs = [], []
    for s in range(NS):
        inp = layer_inputs(shape, seed=1000 + s, device="cuda")
        layers.append(MoELayer.from_shape(shape, inp))
        xs.append(inp["x"])
    for i in range(2 * NS):
        layers[i % NS].forward(xs[i % NS])
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for i in range(NS):
            layers[i].forward(xs[i])
    for _ in range(20):
        g.replay()
    torch.cuda.synchronize()

    rec = np.dtype([("tag", "<u4"), ("cta", "<u4"), ("t", "<u8")])
    readers = {"routing": lib.dmoe_debug_klog_router, "experts": lib.dmoe_debug_klog_decode,
               "combine": lib.dmoe_debug_klog_experts}
    for f in readers.values():
        f.argtypes = [ctypes.c_void_p, ctypes.c_uint]
        f.restype = ctypes.c_int
        f(None, 0)
    lib.dmoe_debug_ctrace_clear()
    g.replay()
    torch.cuda.synchronize()
    launches = {}
    for (name, f), kid in zip(readers.items(), (0, 3, 4)):
        buf = np.zeros(32768, dtype=rec)
        n = f(buf.ctypes.data, 32768)
        log = buf[:n]
        ent = np.sort(log["t"][log["tag"] == 2 * kid].astype(np.int64))
        ext = np.sort(log["t"][log["tag"] == 2 * kid + 1].astype(np.int64))
        pe, px = len(ent) // NS, len(ext) // NS
        launches[name] = [(ent[i * pe:(i + 1) * pe], ext[i * px:(i + 1) * px]) for i in range(NS)]
    r0 = [launches["routing"][i][0].min() for i in range(NS)]
    print(f"workload: {mode}, unique experts per set: {[int(L.n_unique.item()) for L in layers]}")
    print("forward spacing (us):", np.round(np.diff(r0) / 1e3, 2).tolist())
    print("launch      CTAs  first entry  last entry  first exit  last exit   (us from the "
          "routing launch's first entry, mean of forwards 2..8)")
    for name, ls in launches.items():
        v = np.array([[(e.min() - r0[i]), (e.max() - r0[i]), (x.min() - r0[i]), (x.max() - r0[i])]
                      for i, (e, x) in enumerate(ls) if i > 0]) / 1e3
        m = v.mean(0)
        print(f"{name:10s} {len(ls[0][0]):5d} {m[0]:12.2f} {m[1]:11.2f} {m[2]:11.2f} {m[3]:10.2f}")

    ct = np.zeros(64 * 8 * 64, dtype=np.uint64)
    lib.dmoe_debug_ctrace.argtypes = [ctypes.c_void_p]
    lib.dmoe_debug_ctrace(ct.ctypes.data)
    ct = ct.reshape(512, 64).astype(np.int64)[:64]
    clk = ct[:, 32:64]
    # the continuing cluster of the last forward: its stamps after the ticket are fresh
    # (clock64 is per SM, so only differences within one CTA and forward are used)
    last = [c for c in range(64) if 0 < clk[c, 4] - clk[c, 3] < 40000]
    mhz = float(os.environ.get("DMOE_TIMELINE_SM_MHZ", "2070"))
    print(f"routing launch, continuing cluster CTAs {last} (clock64 at {mhz:.0f} MHz, "
          "median over its CTAs, from each CTA's entry):")
    for st, label in ROUTER_STAGES:
        v = [(clk[c, st] - clk[c, 0]) / mhz for c in last if 0 < clk[c, st] - clk[c, 0] < 60000]
        if v:
            print(f"  {label:30s} {np.median(v):7.2f} us")
    dt = np.zeros(320 * 32, dtype=np.uint64)
    lib.dmoe_debug_dtrace.argtypes = [ctypes.c_void_p]
    lib.dmoe_debug_dtrace(dt.ctypes.data)
    nb = len(launches["experts"][0][0])
    dt = dt.reshape(320, 32).astype(np.int64)[:nb]
    print(f"expert launch ({nb} CTAs; globaltimer, us from the routing launch's first entry):")
    for slot, label in EXPERT_SLOTS:
        v = dt[:, slot]
        v = (v[v > r0[-1] - 50_000] - r0[-1]) / 1e3
        if len(v):
            print(f"  {label:30s} min {v.min():6.2f}  median {np.median(v):6.2f}  max {v.max():6.2f}")
    for L in layers:
        st, info = dm.dmoe_get_device_error(L.ws)
        if st != 0:
            raise RuntimeError(f"device fault {info}")


def main(argv=None) -> int:
    argv = list(sys.argv[1:] if argv is None else argv)
    mode = argv[0] if argv else "block"
    if mode not in ("block", "p06", "token"):
        raise SystemExit("usage: python -m paper_2605_30876_gb300.timeline [block | p06 | token]")
    if os.environ.get("DMOE_LIB"):
        _run(mode)
        return 0
    lib = build_trace_lib()
    env = dict(os.environ, DMOE_LIB=lib)
    return subprocess.call([sys.executable, "-m", "paper_2605_30876_gb300.timeline", mode],
                           env=env, cwd=os.path.dirname(PKG))


if __name__ == "__main__":
    sys.exit(main())
