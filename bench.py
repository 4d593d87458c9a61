#!/usr/bin/env python3
"""Benchmark of ARC-KV per-context KV-cache compaction on GB300.

A step is one pass of the whole compaction path over one synthetic context:
every (layer, KV head) pair of a Llama-3.1-8B-shaped cache (32 layers x 8 KV
heads, head dim 128), compacted layer by layer through arckv_compact.  The
default context is the longest single-GPU workload: T = 131072 bf16 tokens,
n_q = 2048 reference queries per KV head and t = 13107 anchors (10%
retention), whose fits run in their n x n dual form.  The metric is context
tokens per second (T / seconds per context); seconds per context are
reported alongside.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gpu|reference]
                       [--workload NAME] [--split contexts|layers]
For N > 1 launch under torchrun.  With --split contexts (the default) every
rank compacts its own context (weak scaling); with --split layers the ranks
take contiguous blocks of one context's layers (strong scaling, no exchange:
each rank keeps its layers' compact cache).  Rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import ctypes
import datetime
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
if str(ROOT) not in sys.path:
    sys.path.insert(0, str(ROOT))

METRIC = "compaction s/context and context tokens/s at Llama-3.1-8B shape; % roofline"
UNIT = "context tokens/s"
DEFAULT_WORKLOAD = "llama8b_T131072_r10"
PROFILE_SUMMARY = ROOT / "profiles" / "assign_argmax_tc_llama8b_T131072.md"
DOMINANT_SOURCES = [ROOT / "paper_2609_36835_gb300" / "csrc" / f
                    for f in ("tc_assign.cu", "tc_gemm.cuh", "tc.cuh", "common.cuh")]
FALLBACK_BF16_SUSTAINED_TFLOPS = 1700.0


def measured_burst():
    """Burst bf16 peak (a kernel timed alone), else the sustained one."""
    try:
        return float(json.loads((ROOT / "MEASURED_PEAKS.json").read_text())["bf16_tflops"])
    except (OSError, ValueError, KeyError):
        return measured_peaks()[0]


def measured_peaks():
    """Measured GB300 peaks (MEASURED_PEAKS.json), else the fallback."""
    p = ROOT / "MEASURED_PEAKS.json"
    try:
        d = json.loads(p.read_text())
        return float(d["bf16_tflops_sustained"]), float(d["hbm_gbs"]), "measured"
    except (OSError, ValueError, KeyError):
        return FALLBACK_BF16_SUSTAINED_TFLOPS, 6800.0, "fallback"


def dominant_source_hash() -> str:
    h = hashlib.sha256()
    for f in DOMINANT_SOURCES:
        h.update(f.read_bytes())
    return h.hexdigest()


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0,
                    help="timed steps (default: 20, or 14 for contexts of 64K tokens and more, so that the "
                         "timed region stays near a minute)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("gpu", "reference"), default="gpu")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--e2e-steps", type=int, default=2)
    ap.add_argument("--streams", type=int, default=0,
                    help="CUDA streams (each with its own workspace) the layers of a context are spread over "
                         "(0: 3 for caches of 64K tokens and more, else 4)")
    ap.add_argument("--cpu-pairs", type=int, default=0,
                    help="(layer, head) pairs the oracle baseline times (0: about 12 s of oracle work, "
                         "at least one pair)")
    ap.add_argument("--split", choices=("contexts", "layers"), default="contexts",
                    help="N > 1: each rank compacts its own context (weak scaling) or a contiguous block of "
                         "one context's layers (strong scaling)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--selector", choices=("indexer", "ha", "vi"), default="indexer",
                    help="anchor scores: the ARC-KV indexer (default) or the HA / VI selectors of App. B.1")
    ap.add_argument("--chunk-len", type=int, default=0, help="App. A.3 chunked selection (0: global top-t)")
    ap.add_argument("--eval-selectors", action="store_true",
                    help="held-out truncated-output error E(S) of the three selectors on one layer (App. B.1)")
    ap.add_argument("--decode", action="store_true",
                    help="time one decode step of attention (App. D shape) instead of the compaction")
    ap.add_argument("--decode-contexts", default="4096,8192,16384,32768")
    ap.add_argument("--decode-iters", type=int, default=50)
    ap.add_argument("--profile-layer", action="store_true",
                    help="compact layer 0 twice and exit (a small case for ncu captures)")
    ap.add_argument("--layer-shape", default="",
                    help="with --profile-layer: T,n_pos,t overriding the workload's sizes (same distributions), "
                         "e.g. 16384,64,2048 for a small case of the dual-form fits (t > n)")
    args = ap.parse_args(argv)
    if args.steps <= 0:
        import synth
        w = synth.WORKLOADS.get(args.workload)
        args.steps = 14 if (w is not None and w.T >= 65536 and args.impl == "gpu") else 20
    return args


# ------------------------------------------------------------ distributed

class Dist:
    """Rank bookkeeping; a real process group only when WORLD_SIZE > 1."""

    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local_rank = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None

    def init(self, backend: str):
        if self.world > 1:
            import torch.distributed as dist
            os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
            dist.init_process_group(backend=backend)
            self.pg = dist

    def barrier(self):
        if self.pg is not None:
            self.pg.barrier()

    def max(self, x: float, device="cpu") -> float:
        if self.pg is None:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64, device=device)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg is not None:
            self.pg.destroy_process_group()


def context_layers(layers: int, rank: int, world: int = 1, split: str = "contexts"):
    """Layer seeds a rank compacts.  ``contexts``: one whole, distinct context
    of ``layers`` layers per rank (weak scaling).  ``layers``: the ranks share
    one context, rank r taking the contiguous block [r L / N, (r + 1) L / N)
    of its layers (strong scaling; no exchange, App. C.2 shards by layer)."""
    if split == "layers":
        return list(range(rank * layers // world, (rank + 1) * layers // world))
    return [rank * layers + l for l in range(layers)]


def default_cpu_pairs(T: int) -> int:
    """Pairs of the oracle baseline: about 12 s of oracle work on 16 cores
    (one pair takes ~1 s at T = 8192 and grows with T), at least one."""
    return max(1, (12 * 8192) // T)


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi clock / throttle sampling in the background (-lms 200).

    Each sample carries nvidia-smi's own query time, so ``stop(window)``
    keeps the samples taken inside the timed region (host wall-clock
    seconds), whatever buffering the pipe adds."""
    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.lines = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.th = threading.Thread(target=self._read, daemon=True)
        self.th.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    @staticmethod
    def _when(field: str):
        """nvidia-smi's 'YYYY/MM/DD HH:MM:SS.mmm' (local time) as epoch seconds, or None."""
        try:
            dt = datetime.datetime.strptime(field.strip(), "%Y/%m/%d %H:%M:%S.%f")
        except ValueError:
            return None
        return time.mktime(dt.timetuple()) + dt.microsecond / 1e6

    @classmethod
    def parse(cls, lines, window=None):
        """Summary of the sample lines: median SM clock, max clock, active
        throttle reasons.  With ``window`` = (t0, t1), host wall-clock seconds,
        only samples queried inside it count; if none were, all samples count
        and ``in_window`` says so."""
        rows = []
        for l in lines:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 10:
                continue
            try:
                sm, mx = float(f[2]), float(f[3])
            except ValueError:
                continue
            act = {nm for nm, v in zip(cls.REASONS, f[6:10]) if v.lower().startswith("active")}
            rows.append((cls._when(f[0]), sm, mx, act))
        if not rows:
            return None
        inside = rows
        if window is not None:
            t0, t1 = window
            inside = [r for r in rows if r[0] is not None and t0 <= r[0] <= t1]
        use = inside if inside else rows
        return {"sm_mhz": statistics.median(r[1] for r in use), "sm_max_mhz": max(r[2] for r in use),
                "reasons": sorted(set().union(*(r[3] for r in use))), "samples": len(use),
                "in_window": bool(inside) if window is not None else None, "samples_total": len(rows)}

    def stop(self, window=None):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.th.join(timeout=5)
        return self.parse(self.lines, window)


# ------------------------------------------------------------- helpers

def blas_threads() -> int:
    """Threads the oracle's BLAS uses (OpenBLAS query when available)."""
    try:
        maps = Path("/proc/self/maps").read_text()
        libs = sorted({l.split()[-1] for l in maps.splitlines() if "openblas" in l.lower() and ".so" in l})
        for path in libs:
            lib = ctypes.CDLL(path)
            for sym in ("scipy_openblas_get_num_threads64_", "openblas_get_num_threads64_",
                        "openblas_get_num_threads"):
                fn = getattr(lib, sym, None)
                if fn is not None:
                    fn.restype = ctypes.c_int
                    return int(fn())
    except OSError:
        pass
    return len(os.sched_getaffinity(0))


def cpu_sample_pairs(layers: int, heads: int, k: int):
    """k distinct (layer, KV head) pairs spread over the context: layers evenly
    spaced from the first to the last with heads stepping by 3, topped up in
    (layer, head) order where those repeat (deterministic)."""
    k = max(1, min(k, layers * heads))
    out = []
    for i in range(k):
        p = ((i * (layers - 1)) // max(1, k - 1), (3 * i) % heads)
        if p not in out:
            out.append(p)
    for l in range(layers):
        for h in range(heads):
            if len(out) < k and (l, h) not in out:
                out.append((l, h))
    return out


def oracle_pair_seconds(w, pairs, selector="indexer", chunk_len=0):
    """Time the fp64 oracle (as it stands) on (layer, head) pairs at full size."""
    import numpy as np
    import oracle
    import synth
    f64 = synth.bf16_to_f64
    times = []
    for (layer, head) in pairs:
        p = synth.make_pair(w, layer, head)
        X = synth.make_layer_activations(w, layer)
        W = {k: f64(v) for k, v in synth.make_indexer(w, layer, head).items()}
        K, V, Q = f64(p["K"]), f64(p["V"]), f64(p["Q"])
        Xr = np.repeat(f64(X), w.G, axis=0)
        t0 = time.perf_counter()
        oracle.compact_pair(K, V, Q, Xr, W, oracle.OracleConfig(t=w.t, selector=selector, chunk_len=chunk_len))
        times.append(time.perf_counter() - t0)
    return times


def gemm_rates(dev, reps: int = 5):
    """Library GEMM rates of this GPU in the precisions the peak file does not
    carry, timed like its bf16 figure (torch.matmul, best of `reps` after two
    warm-up calls, CUDA events): fp64, fp32 on the SIMT pipes (tf32 off) and
    tf32.  Measured outside every timed region; the denominators for the
    fp64-grade solvers and for SIMT work."""
    import torch
    out = {}
    prev = torch.backends.cuda.matmul.allow_tf32
    try:
        for name, dtype, size, tf32 in (("fp64", torch.float64, 4096, False), ("fp32_simt", torch.float32, 8192, False),
                                        ("tf32", torch.float32, 8192, True)):
            torch.backends.cuda.matmul.allow_tf32 = tf32
            g = torch.Generator(device=dev).manual_seed(7)
            a = torch.randn(size, size, device=dev, dtype=dtype, generator=g)
            b = torch.randn(size, size, device=dev, dtype=dtype, generator=g)
            best = float("inf")
            for i in range(reps + 2):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                torch.matmul(a, b)
                e1.record()
                e1.synchronize()
                if i >= 2:
                    best = min(best, e0.elapsed_time(e1) / 1e3)
            out[name] = 2.0 * size ** 3 / best / 1e12
            del a, b
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
    out["how"] = ("torch.matmul (cuBLAS), 4096^3 fp64, 8192^3 fp32 with tf32 off and on; best of %d after 2 "
                  "warm-up calls, CUDA events" % reps)
    return out


def profiled_traffic():
    """dram bytes per launch of the dominant kernel from the committed ncu
    summary, if it was taken on the current source of that kernel."""
    if not PROFILE_SUMMARY.exists():
        return None
    text = PROFILE_SUMMARY.read_text()
    m = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
    h = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    if not m or not h:
        return None
    return float(m.group(1)) if h.group(1) == dominant_source_hash() else None


# ------------------------------------------------------------ reference arm

def oracle_segments(w, pairs, selector="indexer", chunk_len=0):
    """The fp64 oracle (as it stands) on (layer, head) pairs, one bounded
    segment at a time: yields the seconds of each segment of
    oracle.compact_pair_steps (a stage, an index head, a block of keys) and
    marks the end of each pair with None.  Input generation is not timed."""
    import numpy as np
    import oracle
    import synth
    f64 = synth.bf16_to_f64
    for (layer, head) in pairs:
        p = synth.make_pair(w, layer, head)
        X = synth.make_layer_activations(w, layer)
        W = {k: f64(v) for k, v in synth.make_indexer(w, layer, head).items()}
        K, V, Q = f64(p["K"]), f64(p["V"]), f64(p["Q"])
        Xr = np.repeat(f64(X), w.G, axis=0)
        steps = oracle.compact_pair_steps(K, V, Q, Xr, W, oracle.OracleConfig(t=w.t, selector=selector,
                                                                                chunk_len=chunk_len))
        while True:
            t0 = time.perf_counter()
            try:
                next(steps)
            except StopIteration:
                yield time.perf_counter() - t0
                break
            yield time.perf_counter() - t0
        yield None


def run_reference(args, dist: Dist):
    """The reference arm: the fp64 oracle on the host cores.  A step is one
    bounded segment of the oracle's pipeline on one (layer, KV head) pair
    (oracle.compact_pair_steps); pairs are taken in a fixed spread over the
    context.  Seconds per context = the mean seconds of a complete pair x the
    pairs of the context; the pair in progress when the timed steps end is
    completed (untimed steps) so that every stage is counted."""
    if dist.rank != 0:
        return 0
    import synth
    w = synth.WORKLOADS[args.workload]
    pairs = [(l, h) for l in range(w.layers) for h in range(w.H_kv)]
    pick = [pairs[(i * 37) % len(pairs)] for i in range(len(pairs))]
    seg = oracle_segments(w, pick, args.selector, args.chunk_len)
    step_s, pair_s, cur = [], [], 0.0

    def advance():
        nonlocal cur
        while True:
            x = next(seg)
            if x is None:
                pair_s.append(cur)
                cur = 0.0
                continue
            cur += x
            return x

    for _ in range(args.warmup):
        advance()
    for _ in range(args.steps):
        step_s.append(advance())
    if not pair_s or cur > 0.0:
        while not pair_s or cur > 0.0:
            x = next(seg)
            if x is None:
                pair_s.append(cur)
                cur = 0.0
                if len(pair_s) >= 1:
                    break
            else:
                cur += x
    per_pair = statistics.mean(pair_s)
    s_ctx = per_pair * len(pairs)
    value = w.T / s_ctx
    cores = blas_threads()
    sample = ("fp64 oracle, %d complete (layer, KV head) pair(s) of %s at full size timed segment by segment "
              "(%.1f s per pair); seconds per context extrapolated x%d pairs; a step is one segment"
              % (len(pair_s), w.name, per_pair, len(pairs)))
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": (statistics.mean(step_s) * 1e3) if step_s else 0.0, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w, "none (CPU)"), "s_per_context": s_ctx,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def workload_config(w, l2: str):
    return {"workload": "%s: %d layers x %d KV heads (GQA %d), head_dim 128, T=%d bf16, n_q=%d per KV head, "
                        "t=%d (%.0f%% retention), H_I=8, d_I=d_A=128, d_x=%d" %
                        (w.name, w.layers, w.H_kv, w.G, w.T, w.n, w.t, 100.0 * w.t / w.T, w.shape.d_x),
            "layers": w.layers, "kv_heads": w.H_kv, "T": w.T, "n_q": w.n, "t": w.t, "head_dim": 128,
            "l2": l2}


# ------------------------------------------------------------------ GPU arm

def run_gpu(args, dist: Dist):
    import numpy as np
    import torch
    import synth
    import paper_2609_36835_gb300 as pk
    from paper_2609_36835_gb300 import workload

    dist.init("nccl")
    dev = torch.device("cuda", dist.local_rank)
    torch.cuda.set_device(dev)
    pk.load_library()
    w = synth.WORKLOADS[args.workload]
    layers = context_layers(w.layers, dist.rank, dist.world, args.split)
    if args.profile_layer:
        layers = layers[:1]
    sel = {"indexer": pk.SELECTOR_INDEXER, "ha": pk.SELECTOR_HA, "vi": pk.SELECTOR_VI}[args.selector]
    shape = {}
    if args.profile_layer and args.layer_shape:
        T_, np_, t_ = (int(x) for x in args.layer_shape.split(","))
        shape = dict(T=T_, n_pos=np_, t=t_)
    cfg = workload.layer_config(w, w.H_kv, flags=pk.FLAG_NONBLOCKING, selector=sel, chunk_len=args.chunk_len, **shape)
    cfg_block = workload.layer_config(w, w.H_kv, selector=sel, chunk_len=args.chunk_len, **shape)

    # seeded inputs drawn on the device (synth.make_layer_device: the recipe of
    # the host generator, seconds instead of minutes for a 128K context)
    dev_in = [synth.make_layer_device(w, l, list(range(w.H_kv)), dev, T=shape.get("T"), n_pos=shape.get("n_pos"))
              for l in layers]
    torch.cuda.synchronize()
    # layers are independent: they are spread round-robin over `n_str` streams,
    # each with its own workspace (arckv_compact is reentrant per workspace/stream)
    n_str = max(1, min(args.streams or (3 if w.T >= 65536 else 4), len(layers)))
    wss = [torch.empty(pk.workspace_bytes(cfg), dtype=torch.uint8, device=dev) for _ in range(n_str)]
    f32 = dict(dtype=torch.float32, device=dev)
    tp = pk.anchor_count(cfg)   # = w.t without chunking
    outs = [{"C_k": torch.empty(w.H_kv, tp, 128, **f32), "beta": torch.empty(w.H_kv, tp, **f32),
             "C_v": torch.empty(w.H_kv, tp, 128, **f32)} for _ in layers]
    stream = torch.cuda.current_stream(dev)
    streams = [stream] + [torch.cuda.Stream(dev) for _ in range(n_str - 1)]

    def compact(i, events=None, c=cfg, ins=None, out=None):
        t = ins if ins is not None else dev_in[i]
        o = out if out is not None else outs[i]
        ws, s_i = wss[i % n_str], streams[i % n_str]
        st, nl = pk.arckv_compact(c, t["K"], t["V"], t["Q"], t["X"], workload.indexer_dict(t), o["C_k"],
                                  o["beta"], o["C_v"], ws, ws.numel(), stream=s_i, stage_events=events)
        if st != 0:
            raise pk.ArckvError(st, "arckv_compact")
        return nl

    def fork():
        e = torch.cuda.Event()
        e.record(stream)
        for s_i in streams[1:]:
            s_i.wait_event(e)

    def join():
        for s_i in streams[1:]:
            e = torch.cuda.Event()
            e.record(s_i)
            stream.wait_event(e)

    def statuses():
        for ws, s_i in zip(wss, streams):
            code = pk.arckv_query_status(ws, s_i)
            if code != 0:
                raise pk.ArckvError(code, "timed region")

    if args.profile_layer:
        compact(0, c=cfg_block)
        compact(0, c=cfg_block)
        torch.cuda.synchronize()
        print("profile-layer done", flush=True)
        return 0

    # correctness of every layer once (blocking status read per call)
    for i in range(len(layers)):
        compact(i, c=cfg_block)

    def new_events(k, s_i=None):
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(k)]
        for e in evs:
            e.record(s_i if s_i is not None else stream)
        return evs

    def step(handles=None):
        n = 0
        fork()
        for i in range(len(layers)):
            n += compact(i, handles[i] if handles is not None else None)
        join()
        return n

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    n_ev = pk.NUM_STAGES + 1
    ev_sets = [[new_events(n_ev, streams[i % n_str]) for i in range(len(layers))] for _ in range(args.steps)]
    handles = [[[e.cuda_event for e in evs] for evs in st_] for st_ in ev_sets]
    t_start, t_end = new_events(2)
    launches = 0
    clocks = ClockSampler(dist.local_rank)
    clocks.start()
    time.sleep(0.3)
    dist.barrier()
    torch.cuda.synchronize()
    w0 = time.time()
    t_start.record(stream)
    for s in range(args.steps):
        launches += step(handles[s])
    t_end.record(stream)
    torch.cuda.synchronize()
    w1 = time.time()
    dist.barrier()
    clk = clocks.stop((w0, w1))
    ms_total = t_start.elapsed_time(t_end)
    ms_total = dist.max(ms_total, dev)
    ms_step = ms_total / args.steps
    # status of the timed calls: one blocking read per workspace
    statuses()

    # per-stage event spans of every layer call in the timed region (the stage
    # launches of one call, on the stream the call ran on)
    stage_ms = [0.0] * pk.NUM_STAGES
    stage_launch_ms = [[] for _ in range(pk.NUM_STAGES)]
    for s in range(args.steps):
        for evs in ev_sets[s]:
            for k in range(pk.NUM_STAGES):
                v = evs[k].elapsed_time(evs[k + 1])
                stage_ms[k] += v
                stage_launch_ms[k].append(v)
    stage_ms = [x / args.steps for x in stage_ms]

    # the same stages timed alone: layer 0 on one stream, blocking calls
    iso_ms = [[] for _ in range(pk.NUM_STAGES)]
    iso_ev = new_events(n_ev)
    iso_h = [e.cuda_event for e in iso_ev]
    for _ in range(5):
        st_, _ = pk.arckv_compact(cfg_block, dev_in[0]["K"], dev_in[0]["V"], dev_in[0]["Q"], dev_in[0]["X"],
                                  workload.indexer_dict(dev_in[0]), outs[0]["C_k"], outs[0]["beta"], outs[0]["C_v"],
                                  wss[0], wss[0].numel(), stream=stream, stage_events=iso_h)
        if st_ != 0:
            raise pk.ArckvError(st_, "isolated layer")
        for k in range(pk.NUM_STAGES):
            iso_ms[k].append(iso_ev[k].elapsed_time(iso_ev[k + 1]))

    # roofline of the dominant kernel: the assignment GEMM (Eq. anchor_assignment,
    # one launch per layer, stage 5), a split-bf16 tcgen05 GEMM issuing three
    # bf16 MMAs per useful product; 2 n (T - t) t useful flops per head (the
    # anchors' own assignment is fixed, kappa(s_r) = r: the launch scores the
    # T - t other keys against the t anchors)
    flops = 2.0 * w.H_kv * w.n * (w.T - tp) * tp
    avg_s = statistics.mean(stage_launch_ms[5]) / 1e3
    iso_s = statistics.median(iso_ms[5]) / 1e3
    peak, _, peak_src = measured_peaks()
    burst = measured_burst()
    achieved = flops / avg_s / 1e12
    roofline = {"kernel": "tc_gemm_kernel<256, kSplit, TcEpiArgmax8> (assignment, Eq. anchor_assignment)",
                "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                "traffic": profiled_traffic(), "flops_per_launch": flops, "launch_ms": avg_s * 1e3,
                "issued_tflops": 3.0 * achieved, "issued_frac": 3.0 * achieved / peak,
                "launch_ms_isolated": iso_s * 1e3, "frac_isolated": flops / iso_s / 1e12 / burst,
                "timing_note": "launch_ms: live CUDA events over the timed region, where %d streams share the GPU; "
                               "launch_ms_isolated: the same launch with the GPU to itself (median of 5), "
                               "frac_isolated against the burst peak" % n_str,
                "peak_note": "bf16 dense, sustained, of %s (MEASURED_PEAKS.json); achieved counts useful flops, "
                             "issued counts the 3 bf16 MMAs of each split-bf16 product" % peak_src}
    # the solvers of the two fits (stages 8 and 10), timed the same way
    dual = tp > w.n
    m_sys = w.n if dual else tp
    solve_flops = {8: w.H_kv * (m_sys ** 3 / 3.0 + 2.0 * m_sys ** 2),
                   10: w.H_kv * (m_sys ** 3 / 3.0 + 4.0 * m_sys ** 2 * 128)}
    rates = gemm_rates(dev)
    solver = {}
    for k, name in ((8, "beta_solve"), (10, "value_solve")):
        live = statistics.mean(stage_launch_ms[k]) / 1e3
        iso = statistics.median(iso_ms[k]) / 1e3
        solver[name] = {"flops": solve_flops[k], "ms_live": live * 1e3, "ms_isolated": iso * 1e3,
                        "tflops_isolated": solve_flops[k] / iso / 1e12,
                        "frac_isolated": solve_flops[k] / iso / 1e12 / burst,
                        "vs_fp64_gemm": solve_flops[k] / iso / 1e12 / rates["fp64"]}
    roofline["solvers"] = dict(solver, kernel=("blocked Cholesky of the n x n dual systems: fp64 64 x 64 "
                                               "diagonal factors, 5-slice tensor-core block products "
                                               "(sliced_gemm_kernel<5>); the 4-slice Grams and back-projection "
                                               "are counted outside" if dual else
                                               "chol_cluster_kernel<float, 4|8> (tcgen05 trailing updates) "
                                               "+ two refinement steps"),
                               note="Cholesky m^3 / 3 plus the triangular solves (m = %d, 1 and 128 right-hand "
                                    "sides), against the bf16 burst peak; vs_fp64_gemm against this GPU's own "
                                    "fp64 GEMM rate (gemm_rates)" % m_sys)
    roofline["gemm_rates"] = rates

    # end to end: pinned host inputs -> device -> compaction -> host outputs, every step
    pinned = [{k: v.to("cpu").pin_memory() for k, v in d.items()} for d in dev_in]
    host_out = [{k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True) for k, v in o.items()} for o in outs]
    h2d = sum(t.numel() * t.element_size() for p in pinned for t in p.values())
    d2h = sum(t.numel() * t.element_size() for o in host_out for t in o.values())

    h2d_stream, d2h_stream = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

    def e2e_step():
        # the host-to-device copies run ahead on their own stream (one event per
        # layer), each layer's compaction waits only for its own inputs, and its
        # outputs go back on a third stream as soon as it finishes; the step
        # ends when every stream has drained, so the next step's copies never
        # overwrite inputs still in use
        fork()
        start = torch.cuda.Event()
        start.record(stream)
        h2d_stream.wait_event(start)
        d2h_stream.wait_event(start)
        ready = []
        with torch.cuda.stream(h2d_stream):
            for i in range(len(layers)):
                for k, t in pinned[i].items():
                    dev_in[i][k].copy_(t, non_blocking=True)
                e = torch.cuda.Event()
                e.record(h2d_stream)
                ready.append(e)
        for i in range(len(layers)):
            s_i = streams[i % n_str]
            s_i.wait_event(ready[i])
            compact(i)
            done = torch.cuda.Event()
            done.record(s_i)
            d2h_stream.wait_event(done)
            with torch.cuda.stream(d2h_stream):
                for k, t in outs[i].items():
                    host_out[i][k].copy_(t, non_blocking=True)
        join()
        for side in (h2d_stream, d2h_stream):
            e = torch.cuda.Event()
            e.record(side)
            stream.wait_event(e)

    e2e_step()
    torch.cuda.synchronize()
    e0, e1 = new_events(2)
    dist.barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.e2e_steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = dist.max(e0.elapsed_time(e1), dev) / args.e2e_steps
    statuses()

    # contexts split over ranks: the whole job compacts one context per step
    ctx_per_step = 1 if args.split == "layers" else dist.world
    value = ctx_per_step * w.T / (ms_step / 1e3)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "strong" if args.split == "layers" else "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded Llama-3.1-8B-shaped caches)",
        "config": dict(workload_config(w, "inputs larger than L2 (%.2f GB per context)" % (h2d / 1e9)),
                       selector=args.selector, chunk_len=args.chunk_len, anchors_per_head=tp,
                       parallelism=("layer blocks of one context over %d ranks" % dist.world
                                    if args.split == "layers" else "one context per rank"),
                       inputs="seeded, drawn on the device (synth.make_layer_device)"),
        "s_per_context": ms_step / 1e3,
        "streams": n_str,
        "stage_ms_per_step": dict(zip(pk.STAGE_NAMES, stage_ms)),
        "stage_note": "per-layer event spans summed over layers; with several streams the spans overlap",
        "gpu_launches": launches,
        "roofline": roofline,
        "e2e": {"value": ctx_per_step * w.T / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "clocks": clk,
    }
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu_baseline:
        pairs = cpu_sample_pairs(w.layers, w.H_kv, args.cpu_pairs or default_cpu_pairs(w.T))
        times = oracle_pair_seconds(w, pairs, args.selector, args.chunk_len)
        per_pair = statistics.mean(times)
        n_pairs = w.layers * w.H_kv
        line["cpu_baseline"] = {
            "value": w.T / (per_pair * n_pairs), "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
            "sample": "fp64 oracle on %d (layer, KV head) pairs at full size (%.1f s each), seconds per "
                      "context extrapolated x%d pairs" % (len(times), per_pair, n_pairs)}
    if dist.rank == 0:
        print(json.dumps(line), flush=True)
    dist.close()
    return 0


def run_decode(args, dist: Dist):
    """One decode step of attention for a batch of 64 Llama-3.1-8B sequences
    (8 KV heads x 4 query heads, head dim 128) per layer: full bf16 cache
    (plain attention, t = 0) against a 20 % compact cache (bf16 C_k, C_v and
    the bias beta), both through arckv_attend_joint, plus the full-length
    bias-aware path (the whole cache passed as the compact block).  Inputs are
    larger than L2 at every context, so calls run back to back."""
    import torch
    import synth
    import paper_2609_36835_gb300 as pk

    if dist.rank != 0:
        return 0
    torch.cuda.set_device(0)
    pk.load_library()
    B, H_kv, G, d = 64, 8, 4, 128
    H = B * H_kv
    _, hbm_peak, peak_src = measured_peaks()
    flags = pk.FLAG_NONBLOCKING | pk.FLAG_COMPACT_BF16
    stream = torch.cuda.current_stream()

    def timed(fn):
        for _ in range(max(3, args.warmup)):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.decode_iters):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / args.decode_iters   # us per call

    rows = []
    clocks = ClockSampler(0)
    clocks.start()
    for T in [int(x) for x in args.decode_contexts.split(",")]:
        t = int(round(0.2 * T))
        x = synth.decode_batch_device(1000 + T, H, G, T, t, 0, "cuda", compact_bf16=True)
        O = torch.empty(H, G, d, dtype=torch.float32, device="cuda")
        def call(t_, F_, Ck, beta, Cv, Kf, Vf, fl):
            ws = torch.empty(pk.attend_joint_workspace_bytes(H, G, t_, F_), dtype=torch.uint8, device="cuda")
            def fn():
                st = pk.arckv_attend_joint(H, G, t_, F_, d, 0.0, x["Q"], Ck, beta, Cv, Kf, Vf, O, ws, ws.numel(),
                                           flags=fl, stream=stream)
                if st != 0:
                    raise pk.ArckvError(st, "arckv_attend_joint")
            return fn
        us_full = timed(call(0, T, None, None, None, x["K"], x["V"], pk.FLAG_NONBLOCKING))
        us_comp = timed(call(t, 0, x["C_k"], x["beta"], x["C_v"], None, None, flags))
        beta_full = torch.zeros(H, T, dtype=torch.float32, device="cuda")
        us_bias = timed(call(T, 0, x["K"], beta_full, x["V"], None, None, flags))
        io = H * G * d * (2 + 4)                     # Q in, O out
        b_full = H * T * d * 2 * 2 + io              # K and V, bf16
        b_comp = H * t * d * 2 * 2 + H * t * 4 + io  # C_k, C_v bf16 and beta fp32
        b_bias = H * T * d * 2 * 2 + H * T * 4 + io
        rows.append({"T": T, "t": t, "full_us": round(us_full, 2), "compact_us": round(us_comp, 2),
                     "full_bias_us": round(us_bias, 2), "speedup": round(us_full / us_comp, 3),
                     "bias_path_vs_full": round(us_bias / us_full, 3),
                     "kv_gb_full": round(b_full / 1e9, 3), "kv_gb_compact": round(b_comp / 1e9, 3),
                     "full_gbs": round(b_full / us_full / 1e3, 1), "compact_gbs": round(b_comp / us_comp / 1e3, 1),
                     "full_frac": round(b_full / us_full / 1e3 / hbm_peak, 3),
                     "compact_frac": round(b_comp / us_comp / 1e3 / hbm_peak, 3)})
        del x, beta_full
        torch.cuda.empty_cache()
    clk = clocks.stop()
    last = rows[-1]
    line = {
        "metric": "decode-step attention latency per layer, batch 64, Llama-3.1-8B GQA (8 KV x 4 q heads), "
                  "20% compact cache with beta vs full cache",
        "value": last["compact_us"], "unit": "us/layer", "higher_is_better": False, "n_gpus": 1,
        "steps": args.decode_iters, "warmup": max(3, args.warmup), "dtype": "bf16 cache, f32 accumulate",
        "data": "synthetic (seeded N(0,1) bf16 caches on the device)",
        "config": {"workload": "decode step: 64 sequences x 8 KV heads x 4 query rows, head_dim 128, t = 0.2 T",
                   "l2": "inputs larger than L2 at every context; calls back to back"},
        "contexts": rows,
        "roofline": {"kernel": "attend_bulk_kernel (split-key decode attention, bulk-copy K/V ring)", "bound": "hbm",
                     "achieved": last["compact_gbs"], "peak": hbm_peak, "unit": "GB/s",
                     "frac": last["compact_frac"], "traffic": None,
                     "peak_note": "HBM copy bandwidth, of %s (MEASURED_PEAKS.json)" % peak_src},
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    return 0


def run_eval_selectors(args, dist: Dist):
    """App. B.1 on synthetic caches: compact one layer with each selector, then
    the held-out truncated-output error E(S) of each anchor set (64 held-out
    queries per head, drawn like the reference queries)."""
    import numpy as np
    import torch
    import synth
    import paper_2609_36835_gb300 as pk
    from paper_2609_36835_gb300 import workload

    if dist.rank != 0:
        return 0
    torch.cuda.set_device(0)
    pk.load_library()
    w = synth.WORKLOADS[args.workload]
    rows = {}
    for layer in (0, w.layers // 2, w.layers - 1):
        heads = list(range(w.H_kv))
        arr = workload.layer_inputs_np(w, layer, heads)
        ten = workload.to_device(arr, "cuda")
        Qh = np.stack([synth.make_heldout(w, layer, h, arr["K"][i], 64) for i, h in enumerate(heads)])
        Qt = workload.bf16_tensor(Qh, "cuda")
        for name, sel in (("indexer", pk.SELECTOR_INDEXER), ("ha", pk.SELECTOR_HA), ("vi", pk.SELECTOR_VI)):
            cfg = workload.layer_config(w, w.H_kv, selector=sel)
            out = pk.compact_layer(cfg, ten["K"], ten["V"], ten["Q"], ten["X"], workload.indexer_dict(ten))
            E = pk.truncated_error(Qt, ten["K"], ten["V"], out["anchors"]).cpu().numpy()
            rows.setdefault(name, []).extend(float(x) for x in E)
    mean = {k: float(np.mean(v)) for k, v in rows.items()}
    line = {"metric": "held-out truncated-output error E(S), App. B.1 (lower is better)", "unit": "relative error",
            "higher_is_better": False, "config": {"workload": args.workload, "layers": [0, w.layers // 2, w.layers - 1],
                                                  "heads": w.H_kv, "t": w.t, "held_out_queries": 64},
            "data": "synthetic (seeded Llama-3.1-8B-shaped caches)",
            "E_mean": mean, "E_per_pair": rows,
            "vi_vs_ha_relative_reduction": (mean["ha"] - mean["vi"]) / mean["ha"]}
    print(json.dumps(line), flush=True)
    return 0


def main(argv=None):
    args = parse_args(argv)
    if args.warmup < 3 and not args.profile_layer:
        sys.stderr.write("note: fewer than 3 warm-up steps\n")
    dist = Dist()
    if args.impl == "reference":
        return run_reference(args, dist)
    if args.decode:
        return run_decode(args, dist)
    if args.eval_selectors:
        return run_eval_selectors(args, dist)
    return run_gpu(args, dist)


if __name__ == "__main__":
    sys.exit(main())
