#!/usr/bin/env python
"""Throughput benchmark of the group-sparse linear layer y = x (W (.) M)^T.

Workload: one LLaMA-2-7B-shaped decoder block (q/k/v/o 4096x4096, gate/up
11008x4096, down 4096x11008), bf16 weights ~ N(0, 0.02^2), 1x256 groups along
the input dimension, per-module keep ratios U[0.3, 0.7] rescaled so the block
keeps exactly 50 % of its 790,528 groups, decode batches of 1, 4 and 16 tokens.

One step = the seven projections at T = 1, 4 and 16 (three batched launches of
the decode kernel, 21 tokens through the block), on one of R rotated packed
copies so that the weights streamed per step never sit in L2.  Packing is a
one-time transform of frozen weights and is timed separately ("pack").  The
tensor-core prefill kernel is measured on the first block of the 7B stack at
T = 2048 with activation outliers ("prefill").

  python bench.py [--gpus N --steps K --warmup W] [--impl reference]

N > 1 runs under torch.distributed.run: each rank holds an independent replica
(the layer shards into independent problems, no collective on the data path).
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
import time
from pathlib import Path

import numpy as np

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

from paper_2609_33977_gb300 import workload as wl  # noqa: E402

METRIC = "group-sparse linear tokens/s; decode HBM GB/s and prefill TFLOP/s vs GB300 peak"
DECODE_T = (1, 4, 16)
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def load_peaks():
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        d = json.loads(p.read_text())
        return d, "measured"
    return dict(PEAKS_FALLBACK), "fallback"


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, interval_ms: int = 50):
        self.gpu = gpu_index
        self.interval = interval_ms
        self.proc = None
        self.path = Path(os.environ.get("TMPDIR", "/tmp")) / f"gs_clocks_{os.getpid()}.csv"

    def start(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 f"-lms={self.interval}"], stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        rows = []
        for line in self.path.read_text().splitlines():
            parts = [s.strip() for s in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        try:
            self.path.unlink()
        except OSError:
            pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max((float(r[3]) for r in rows if r[3].replace(".", "").isdigit()), default=None)}


# ----------------------------------------------------------------------------- multi-rank helpers
def max_over_ranks(x: float, dist=None, device=None) -> float:
    """The maximum of a per-rank float over all ranks (the job's wall time is the
    slowest rank's); identity without a process group."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank_step: float, steps: int, elapsed_max: float, world: int) -> float:
    """Throughput of the whole job: every rank processes the same units per step
    (independent replicas), divided by the slowest rank's time."""
    return world * units_per_rank_step * steps / elapsed_max


# ----------------------------------------------------------------------------- traffic record
def kernel_source_hash(name: str) -> str:
    return hashlib.sha256((ROOT / "paper_2609_33977_gb300" / "csrc" / name).read_bytes()).hexdigest()[:16]


def recorded_traffic(kernel: str, source: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if the kernel source is unchanged since."""
    p = ROOT / "profiles" / "traffic.json"
    if not p.exists():
        return None
    try:
        d = json.loads(p.read_text())
        e = d.get(kernel, {}).get(workload)
        if e and e.get("source_sha256_16") == kernel_source_hash(source):
            return e["dram_bytes_per_launch"]
    except Exception:
        return None
    return None


# ----------------------------------------------------------------------------- workload
def block_inputs():
    w = wl.workload(2)
    k = wl.keep_counts(w)
    layers = []
    for i, L in enumerate(w.layers):
        layers.append({"L": L, "k": int(k[i]), "W": wl.weight_bits(w, i), "B": wl.group_mask(w, i, int(k[i])),
                       "x": {T: wl.activation_bits(w, i, T) for T in DECODE_T}})
    return w, layers


def decode_bytes(layers, T):
    """Algorithmic bytes of one decode launch over the block: kept weights + the index
    metadata the kernel reads (16-bit window mask + 32-bit offset per chunk x 16-row
    window) + x + y."""
    b = 0
    for d in layers:
        L = d["L"]
        nw16 = (L.out + 15) // 16
        b += 512 * d["k"] + 6 * L.G * nw16 + 2 * T * L.inp + 2 * T * L.out
    return b


# ----------------------------------------------------------------------------- CPU oracle timing
def oracle_sample_rate(layers, seconds: float, rows_per_call: int = 256):
    """Times the fp64 oracle on bounded samples: one token through `rows_per_call`
    output rows of one projection per call, rotating over the projections, for
    about `seconds`.  Returns block tokens/s extrapolated by weight count."""
    from oracle import groupsparse_oracle as orc
    total_weights = sum(d["L"].out * d["L"].inp for d in layers)
    done_weights = 0
    t_used = 0.0
    calls = 0
    i = 0
    t_end = time.perf_counter() + seconds
    cpu0 = time.process_time()
    while time.perf_counter() < t_end or calls < len(layers):
        d = layers[i % len(layers)]
        L = d["L"]
        r0 = (calls * 977) % max(1, L.out - rows_per_call)
        rows = slice(r0, r0 + rows_per_call)
        x1 = d["x"][1]
        t0 = time.perf_counter()
        orc.linear(x1, d["W"][rows], d["B"][rows])
        t_used += time.perf_counter() - t0
        done_weights += rows_per_call * L.inp
        calls += 1
        i += 1
    sec_per_weight = t_used / done_weights
    tokens_per_s = 1.0 / (sec_per_weight * total_weights)
    cores = _cores_used(time.process_time() - cpu0, t_used)
    return {"value": tokens_per_s, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{calls} oracle calls, each 1 token x {rows_per_call} output rows of one projection "
                      f"(rotating over the 7), {t_used:.1f} s wall; block tokens/s extrapolated by "
                      f"weight count ({total_weights} weights per block); cores = process CPU time / wall "
                      f"time over the calls"}


def oracle_single_thread_rate(seconds: float):
    """The same bounded oracle sample in a child process whose BLAS and OpenMP
    pools are limited to one thread (the variables must be set before numpy
    loads, hence the child).  The child generates its own copy of the seeded
    block inputs and touches no GPU."""
    env = dict(os.environ)
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
        env[k] = "1"
    env.pop("RANK", None)
    env.pop("WORLD_SIZE", None)
    try:
        r = subprocess.run([sys.executable, str(Path(__file__).resolve()), "--oracle-single-thread", "--warmup", "3",
                            "--cpu-seconds", str(seconds)], env=env, capture_output=True, text=True, timeout=600)
        if r.returncode != 0:
            return {"error": r.stderr.strip().splitlines()[-1] if r.stderr.strip() else f"exit {r.returncode}"}
        d = json.loads(r.stdout.strip().splitlines()[-1])
        return {"value": d["value"], "unit": d["unit"], "cores": d["cores"], "sample": d["sample"]}
    except Exception as e:   # reported in the line, never hidden; the GPU figures stand without it
        return {"error": f"{type(e).__name__}: {e}"}


def _cores_used(cpu_seconds: float, wall_seconds: float) -> int:
    """Threads the oracle kept busy on average: process CPU time over wall time."""
    if wall_seconds <= 0:
        return 1
    return max(1, int(round(cpu_seconds / wall_seconds)))


# ----------------------------------------------------------------------------- reference arm
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    _, layers = block_inputs()
    from oracle import groupsparse_oracle as orc
    total_weights = sum(d["L"].out * d["L"].inp for d in layers)
    rows_per_step = 64

    def one(i):
        d = layers[i % len(layers)]
        L = d["L"]
        r0 = (i * 977) % max(1, L.out - rows_per_step)
        orc.linear(d["x"][1], d["W"][r0:r0 + rows_per_step], d["B"][r0:r0 + rows_per_step])
        return rows_per_step * L.inp

    for i in range(args.warmup):
        one(i)
    t0 = time.perf_counter()
    cpu0 = time.process_time()
    weights = 0
    for i in range(args.steps):
        weights += one(i)
    dt = time.perf_counter() - t0
    cores = _cores_used(time.process_time() - cpu0, dt)
    tokens_per_s = weights / total_weights / dt
    sample = (f"each step: the fp64 oracle on 1 token x {rows_per_step} output rows of one projection "
              f"(rotating over the 7); block tokens/s extrapolated by weight count; cores = process CPU time / "
              f"wall time")
    line = {"impl": "reference", "metric": METRIC, "value": tokens_per_s, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / max(1, args.steps),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": "llama2-7b-block decode T=1 (sampled rows)", "layers": 7},
            "cpu_baseline": {"value": tokens_per_s, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": tokens_per_s, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- our arm
def run_ours(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_33977_gb300 import groupsparse as gs

    peaks, peaks_src = load_peaks()
    t_gen = time.perf_counter()
    w, layers = block_inputs()
    log(f"[bench] inputs generated in {time.perf_counter() - t_gen:.1f}s")

    def dev_bits(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(dev)

    Wd = [dev_bits(d["W"]) for d in layers]
    Md = [torch.from_numpy(d["B"]).to(dev) for d in layers]

    # ---- pack (one-time transform), timed on its own
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    packs0 = [gs.pack(Wd[i], Md[i]) for i in range(len(layers))]
    torch.cuda.synchronize()
    pack_s = time.perf_counter() - t0
    kept = sum(p.kept for p in packs0)
    assert kept == w.budget, (kept, w.budget)
    pack_bytes = sum(512 * d["k"] * 2 + d["L"].groups + 6 * d["L"].G * ((d["L"].out + 15) // 16) + 4 * d["k"]
                     for d in layers)

    # ---- rotated copies so each step streams weights that are not L2-resident
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    kept_bytes = 512 * kept
    R = max(2, int(math.ceil(3 * l2 / kept_bytes)) + 1) if args.rotate <= 0 else args.rotate
    packs = [packs0] + [[gs.pack(Wd[i], Md[i]) for i in range(len(layers))] for _ in range(R - 1)]
    xs = {T: [dev_bits(d["x"][T]) for d in layers] for T in DECODE_T}
    ys = {T: [torch.empty((T, d["L"].out), dtype=torch.bfloat16, device=dev) for d in layers] for T in DECODE_T}

    stream = torch.cuda.Stream(device=dev)
    graphs = []
    with torch.cuda.stream(stream):
        for c in range(R):                       # warm-up launches outside capture
            for T in DECODE_T:
                gs.linear_batched_into(xs[T], packs[c], ys[T], stream=stream)
        stream.synchronize()
        for c in range(R):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for T in DECODE_T:
                    gs.linear_batched_into(xs[T], packs[c], ys[T], stream=stream)
            graphs.append(g)
    stream.synchronize()
    launches_per_step = len(DECODE_T)

    def barrier():
        if dist is not None:
            dist.barrier()

    # ---- warm-up, then exactly K timed steps
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            graphs[i % R].replay()
    stream.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    barrier()
    torch.cuda.synchronize(dev)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    n0 = gs.launch_count()
    with torch.cuda.stream(stream):
        ev0.record(stream)
        for i in range(args.steps):
            graphs[i % R].replay()
        ev1.record(stream)
    ev1.synchronize()
    torch.cuda.synchronize(dev)
    barrier()
    clock_rec = clocks.stop()
    # graph replays do not go through the library's launch counter: count the
    # kernels they contain (one decode launch per token batch per step)
    launches = args.steps * launches_per_step + (gs.launch_count() - n0)
    elapsed = max_over_ranks(ev0.elapsed_time(ev1) / 1e3, dist, dev)
    tokens_per_step = sum(DECODE_T)
    value = whole_job_rate(tokens_per_step, args.steps, elapsed, world)
    bytes_per_step = sum(decode_bytes(layers, T) for T in DECODE_T)
    achieved_gbs = bytes_per_step * args.steps / elapsed / 1e9

    # ---- per-T kernel timing (decode alone, one graph per T) for the breakdown
    per_T = {}
    with torch.cuda.stream(stream):
        for T in DECODE_T:
            gT = []
            for c in range(R):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    gs.linear_batched_into(xs[T], packs[c], ys[T], stream=stream)
                gT.append(g)
            n = max(50, min(2000, args.steps))
            for i in range(10):
                gT[i % R].replay()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for i in range(n):
                gT[i % R].replay()
            b.record(stream)
            b.synchronize()
            us = a.elapsed_time(b) * 1e3 / n
            per_T[str(T)] = {"us_per_launch": us, "GB/s": decode_bytes(layers, T) / us / 1e3,
                             "tokens/s": T / us * 1e6}

    # ---- end to end through the public API with host buffers
    # One pinned host buffer per direction holds a step's inputs (x of every
    # projection for T = 1, 4, 16, back to back) and its results.  The device
    # side alternates between two copies of each, so a step's copies overlap
    # the neighbouring steps' launches; events order every buffer's reuse.
    y_len = {T: sum(T * d["L"].out for d in layers) for T in DECODE_T}
    xh_all = torch.cat([torch.cat([xx.reshape(-1) for xx in xs[T]]) for T in DECODE_T]).cpu().pin_memory()
    yh_all = torch.empty(sum(y_len.values()), dtype=torch.bfloat16).pin_memory()
    xd_all = [torch.empty_like(xh_all, device=dev) for _ in range(2)]
    yd_all = [torch.empty_like(yh_all, device=dev) for _ in range(2)]

    def layer_views(buf, dim):
        out, off = {}, 0
        for T in DECODE_T:
            views = []
            for d in layers:
                n = T * getattr(d["L"], dim)
                views.append(buf[off:off + n].view(T, getattr(d["L"], dim)))
                off += n
            out[T] = views
        return out

    xv = [layer_views(xd_all[k], "inp") for k in range(2)]
    yv = [layer_views(yd_all[k], "out") for k in range(2)]
    h2d = xh_all.numel() * 2
    d2h = yh_all.numel() * 2
    e2e_steps = max(20, min(args.steps, 2000))
    h2d_stream = torch.cuda.Stream(device=dev)
    d2h_stream = torch.cuda.Stream(device=dev)
    x_ready = [torch.cuda.Event() for _ in range(2)]
    k_done = [torch.cuda.Event() for _ in range(2)]
    y_read = [torch.cuda.Event() for _ in range(2)]
    used = [False, False]

    def e2e_step(i):
        c, k = i % R, i % 2
        if used[k]:
            h2d_stream.wait_event(k_done[k])    # the launches two steps back have read this x buffer
        with torch.cuda.stream(h2d_stream):
            xd_all[k].copy_(xh_all, non_blocking=True)
            x_ready[k].record(h2d_stream)
        stream.wait_event(x_ready[k])
        if used[k]:
            stream.wait_event(y_read[k])        # the copy two steps back has read this y buffer
        with torch.cuda.stream(stream):
            for T in DECODE_T:
                gs.linear_batched_into(xv[k][T], packs[c], yv[k][T], stream=stream)
            k_done[k].record(stream)
        d2h_stream.wait_event(k_done[k])
        with torch.cuda.stream(d2h_stream):
            yh_all.copy_(yd_all[k], non_blocking=True)
            y_read[k].record(d2h_stream)
        used[k] = True

    for i in range(5):
        e2e_step(i)
    torch.cuda.synchronize(dev)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    h2d_stream.wait_event(a)
    for i in range(e2e_steps):
        e2e_step(i)
    stream.wait_event(y_read[(e2e_steps - 1) % 2])    # the last step's results are on the host
    b.record(stream)
    b.synchronize()
    torch.cuda.synchronize(dev)
    e2e_s = a.elapsed_time(b) / 1e3
    e2e_value = world * tokens_per_step * e2e_steps / e2e_s
    # results of the e2e path equal the device-resident path
    y_dev = torch.cat([torch.cat([yy.reshape(-1) for yy in ys[T]]) for T in DECODE_T])
    assert torch.equal(yh_all.to(dev), y_dev), "e2e result mismatch"

    # ---- dense bf16 torch matmul on the unpruned weights (reference point)
    dense = {}
    with torch.cuda.stream(stream):
        for T in DECODE_T:
            Wd_rot = [Wd] + [[wt.clone() for wt in Wd] for _ in range(1)]
            for i in range(5):
                for j, d in enumerate(layers):
                    torch.matmul(xs[T][j], Wd_rot[i % 2][j].t())
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            n = 50
            a.record(stream)
            for i in range(n):
                for j, d in enumerate(layers):
                    torch.matmul(xs[T][j], Wd_rot[i % 2][j].t())
            b.record(stream)
            b.synchronize()
            us = a.elapsed_time(b) * 1e3 / n
            dense[str(T)] = {"us_per_block": us, "tokens/s": T / us * 1e6}
            del Wd_rot
    torch.cuda.empty_cache()

    # ---- per-GPU characterisations (N = 1 only: at N > 1 every rank would repeat them
    # while all GPUs are held, and they are not part of the scaled metric)
    # tensor-core prefill on the first block of the 7B stack, T = 2048 (outliers)
    prefill = None
    prefill_sweep = None
    decode_sweep = None
    mask_export = None
    if not args.no_prefill and world == 1:
        prefill = measure_prefill(gs, torch, dev, stream, peaks)
        prefill_sweep = measure_prefill_sweep(gs, torch, dev, stream, peaks)
        decode_sweep = measure_decode_sweep(gs, torch, dev, stream, peaks)

    # selector export (the step that produces the masks), measured last
    if world == 1:
        try:
            mask_export = measure_select(gs, torch, dev, stream, peaks)
        except Exception as e:   # reported in the line, never hidden
            mask_export = {"error": f"{type(e).__name__}: {e}"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = oracle_sample_rate(layers, args.cpu_seconds)
        cpu["single_thread"] = oracle_single_thread_rate(args.cpu_seconds / 2)

    hbm_peak = float(peaks.get("hbm_gbs", PEAKS_FALLBACK["hbm_gbs"]))
    traffic = recorded_traffic("k_decode", "gs_decode.cu", "llama2-7b-block")
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * elapsed / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "llama2-7b-block decode: 7 projections x T=1,4,16 (21 tokens per step)",
                   "layers": 7, "kept_groups": kept, "total_groups": w.total_groups, "density": kept / w.total_groups,
                   "kept_weight_bytes": kept_bytes,
                   "l2": f"inputs larger than L2: {R} rotated packed copies ({R * kept_bytes / 1e6:.0f} MB) vs "
                         f"L2 {l2 / 1e6:.0f} MB", "parallelism": f"replicas x{world}", "graph": "one CUDA graph per step"},
        "roofline": {"kernel": "k_decode", "bound": "hbm", "achieved": achieved_gbs, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved_gbs / hbm_peak, "peak_source": f"{peaks_src} hbm_gbs",
                     "bytes_per_step": bytes_per_step, "traffic": traffic,
                     "frac_of_8TBs_nominal": achieved_gbs / 8000.0},
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "steps": e2e_steps, "how": "per step: one pinned host -> device copy of every x (T = 1, 4, 16), three "
                                         "gs_linear_batched calls through the Python binding (no graph), one device -> "
                                         "pinned host copy of every y; copies on their own streams, device buffers "
                                         "alternating between steps so copies overlap neighbouring launches"},
        "gpu_launches": launches,
        "clocks": clock_rec,
        "per_T": per_T,
        "dense_torch_bf16": dense,
        "pack": {"seconds": pack_s, "layers": 7, "GB/s_incl_alloc_and_sync": pack_bytes / pack_s / 1e9},
        "prefill": prefill,
        "prefill_sweep": prefill_sweep,
        "decode_sweep": decode_sweep,
        "mask_export": mask_export,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def _time_block(gs, torch, stream, xd, ps, ys, algo, n=10):
    """Seconds per pass over one block's 7 projections (CUDA events, after warm-up);
    one batched call per pass (T >= 33 takes the tensor-core prefill kernel)."""
    assert algo == gs.ALGO_PREFILL and xd[0].shape[0] >= 33
    with torch.cuda.stream(stream):
        for _ in range(3):
            gs.linear_batched_into(xd, ps, ys, stream=stream)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n):
            gs.linear_batched_into(xd, ps, ys, stream=stream)
        b.record(stream)
        b.synchronize()
    return a.elapsed_time(b) / 1e3 / n


def measure_prefill(gs, torch, dev, stream, peaks):
    w = wl.workload(3, blocks=1)
    k = wl.keep_counts(w)
    T = 2048
    # device-side draws of the same distributions (numpy draws of 7 full layers are slow)
    Wd = [wl.weight_device(w, i, device=dev) for i in range(7)]
    Bd = [torch.from_numpy(wl.group_mask(w, i, int(k[i]))).to(dev) for i in range(7)]
    xd = [wl.activation_device(w, i, T, device=dev) for i in range(7)]
    ps = [gs.pack(Wd[i], Bd[i]) for i in range(7)]
    ys = [torch.empty((T, L.out), dtype=torch.bfloat16, device=dev) for L in w.layers]
    kept = sum(p.kept for p in ps)
    flops = 2.0 * T * 256 * kept
    s_block = _time_block(gs, torch, stream, xd, ps, ys, gs.ALGO_PREFILL)
    n = 10
    with torch.cuda.stream(stream):
        # dense bf16 reference point on the unpruned weights
        for i in range(7):
            torch.matmul(xd[i], Wd[i].t())
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n):
            for i in range(7):
                torch.matmul(xd[i], Wd[i].t())
        b.record(stream)
        b.synchronize()
        s_dense = a.elapsed_time(b) / 1e3 / n
    tflops = flops / s_block / 1e12
    peak = float(peaks.get("bf16_tflops", PEAKS_FALLBACK["bf16_tflops"]))
    dense_flops = 2.0 * T * sum(L.out * L.inp for L in w.layers)
    assert gs.device_status() == gs.GS_OK
    out = {"workload": "llama2-7b block 0 (7 projections), T=2048, 1% outlier channels x20, layer-adaptive 50%",
           "kept_groups": kept, "kept_tflop_per_block": flops / 1e12, "ms_per_block": s_block * 1e3,
           "tokens/s": T / s_block, "TFLOP/s": tflops, "peak_TFLOP/s": peak, "frac": tflops / peak,
           "peak_source": "measured bf16_tflops (burst)",
           "dense_torch_ms_per_block": s_dense * 1e3,
           "dense_torch_TFLOP/s": dense_flops / s_dense / 1e12, "speedup_vs_dense": s_dense / s_block}
    del Wd, Bd, xd, ps, ys
    torch.cuda.empty_cache()
    return out


def measure_prefill_sweep(gs, torch, dev, stream, peaks):
    """Prefill kernel over the token counts of the 13B and Qwen stacks (first block
    of each).  The attainable rate at a token count is min(tensor peak, kept FLOPs
    over the time to stream the block's bytes at the measured HBM bandwidth)."""
    tpk = float(peaks.get("bf16_tflops", PEAKS_FALLBACK["bf16_tflops"]))
    bw = float(peaks.get("hbm_gbs", PEAKS_FALLBACK["hbm_gbs"])) * 1e9
    rows = []
    for cfg, d, Ts, name in ((4, 0.5, (128, 512, 2048), "llama2-13b block 0"),
                             (5, 0.5, (1024,), "qwen2.5-7b block 0, d=0.5")):
        w = wl.workload(cfg, d, blocks=1)
        k = wl.keep_counts(w)
        Wd = [wl.weight_device(w, i, device=dev) for i in range(7)]
        ps = [gs.pack(Wd[i], torch.from_numpy(wl.group_mask(w, i, int(k[i]))).to(dev)) for i in range(7)]
        del Wd
        kept = sum(p.kept for p in ps)
        for T in Ts:
            xd = [wl.activation_device(w, i, T, device=dev) for i in range(7)]
            ys = [torch.empty((T, L.out), dtype=torch.bfloat16, device=dev) for L in w.layers]
            s_block = _time_block(gs, torch, stream, xd, ps, ys, gs.ALGO_PREFILL)
            flops = 2.0 * T * 256 * kept
            nbytes = 512.0 * kept + sum(2.0 * T * (L.inp + L.out) for L in w.layers)
            attainable = min(tpk, flops / (nbytes / bw) / 1e12)
            tflops = flops / s_block / 1e12
            rows.append({"workload": f"{name}, T={T}", "T": T, "kept_groups": kept, "ms_per_block": s_block * 1e3,
                         "tokens/s": T / s_block, "TFLOP/s": tflops, "attainable_TFLOP/s": attainable,
                         "frac_of_attainable": tflops / attainable, "frac_of_tensor_peak": tflops / tpk})
            del xd, ys
        del ps
        torch.cuda.empty_cache()
    assert gs.device_status() == gs.GS_OK
    return rows


def measure_decode_sweep(gs, torch, dev, stream, peaks):
    """Decode kernel on the first block of the 13B stack (T = 1, 16), of the Qwen
    stack (d = 0.5, T = 1), and on block 25 of the 7B stack under the paper-shaped
    allocation (Q/K near 8 %, down above 53 %; T = 1): one batched launch per pass
    over the block's 7 projections, alternating between two packed copies (each
    larger than L2)."""
    bw = float(peaks.get("hbm_gbs", PEAKS_FALLBACK["hbm_gbs"]))
    rows = []
    for w, blk, Ts, name in ((wl.workload(4, 0.5, blocks=1), 0, (1, 16), "llama2-13b block 0"),
                             (wl.workload(5, 0.5, blocks=1), 0, (1,), "qwen2.5-7b block 0, d=0.5"),
                             (wl.workload(3, allocation="paper"), 25, (1,),
                              "llama2-7b block 25, paper-shaped allocation")):
        k = wl.keep_counts(w)
        ids = list(range(7 * blk, 7 * blk + 7))
        Wd = [wl.weight_device(w, i, device=dev) for i in ids]
        Md = [torch.from_numpy(wl.group_mask(w, i, int(k[i]))).to(dev) for i in ids]
        copies = [[gs.pack(Wd[j], Md[j]) for j in range(7)] for _ in range(2)]
        del Wd, Md
        kept = sum(p.kept for p in copies[0])
        layers = [w.layers[i] for i in ids]
        for T in Ts:
            xd = [wl.activation_device(w, i, T, device=dev) for i in ids]
            ys = [torch.empty((T, L.out), dtype=torch.bfloat16, device=dev) for L in layers]
            n = 50
            with torch.cuda.stream(stream):
                for i in range(4):
                    gs.linear_batched_into(xd, copies[i % 2], ys, stream=stream)
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record(stream)
                for i in range(n):
                    gs.linear_batched_into(xd, copies[i % 2], ys, stream=stream)
                b.record(stream)
                b.synchronize()
            s_pass = a.elapsed_time(b) / 1e3 / n
            nbytes = sum(512.0 * p.kept + 6.0 * (L.inp // 256) * ((L.out + 15) // 16) + 2.0 * T * (L.inp + L.out)
                         for p, L in zip(copies[0], layers))
            gbs = nbytes / s_pass / 1e9
            rows.append({"workload": f"{name}, T={T}", "T": T, "kept_groups": kept, "us_per_block": s_pass * 1e6,
                         "tokens/s": T / s_pass, "GB/s": gbs, "frac_of_measured_hbm": gbs / bw})
            del xd, ys
        del copies
        torch.cuda.empty_cache()
    assert gs.device_status() == gs.GS_OK
    return rows


def measure_select(gs, torch, dev, stream, peaks):
    """Selector export (gs_select_groups) over all selectors of the 13B stack (40
    blocks, 49,561,600 groups): float32 logits (198 MB) in, uint8 masks (50 MB) out,
    together larger than L2.  Algorithmic bytes: 4 read + 1 written per selector."""
    bw = float(peaks.get("hbm_gbs", PEAKS_FALLBACK["hbm_gbs"]))
    w = wl.workload(4, 0.5)
    n = w.total_groups
    lg = wl.selector_logits_device(n, 0.5, seed=1, device=dev)
    mask = torch.empty((n,), dtype=torch.uint8, device=dev)
    kept = torch.empty((1,), dtype=torch.int64, device=dev)
    reps = 50
    with torch.cuda.stream(stream):
        for _ in range(5):
            gs.select_groups(lg, mask, kept, stream=stream)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            gs.select_groups(lg, mask, kept, stream=stream)
        b.record(stream)
        b.synchronize()
    s_launch = a.elapsed_time(b) / 1e3 / reps
    k = int(kept.cpu()[0])
    del lg, mask, kept
    torch.cuda.empty_cache()
    gbs = 5.0 * n / s_launch / 1e9
    return {"workload": "selectors of the llama2-13b stack (40 blocks), logits ~ N(0, 1)", "kernel": "k_select",
            "selectors": n, "kept": k, "bytes_per_launch": 5 * n, "us_per_launch": s_launch * 1e6, "GB/s": gbs,
            "frac_of_measured_hbm": gbs / bw}


def run_mask_export(args):
    """The selector export measurement alone; prints one JSON line."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_33977_gb300 import groupsparse as gs
    peaks, _ = load_peaks()
    stream = torch.cuda.Stream()
    rec = measure_select(gs, torch, torch.device("cuda", 0), stream, peaks)
    assert gs.device_status() == gs.GS_OK
    print(json.dumps(rec), flush=True)
    return 0


def run_layer(args):
    """One synthetic layer (random mask of the given density), one kernel family,
    timed with CUDA events; prints one JSON line.  Used for sweeps and for the
    small cases that ncu captures."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_33977_gb300 import groupsparse as gs
    T = args.tokens
    dev = torch.device("cuda", 0)
    if args.layer == "llama2-7b-block":
        return run_block_layers(args, gs, torch, dev)
    out, inp = (int(v) for v in args.layer.lower().split("x"))
    g = torch.Generator(device=dev)
    g.manual_seed(1234)
    W = (torch.randn((out, inp), generator=g, device=dev) * 0.02).to(torch.bfloat16)
    B = (torch.rand((out, inp // 256), generator=g, device=dev) < args.density).to(torch.uint8)
    x = torch.randn((T, inp), generator=g, device=dev).to(torch.bfloat16)
    p = gs.pack(W, B)
    y = torch.empty((T, out), dtype=torch.bfloat16, device=dev)
    algo = {"auto": gs.ALGO_AUTO, "decode": gs.ALGO_DECODE, "prefill": gs.ALGO_PREFILL}[args.algo]
    for _ in range(args.warmup):
        gs.linear_into(x, p, y, algo=algo)
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        gs.linear_into(x, p, y, algo=algo)
    b.record()
    b.synchronize()
    s = a.elapsed_time(b) / 1e3 / args.steps
    kept = p.kept
    G, nw16 = inp // 256, (out + 15) // 16
    nbytes = 512 * kept + 6 * G * nw16 + 2 * T * inp + 2 * T * out
    flops = 2.0 * T * 256 * kept
    assert gs.device_status() == gs.GS_OK
    print(json.dumps({"layer": f"{out}x{inp}", "T": T, "density": args.density, "algo": args.algo, "kept": kept,
                      "us": s * 1e6, "GB/s": nbytes / s / 1e9, "TFLOP/s": flops / s / 1e12}), flush=True)
    return 0


def run_block_layers(args, gs, torch, dev):
    """The seven LLaMA-2-7B block projections (random masks of --density) in one
    batched call per step, timed with CUDA events over R rotated packed copies."""
    shapes = [(o, i) for (_, o, i) in wl.LLAMA2_7B_BLOCK]
    T = args.tokens
    g = torch.Generator(device=dev)
    g.manual_seed(1234)
    R = 4
    packs = []
    for _ in range(R):
        hs = []
        for (o, i) in shapes:
            W = (torch.randn((o, i), generator=g, device=dev) * 0.02).to(torch.bfloat16)
            B = (torch.rand((o, i // 256), generator=g, device=dev) < args.density).to(torch.uint8)
            hs.append(gs.pack(W, B))
        packs.append(hs)
    xs = [torch.randn((T, i), generator=g, device=dev).to(torch.bfloat16) for (o, i) in shapes]
    ys = [torch.empty((T, o), dtype=torch.bfloat16, device=dev) for (o, i) in shapes]
    for r in range(args.warmup):
        gs.linear_batched_into(xs, packs[r % R], ys)
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    for r in range(args.steps):
        gs.linear_batched_into(xs, packs[r % R], ys)
    b.record()
    b.synchronize()
    s = a.elapsed_time(b) / 1e3 / args.steps
    kept = sum(p.kept for p in packs[0])
    nbytes = 512 * kept + sum(16 * (i // 256) * ((o + 63) // 64) + 2 * T * (i + o) for (o, i) in shapes)
    assert gs.device_status() == gs.GS_OK
    print(json.dumps({"layer": "llama2-7b-block x7 batched", "T": T, "density": args.density, "kept": kept,
                      "us": s * 1e6, "GB/s": nbytes / s / 1e9}), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--rotate", type=int, default=0, help="rotated packed copies (0 = enough to exceed 3x L2)")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--oracle-single-thread", action="store_true",
                    help="internal: time the oracle sample only and print it (run with one BLAS thread)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-prefill", action="store_true")
    ap.add_argument("--layer", default=None, help="single-layer mode: OUTxIN (random mask of --density)")
    ap.add_argument("--tokens", type=int, default=16)
    ap.add_argument("--density", type=float, default=0.5)
    ap.add_argument("--algo", choices=["auto", "decode", "prefill"], default="auto")
    ap.add_argument("--mask-export", action="store_true",
                    help="time only the selector export kernel over the 13B stack's selectors")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.oracle_single_thread:
        _, layers = block_inputs()
        print(json.dumps(oracle_sample_rate(layers, args.cpu_seconds)), flush=True)
        return 0
    if args.impl == "reference":
        return run_reference(args)
    if args.layer:
        return run_layer(args)
    if args.mask_export:
        return run_mask_export(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
