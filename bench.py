#!/usr/bin/env python
"""Throughput benchmark of the group-sparse linear layer y = x (W (.) M)^T.

Headline workload: the full LLaMA-2-13B-shaped linear stack (40 blocks of
q/k/v/o 5120x5120, gate/up 13824x5120, down 5120x13824; 280 layers, bf16
weights ~ N(0, 0.02^2), 1x256 groups along the input dimension, per-layer keep
ratios U[0.2, 0.8] rescaled so the stack keeps exactly 50 % of its 49,561,600
groups: 12.69 GB of kept weights).  This is the largest configuration of the
five; it fits one GB300.

One step = one decode pass over the whole stack at T = 1 and one at T = 16
(17 tokens): per pass one gs_linear_batched call per block (the block's 7
projections share one launch), captured as one CUDA graph per step.  The
stack's kept weights (12.7 GB) are far larger than L2, so every pass streams
them from HBM.  tokens/s = tokens per step / step time, which is T / (sum of
the layer times) per pass.  Packing is a one-time transform of frozen weights
and is timed separately ("pack").

Extra keys (N = 1 only): per-T decode passes, the same passes with one call per
layer, the tensor-core prefill over the whole 13B stack at T = 128, 512 and
2048, the whole LLaMA-2-7B stack at T = 2048 with activation outliers, the
whole Qwen2.5-7B stack at densities 0.3 / 0.5 / 0.7 (decode T = 1, prefill
T = 1024), the single 1024x1024 layer at T = 8 (a graph over 256 rotated
packed copies), one LLaMA-2-7B block at T = 1, 4, 16, the selector export,
dense bf16 torch matmuls on unpruned weights as reference points, and the CPU
oracle on a bounded sample.

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
HEADLINE_CFG = 4            # the LLaMA-2-13B-shaped stack, 40 blocks
DECODE_T = (1, 16)          # decode token counts of the headline step
PREFILL_T = (128, 512, 2048)
BLOCK_T = (1, 4, 16)        # the single LLaMA-2-7B block (second configuration)
NOMINAL_HBM_GBS = 8000.0    # the ~8 TB/s nominal HBM3e bandwidth the target is stated against
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



# ----------------------------------------------------------------------------- algorithmic work
def layer_decode_bytes(L, k: int, T: int) -> int:
    """Bytes one decode pass moves for one layer: kept weights, the index metadata
    the kernel reads (16-bit window mask + 32-bit offset per chunk x 16-row window),
    x and y."""
    return 512 * int(k) + 6 * L.G * ((L.out + 15) // 16) + 2 * T * (L.inp + L.out)


def stack_decode_bytes(layers, ks, T: int) -> int:
    return sum(layer_decode_bytes(L, k, T) for L, k in zip(layers, ks))


def kept_flops(ks, T: int) -> float:
    """Kept FLOPs of a pass: 2 T 256 per kept group (pruned groups cost nothing)."""
    return 2.0 * T * 256 * float(sum(int(k) for k in ks))


# ----------------------------------------------------------------------------- packed stacks
class Stack:
    """Every layer of a workload packed on the device.  Weights are drawn on the
    device (torch Philox seeded from the workload's SeedSequence), masks on the host
    (numpy top-k of seeded scores, several layers at once in a thread pool); each
    dense weight is freed once packed."""

    def __init__(self, gs, torch, dev, w, pool, blocks_of: int = 7):
        self.w = w
        self.layers = list(w.layers)
        ks = wl.keep_counts(w)
        futs = [pool.submit(wl.group_mask, w, i, int(ks[i])) for i in range(len(self.layers))]
        self.packs = []
        pack_s = 0.0
        for i in range(len(self.layers)):
            W = wl.weight_device(w, i, device=dev)
            M = torch.from_numpy(futs[i].result()).to(dev)
            torch.cuda.synchronize(dev)
            t0 = time.perf_counter()
            self.packs.append(gs.pack(W, M))
            torch.cuda.synchronize(dev)
            pack_s += time.perf_counter() - t0
            del W, M
        self.kept = [p.kept for p in self.packs]
        assert sum(self.kept) == w.budget, (sum(self.kept), w.budget)
        assert self.kept == [int(k) for k in ks]
        self.pack_s = pack_s
        n = len(self.layers)
        self.blocks = [list(range(b, min(n, b + blocks_of))) for b in range(0, n, blocks_of)]
        torch.cuda.empty_cache()

    @property
    def kept_groups(self) -> int:
        return int(sum(self.kept))

    def pack_bytes(self) -> int:
        """HBM bytes of packing: kept W read + tiles written + mask + metadata + row indices."""
        return sum(1024 * k + L.groups + 6 * L.G * ((L.out + 15) // 16) + 4 * k for L, k in zip(self.layers, self.kept))

    def free(self):
        for p in self.packs:
            p.free()
        self.packs = []


def stack_inputs(torch, w, dev, T: int):
    xs = [wl.activation_device(w, i, T, device=dev) for i in range(len(w.layers))]
    ys = [torch.empty((T, L.out), dtype=torch.bfloat16, device=dev) for L in w.layers]
    return xs, ys


def stack_pass(gs, S, xs, ys, stream, per_layer: bool = False):
    """One pass over the stack: one batched call per block (or one call per layer)."""
    if per_layer:
        for i, p in enumerate(S.packs):
            gs.linear_into(xs[i], p, ys[i], stream=stream)
        return
    for blk in S.blocks:
        gs.linear_batched_into([xs[i] for i in blk], [S.packs[i] for i in blk], [ys[i] for i in blk], stream=stream)


def capture(torch, stream, fn):
    """A CUDA graph of fn() (launches on `stream`); fn runs once first, outside capture."""
    with torch.cuda.stream(stream):
        fn()
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    stream.synchronize()
    return g


def time_replays(torch, stream, graphs, reps: int, warm: int = 3) -> float:
    """Seconds per graph replay (CUDA events on `stream`, replays cycling over `graphs`)."""
    with torch.cuda.stream(stream):
        for i in range(warm):
            graphs[i % len(graphs)].replay()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(reps):
            graphs[i % len(graphs)].replay()
        b.record(stream)
        b.synchronize()
    return a.elapsed_time(b) / 1e3 / reps


def time_calls(torch, stream, fn, reps: int, warm: int = 1) -> float:
    """Seconds per fn() (launches on `stream`, no graph)."""
    with torch.cuda.stream(stream):
        for _ in range(warm):
            fn()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            fn()
        b.record(stream)
        b.synchronize()
    return a.elapsed_time(b) / 1e3 / reps


def dense_block_seconds(torch, w, dev, stream, T: int, reps: int = 10, block: int = 0) -> float:
    """Seconds per pass of dense bf16 torch.matmul over one block's unpruned weights
    (the reference point; a block's dense weights are larger than L2)."""
    ids = list(range(7 * block, 7 * block + 7))
    Wd = [wl.weight_device(w, i, device=dev) for i in ids]
    xd = [wl.activation_device(w, i, T, device=dev) for i in ids]

    def run():
        for W, x in zip(Wd, xd):
            torch.matmul(x, W.t())
    s = time_calls(torch, stream, run, reps, warm=2)
    del Wd, xd
    torch.cuda.empty_cache()
    return s


# ----------------------------------------------------------------------------- CPU oracle timing
def oracle_block_inputs(cfg: int = HEADLINE_CFG):
    """Host (numpy) copies of block 0 of a stack: the sample the CPU oracle is timed on."""
    w = wl.workload(cfg)
    ks = wl.keep_counts(w)
    layers = []
    for i in range(7):
        layers.append({"L": w.layers[i], "W": wl.weight_bits(w, i), "B": wl.group_mask(w, i, int(ks[i])),
                       "x1": wl.activation_bits(w, i, 1)})
    return w, layers


def oracle_sample_rate(w, layers, seconds: float, rows_per_call: int = 256):
    """Times the fp64 oracle on bounded samples: one token through `rows_per_call`
    output rows of one projection of block 0 per call, rotating over its 7
    projections, for about `seconds`.  Returns stack tokens/s extrapolated by
    weight count (every block has the same shapes)."""
    from oracle import groupsparse_oracle as orc
    total_weights = sum(L.out * L.inp for L in w.layers)
    done_weights = 0
    t_used = 0.0
    calls = 0
    t_end = time.perf_counter() + seconds
    cpu0 = time.process_time()
    while time.perf_counter() < t_end or calls < len(layers):
        d = layers[calls % len(layers)]
        L = d["L"]
        r0 = (calls * 977) % max(1, L.out - rows_per_call)
        rows = slice(r0, r0 + rows_per_call)
        t0 = time.perf_counter()
        orc.linear(d["x1"], d["W"][rows], d["B"][rows])
        t_used += time.perf_counter() - t0
        done_weights += rows_per_call * L.inp
        calls += 1
    tokens_per_s = done_weights / t_used / total_weights
    cores = _cores_used(time.process_time() - cpu0, t_used)
    return {"value": tokens_per_s, "unit": "tokens/s", "cores": cores, "host_cpus": os.cpu_count(),
            "kind": "oracle",
            "sample": f"{calls} oracle calls, each 1 token x {rows_per_call} output rows of one projection of "
                      f"block 0 (rotating over its 7), {t_used:.1f} s wall; stack tokens/s extrapolated by weight "
                      f"count ({total_weights} weights in the {len(w.layers)} layers); cores = process CPU time / "
                      f"wall time over the calls; host_cpus = os.cpu_count()"}


def oracle_single_thread_rate(seconds: float):
    """The same bounded oracle sample in a child process whose BLAS and OpenMP
    pools are limited to one thread (the variables must be set before numpy
    loads, hence the child).  The child generates its own copy of the seeded
    inputs and touches no GPU."""
    env = dict(os.environ)
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
        env[k] = "1"
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        env.pop(k, None)
    try:
        r = subprocess.run([sys.executable, str(Path(__file__).resolve()), "--oracle-single-thread", "--warmup", "3",
                            "--cpu-seconds", str(seconds)], env=env, capture_output=True, text=True, timeout=600)
        if r.returncode != 0:
            return {"error": r.stderr.strip().splitlines()[-1] if r.stderr.strip() else f"exit {r.returncode}"}
        d = json.loads(r.stdout.strip().splitlines()[-1])
        return {"value": d["value"], "unit": d["unit"], "cores": d["cores"],
                "sample": "the same sample in a child process with one BLAS / OpenMP thread"}
    except Exception as e:   # reported in the line, never hidden; the GPU figures stand without it
        return {"error": f"{type(e).__name__}: {e}"}


def _cores_used(cpu_seconds: float, wall_seconds: float) -> int:
    """Threads the oracle kept busy on average: process CPU time over wall time."""
    if wall_seconds <= 0:
        return 1
    return max(1, int(round(cpu_seconds / wall_seconds)))


# ----------------------------------------------------------------------------- reference arm
def run_reference(args):
    """The CPU oracle, as it stands, on the headline workload: each step times the
    fp64 oracle on one token through a bounded sample of output rows of block 0's
    projections, extrapolated to the stack by weight count."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w, layers = oracle_block_inputs()
    from oracle import groupsparse_oracle as orc
    total_weights = sum(L.out * L.inp for L in w.layers)
    rows_per_step = 64

    def one(i):
        d = layers[i % len(layers)]
        L = d["L"]
        r0 = (i * 977) % max(1, L.out - rows_per_step)
        orc.linear(d["x1"], d["W"][r0:r0 + rows_per_step], d["B"][r0:r0 + rows_per_step])
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
    sample = (f"each step: the fp64 oracle on 1 token x {rows_per_step} output rows of one projection of block 0 "
              f"(rotating over its 7); stack tokens/s extrapolated by weight count; cores = process CPU time / "
              f"wall time; host_cpus = os.cpu_count()")
    line = {"impl": "reference", "metric": METRIC, "value": tokens_per_s, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / max(1, args.steps),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{w.name} decode, T=1 (sampled rows of block 0)", "layers": len(w.layers)},
            "cpu_baseline": {"value": tokens_per_s, "unit": "tokens/s", "cores": cores, "host_cpus": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": tokens_per_s, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- our arm
def run_ours(args):
    import concurrent.futures as cf
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
    hbm_peak = float(peaks.get("hbm_gbs", PEAKS_FALLBACK["hbm_gbs"]))
    tpk = float(peaks.get("bf16_tflops", PEAKS_FALLBACK["bf16_tflops"]))
    tpk_sus = float(peaks.get("bf16_tflops_sustained", PEAKS_FALLBACK["bf16_tflops_sustained"]))
    pool = cf.ThreadPoolExecutor(max_workers=8)
    stream = torch.cuda.Stream(device=dev)

    # ---- the headline stack, packed once (one-time transform of frozen weights)
    t_gen = time.perf_counter()
    w4 = wl.workload(HEADLINE_CFG)
    S = Stack(gs, torch, dev, w4, pool)
    log(f"[bench] {w4.name}: {len(S.layers)} layers packed in {time.perf_counter() - t_gen:.1f}s "
        f"({S.kept_groups} kept groups)")
    xs = {}
    ys = {}
    for T in DECODE_T:
        xs[T], ys[T] = stack_inputs(torch, w4, dev, T)

    def step():
        for T in DECODE_T:
            stack_pass(gs, S, xs[T], ys[T], stream)

    g_step = capture(torch, stream, step)
    launches_per_step = len(DECODE_T) * len(S.blocks)

    def barrier():
        if dist is not None:
            dist.barrier()

    # ---- warm-up, then exactly K timed steps
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g_step.replay()
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
        for _ in range(args.steps):
            g_step.replay()
        ev1.record(stream)
    ev1.synchronize()
    torch.cuda.synchronize(dev)
    barrier()
    clock_rec = clocks.stop()
    # graph replays bypass the library's launch counter: count the kernels they hold
    launches = args.steps * launches_per_step + (gs.launch_count() - n0)
    elapsed = max_over_ranks(ev0.elapsed_time(ev1) / 1e3, dist, dev)
    tokens_per_step = sum(DECODE_T)
    value = whole_job_rate(tokens_per_step, args.steps, elapsed, world)
    bytes_per_step = sum(stack_decode_bytes(S.layers, S.kept, T) for T in DECODE_T)
    achieved_gbs = bytes_per_step * args.steps / elapsed / 1e9
    assert gs.device_status() == gs.GS_OK

    # ---- each decode pass alone, per-block batched calls and per-layer calls
    per_T = {}
    for T in DECODE_T:
        nb = stack_decode_bytes(S.layers, S.kept, T)
        s_b = time_replays(torch, stream, [capture(torch, stream, lambda: stack_pass(gs, S, xs[T], ys[T], stream))],
                           reps=20)
        s_l = time_replays(torch, stream, [capture(torch, stream,
                                                   lambda: stack_pass(gs, S, xs[T], ys[T], stream, per_layer=True))],
                           reps=20)
        per_T[str(T)] = {"ms_per_pass": s_b * 1e3, "tokens/s": T / s_b, "GB/s": nb / s_b / 1e9,
                         "frac_of_measured_hbm": nb / s_b / 1e9 / hbm_peak,
                         "frac_of_8TBs_nominal": nb / s_b / 1e9 / NOMINAL_HBM_GBS,
                         "launches_per_pass": len(S.blocks),
                         "per_layer_calls": {"ms_per_pass": s_l * 1e3, "GB/s": nb / s_l / 1e9,
                                             "launches_per_pass": len(S.layers)}}
    torch.cuda.empty_cache()

    # ---- end to end through the public API with host buffers (no graph); the
    # step graph (per-block batched calls, as the e2e path makes) writes the
    # device-resident results it is compared with
    with torch.cuda.stream(stream):
        g_step.replay()
    stream.synchronize()
    e2e = measure_e2e(gs, torch, dev, stream, S, xs, ys, tokens_per_step, world, args)

    # ---- per-GPU characterisations (N = 1 only: at N > 1 every rank would repeat them
    # while all GPUs are held, and they are not part of the scaled metric)
    extras = {}
    if world == 1 and not args.headline_only:
        dense = {}
        for T in DECODE_T:
            s = dense_block_seconds(torch, w4, dev, stream, T) * len(S.blocks)
            dense[str(T)] = {"ms_per_stack_pass": s * 1e3, "tokens/s": T / s,
                             "how": "dense bf16 torch.matmul on block 0's unpruned weights, x 40 blocks"}
        extras["dense_torch_bf16"] = dense
        del xs, ys
        torch.cuda.empty_cache()
        extras["prefill_stack"] = measure_prefill_stack(gs, torch, dev, stream, S, PREFILL_T, tpk, tpk_sus,
                                                        hbm_peak, dense_ref=True)
        extras["pack"] = {"workload": w4.name, "seconds": S.pack_s, "layers": len(S.layers),
                          "GB/s_incl_alloc_and_sync": S.pack_bytes() / S.pack_s / 1e9}
        S.free()
        del S
        torch.cuda.empty_cache()
        extras["stack_7b"] = measure_stack_7b(gs, torch, dev, stream, pool, tpk, tpk_sus, hbm_peak)
        extras["stack_qwen"] = measure_stack_qwen(gs, torch, dev, stream, pool, tpk, tpk_sus, hbm_peak)
        extras["single_layer"] = measure_single_layer(gs, torch, dev, stream, hbm_peak)
        extras["block_7b"] = measure_block_7b(gs, torch, dev, stream, pool, hbm_peak)
        extras["group_shapes"] = measure_group_shapes(gs, torch, dev, stream, pool, tpk, hbm_peak)
        extras["train_op"] = measure_train_op(gs, torch, dev, stream, tpk, hbm_peak)
        try:
            extras["mask_export"] = measure_select(gs, torch, dev, stream, peaks)
        except Exception as e:   # reported in the line, never hidden
            extras["mask_export"] = {"error": f"{type(e).__name__}: {e}"}
        assert gs.device_status() == gs.GS_OK

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        w_o, layers_o = oracle_block_inputs()
        cpu = oracle_sample_rate(w_o, layers_o, args.cpu_seconds)
        cpu["single_thread"] = oracle_single_thread_rate(args.cpu_seconds / 2)

    traffic = recorded_traffic("k_decode", "gs_decode.cu", "llama2-13b-block")
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * elapsed / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "gpu_launches": launches,
        "config": {"workload": f"{w4.name} decode: {len(w4.layers)} layers x T=1,16 (17 tokens per step)",
                   "layers": len(w4.layers), "kept_groups": w4.budget, "total_groups": w4.total_groups,
                   "density": w4.budget / w4.total_groups, "kept_weight_bytes": 512 * w4.budget,
                   "l2": f"inputs larger than L2: {512 * w4.budget / 1e9:.2f} GB of kept weights per pass",
                   "parallelism": f"replicas x{world}",
                   "graph": f"one CUDA graph per step: {launches_per_step} batched decode launches "
                            f"(one per block per T)"},
        "roofline": {"kernel": "k_decode", "bound": "hbm", "achieved": achieved_gbs, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved_gbs / hbm_peak, "peak_source": f"{peaks_src} hbm_gbs",
                     "bytes_per_step": bytes_per_step, "launches_per_step": launches_per_step,
                     "algorithmic_bytes_per_launch": bytes_per_step / launches_per_step, "traffic": traffic,
                     "traffic_source": "profiles/traffic.json: DRAM bytes of one block's launch (mean over T = 1, 16)",
                     "frac_of_8TBs_nominal": achieved_gbs / NOMINAL_HBM_GBS},
        "cpu_baseline": cpu,
        "e2e": e2e,
        "clocks": clock_rec,
        "per_T": per_T,
    }
    line.update(extras)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def measure_e2e(gs, torch, dev, stream, S, xs, ys, tokens_per_step, world, args):
    """The headline step through the public API (gs_linear_batched via the Python
    binding, no graph) with host buffers: every step copies all x of both passes
    from pinned host memory and all y back.  Two schedules: `value` overlaps a
    step's copies with the neighbouring steps' launches (copies on their own
    streams, device buffers alternating between steps); `serialised` runs copy,
    launches and copy back in order on one stream."""
    layers = S.layers
    xh = torch.cat([torch.cat([x.reshape(-1) for x in xs[T]]) for T in DECODE_T]).cpu().pin_memory()
    yh = torch.empty(sum(T * L.out for T in DECODE_T for L in layers), dtype=torch.bfloat16).pin_memory()
    xd = [torch.empty_like(xh, device=dev) for _ in range(2)]
    yd = [torch.empty_like(yh, device=dev) for _ in range(2)]

    def views(buf, dim):
        out, off = {}, 0
        for T in DECODE_T:
            v = []
            for L in layers:
                n = T * getattr(L, dim)
                v.append(buf[off:off + n].view(T, getattr(L, dim)))
                off += n
            out[T] = v
        return out

    xv = [views(xd[k], "inp") for k in range(2)]
    yv = [views(yd[k], "out") for k in range(2)]
    h2d = xh.numel() * 2
    d2h = yh.numel() * 2
    n_steps = max(10, min(args.steps, 200))
    h2d_stream = torch.cuda.Stream(device=dev)
    d2h_stream = torch.cuda.Stream(device=dev)
    x_ready = [torch.cuda.Event() for _ in range(2)]
    k_done = [torch.cuda.Event() for _ in range(2)]
    y_read = [torch.cuda.Event() for _ in range(2)]
    used = [False, False]

    def overlapped(i):
        k = i % 2
        if used[k]:
            h2d_stream.wait_event(k_done[k])   # the launches two steps back have read this x buffer
        with torch.cuda.stream(h2d_stream):
            xd[k].copy_(xh, non_blocking=True)
            x_ready[k].record(h2d_stream)
        stream.wait_event(x_ready[k])
        if used[k]:
            stream.wait_event(y_read[k])       # the copy two steps back has read this y buffer
        for T in DECODE_T:
            stack_pass(gs, S, xv[k][T], yv[k][T], stream)
        k_done[k].record(stream)
        d2h_stream.wait_event(k_done[k])
        with torch.cuda.stream(d2h_stream):
            yh.copy_(yd[k], non_blocking=True)
            y_read[k].record(d2h_stream)
        used[k] = True

    def serialised(i):
        with torch.cuda.stream(stream):
            xd[0].copy_(xh, non_blocking=True)
            for T in DECODE_T:
                stack_pass(gs, S, xv[0][T], yv[0][T], stream)
            yh.copy_(yd[0], non_blocking=True)

    out = {}
    for name, fn in (("overlapped", overlapped), ("serialised", serialised)):
        for i in range(3):
            fn(i)
        torch.cuda.synchronize(dev)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        h2d_stream.wait_event(a)
        for i in range(n_steps):
            fn(i)
        if name == "overlapped":
            stream.wait_event(y_read[(n_steps - 1) % 2])   # the last step's results are on the host
        b.record(stream)
        b.synchronize()
        torch.cuda.synchronize(dev)
        out[name] = world * tokens_per_step * n_steps / (a.elapsed_time(b) / 1e3)
        # the host copy of the results equals the device-resident path's results
        y_ref = torch.cat([torch.cat([y.reshape(-1) for y in ys[T]]) for T in DECODE_T])
        assert torch.equal(yh.to(dev), y_ref), f"e2e ({name}) result mismatch"
    return {"value": out["overlapped"], "unit": "tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": n_steps, "serialised": out["serialised"],
            "how": "per step: one pinned host -> device copy of every layer's x (T = 1 and 16), one "
                   "gs_linear_batched call per block and T through the Python binding (no graph), one device -> "
                   "pinned host copy of every y.  value: copies on their own streams, device buffers alternating "
                   "between steps; serialised: copy, launches, copy back in order on one stream"}


def measure_prefill_stack(gs, torch, dev, stream, S, Ts, tpk, tpk_sus, hbm_peak, dense_ref=False):
    """Tensor-core prefill over a whole packed stack: one batched call per block
    (7 layers per launch).  tokens/s = T / pass time; kept TFLOP/s against the
    measured dense bf16 peak (burst, and sustained: a pass is a long step); at
    small T the attainable rate is min(tensor peak, kept FLOPs / time to stream
    the pass's bytes at the measured HBM bandwidth)."""
    rows = []
    w = S.w
    for T in Ts:
        xs, ys = stack_inputs(torch, w, dev, T)
        reps = 3 if T >= 1024 else 5
        s = time_calls(torch, stream, lambda: stack_pass(gs, S, xs, ys, stream), reps, warm=1)
        flops = kept_flops(S.kept, T)
        nbytes = 512.0 * S.kept_groups + sum(2.0 * T * (L.inp + L.out) for L in S.layers)
        attainable = min(tpk, flops / (nbytes / (hbm_peak * 1e9)) / 1e12)
        tf = flops / s / 1e12
        row = {"workload": f"{w.name}, T={T}", "T": T, "kept_groups": S.kept_groups, "ms_per_pass": s * 1e3,
               "tokens/s": T / s, "kept_TFLOP/s": tf, "frac_of_burst_peak": tf / tpk,
               "frac_of_sustained_peak": tf / tpk_sus, "attainable_TFLOP/s": attainable,
               "frac_of_attainable": tf / attainable, "launches_per_pass": len(S.blocks)}
        del xs, ys
        torch.cuda.empty_cache()
        if dense_ref:
            sd = dense_block_seconds(torch, w, dev, stream, T, reps=3) * len(S.blocks)
            row["dense_torch_ms_per_pass"] = sd * 1e3
            row["speedup_vs_dense"] = sd / s
            row["dense_how"] = "dense bf16 torch.matmul on block 0's unpruned weights, x blocks"
        rows.append(row)
    assert gs.device_status() == gs.GS_OK
    return rows


def measure_stack_7b(gs, torch, dev, stream, pool, tpk, tpk_sus, hbm_peak):
    """The whole LLaMA-2-7B stack (32 blocks, 224 layers) at T = 2048 with 1 % of
    input channels scaled x20 (the third configuration)."""
    w = wl.workload(3)
    S = Stack(gs, torch, dev, w, pool)
    rows = measure_prefill_stack(gs, torch, dev, stream, S, (2048,), tpk, tpk_sus, hbm_peak, dense_ref=True)
    S.free()
    torch.cuda.empty_cache()
    return rows[0]


def measure_stack_qwen(gs, torch, dev, stream, pool, tpk, tpk_sus, hbm_peak):
    """The whole Qwen2.5-7B stack (28 blocks, 196 layers) at global densities 0.3,
    0.5 and 0.7: a decode pass at T = 1 (graph of one batched call per block) and a
    prefill pass at T = 1024 (the fifth configuration)."""
    out = []
    for d in (0.3, 0.5, 0.7):
        w = wl.workload(5, d)
        S = Stack(gs, torch, dev, w, pool)
        xs, ys = stack_inputs(torch, w, dev, 1)
        s = time_replays(torch, stream, [capture(torch, stream, lambda: stack_pass(gs, S, xs, ys, stream))], reps=30)
        nb = stack_decode_bytes(S.layers, S.kept, 1)
        row = {"workload": w.name, "density": d, "kept_groups": S.kept_groups,
               "decode_T1": {"ms_per_pass": s * 1e3, "tokens/s": 1 / s, "GB/s": nb / s / 1e9,
                             "frac_of_measured_hbm": nb / s / 1e9 / hbm_peak,
                             "frac_of_8TBs_nominal": nb / s / 1e9 / NOMINAL_HBM_GBS}}
        del xs, ys
        row["prefill_T1024"] = measure_prefill_stack(gs, torch, dev, stream, S, (1024,), tpk, tpk_sus, hbm_peak)[0]
        S.free()
        torch.cuda.empty_cache()
        out.append(row)
    return out


def measure_single_layer(gs, torch, dev, stream, hbm_peak, copies: int = 256):
    """The single 1024x1024 layer (first configuration: exactly half of its 4096
    groups kept, T = 8): one graph of `copies` calls, each on its own packed copy
    (256 MiB of kept weights in all, larger than L2)."""
    w = wl.workload(1)
    ks = wl.keep_counts(w)
    W = wl.weight_device(w, 0, device=dev)
    M = torch.from_numpy(wl.group_mask(w, 0, int(ks[0]))).to(dev)
    ps = [gs.pack(W, M) for _ in range(copies)]
    x = wl.activation_device(w, 0, 8, device=dev)
    ys = [torch.empty((8, 1024), dtype=torch.bfloat16, device=dev) for _ in range(copies)]

    def run():
        for p, y in zip(ps, ys):
            gs.linear_into(x, p, y, stream=stream)
    s = time_replays(torch, stream, [capture(torch, stream, run)], reps=20) / copies
    nb = layer_decode_bytes(w.layers[0], ks[0], 8)
    out = {"workload": "single 1024x1024 layer, 2048 of 4096 groups kept, T=8", "us_per_call": s * 1e6,
           "tokens/s": 8 / s, "GB/s": nb / s / 1e9, "frac_of_measured_hbm": nb / s / 1e9 / hbm_peak,
           "how": f"one CUDA graph of {copies} gs_linear calls, each on its own packed copy"}
    for p in ps:
        p.free()
    del ps, W, M
    torch.cuda.empty_cache()
    return out


def measure_block_7b(gs, torch, dev, stream, pool, hbm_peak, copies: int = 4):
    """One LLaMA-2-7B block (second configuration: per-module keep U[0.3, 0.7]
    rescaled to 50 %) at T = 1, 4 and 16: one batched call per T, graphs cycling
    over `copies` packed copies (together larger than L2)."""
    w = wl.workload(2)
    Ss = [Stack(gs, torch, dev, w, pool) for _ in range(copies)]
    rows = []
    for T in BLOCK_T:
        xs, ys = stack_inputs(torch, w, dev, T)
        gr = [capture(torch, stream, lambda S=S: stack_pass(gs, S, xs, ys, stream)) for S in Ss]
        s = time_replays(torch, stream, gr, reps=200)
        nb = stack_decode_bytes(Ss[0].layers, Ss[0].kept, T)
        rows.append({"T": T, "us_per_launch": s * 1e6, "tokens/s": T / s, "GB/s": nb / s / 1e9,
                     "frac_of_measured_hbm": nb / s / 1e9 / hbm_peak})
        del xs, ys, gr
    for S in Ss:
        S.free()
    torch.cuda.empty_cache()
    return {"workload": "llama2-7b block (7 projections), one batched launch per T", "per_T": rows}


def measure_group_shapes(gs, torch, dev, stream, pool, tpk, hbm_peak,
                         shapes=((1, 128), (16, 16), (32, 32), (64, 64), (128, 128))):
    """The other group shapes (1x128 and square g x g; Sec. 3.5 ablation, App. E) on the
    LLaMA-2-7B block's seven projections, each keeping the same fraction of its
    groups as under the second configuration's 1x256 allocation (50 % overall):
    prefill at T = 2048 (one batched call per pass, kept TFLOP/s against the
    measured bf16 peak) and decode at T = 1 and 16 (two packed copies
    alternating, together larger than L2), next to the 1x256 kernels."""
    w = wl.workload(2)
    ks = wl.keep_counts(w)
    n = len(w.layers)
    rows = []
    for go, gi in shapes:
        masks = [pool.submit(wl.group_mask_shaped, w, i, int(ks[i]), go, gi) for i in range(n)]
        copies = [[], []]
        for i in range(n):
            W = wl.weight_device(w, i, device=dev)
            M = torch.from_numpy(masks[i].result()).to(dev)
            for c in range(2):
                copies[c].append(gs.pack_groups(W, M, go, gi))
            del W, M
        kept_tiles = sum(p.kept for p in copies[0])
        kept_w = kept_tiles * go * gi
        row = {"group": f"{go}x{gi}", "kept_weights": kept_w,
               "kept_fraction": kept_w / sum(L.out * L.inp for L in w.layers)}
        for T in (1, 16, 2048):
            xs, ys = stack_inputs(torch, w, dev, T)

            def run(c, xs=xs, ys=ys):
                gs.linear_batched_into(xs, copies[c], ys, stream=stream)
            if T <= 16:
                gr = [capture(torch, stream, lambda c=c: run(c)) for c in range(2)]
                s = time_replays(torch, stream, gr, reps=100)
                meta = (lambda p, L: 6.0 * (L.inp // gi) * ((L.out + 15) // 16)) if go == 1 else \
                    (lambda p, L: 4.0 * p.kept)
                nb = 2.0 * kept_w + sum(meta(p, L) + 2.0 * T * (L.inp + L.out) for p, L in zip(copies[0], w.layers))
                row[f"decode_T{T}"] = {"us_per_block": s * 1e6, "GB/s": nb / s / 1e9,
                                       "frac_of_measured_hbm": nb / s / 1e9 / hbm_peak}
            else:
                s = time_calls(torch, stream, lambda: run(0), reps=10, warm=2)
                tf = 2.0 * T * kept_w / s / 1e12
                row[f"prefill_T{T}"] = {"ms_per_block": s * 1e3, "kept_TFLOP/s": tf, "frac_of_burst_peak": tf / tpk}
            del xs, ys
        for c in copies:
            for p in c:
                p.free()
        torch.cuda.empty_cache()
        rows.append(row)
    assert gs.device_status() == gs.GS_OK
    return {"workload": "llama2-7b block (7 projections), square groups at the 1x256 allocation's per-layer "
                        "fractions", "shapes": rows}


def measure_train_op(gs, torch, dev, stream, tpk, hbm_peak):
    """The training-side op (Sec. 2.2): one Gumbel-Sigmoid sample over all selectors
    of the 13B stack (logits + noise + ds/dl float32, mask uint8: 13 B per selector),
    and the straight-through backward of one 13B down projection (5120 x 13824,
    1x256 groups) at T = 2048 with and without the input gradient."""
    w = wl.workload(4, 0.5)
    n = w.total_groups
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    lg = torch.randn((n,), generator=g, device=dev)
    u = torch.rand((n,), generator=g, device=dev).clamp_(1e-7, 1 - 1e-7)
    noise = (torch.log(u) - torch.log1p(-u)).float()
    s = time_calls(torch, stream, lambda: gs.gumbel_select(lg, noise, 0.4, stream=stream), reps=20, warm=3)
    out = {"sample": {"selectors": n, "us_per_call": s * 1e6, "GB/s": 13.0 * n / s / 1e9,
                      "frac_of_measured_hbm": 13.0 * n / s / 1e9 / hbm_peak}}
    del lg, u, noise
    o, i, T = 5120, 13824, 2048
    W = (torch.randn((o, i), generator=g, device=dev) * 0.02).to(torch.bfloat16)
    lgl = torch.randn((o, i // 256), generator=g, device=dev)
    nz = torch.zeros_like(lgl)
    mask, dsdl, _ = gs.gumbel_select(lgl, nz, 0.4)
    p = gs.pack(W, mask)
    x = torch.randn((T, i), generator=g, device=dev).to(torch.bfloat16)
    dy = torch.randn((T, o), generator=g, device=dev).to(torch.bfloat16)
    for want_dx in (False, True):
        sb = time_calls(torch, stream, lambda: gs.masked_linear_backward(x, W, p, dy, dsdl, want_dx=want_dx,
                                                                          stream=stream), reps=5, warm=2)
        fl = 2.0 * T * o * i * (2 if want_dx else 1)
        out["backward_dx" if want_dx else "backward"] = {"layer": f"{o}x{i}", "T": T, "ms": sb * 1e3,
                                                         "dense_TFLOP/s": fl / sb / 1e12,
                                                         "frac_of_burst_peak": fl / sb / 1e12 / tpk}
    assert gs.device_status() == gs.GS_OK
    del W, x, dy, p
    torch.cuda.empty_cache()
    return out


def run_train_op(args):
    """The training-side op measurement alone; prints one JSON line."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_33977_gb300 import groupsparse as gs
    peaks, _ = load_peaks()
    dev = torch.device("cuda", 0)
    stream = torch.cuda.Stream(device=dev)
    print(json.dumps(measure_train_op(gs, torch, dev, stream, float(peaks.get("bf16_tflops", 1900.0)),
                                      float(peaks.get("hbm_gbs", 6800.0)))), flush=True)
    return 0


def run_group_shapes(args):
    """The group-shape measurement alone; prints one JSON line."""
    import concurrent.futures as cf
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_33977_gb300 import groupsparse as gs
    peaks, _ = load_peaks()
    dev = torch.device("cuda", 0)
    stream = torch.cuda.Stream(device=dev)
    pool = cf.ThreadPoolExecutor(max_workers=8)
    rec = measure_group_shapes(gs, torch, dev, stream, pool, float(peaks.get("bf16_tflops", 1900.0)),
                               float(peaks.get("hbm_gbs", 6800.0)))
    print(json.dumps(rec), flush=True)
    return 0


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
    s = time_calls(torch, stream, lambda: gs.select_groups(lg, mask, kept, stream=stream), reps=50, warm=5)
    k = int(kept.cpu()[0])
    del lg, mask, kept
    torch.cuda.empty_cache()
    gbs = 5.0 * n / s / 1e9
    return {"workload": "selectors of the llama2-13b stack (40 blocks), logits ~ N(0, 1)", "kernel": "k_select",
            "selectors": n, "kept": k, "bytes_per_launch": 5 * n, "us_per_launch": s * 1e6, "GB/s": gbs,
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


def run_block(args):
    """One block of a stack (--block-of 4: the 13B stack, 2: the 7B block, 3: the
    7B stack, 5: the Qwen stack at --density) at --tokens, one batched call per
    step, cycling over two packed copies; prints one JSON line.  Used for the
    small cases that ncu captures."""
    import concurrent.futures as cf
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_33977_gb300 import groupsparse as gs
    dev = torch.device("cuda", 0)
    w = wl.workload(args.block_of, args.density, blocks=1)
    pool = cf.ThreadPoolExecutor(max_workers=8)
    Ss = [Stack(gs, torch, dev, w, pool) for _ in range(2)]
    T = args.tokens
    xs, ys = stack_inputs(torch, w, dev, T)
    stream = torch.cuda.current_stream()
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            stack_pass(gs, Ss[i % 2], xs, ys, stream)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(args.steps):
            stack_pass(gs, Ss[i % 2], xs, ys, stream)
        b.record(stream)
        b.synchronize()
    s = a.elapsed_time(b) / 1e3 / args.steps
    nb = stack_decode_bytes(Ss[0].layers, Ss[0].kept, T)
    fl = kept_flops(Ss[0].kept, T)
    assert gs.device_status() == gs.GS_OK
    print(json.dumps({"workload": f"{w.name} block 0", "T": T, "kept": Ss[0].kept_groups, "us": s * 1e6,
                      "GB/s": nb / s / 1e9, "kept_TFLOP/s": fl / s / 1e12}), flush=True)
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
    out, inp = (int(v) for v in args.layer.lower().split("x"))
    g = torch.Generator(device=dev)
    g.manual_seed(1234)
    W = (torch.randn((out, inp), generator=g, device=dev) * 0.02).to(torch.bfloat16)
    gsz = args.group
    gin = args.group_in
    if gsz:
        B = (torch.rand((out // gsz, inp // gsz), generator=g, device=dev) < args.density).to(torch.uint8)
    else:
        B = (torch.rand((out, inp // gin), generator=g, device=dev) < args.density).to(torch.uint8)
    x = torch.randn((T, inp), generator=g, device=dev).to(torch.bfloat16)
    p = gs.pack_groups(W, B, gsz, gsz) if gsz else gs.pack_groups(W, B, 1, gin)
    y = torch.empty((T, out), dtype=torch.bfloat16, device=dev)
    algo = {"auto": gs.ALGO_AUTO, "decode": gs.ALGO_DECODE, "prefill": gs.ALGO_PREFILL,
            "prefill_dense": gs.ALGO_PREFILL_DENSE}[args.algo]
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
    if gsz:
        kept_w = kept * gsz * gsz
        nbytes = 2 * kept_w + 4 * kept + 2 * T * inp + 2 * T * out
    else:
        kept_w = gin * kept
        G, nw16 = inp // gin, (out + 15) // 16
        nbytes = 2 * kept_w + 6 * G * nw16 + 2 * T * inp + 2 * T * out
    flops = 2.0 * T * kept_w
    assert gs.device_status() == gs.GS_OK
    print(json.dumps({"layer": f"{out}x{inp}", "group": f"{gsz}x{gsz}" if gsz else f"1x{gin}", "T": T,
                      "density": args.density, "algo": args.algo, "kept": kept,
                      "us": s * 1e6, "GB/s": nbytes / s / 1e9, "TFLOP/s": flops / s / 1e12}), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--oracle-single-thread", action="store_true",
                    help="internal: time the oracle sample only and print it (run with one BLAS thread)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--headline-only", action="store_true", help="skip the per-GPU characterisations")
    ap.add_argument("--layer", default=None, help="single-layer mode: OUTxIN (random mask of --density)")
    ap.add_argument("--block-of", type=int, default=0,
                    help="block mode: block 0 of workload 2, 3, 4 or 5, at --tokens")
    ap.add_argument("--tokens", type=int, default=16)
    ap.add_argument("--group", type=int, default=0, help="single-layer mode: square g x g groups (0 = 1x256)")
    ap.add_argument("--density", type=float, default=0.5)
    ap.add_argument("--algo", choices=["auto", "decode", "prefill", "prefill_dense"], default="auto")
    ap.add_argument("--group-in", type=int, default=256, choices=[128, 256],
                    help="single-layer mode with --group 0: 1 x group_in groups")
    ap.add_argument("--train-op", action="store_true",
                    help="time only the Gumbel-Sigmoid sample and the straight-through backward")
    ap.add_argument("--group-shapes", action="store_true",
                    help="time only the square-group kernels on the 7B block")
    ap.add_argument("--mask-export", action="store_true",
                    help="time only the selector export kernel over the 13B stack's selectors")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.oracle_single_thread:
        w, layers = oracle_block_inputs()
        print(json.dumps(oracle_sample_rate(w, layers, args.cpu_seconds)), flush=True)
        return 0
    if args.impl == "reference":
        return run_reference(args)
    if args.layer:
        return run_layer(args)
    if args.block_of:
        return run_block(args)
    if args.mask_export:
        return run_mask_export(args)
    if args.group_shapes:
        return run_group_shapes(args)
    if args.train_op:
        return run_train_op(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
