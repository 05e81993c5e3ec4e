#!/usr/bin/env python3
"""Benchmark of the regulated streaming-attention hot path on GB300.

A step is one frame through every global-attention layer: per layer, the
regulated attention over [memory ; frame] with LSE (Eq. 3), the LSE-saliency
(Sec. 3.3) and the top-k admission into the layer's bank (Eq. 4 / Eq. 6),
issued as one regmem_attend_admit call per layer (the admission runs inside
the saliency kernel).
Default workload: the long-horizon stream -- 24 layers, 16 heads x 64,
1374 tokens per frame (37x37 patches + 5 special tokens), k = 14 admitted
rows per head per frame, 2000 frames, so each layer's memory grows from 0 to
29,360 rows.  `value` is frames/s over the timed frames.  With --steps K
shorter than the stream, the K timed frames are a window centred on the
stream's middle frame, where a frame attends the stream's mean number of
keys (Eq. 6: the memory grows linearly, so the middle frame's length is the
mean): frames 991-1010 for K = 20 on the 2000-frame stream.  Each layer's
bank then starts with the rows that frame would see (seeded synthetic rows
imported through regmem_import_bank), restored after the W warm-up frames.
--start-frame overrides the window; --steps 0 times the whole stream.

Inputs: Q/K/V come from a pool of distinct seeded synthetic frames resident
in HBM (frame t uses pool entry (t-1) mod P); every step touches more than
L2 holds (>= 202 MB of inputs per frame, plus the banks), so no L2 flush is
needed.

Also reported:
  roofline      attention kernel: algorithmic FLOPs / the kernel's own launch
                clock over every launch of the timed region, against the
                measured bf16 peak (burst for a timed region under a second,
                sustained for longer ones)
  e2e           same metric through regmem_attend_admit_host: pinned host
                Q/K/V in, O and saliency back to host, copies inside the timed
                region; the window is timed three times (banks restored
                between, untimed) and the value is all frames / all time
  cpu_baseline  the fp64 oracle on the host cores, timed on a bounded sample
                of the same frames (single layer-frames at the window's ends,
                cost linear in the attended length)
  clocks        nvidia-smi samples taken during the timed region

--impl reference runs only the oracle (the reference arm) on the same frames:
each step is one (layer, head) of a layer-frame of the window.
Under torchrun with --gpus N each rank runs an independent replica stream
(distinct seed): weak scaling, no collective on the data path.
"""
from __future__ import annotations

import argparse
import gc
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

METRIC = "frames/s of regulated attn+saliency+admit at 1374 tok/frame; TC util %"
UNIT = "frames/s"

CONFIGS = {
    # name: layers, heads, n_special, grid_h, grid_w, frames, k, seed, frame_attention
    "tiny": dict(layers=1, heads=2, ns=5, gh=8, gw=8, frames=8, k=1, seed=0, fa=False),
    "layer": dict(layers=1, heads=16, ns=5, gh=37, gw=37, frames=100, k=14, seed=1, fa=False),
    "full": dict(layers=24, heads=16, ns=5, gh=37, gw=37, frames=500, k=14, seed=2, fa=False),
    "long": dict(layers=24, heads=16, ns=5, gh=37, gw=37, frames=2000, k=14, seed=3, fa=False),
    "nonsquare": dict(layers=24, heads=16, ns=5, gh=37, gw=28, frames=1000, k=11, seed=4, fa=True),
}

# dram__bytes_read.sum + dram__bytes_write.sum of one attention-kernel launch,
# from ncu captures of single launches (profiles/attn_fwd_long_stream.md):
# {(config, attended rows L): bytes}.  The line reports the capture whose L
# lies within 2 % of the timed launches' mean L, else null; the table is
# emptied whenever the attention kernel changes until it is captured again.
ATTN_TRAFFIC_CAPTURES = {("long", 16734): 73.76e6, ("long", 30720): 135.28e6}


def traffic_for(cfg_name, mean_L):
    """(bytes per launch, note) of a capture matching the timed launches."""
    for (name, L), b in ATTN_TRAFFIC_CAPTURES.items():
        if name == cfg_name and abs(L - mean_L) <= 0.02 * mean_L:
            return b, (f"ncu dram bytes (read + write) of one attention launch at L = {L} "
                       f"(timed launches: mean L = {mean_L:.0f})")
    return None, "no ncu capture of the attention kernel at this attended length"


def default_start_frame(frames, K):
    """First timed frame: K frames centred on the stream's middle frame, whose
    attended length is the stream's mean (the memory grows linearly, Eq. 6);
    the whole stream when K covers it."""
    if K <= 0 or K >= frames:
        return 1
    mid = frames // 2 + 1
    return max(1, min(mid - K // 2, frames - K + 1))


def window_frames(S0, K):
    return list(range(S0, S0 + K))


def mean_attended(cfg, frames):
    Ls = [attended_rows(cfg, t, l) for t in frames for l in range(cfg["layers"])]
    return sum(Ls) / len(Ls)


def bench_config(cfg, name, S0, K, world):
    """The `config` object, identical in both arms' lines."""
    frames = window_frames(S0, K)
    return {
        "workload": describe(cfg, name),
        "first_frame": S0,
        "frames_timed": K,
        "stream_frames": cfg["frames"],
        "mean_attended_rows": round(mean_attended(cfg, frames), 1),
        "window": ("whole stream" if S0 == 1 and K >= cfg["frames"] else
                   f"frames {S0}-{S0 + K - 1} of the stream, banks pre-filled with the rows "
                   "those frames see"),
        "l2": "no flush: inputs larger than L2 (>= 202 MB of Q/K/V per step plus the banks)",
        "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
        **({"variant": cfg["variant"]} if cfg.get("variant") else {}),
    }


# Attention launches bracketed by CUDA events inside the timed region: every
# 61st (prime to the layer count, so the sample walks through all layers).
# Kernels are launched to overlap their predecessor's tail; an event pair
# removes that overlap at its two boundaries, so the sample is kept sparse:
# every 8th launch measured 1.7 % off the frame rate, every 64th 0.2 %.  The
# roofline itself comes from the attention's launch clock, which times every
# launch without events.
PROFILE_EVERY = 61

# Times the e2e leg runs the timed window (value: all frames / all time).
E2E_REPS = 3


def describe(cfg, name):
    N = cfg["ns"] + cfg["gh"] * cfg["gw"]
    s = (f"{name}: {cfg['layers']} layers x {cfg['heads']} heads x 64, {N} tok/frame "
         f"({cfg['gh']}x{cfg['gw']} patches + {cfg['ns']} special), k={cfg['k']}/head/frame, "
         f"{cfg['frames']}-frame stream, 2x2 query sampling")
    if cfg["fa"]:
        s += ", each global layer paired with a non-causal frame-attention layer"
    return s


def layer_k(cfg, layer):
    """Rows a frame admits per head in `layer` (Eq. 5 layers: 0)."""
    ks = cfg.get("k_layers")
    return ks[layer] if ks else cfg["k"]


def attended_rows(cfg, t, layer=None):
    """L = M + N attended by frame t (memory rows before frame t plus N)."""
    N = cfg["ns"] + cfg["gh"] * cfg["gw"]
    k = cfg["k"] if layer is None else layer_k(cfg, layer)
    M = 0 if t == 1 else N + (t - 2) * k
    return M + N


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------
class ClockSampler:
    """nvidia-smi sampling of SM clock, power and throttle reasons."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)

    def summary(self):
        return parse_clock_lines(self.lines)


def parse_clock_lines(lines):
    sm, mx, pw, reasons = [], [], [], set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for ln in lines:
        parts = [p.strip() for p in ln.split(",")]
        if len(parts) < 7:
            continue
        try:
            sm.append(float(parts[0]))
            mx.append(float(parts[1]))
            pw.append(float(parts[2]))
        except ValueError:
            continue
        for n, v in zip(names, parts[3:7]):
            if v.lower().startswith("active"):
                reasons.add(n)
    if not sm:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
    busy = [s for s in sm if s > 0.5 * max(sm)] or sm
    return {"sm_mhz": statistics.median(busy), "sm_max_mhz": max(mx),
            "power_w_max": max(pw), "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# distributed helpers (torchrun)
# ---------------------------------------------------------------------------
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    return int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")), ws


def max_over_ranks(x: float, device=None) -> float:
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: float, device=None) -> float:
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


# ---------------------------------------------------------------------------
# oracle timing (runs in a fresh process: no CUDA, BLAS threads pinned)
# ---------------------------------------------------------------------------
def oracle_layer_frame_seconds(cfg, t, heads=None, seed=7):
    """Times the fp64 oracle on one layer-frame of the workload at frame t
    (memory of the size frame t sees, random bf16-valued rows): attention,
    saliency and top-k for `heads` heads (default all)."""
    import numpy as np
    import oracle as orc
    H = cfg["heads"] if heads is None else heads
    N = cfg["ns"] + cfg["gh"] * cfg["gw"]
    M = attended_rows(cfg, t) - N
    rng = np.random.default_rng(seed + t)

    def bf(a):  # round to bf16-representable values
        a = a.astype(np.float32)
        b = (a.view(np.uint32) + 0x7FFF + ((a.view(np.uint32) >> 16) & 1)) & 0xFFFF0000
        return b.view(np.float32).astype(np.float64)

    q = bf(rng.standard_normal((N, H, 64)))
    k = bf(rng.standard_normal((N, H, 64)))
    v = bf(rng.standard_normal((N, H, 64)))
    bk = [bf(rng.standard_normal((M, 64))) for _ in range(H)]
    bv = [bf(rng.standard_normal((M, 64))) for _ in range(H)]
    qidx = orc.sampled_query_tokens(cfg["ns"], cfg["gh"], cfg["gw"], 2)
    t0 = time.perf_counter()
    res = orc.attend_frame(q, k, v, bk, bv, 0.125, qidx)
    for h in range(H):
        orc.topk_admission(res["S"][h], cfg["ns"], cfg["k"])
    return time.perf_counter() - t0


def oracle_baseline(cfg, S0, K):
    """Bounded CPU baseline on the timed frames S0 .. S0+K-1: single
    layer-frames (all heads) at the window's first and last frame, cost
    fitted linear in the attended length L and summed over the window's
    layer-frames (plus, with frame-attention layers, one frame-attention
    layer-frame timed at L = N for each)."""
    frames = window_frames(S0, K)
    ts = sorted(set([frames[0], frames[-1]]))
    pts = [(attended_rows(cfg, t), oracle_layer_frame_seconds(cfg, t)) for t in ts]
    if len(pts) >= 2:
        (l0, s0), (l1, s1) = pts[0], pts[-1]
        a = (s1 - s0) / (l1 - l0) if l1 != l0 else 0.0
        b = s0 - a * l0
    else:
        a, b = pts[0][1] / pts[0][0], 0.0
    total = sum(max(a * attended_rows(cfg, t, l) + b, 0.0)
                for t in frames for l in range(cfg["layers"]))
    fa = None
    if cfg["fa"]:
        fa = oracle_layer_frame_seconds(cfg, 1)
        total += fa * cfg["layers"] * len(frames)
    return {"frames_per_s": len(frames) / total, "samples": pts, "frame_attention_s": fa}


def run_oracle_subprocess(cfg, what="baseline", steps=0, warmup=0, S0=1, K=1):
    threads = os.cpu_count() or 1
    env = dict(os.environ, OPENBLAS_NUM_THREADS=str(threads), OMP_NUM_THREADS=str(threads),
               MKL_NUM_THREADS=str(threads), CUDA_VISIBLE_DEVICES="")
    code = (f"import json, bench; print(json.dumps(bench._oracle_entry({json.dumps(cfg)!r}, "
            f"{what!r}, {steps}, {warmup}, {S0}, {K})))")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True,
                       text=True)
    if r.returncode != 0:
        raise RuntimeError(f"oracle timing failed:\n{r.stderr[-2000:]}")
    out = json.loads(r.stdout.strip().splitlines()[-1])
    out["threads"] = threads
    return out


def _oracle_entry(cfg_json, what, steps, warmup, S0, K):
    cfg = json.loads(cfg_json)
    if what == "baseline":
        return oracle_baseline(cfg, S0, K)
    # reference arm: step i = one (layer, head) of a layer-frame at frame
    # S0 + (i mod K) of the timed window (plus, with frame-attention layers,
    # one (layer, head) of a frame-attention layer-frame)
    frames = window_frames(S0, K)
    # with fewer steps than timed frames, the steps spread evenly over them
    picks = [frames[(i * len(frames)) // max(steps, 1)] for i in range(steps)]

    def step(t, seed):
        s = oracle_layer_frame_seconds(cfg, t, heads=1, seed=seed)
        if cfg["fa"]:
            s += oracle_layer_frame_seconds(cfg, 1, heads=1, seed=seed + 1)
        return s

    for i in range(warmup):
        step(picks[i % len(picks)] if picks else frames[0], 5)
    times = [step(t, 11 + i) for i, t in enumerate(picks)]
    return {"step_s": times, "frames": picks}


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def parse_cpulist(text):
    cpus = set()
    for part in text.strip().split(","):
        if not part:
            continue
        lo, _, hi = part.partition("-")
        cpus.update(range(int(lo), int(hi or lo) + 1))
    return cpus


def bind_near_gpu(index):
    """Restricts this process to the CPUs attached to GPU `index` (its NUMA
    node, from sysfs), so that host buffers pinned afterwards are placed in
    the memory nearest the GPU and its copy engines do not cross the
    socket link.  Returns what was done, or None where sysfs does not say."""
    import torch
    try:
        pr = torch.cuda.get_device_properties(index)
        bus = f"{pr.pci_domain_id:04x}:{pr.pci_bus_id:02x}:{pr.pci_device_id:02x}.0"
        base = f"/sys/bus/pci/devices/{bus}"
        cpus = parse_cpulist(open(f"{base}/local_cpulist").read()) & os.sched_getaffinity(0)
        node = open(f"{base}/numa_node").read().strip()
    except (AttributeError, OSError, ValueError):
        return None
    if not cpus:
        return None
    os.sched_setaffinity(0, cpus)
    return {"pci": bus, "numa_node": int(node), "cpus": len(cpus)}


def make_pool(cfg, P, seed, device):
    import torch
    from paper_2609_23286_gb300 import synth
    N = cfg["ns"] + cfg["gh"] * cfg["gw"]
    pool = []
    for layer in range(cfg["layers"]):
        ks = synth.key_scale(seed, layer, N, device=device)
        frames = []
        for f in range(P):
            frames.append(synth.frame_qkv(seed, layer, f + 1, N, cfg["heads"], 64,
                                          device=device, scale_cache=ks))
        pool.append(frames)
    torch.cuda.synchronize()
    return pool


def run_frames(rm, cfg, pool, t0, count, out, sal, fa_out=None, two_call=False):
    """Enqueue frames t0 .. t0+count-1 (all layers) through the C ABI: one
    regmem_attend_admit per layer (regmem_attend_admit_shared for the
    head-averaged selection), or with `two_call` regmem_attend_frame +
    regmem_admit (regmem_admit_shared)."""
    P = len(pool[0])
    shared = cfg.get("selection") == "head-averaged"
    for t in range(t0, t0 + count):
        for layer in range(cfg["layers"]):
            q, k, v = pool[layer][(t - 1) % P]
            kk = layer_k(cfg, layer)
            if fa_out is not None:
                fq, fk, fv = pool[layer][t % P]
                rm.frame_attention(fq, fk, fv, fa_out)
            if two_call:
                rm.attend_frame(layer, q, k, v, out, sal)
                (rm.admit_shared if shared else rm.admit)(layer, kk)
            else:
                (rm.attend_admit_shared if shared else rm.attend_admit)(layer, q, k, v, out, sal, kk)


def synthetic_bank(cfg, rows, seed, device):
    """Random bf16 bank rows standing in for the memory frame `start` would
    see: K rows with the per-token log-normal key scale, V rows N(0,1)."""
    import torch
    g = torch.Generator(device=device).manual_seed(seed)
    H = cfg["heads"]
    k = torch.randn(H, rows, 64, generator=g, device=device)
    k *= torch.exp(0.5 * torch.randn(1, rows, 1, generator=g, device=device))
    v = torch.randn(H, rows, 64, generator=g, device=device)
    return k.to(torch.bfloat16).cpu(), v.to(torch.bfloat16).cpu()


def timed_window(args, cfg):
    """(first timed frame, frames timed) for the command line: --start-frame
    if given, else the window centred on the stream's middle frame."""
    if args.steps:
        K = args.steps
        S0 = args.start_frame if args.start_frame else default_start_frame(cfg["frames"], K)
    else:
        S0 = args.start_frame or 1
        K = max(cfg["frames"] - S0 + 1, 1)
    return S0, K


def gpu_arm(args, cfg, cfg_name):
    import torch
    import torch.distributed as dist
    from paper_2609_23286_gb300 import regmem

    rank, local_rank, world = dist_env()
    if world > 1 and not dist.is_initialized():
        dist.init_process_group("nccl")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    # with --overlap the saliency and admission run on the library's side
    # stream (lowest priority); the attention chain gets a high-priority stream
    # so that its CTAs are dispatched first when both wait for SMs
    stream = (torch.cuda.Stream(device=dev, priority=-1) if args.overlap
              else torch.cuda.current_stream())
    N = cfg["ns"] + cfg["gh"] * cfg["gw"]
    H, L = cfg["heads"], cfg["layers"]
    S0, K = timed_window(args, cfg)
    W = args.warmup
    seed = cfg["seed"] + 1000 * rank

    # CPU baseline first (fresh process, before this process's GPU work grows)
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = run_oracle_subprocess(cfg, "baseline", S0=S0, K=K)

    # after the oracle baseline (which uses every core): this process keeps
    # to the GPU's own CPUs, where its pinned host buffers are then placed
    placement = bind_near_gpu(local_rank)

    P = min(args.pool, max(K, W, 1))
    pool = make_pool(cfg, P, seed, dev)
    out = torch.empty(N, H, 64, dtype=torch.bfloat16, device=dev)
    fa_out = torch.empty_like(out) if cfg["fa"] else None
    sal = torch.empty(H, N, dtype=torch.float32, device=dev)

    budget = max(layer_k(cfg, l) for l in range(L))
    rm = regmem.RegMem(L, H, 64, budget)
    rm.set_frame(cfg["ns"], cfg["gh"], cfg["gw"], ds=cfg.get("ds", 2),
                 max_frames=S0 - 1 + max(K, W, 1), candidates=cfg.get("candidates", 0))
    torch.cuda.synchronize()  # inputs made on the current stream
    rm.set_stream(stream)
    rm.set_overlap(args.overlap)

    # Starting later in the stream: each layer's bank holds the rows frame S0
    # would see (synthetic rows), restored again after the warm-up.
    banks = None
    if S0 > 1:
        banks = [synthetic_bank(cfg, attended_rows(cfg, S0, l) - N, seed * 7919 + l, dev)
                 for l in range(L)]

    def restore():
        rm.reset()
        if banks is not None:
            for l, (bk, bv) in enumerate(banks):
                rm.import_bank(l, bk, bv, bk.shape[1])

    # warm-up frames, then a fresh stream (or the restored late-stream banks)
    restore()
    run_frames(rm, cfg, pool, S0, W, out, sal, fa_out, args.two_call)
    rm.synchronize()
    restore()

    clocks = ClockSampler(local_rank)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    every = PROFILE_EVERY
    rm.profile_enable(every)
    barrier()
    torch.cuda.synchronize()
    clocks.start()
    # no collector pass of Python's own inside a timed region (a full pass
    # can hold the enqueueing thread for tens of milliseconds)
    gc.collect()
    gc.disable()
    ev0.record(stream)
    run_frames(rm, cfg, pool, S0, K, out, sal, fa_out, args.two_call)
    rm.join()  # the last layers' side work ends inside the timed region
    ev1.record(stream)
    torch.cuda.synchronize()
    gc.enable()
    barrier()
    clocks.stop()
    prof = rm.profile_read()
    ms_local = ev0.elapsed_time(ev1)
    ms = max_over_ranks(ms_local, dev)
    mem_rows = rm.memory_len(0)
    mem_rows_layers = [rm.memory_len(l) for l in range(L)]

    # e2e: host buffers through the public host-buffer entry point
    e2e = None
    if not args.no_e2e:
        Ph = min(4, P)
        hpool = [[tuple(x.cpu().pin_memory() for x in pool[l][f]) for f in range(Ph)]
                 for l in range(L)]
        hout = torch.empty(N, H, 64, dtype=torch.bfloat16).pin_memory()
        hsal = torch.empty(H, N, dtype=torch.float32).pin_memory()
        hfa = torch.empty_like(hout).pin_memory() if cfg["fa"] else None

        def host_frames(t0, count):
            for t in range(t0, t0 + count):
                for layer in range(L):
                    q, k, v = hpool[layer][(t - 1) % Ph]
                    if hfa is not None:
                        fq, fk, fv = pool[layer][t % P]
                        rm.frame_attention(fq, fk, fv, fa_out)  # frame-attention layer: device inputs
                    rm.attend_admit_host(layer, q, k, v, hout, hsal, layer_k(cfg, layer))

        # untimed warm-up frames through the host path, then the same banks
        # as the device leg's timed region
        restore()
        rm.profile_enable(0)
        host_frames(S0, W)
        rm.synchronize()
        # the window is timed E2E_REPS times (banks restored, untimed, in
        # between): one short window's host-to-device copies are exposed to
        # whatever else the host does at that moment
        rep_ms, enqueue_ms = [], 0.0
        for _ in range(E2E_REPS):
            restore()
            barrier()
            torch.cuda.synchronize()
            gc.collect()
            gc.disable()
            # host clock around the calls and the final synchronisation: the
            # library's copies run on a stream of its own
            t_e0 = time.perf_counter()
            host_frames(S0, K)
            t_enq = time.perf_counter()
            rm.synchronize()
            rep_ms.append((time.perf_counter() - t_e0) * 1e3)
            gc.enable()
            enqueue_ms += (t_enq - t_e0) * 1e3
        e2e_ms = max_over_ranks(sum(rep_ms), dev)
        barrier()
        tb = N * H * 64 * 2
        e2e = {"value": round(E2E_REPS * K * world / (e2e_ms / 1e3), 3), "unit": UNIT,
               "h2d_bytes_per_step": 3 * tb * L, "d2h_bytes_per_step": (tb + H * N * 4) * L,
               "api": "regmem_attend_admit_host (pinned host buffers)",
               "repetitions_of_the_window": E2E_REPS,
               "repetition_values": [round(K * world / (m / 1e3), 3) for m in rep_ms],
               "host_enqueue_ms_per_step": round(enqueue_ms / (E2E_REPS * K), 4)}

    launches = int(sum_over_ranks(prof.launches(), dev))
    rm.close()
    if rank != 0:
        return None

    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except OSError:
        pass
    peak_sust = peaks.get("bf16_tflops_sustained")
    peak_burst = peaks.get("bf16_tflops")
    measured = peak_sust is not None and peak_burst is not None
    if not measured:
        peak_sust, peak_burst = 1700.0, 1900.0
    # the burst peak for a timed region shorter than a second (the GPU has no
    # time to settle under its power cap), the sustained one for longer runs
    long_run = ms >= 1000.0
    peak = peak_sust if long_run else peak_burst
    peak_src = ("measured" if measured else "fallback") + (
        " bf16 sustained peak (timed region >= 1 s)" if long_run
        else " bf16 burst peak (timed region < 1 s)")
    attn_tflops = prof.attention_flops / (prof.attention_ms / 1e3) / 1e12 if prof.attention_ms else 0.0
    attn_ms_mean = prof.attention_ms / max(prof.attention_timed, 1)
    if prof.attention_clocked:
        roof_ms_mean = prof.attention_clock_ms / prof.attention_clocked
        roof_flops_per_launch = prof.attention_clock_flops / prof.attention_clocked
    else:
        roof_ms_mean = attn_ms_mean
        roof_flops_per_launch = prof.attention_flops / max(prof.attention_timed, 1)
    roof_tflops = roof_flops_per_launch / (roof_ms_mean / 1e3) / 1e12 if roof_ms_mean else 0.0
    merge_ms_mean = prof.merge_ms / max(prof.attention_timed, 1)
    flops_total = sum(4.0 * N * attended_rows(cfg, t, l) * 64 * H
                      for t in range(S0, S0 + K) for l in range(L))
    if cfg["fa"]:
        flops_total += 4.0 * N * N * 64 * H * L * K
    clk = clocks.summary()
    traffic = traffic_for(cfg_name, mean_attended(cfg, window_frames(S0, K)))
    line = {
        "metric": METRIC,
        "value": round(K * world / (ms / 1e3), 3),
        "unit": UNIT,
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": round(ms / K, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) Q/K/V, log-normal(0,0.5) per-token key scale, bf16)",
        "config": bench_config(cfg, cfg_name, S0, K, world),
        "run": {
            "final_memory_rows_per_head": mem_rows,
            "input_pool_frames": P,
            "overlap": ("saliency + admission on a side stream" if args.overlap
                        else "all kernels on one stream"),
            "timed_region_ms": round(ms, 3),
            "host_placement": placement,
        },
        "tflops_attention_path": round(flops_total / (ms / 1e3) / 1e12 * world, 2),
        "roofline": {
            "kernel": "attn_fwd_kernel (tcgen05 attention + LSE)",
            "bound": "tensor",
            # every launch of the timed region, timed inside the kernel by the
            # GPU's global timer (first CTA past its dependency wait -> last
            # CTA's end): nothing is recorded between launches, so no launch
            # loses its programmatic overlap with the previous kernel
            "achieved": round(roof_tflops, 2),
            "peak": peak,
            "unit": "TFLOP/s",
            "frac": round(roof_tflops / peak, 4),
            "frac_of_burst_peak": round(roof_tflops / peak_burst, 4),
            "frac_of_sustained_peak": round(roof_tflops / peak_sust, 4),
            "peak_source": peak_src,
            "timing": ("launch clock: every attention launch, device global timer"
                       if prof.attention_clocked else "CUDA events on sampled launches"),
            "traffic": traffic[0],
            "traffic_note": traffic[1],
            "launches": prof.attention_clocked or prof.attention_timed,
            "launches_total": prof.launches_attention - prof.launches_frame_attention,
            "ctas": prof.attention_ctas,
            "ctas_per_sm": prof.attention_ctas_per_sm,
            "mean_launch_ms": round(roof_ms_mean, 5),
            "algorithmic_flops_per_launch": roof_flops_per_launch,
            "algorithmic_bytes_per_launch": prof.attention_bytes / max(prof.attention_timed, 1),
            # CUDA events on the handle's stream around every n-th attention
            # launch and its merge: the event before the attention removes its
            # programmatic launch behind the previous kernel (and, with the
            # side stream, lets the previous layer's saliency take SMs first),
            # so these sampled launches run longer than the unobserved ones
            "events": {
                "achieved": round(attn_tflops, 2),
                "frac": round(attn_tflops / peak, 4),
                "launches": prof.attention_timed,
                "launches_sampled_every": every,
                "mean_launch_ms": round(attn_ms_mean, 5),
                "merge_mean_ms": round(merge_ms_mean, 5),
            },
            # attention kernel plus the merge of split units behind it
            "share_of_step": (round((roof_ms_mean * (prof.launches_attention - prof.launches_frame_attention)
                                     + prof.frame_attention_clock_ms
                                     + merge_ms_mean * prof.launches_attention) / ms_local, 4)
                              if ms_local else None),
        },
        "gpu_launches": launches,
        "clocks": clk,
        "e2e": e2e,
    }
    if cfg["fa"] and prof.frame_attention_clocked:
        # the non-causal frame-attention layers (Sec. 3.1) run the same kernel
        # with no memory: their own launch clock and algorithmic FLOPs
        fa_ms = prof.frame_attention_clock_ms / prof.frame_attention_clocked
        fa_flops = prof.frame_attention_clock_flops / prof.frame_attention_clocked
        fa_tf = fa_flops / (fa_ms / 1e3) / 1e12 if fa_ms else 0.0
        line["roofline_frame_attention"] = {
            "kernel": "attn_fwd_kernel on the frame's own N keys (regmem_frame_attention)",
            "bound": "tensor", "achieved": round(fa_tf, 2), "peak": peak, "unit": "TFLOP/s",
            "frac": round(fa_tf / peak, 4), "launches": prof.frame_attention_clocked,
            "mean_launch_ms": round(fa_ms, 5), "algorithmic_flops_per_launch": fa_flops,
        }
    # The paper's own figures for this path, beside ours as context (not a
    # target): it reports no throughput and no memory measurement in its text,
    # only the saliency's added latency (the query-downsampling sensitivity
    # table and the head-specific retention ablation table), all on one
    # NVIDIA RTX 3090 (24 GB, Sec. 4 implementation details), and the memory
    # law |M_t| = |M_1| + (t - 1) floor(gamma N) of Eq. 6.
    n_tok = cfg["ns"] + cfg["gh"] * cfg["gw"]
    end_rows = [attended_rows(cfg, cfg["frames"] + 1, l) - n_tok for l in range(L)]
    line["paper_context"] = {
        "hardware": "NVIDIA RTX 3090, 24 GB",
        "throughput_reported": None,
        "saliency_latency_ms": {"ds 2x2 (default)": 8.29, "ds 1x1": 17.64, "ds 3x3": 7.69,
                                "ds 4x4": 7.45, "without head-specific retention": 17.66},
        "saliency_latency_note": "extra inference latency of the saliency estimate; precision, "
                                 "sequence length and unit (per frame or per sequence) not stated",
        "memory_law": "|M_t| = |M_1| + (t - 1) floor(gamma N), gamma = 0.01 (Eq. 6)",
        "this_workload_bank_rows_per_layer_at_stream_end": max(end_rows),
        "this_workload_bank_bytes_at_stream_end": int(sum(end_rows) * H * 64 * 2 * 2),
    }
    if cfg.get("variant"):
        share = line["roofline"]["share_of_step"] or 0.0
        line["memory"] = {
            "bank_rows_per_layer": mem_rows_layers,
            "bank_bytes": int(sum(mem_rows_layers) * H * 64 * 2 * 2),
            "bank_rows_law": "N + (t - 1) k_l per layer (t N when every frame is kept)",
        }
        line["non_attention_ms_per_layer_frame"] = round((1.0 - share) * ms / K / L, 5)
    if cpu is not None:
        line["cpu_baseline"] = {
            "value": round(cpu["frames_per_s"], 6), "unit": UNIT, "cores": cpu["threads"],
            "kind": "oracle",
            "sample": ("fp64 numpy oracle, one layer-frame (all heads) at each end of the "
                       "timed window: "
                       + ", ".join(f"L={l} ({s:.2f}s)" for l, s in cpu["samples"])
                       + (f", frame attention L={N} ({cpu['frame_attention_s']:.2f}s)"
                          if cpu.get("frame_attention_s") else "")
                       + f"; cost fitted linear in L and summed over the {K} timed frames x "
                       f"{L} layers; BLAS matmuls on {cpu['threads']} threads, "
                       "elementwise exp single-threaded"),
        }
    return line


def reference_arm(args, cfg, cfg_name):
    rank, _, world = dist_env()
    if rank != 0:
        return None
    S0, Kw = timed_window(args, cfg)
    steps = args.steps if args.steps else 5
    W = args.warmup
    r = run_oracle_subprocess(cfg, "reference", steps, W, S0=S0, K=Kw)
    step = statistics.mean(r["step_s"])
    units = cfg["layers"] * cfg["heads"]
    fps = 1.0 / (step * units)
    fr = r["frames"]
    what = "one (layer, head) of a regulated layer-frame" + (
        " plus one (layer, head) of a frame-attention layer-frame" if cfg["fa"] else "")
    return {
        "impl": "reference",
        "metric": METRIC, "value": round(fps, 8), "unit": UNIT, "n_gpus": world,
        "steps": steps, "warmup": W, "ms_per_step": round(step * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded N(0,1) Q/K/V, log-normal(0,0.5) per-token key scale, bf16)",
        "config": bench_config(cfg, cfg_name, S0, Kw, world),
        "cpu_baseline": {"kind": "oracle", "cores": r["threads"], "value": round(fps, 8),
                         "unit": UNIT,
                         "sample": (f"fp64 numpy oracle; each step = {what} at frames "
                                    f"{fr[0]}..{fr[-1]} of the timed window (mean attended "
                                    f"length {mean_attended(cfg, fr):.0f}); frames/s = 1 / "
                                    f"({units} x mean step time)")},
        "e2e": {"value": round(fps, 8), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0, help="frames timed (default: whole stream)")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", choices=sorted(CONFIGS), default="long")
    ap.add_argument("--pool", type=int, default=16, help="distinct input frames kept in HBM")
    ap.add_argument("--start-frame", type=int, default=0,
                    help="first timed frame (default: a window centred on the stream's middle "
                         "frame); banks are pre-filled with the rows it would see")
    ap.add_argument("--layers", type=int, default=0, help="override the config's layer count")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--overlap", type=int, choices=[0, 1], default=None,
                    help="1: saliency and admission on the library's side stream, overlapping "
                         "the next layer's attention (default: 1 with several layers; 0 for a "
                         "single layer, whose next attention always waits for that side work)")
    ap.add_argument("--two-call", action="store_true",
                    help="per layer regmem_attend_frame + regmem_admit instead of regmem_attend_admit")
    ap.add_argument("--frames", type=int, default=0, help="override the config's stream length")
    # variants the paper studies around its default (each prints the same
    # JSON line with config.variant and a memory footprint)
    ap.add_argument("--layer-split", action="store_true",
                    help="Sec. 4.1: layers 11-17 admit k per frame, the others keep only the anchor")
    ap.add_argument("--gamma", type=float, default=0.0,
                    help="retention rate: k = floor(gamma N) on the admitting layers (Eq. 6)")
    ap.add_argument("--ds", type=int, default=0,
                    help="query down-sampling window for saliency (default 2, Sec. 3.3)")
    ap.add_argument("--head-avg", action="store_true",
                    help="one index set for all heads from the head-averaged saliency (Table 4)")
    ap.add_argument("--unregulated", action="store_true",
                    help="full-KV memory: every frame's N rows kept (default 200 frames)")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "ours":
        ap.error("--warmup must be >= 3")
    cfg = dict(CONFIGS[args.config])
    if args.layers:
        cfg["layers"] = args.layers
    if args.overlap is None:
        args.overlap = 1 if cfg["layers"] > 1 else 0
    if args.frames:
        cfg["frames"] = args.frames
    variant = {}
    N = cfg["ns"] + cfg["gh"] * cfg["gw"]
    if args.gamma:
        if not 0.0 < args.gamma <= 1.0:
            ap.error("--gamma must be in (0, 1]")
        cfg["k"] = int(math.floor(args.gamma * N))
        variant["gamma"] = args.gamma
    if args.unregulated:
        cfg["k"], cfg["candidates"] = N, 1
        if not args.frames:
            cfg["frames"] = 200
        variant["memory"] = "unregulated full-KV (every frame's N rows kept)"
    if args.layer_split:
        cfg["k_layers"] = [cfg["k"] if 11 <= l + 1 <= 17 else 0 for l in range(cfg["layers"])]
        variant["layer_split"] = "layers 11-17 admit k, the others keep only the anchor (Sec. 4.1)"
    if args.ds:
        if args.ds < 1:
            ap.error("--ds must be >= 1")
        cfg["ds"] = args.ds
        variant["ds"] = args.ds
    if args.head_avg:
        cfg["selection"] = "head-averaged"
        variant["selection"] = "head-averaged (one index set for all heads)"
        args.no_e2e = True  # the host-buffer call selects per head: no e2e leg for this variant
    if variant:
        variant["k_per_layer"] = [layer_k(cfg, l) for l in range(cfg["layers"])]
        cfg["variant"] = variant
        args.no_cpu_baseline = True  # the oracle baseline models the default stream only
    if args.start_frame < 0 or args.start_frame > cfg["frames"]:
        ap.error("--start-frame must be in [1, frames] (0: the default window)")
    if args.impl == "reference":
        line = reference_arm(args, cfg, args.config)
    else:
        line = gpu_arm(args, cfg, args.config)
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
