#!/usr/bin/env python3
"""Benchmark of the InfiniPot-V compression pass on GB300.

`python bench.py [--gpus N] [--steps K] [--warmup W] [--config llava]`
prints one JSON line. A step is one whole compression pass (recent-frame
mean, TaR/VaN scoring, split-budget selection, compaction) over every
(layer, KV head) slab of a seeded synthetic cache already resident in HBM;
the L2 is flushed (256 MiB write) between timed passes. Under torchrun each
rank runs its own independent stream (weak scaling; no data-path
collective). `--impl reference` times the CPU oracle instead (rank 0 only).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "compress-pass latency (ms) and HBM GB/s vs GB300 peak, 7B shape 6K budget"
KERNELS = ("recent_mean", "score", "select", "gather", "fused", "pool", "combine")
FALLBACK_HBM_GBS = 6800.0


def workload_desc(w: synth.Workload) -> str:
    """The workload in under 120 characters (the options go in config keys)."""
    return (f"{w.name}: {w.n_streams}x{w.n_layers}L x {w.n_kv_heads} KV heads x {w.head_dim} {w.dtype}, "
            f"{w.grid_h}x{w.grid_w}/frame, {w.n_frames} frames ({w.n_tokens} tok) -> {w.budget}, "
            f"alpha {w.tar_ratio}")


def workload_options(w: synth.Workload) -> dict:
    opts = {}
    if w.van_pool:
        opts["van"] = f"layer-adaptive pooled, CV thresholds {tuple(w.cv_tau)}"
    if w.head_shared:
        opts["index_set"] = "one per layer, shared by its KV heads"
    if w.ablation != "none":
        opts["ablation"] = w.ablation
    return opts


def run_config(w: synth.Workload, S: int, r: int, world: int, n_streams: int) -> dict:
    """The config object of a bench line; both arms print the same one."""
    return {"workload": workload_desc(w), **workload_options(w), "storage_dtype": w.dtype,
            "streams_per_gpu": n_streams, "slabs_per_gpu": S, "recent_frames": r,
            "l2": "flushed (256 MiB write) before every timed pass; inputs "
                  f"{2 * S * w.n_tokens * w.head_dim * w.elem_bytes / 1e6:.0f} MB > L2",
            "parallelism": f"independent streams, {world} GPU(s), no collective"}


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            return float(json.load(fh)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def bytes_model(w: synth.Workload, S: int, r: int):
    """Algorithmic bytes: the pass total of the design contract and per kernel."""
    s, D, N, C, p = w.elem_bytes, w.head_dim, w.n_tokens, w.budget, w.p
    rp = r * p
    n_past = N - rp
    row = D * s
    pass_bytes = S * row * (2 * N + 4 * C) + S * C * 4
    tight = S * row * (2 * N - rp + 4 * C) + S * C * 4
    per_kernel = {
        "recent_mean": S * (rp * row + p * D * 4),
        "score": S * (2 * n_past * row + 8 * n_past),
        "select": S * (8 * n_past + 4 * C),
        "gather": S * (4 * C * row + 4 * C),
        "fused": pass_bytes,  # the fused pass does all four steps
        "pool": 0,
        "combine": 0,
    }
    if w.van_pool:
        # the recent rows' V (and their VaN) for the layer's CV; the pooling
        # reads the VaN of every row and writes the pooled VaN of past rows
        per_kernel["recent_mean"] += S * (rp * row + 4 * rp)
        per_kernel["pool"] = S * (4 * N + 4 * n_past)
    if w.head_shared:
        # partial sums (k.m, |k|^2, |v|^2) of every head in, the layer's TaR and
        # VaN out; the selection reads per-layer scores and writes per-layer kept
        L = S // w.n_kv_heads
        per_kernel["combine"] = S * 12 * n_past + L * 8 * n_past
        per_kernel["score"] += S * 4 * n_past
        per_kernel["select"] = L * (8 * n_past + 4 * C)
        per_kernel["gather"] = S * 4 * C * row + L * 4 * C
        if w.van_pool:
            per_kernel["pool"] = L * (4 * N + 4 * n_past)
    if w.ablation == "uniform":
        # Uniform Select reads no score: kept indices out, the kept rows copied
        pass_bytes = tight = S * row * 4 * C + S * C * 4
        per_kernel.update(recent_mean=0, score=0, select=S * 4 * C, pool=0, combine=0)
    return pass_bytes, tight, per_kernel


def oracle_pass(w: synth.Workload, k_np, v_np, r: int):
    """One oracle pass over the given slabs (pooled VaN if the workload asks
    for it; then the slabs are whole layers)."""
    import oracle
    if w.ablation != "none":
        return oracle.compress_ablation(k_np, v_np, w.n_tokens, w.grid_h, w.grid_w, r, w.budget,
                                        w.tar_ratio, w.ablation)
    if w.head_shared:
        return oracle.compress_shared(k_np, v_np, w.n_tokens, w.grid_h, w.grid_w, r, w.budget,
                                      w.tar_ratio, w.n_kv_heads,
                                      tau=w.cv_tau if w.van_pool else None)
    if w.van_pool:
        return oracle.compress_pooled(k_np, v_np, w.n_tokens, w.grid_h, w.grid_w, r, w.budget,
                                      w.tar_ratio, w.cv_tau, w.n_kv_heads)
    return oracle.compress(k_np, v_np, w.n_tokens, w.p, r, w.budget, w.tar_ratio)


def dram_min_bytes(w: synth.Workload, S: int, r: int) -> int:
    """Least DRAM traffic any pass can have: read every K and V row once (the
    V of recent rows is not needed), write the kept K and V rows and indices."""
    row = w.head_dim * w.elem_bytes
    return S * row * (2 * w.n_tokens - r * w.p + 2 * w.budget) + S * w.budget * 4


def source_digest() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2506_15745_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, name), "rb") as fh:
            h.update(name.encode() + fh.read())
    return h.hexdigest()[:16]


def ncu_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources (else None)."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        with open(path) as fh:
            rec = json.load(fh)
    except Exception:
        return None
    ent = rec.get("kernels", {}).get(kernel)
    if not ent or rec.get("source_digest") != source_digest() or rec.get("workload") != workload:
        return None
    return ent.get("dram_bytes_per_launch_full_size")


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"],
                    "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=10)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def time_oracle(w: synth.Workload, k_np, v_np, r: int, budget_s: float = 12.0):
    """Oracle ms per full pass, from a bounded sample of slabs (single thread)."""
    import oracle
    oracle.build()
    S_total = w.n_slabs
    unit = w.n_kv_heads if (w.van_pool or w.head_shared) else 1  # whole layers
    t0 = time.perf_counter()
    oracle_pass(w, k_np[:unit], v_np[:unit], r)
    t1 = (time.perf_counter() - t0) / unit
    n = int(max(1, min(k_np.shape[0], round(budget_s / max(t1, 1e-6)))))
    n = max(unit, n // unit * unit)
    t0 = time.perf_counter()
    oracle_pass(w, k_np[:n], v_np[:n], r)
    dt = time.perf_counter() - t0
    ms_pass = dt * 1e3 * S_total / n
    return ms_pass, n, dt


def _host_part(args):
    w, s0, s1 = args
    return synth.host_generate(w, slabs=s1 - s0, slab0=s0)


def host_inputs(w: synth.Workload, S: int):
    """K, V of the first S slabs of stream 0, generated on the host by a pool
    of processes (spawned: no forked copy of an initialised runtime)."""
    import concurrent.futures as cf
    import multiprocessing as mp
    n_proc = max(1, min(len(os.sched_getaffinity(0)), 16, S))
    bounds = [(S * i // n_proc, S * (i + 1) // n_proc) for i in range(n_proc)]
    if n_proc == 1:
        return synth.host_generate(w, slabs=S)
    with cf.ProcessPoolExecutor(n_proc, mp_context=mp.get_context("spawn")) as ex:
        parts = list(ex.map(_host_part, [(w, a, b) for a, b in bounds]))
    return np.concatenate([k for k, _ in parts]), np.concatenate([v for _, v in parts])


def run_reference(args, w: synth.Workload):
    """The reference arm: the CPU oracle as it stands, on host cores, rank 0
    only. A step is one whole pass over every slab of one stream, as the GPU
    arm's; only if K + W such passes would not end within --ref-seconds does a
    step take the first slabs only, and the line says so."""
    world, rank, _ = dist_setup()
    if rank != 0:
        return
    import oracle
    oracle.build()
    from paper_2506_15745_gb300.shard import shard_range
    r = oracle.recent_frames(w.n_frames)
    unit = w.n_kv_heads if (w.van_pool or w.head_shared) else 1  # whole layers
    # The slabs one GPU's pass covers, as in the GPU arm: rank 0's share of
    # the streams of a multi-stream workload, else one stream.
    n_str = 1
    if w.n_streams > 1:
        s0, s1 = shard_range(w.n_streams, 0, world)
        n_str = s1 - s0
    S = w.slabs_per_stream * n_str
    K1, V1 = synth.host_generate(w.scaled(n_streams=1), slabs=unit)
    t0 = time.perf_counter()
    oracle_pass(w, K1, V1, r)
    t_slab = (time.perf_counter() - t0) / unit
    fit = int(args.ref_seconds / max(1e-6, (args.steps + args.warmup) * t_slab))
    per_step_slabs = max(unit, min(S, w.slabs_per_stream, fit) // unit * unit)
    K, V = host_inputs(w.scaled(n_streams=1), per_step_slabs)
    for _ in range(args.warmup):
        oracle_pass(w, K, V, r)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_pass(w, K, V, r)
        times.append(time.perf_counter() - t0)
    ms = float(np.mean(times)) * 1e3 * S / per_step_slabs
    if per_step_slabs == S:
        sample = f"every one of the {S} slabs of the pass in every step (host-generated, same recipe)"
    else:
        sample = (f"{per_step_slabs} of {S} slabs per step (host-generated, same recipe), "
                  f"extrapolated x{S / per_step_slabs:.1f} to a full pass")
    line = {
        "impl": "reference", "metric": METRIC, "value": ms, "unit": "ms", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": run_config(w, S, r, world, n_str),
        "cpu_baseline": {"value": ms, "unit": "ms", "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": ms, "unit": "ms", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_e2e(args, w, cache, kept, flush, one_pass, S, N, C, D):
    """End to end through the public API with host buffers: every step copies
    its K and V from pinned host memory, runs the pass and reads back the kept
    indices and the compacted K and V rows. Slabs are independent, so a step
    is cut into layer-aligned chunks: the host-to-device copies of chunk g+1,
    the pass on chunk g and the device-to-host copies of chunk g-1 overlap, K
    and V each on a stream of their own in each direction (events order each
    chunk's halves across chunks and steps). The value is the time of all
    steps divided by their number."""
    import torch
    from paper_2506_15745_gb300 import ipv
    from paper_2506_15745_gb300.shard import max_over_ranks
    e2e_steps = max(3, min(args.e2e_steps, args.steps))
    H = w.n_kv_heads
    k_host = torch.empty((S, N, D), dtype=cache.k.dtype, pin_memory=True)
    v_host = torch.empty_like(k_host, pin_memory=True)
    k_host.copy_(cache.k[0])
    v_host.copy_(cache.v[0])
    kept_host = torch.empty(tuple(kept.shape), dtype=torch.int32, pin_memory=True)
    k_out = torch.empty((S, C, D), dtype=cache.k.dtype, pin_memory=True)
    v_out = torch.empty_like(k_out, pin_memory=True)
    n_layers = S // H
    # A small step (under 64 MB of K and V) is latency-bound: one chunk, all on one stream.
    small = 2 * S * N * D * cache.k.element_size() < 64e6
    per = n_layers if small else max(1, -(-n_layers // max(1, args.e2e_chunks)))  # layers per chunk
    chunks = [(l0 * H, min(n_layers, l0 + per) * H) for l0 in range(0, n_layers, per)]
    comp = torch.cuda.current_stream()
    # K and V travel on streams of their own in each direction (one copy engine each)
    h2d = (comp, comp) if small else (torch.cuda.Stream(), torch.cuda.Stream())
    d2h = (comp, comp) if small else (torch.cuda.Stream(), torch.cuda.Stream())
    consumed = {c: None for c in chunks}   # the pass has read this chunk's input half
    drained = {c: [None, None] for c in chunks}  # the output halves have been read back

    def kept_rows(lo, hi):
        return (lo // H, hi // H) if w.head_shared else (lo, hi)

    def e2e_step():
        for lo, hi in chunks:
            ready = []
            for t, (dev_t, host_t) in enumerate(((cache.k, k_host), (cache.v, v_host))):
                with torch.cuda.stream(h2d[t]):
                    if consumed[(lo, hi)] is not None:
                        h2d[t].wait_event(consumed[(lo, hi)])
                    dev_t[0, lo:hi].copy_(host_t[lo:hi], non_blocking=True)
                    ready.append(h2d[t].record_event())
            for ev in ready:
                comp.wait_event(ev)
            for ev in drained[(lo, hi)]:
                if ev is not None:
                    comp.wait_event(ev)
            k = ipv.KV.from_tensors((cache.k[0, lo:hi], cache.k[1, lo:hi]), (None, None), 0)
            v = ipv.KV.from_tensors((cache.v[0, lo:hi], cache.v[1, lo:hi]), (None, None), 0)
            r0, r1 = kept_rows(lo, hi)
            ipv.compress(k, v, (hi - lo) // H, H, D, N, w.grid_h, w.grid_w, C, w.tar_ratio,
                         kept[r0:r1], comp)
            done = comp.record_event()
            consumed[(lo, hi)] = done
            for t, (dev_t, out_t) in enumerate(((cache.k, k_out), (cache.v, v_out))):
                with torch.cuda.stream(d2h[t]):
                    d2h[t].wait_event(done)
                    if t == 0:
                        kept_host[r0:r1].copy_(kept[r0:r1], non_blocking=True)
                    out_t[lo:hi].copy_(dev_t[1, lo:hi, :C], non_blocking=True)
                    drained[(lo, hi)][t] = d2h[t].record_event()

    if small:  # latency-bound: the host's enqueue cost is the step, so keep it to six calls
        k_all = ipv.KV.from_tensors((cache.k[0], cache.k[1]), (None, None), 0)
        v_all = ipv.KV.from_tensors((cache.v[0], cache.v[1]), (None, None), 0)

        def e2e_step():
            cache.k[0].copy_(k_host, non_blocking=True)
            cache.v[0].copy_(v_host, non_blocking=True)
            k_all.cur = v_all.cur = 0
            ipv.compress(k_all, v_all, n_layers, H, D, N, w.grid_h, w.grid_w, C, w.tar_ratio, kept, comp)
            kept_host.copy_(kept, non_blocking=True)
            k_out.copy_(cache.k[1, :, :C], non_blocking=True)
            v_out.copy_(cache.v[1, :, :C], non_blocking=True)

    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(comp)
    for st in h2d + d2h:
        if st is not comp:
            st.wait_event(e0)
    for _ in range(e2e_steps):
        e2e_step()
    for st in d2h:
        if st is not comp:
            comp.wait_stream(st)
    e1.record(comp)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps)
    h2d_b = 2 * k_host.numel() * k_host.element_size()
    d2h_b = kept_host.numel() * 4 + 2 * k_out.numel() * k_out.element_size()
    return {"value": e2e_ms, "unit": "ms", "h2d_bytes_per_step": h2d_b, "d2h_bytes_per_step": d2h_b,
            "steps": e2e_steps, "chunks_per_step": len(chunks),
            "method": ("one stream (a small step)" if small else
                       "layer-aligned chunks; K and V copies on their own streams each way, "
                       "overlapping the pass and each other")}


def steady_steps(w: synth.Workload, cache, S, C, D, p, rank, n_steps: int = 100):
    """The stream's steady-state step (append the next frames behind the C
    survivors with ipv_append_frames, then compress), launched eagerly and as
    replays of two captured CUDA graphs (one per ping-pong parity). Host
    submission time is taken while a sleep kernel holds the GPU, so it counts
    only the enqueue cost; device time is events around all the steps."""
    import torch

    from paper_2506_15745_gb300 import ipv
    if n_steps <= 0:
        return None
    gen = synth.DeviceGenerator(w, S, stream=rank)
    nf = w.append_frames
    k_new = torch.empty((S, nf * p, D), dtype=cache.k.dtype, device="cuda")
    v_new = torch.empty_like(k_new)
    gen.fill(k_new, v_new, 0, nf)
    kept = torch.empty((S // w.n_kv_heads if w.head_shared else S, C), dtype=torch.int32, device="cuda")

    def structs(c):
        fids = (cache.fid[0], cache.fid[1]) if cache.fid is not None else (None, None)
        k = ipv.KV.from_tensors((cache.k[0], cache.k[1]), (cache.pid[0], cache.pid[1]), c, fids)
        v = ipv.KV.from_tensors((cache.v[0], cache.v[1]), (None, None), c)
        return k, v

    def step(c):
        k, v = structs(c)
        ipv.append_frames(k, v, k_new, v_new, w.n_layers, w.n_kv_heads, D, C, nf, w.grid_h, w.grid_w)
        ipv.compress(k, v, w.n_layers, w.n_kv_heads, D, w.n_tokens, w.grid_h, w.grid_w, C,
                     w.tar_ratio, kept)
        return k.cur

    torch.cuda.synchronize()
    graphs = {}
    for c in (0, 1):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            step(c)
        graphs[c] = g
    out = {"steps": n_steps, "appended_frames": nf}
    for mode in ("eager", "graph"):
        cur = cache.cur
        for _ in range(3):  # warm-up
            if mode == "graph":
                graphs[cur].replay()
                cur = 1 - cur
            else:
                cur = step(cur)
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda._sleep(200_000_000)  # ~0.1 s: the host enqueues every step meanwhile
        e0.record()
        t0 = time.perf_counter()
        for _ in range(n_steps):
            if mode == "graph":
                graphs[cur].replay()
                cur = 1 - cur
            else:
                cur = step(cur)
        submit = time.perf_counter() - t0
        e1.record()
        torch.cuda.synchronize()
        out[f"{mode}_submit_us_per_step"] = submit * 1e6 / n_steps
        out[f"{mode}_device_ms_per_step"] = e0.elapsed_time(e1) / n_steps
        cache.cur = cur
    return out


def run_stream(args, w: synth.Workload):
    """Streaming run (Algorithm 1 loop): frames are generated on the device and
    appended 16 at a time; whenever the cache holds n_tokens rows the pass
    compresses it to budget rows. Each pass is timed alone; the stream is
    timed whole (generation included). No L2 flush: as in deployment, every
    pass follows the appends that filled the cache."""
    import torch
    import torch.distributed as dist

    from paper_2506_15745_gb300 import ipv
    from paper_2506_15745_gb300.cache import PingPongCache
    from paper_2506_15745_gb300.shard import max_over_ranks

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    S, N, C, D, p = w.slabs_per_stream, w.n_tokens, w.budget, w.head_dim, w.p
    ipv.init(device=local, dtype=w.dtype, max_head_dim=D, max_frame_tokens=p, max_slabs=S,
             token_capacity=N, single_kernel=args.single_kernel, van_pool=w.van_pool,
             cv_tau=w.cv_tau, head_shared=w.head_shared, ablation=w.ablation)
    r = ipv.recent_frames(w.n_frames)
    kept = torch.empty((S // w.n_kv_heads if w.head_shared else S, C), dtype=torch.int32,
                       device="cuda")
    pid_block = torch.arange(w.append_frames * p, device="cuda").remainder(p).to(torch.int16)

    def stream(timed: bool, profile_passes: int = 0):
        cache = PingPongCache(S, N, D, w.dtype, patch_ids=True,
                              frame_ids=w.van_pool or w.ablation == "tar_frame")
        gen = synth.DeviceGenerator(w, S, stream=rank)
        evs, frames, n_pass = [], 0, 0
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        while frames < w.stream_frames:
            nf = min(w.append_frames, w.stream_frames - frames)
            row0 = cache.n_tokens
            gen.fill(cache.k_live, cache.v_live, row0, nf)
            cache.pid_live[:, row0:row0 + nf * p] = pid_block[:nf * p]
            if cache.fid is not None:  # frame ids: the stream's frame counter
                cache.fid[cache.cur][:, row0:row0 + nf * p] = (
                    torch.arange(frames, frames + nf, dtype=torch.int32, device="cuda").repeat_interleave(p))
            cache.n_tokens += nf * p
            frames += nf
            if cache.n_tokens >= N:
                if profile_passes and n_pass == 0:
                    ipv.profile_enable(True)
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record()
                cache.compress(w.n_layers, w.n_kv_heads, w.grid_h, w.grid_w, C, w.tar_ratio, kept)
                b.record()
                evs.append((a, b))
                n_pass += 1
                if profile_passes and n_pass == profile_passes:
                    ipv.profile_enable(False)
        t1.record()
        torch.cuda.synchronize()
        return evs, t0.elapsed_time(t1), cache

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)  # let the sampler start; the warm-up stream then keeps the GPU busy
    for _ in range(max(1, args.warmup // 10)):
        stream(False)  # warm-up stream
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    evs, total_ms, cache = stream(True)
    t_wall = time.perf_counter() - t_wall
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    per_pass = np.array([a.elapsed_time(b) for a, b in evs])
    ipv.profile_collect()
    prof_passes = min(len(evs), args.prof_steps)
    stream(False, profile_passes=prof_passes)
    prof = ipv.profile_collect()
    p50 = max_over_ranks(float(np.percentile(per_pass, 50)))
    p99 = max_over_ranks(float(np.percentile(per_pass, 99)))
    total_ms = max_over_ranks(total_ms)
    steady = steady_steps(w, cache, S, C, D, p, rank, n_steps=args.graph_steps) if world == 1 else None

    pass_bytes, tight_bytes, kbytes = bytes_model(w, S, r)
    peak, peak_kind = peaks()
    kern_ms = {k: (prof[k][0] / prof[k][1] if prof[k][1] else 0.0) for k in KERNELS}
    dominant = max(KERNELS, key=lambda k: prof[k][0])
    achieved = kbytes[dominant] / (kern_ms[dominant] * 1e-3) / 1e9
    line = None
    if rank == 0:
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            n_s = min(S, 16)  # the first pass's input shape, generated on the host
            K, V = synth.host_generate(w, slabs=n_s)
            ms_cpu, n_used, secs = time_oracle(w, K, V, r, args.cpu_seconds)
            cpu = {"value": ms_cpu, "unit": "ms", "cores": 1, "kind": "oracle",
                   "sample": f"{n_used} of {S} slabs of one pass ({secs:.1f} s, single thread), "
                             f"extrapolated x{S / n_used:.1f} to a full pass",
                   "host_cores_available": len(os.sched_getaffinity(0))}
        line = {
            "metric": METRIC, "value": p50, "unit": "ms", "n_gpus": world,
            "steps": len(evs), "warmup": max(1, args.warmup // 10), "ms_per_step": float(per_pass.mean()),
            "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": workload_desc(w), **workload_options(w),
                       "stream": f"{w.stream_frames} frames, {w.append_frames} appended per step",
                       "storage_dtype": w.dtype, "streams_per_gpu": 1, "slabs_per_gpu": S,
                       "recent_frames": r,
                       "l2": "not flushed: each pass follows the appends, as in deployment",
                       "parallelism": f"independent streams, {world} GPU(s), no collective"},
            "path": "fused single kernel" if args.single_kernel else "step kernels",
            "passes": len(evs),
            "per_pass_ms_p50": p50, "per_pass_ms_p99": p99,
            "per_pass_ms_mean": float(per_pass.mean()), "per_pass_ms_max": float(per_pass.max()),
            "total_stream_ms": total_ms,
            "pass_bytes": pass_bytes,
            "pass_roofline_frac_p50": pass_bytes / (p50 * 1e-3) / 1e9 / peak,
            "kernel_ms": {k: round(kern_ms[k], 5) for k in KERNELS},
            "kernel_ms_source": f"CUDA events around each kernel over the first {prof_passes} passes of a second stream",
            "roofline": {"bound": "hbm", "kernel": dominant, "achieved": achieved, "peak": peak,
                         "peak_source": f"{peak_kind} hbm_gbs (MEASURED_PEAKS.json)",
                         "unit": "GB/s", "frac": achieved / peak, "traffic": None,
                         "algorithmic_bytes": kbytes[dominant]},
            "cpu_baseline": cpu,
            "e2e": {"value": None, "unit": "ms",
                    "skipped": "the stream is generated on the device; no host input exists"},
            "gpu_launches": sum(prof[k][1] for k in KERNELS) * len(evs) // max(1, prof_passes),
            "timed_wall_s": t_wall,
            "clocks": clk,
            "steady_step": steady,
        }
        print(json.dumps(line), flush=True)
    ipv.shutdown()
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return line


def run_gpu(args, w: synth.Workload):
    import torch
    import torch.distributed as dist

    from paper_2506_15745_gb300 import ipv
    from paper_2506_15745_gb300.cache import PingPongCache
    from paper_2506_15745_gb300.shard import max_over_ranks, shard_range

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    # Units of work on this rank: whole streams. Single-stream configs run one
    # independent replica stream per rank; multi-stream configs are sharded.
    if w.n_streams > 1:
        s0, s1 = shard_range(w.n_streams, rank, world)
        streams = list(range(s0, s1))
    else:
        streams = [rank]
    per = w.slabs_per_stream
    S = per * len(streams)
    N, C, D, p = w.n_tokens, w.budget, w.head_dim, w.p

    ipv.init(device=local, dtype=w.dtype, max_head_dim=D, max_frame_tokens=p, max_slabs=S,
             token_capacity=N, single_kernel=args.single_kernel, van_pool=w.van_pool,
             cv_tau=w.cv_tau, head_shared=w.head_shared, ablation=w.ablation)
    r = ipv.recent_frames(w.n_frames)
    cache = PingPongCache(S, N, D, w.dtype, patch_ids=False)
    for i, st in enumerate(streams):
        synth.device_generate(w, cache.k[0, i * per:(i + 1) * per], cache.v[0, i * per:(i + 1) * per],
                              stream=st)
    kept = torch.empty((S // w.n_kv_heads if w.head_shared else S, C), dtype=torch.int32,
                       device="cuda")
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    L = len(streams) * w.n_layers

    def one_pass():
        k, v = cache.structs(pid_valid=False)
        k.cur = v.cur = 0
        ipv.compress(k, v, L, w.n_kv_heads, D, N, w.grid_h, w.grid_w, C, w.tar_ratio, kept)

    n_ev = args.steps
    ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(n_ev)]
    ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(n_ev)]
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)  # let the sampler start before the timed region
    # Warm-up after the sampler's start-up, so that the GPU is busy up to the
    # timed region (an idle gap before it slowed the first timed pass).
    for _ in range(max(3, args.warmup)):
        flush.zero_()
        one_pass()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    for i in range(args.steps):
        flush.zero_()
        ev0[i].record()
        one_pass()
        ev1[i].record()
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    per_pass = np.array([a.elapsed_time(b) for a, b in zip(ev0, ev1)])

    # Per-kernel device times: events around every kernel would serialise the
    # overlapped launches of the timed loop, so they are taken over a second
    # loop of the same passes.
    prof_steps = max(3, min(args.steps, args.prof_steps))
    ipv.profile_enable(True)
    for i in range(prof_steps):
        flush.zero_()
        one_pass()
    torch.cuda.synchronize()
    ipv.profile_enable(False)
    prof = ipv.profile_collect()
    ms_pass = float(per_pass.mean())
    ms_pass_max = max_over_ranks(ms_pass)
    wall_max = max_over_ranks(t_wall)

    pass_bytes, tight_bytes, kbytes = bytes_model(w, S, r)
    peak, peak_kind = peaks()
    kern_ms = {k: (prof[k][0] / prof[k][1] if prof[k][1] else 0.0) for k in KERNELS}
    dominant = max(KERNELS, key=lambda k: prof[k][0])
    achieved = kbytes[dominant] / (kern_ms[dominant] * 1e-3) / 1e9
    traffic = ncu_traffic(dominant, w.name) if S == w.slabs_per_stream else None
    launches = sum(prof[k][1] for k in KERNELS) * args.steps // prof_steps

    # End to end through the public API with host buffers: pinned H2D of the
    # step's K and V, the pass, D2H of the kept indices and compacted rows.
    # Skipped when a step's K and V exceed the pinned-host budget.
    e2e = None
    if 2 * S * N * D * w.elem_bytes <= args.e2e_max_gb * 1e9:
        e2e = run_e2e(args, w, cache, kept, flush, one_pass, S, N, C, D)
    else:
        e2e = {"value": None, "unit": "ms", "skipped": f"K and V of a step exceed --e2e-max-gb {args.e2e_max_gb}"}

    line = None
    if rank == 0:
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            n_s = min(S, 128)
            k_np = cache.k[0, :n_s].contiguous()
            v_np = cache.v[0, :n_s].contiguous()
            if w.is_bf16:
                k_np = k_np.view(torch.int16).cpu().numpy().view(np.uint16)
                v_np = v_np.view(torch.int16).cpu().numpy().view(np.uint16)
            else:
                k_np, v_np = k_np.cpu().numpy(), v_np.cpu().numpy()
            wc = w.scaled(n_streams=len(streams))
            ms_cpu, n_used, secs = time_oracle(wc, k_np, v_np, r, args.cpu_seconds)
            cpu = {"value": ms_cpu, "unit": "ms", "cores": 1, "kind": "oracle",
                   "sample": f"{n_used} of {S} slabs of this workload ({secs:.1f} s, single "
                             f"thread), extrapolated x{S / n_used:.1f} to a full pass",
                   "host_cores_available": len(os.sched_getaffinity(0))}
        tokens_scored = world * S * N / (ms_pass_max * 1e-3)
        line = {
            "metric": METRIC, "value": ms_pass_max, "unit": "ms", "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_pass_max,
            "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": run_config(w, S, r, world, len(streams)),
            "pass_bytes": pass_bytes,
            "pass_gbs": pass_bytes / (ms_pass_max * 1e-3) / 1e9,
            "pass_roofline_frac": pass_bytes / (ms_pass_max * 1e-3) / 1e9 / peak,
            "pass_bytes_tight": tight_bytes,
            "tokens_scored_per_s": tokens_scored,
            "per_pass_ms_p50": float(np.percentile(per_pass, 50)),
            "per_pass_ms_p99": float(np.percentile(per_pass, 99)),
            "per_pass_ms": [round(float(x), 5) for x in per_pass[:64]],
            "kernel_ms": {k: round(kern_ms[k], 5) for k in KERNELS},
            "kernel_ms_source": f"CUDA events around each kernel over {prof_steps} further passes",
            "path": "fused single kernel" if args.single_kernel else "step kernels",
            "dram_min_bytes": dram_min_bytes(w, S, r),
            "dram_min_frac": dram_min_bytes(w, S, r) / (ms_pass_max * 1e-3) / 1e9 / peak,
            "roofline": {"bound": "hbm", "kernel": dominant, "achieved": achieved, "peak": peak,
                         "peak_source": f"{peak_kind} hbm_gbs (MEASURED_PEAKS.json)" if peak_kind == "measured" else "fallback 6.8 TB/s",
                         "unit": "GB/s", "frac": achieved / peak, "traffic": traffic,
                         "algorithmic_bytes": kbytes[dominant]},
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches,
            "timed_wall_s": wall_max,
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    ipv.shutdown()
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return line


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", default="llava", choices=sorted(synth.CONFIGS))
    ap.add_argument("--e2e-chunks", type=int, default=7,
                    help="layer-aligned chunks per end-to-end step (copies overlap the pass)")
    ap.add_argument("--graph-steps", type=int, default=100,
                    help="streaming configs: steady-state steps timed eager and as CUDA-graph replays")
    ap.add_argument("--impl", default="gpu", choices=["gpu", "reference"])
    ap.add_argument("--seed", type=int, default=None,
                    help="seed of the synthetic inputs (default: the workload's own)")
    ap.add_argument("--ablation", default="none",
                    choices=["none", "tar_reverse", "van_reverse", "tar_frame", "uniform"],
                    help="run a variant of the ablation table (Sec. 4) on the chosen workload")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--e2e-max-gb", type=float, default=8.0)
    ap.add_argument("--prof-steps", type=int, default=200)
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--ref-seconds", type=float, default=150.0,
                    help="reference arm: time budget of its K + W oracle passes")
    ap.add_argument("--single-kernel", action="store_true",
                    help="run the pass as the fused persistent kernel instead of the step kernels")
    args = ap.parse_args(argv)
    w = synth.CONFIGS[args.config]
    if args.seed is not None:
        w = w.scaled(seed=args.seed)
    if args.ablation != "none":  # a variant of the ablation table on the same workload
        if w.van_pool or w.head_shared:
            ap.error("--ablation runs on the per-head, raw-VaN workloads")
        w = w.scaled(name=f"{w.name}+{args.ablation}", ablation=args.ablation)
    if args.impl == "reference":
        run_reference(args, w)
    elif w.stream_frames:
        run_stream(args, w)
    else:
        run_gpu(args, w)


if __name__ == "__main__":
    main()
