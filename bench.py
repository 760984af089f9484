#!/usr/bin/env python3
"""Benchmark of the hot path: policy-indexed chunk-causal attention with its
fused 3D-RoPE + KV-cache write, on seeded synthetic inputs shaped like the
paper's workloads (Wan2.1 geometry, 3-latent-frame chunks of 30x52 patches).

One step = one pass of the whole path over one launch's nodes: context
selection and availability check on the host, sva_rope_kv_write, and
sva_attend_nodes, with inputs resident in HBM.  The L2 is flushed between
timed steps, outside the timed intervals (a 256 MiB write, then a 256 MiB
read so that the flush's own dirty lines are written back before the next
timed step rather than during it).  `value` is the
attention's algorithmic TFLOP/s over whole steps (4*T*Lkv*d*H per node).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the fp64 CPU oracle on the same workload

Under torchrun (N > 1) each rank runs an independent replica of the workload
on its own GPU (the path has no exchange step); the step time is the max over
ranks and `value` counts the work of all ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "chunk-attention TFLOP/s (% of GB300 BF16 peak) and denoising nodes/s per layer"
DEFAULT_WORKLOAD = "stress14b"
KERNEL_SOURCES = ["paper_2609_22283_gb300/csrc/attend.cu", "paper_2609_22283_gb300/csrc/ptx.cuh",
                  "paper_2609_22283_gb300/csrc/internal.h"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "attend_dram_traffic.json")
# Further full-geometry configurations timed beside the default one (attention
# and RoPE + cache write only), each in the same run.
PER_CONFIG = ("clean1", "same4", "prog4")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


class L2Flush:
    """Evicts the path's data from the 129 MB L2 between timed steps.

    A 256 MiB write leaves every L2 line holding the flush buffer, dirty; the
    256 MiB read of a second buffer that follows makes the L2 write those
    lines back now, so that the write-back of the flush is not charged to
    the next timed kernel (it cost the RoPE kernel ~4-5 us per step).
    """

    def __init__(self, dev):
        import torch

        self.w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        self.r = torch.ones(256 << 20, dtype=torch.uint8, device=dev)

    def __call__(self):
        self.w.zero_()
        self.r.max()  # a reduction reads the buffer in place (no widened copy)

def attn_flops(w) -> float:
    """Algorithmic FLOPs of one step's attention: 4*T*Lkv*d*H per node (QK^T + PV),
    counting under frame causality only the visible (query, own key) pairs.
    With a block-sparse mask only the (query tile, key tile) pairs the mask
    keeps count, each as 4 * rows * keys * d * H (ragged last tiles included
    at their true size)."""
    total = 0.0
    if w.sparse is not None:
        from paper_2609_22283_gb300 import inputs as I
        nt = w.tiles
        keep = I.unpack_bits(I.tile_mask(w), (1 + w.W) * nt).numpy()
        size = [min(128, w.T - 128 * t) for t in range(nt)]
        for i, (_, b, _) in enumerate(w.nodes):
            n_ctx = max(0, min(w.W, b - 1))
            for qt in range(nt):
                for k in range((1 + n_ctx) * nt):
                    if keep[i, qt, k]:
                        total += 4.0 * size[qt] * size[k % nt] * w.d * w.H
        return total
    # own chunk: every key, or under frame causality the keys up to the end
    # of the query's latent frame
    ft = w.Hp * w.Wp
    own = (float(w.T) * w.T if w.within != "frame_causal"
           else float(sum(ft * min(T_end, w.T) for T_end in range(ft, w.T + ft, ft))))
    for (_, b, _) in w.nodes:
        n_ctx = max(0, min(w.W, b - 1))
        total += 4.0 * (own + float(w.T) * n_ctx * w.T) * w.d * w.H
    return total


def attn_bytes(w) -> float:
    """Algorithmic DRAM bytes of one attention launch: the K and V of every
    distinct state the nodes read (once per head), Q read and O written once."""
    read = set()
    for (s, b, j) in w.nodes:
        read.add((s, b, j))
        for r in range(1, max(0, min(w.W, b - 1)) + 1):
            lvl = 0 if w.policy == "clean" else (j if w.policy == "same" else max(j - r, 0))
            read.add((s, b - r, lvl))
    kv = len(read) * 2 * w.H * w.T * w.d * 2.0
    return kv + 2 * w.n_nodes * w.T * w.H * w.d * 2.0


def rope_bytes(w) -> float:
    """Algorithmic bytes of one rope_kv_write launch: K, V, Q read once, written once."""
    return 3 * 2 * w.n_nodes * w.T * w.H * w.d * 2.0


def kernel_hash() -> str:
    """Hash of the attention kernel's code: its sources with comments and
    whitespace removed, so that a comment edit keeps the ncu counters valid
    and any change to the code voids them."""
    import re
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, f), encoding="utf-8") as fh:
            src = fh.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update("".join(src.split()).encode())
    return h.hexdigest()[:16]


def read_traffic(workload: str):
    """DRAM bytes per attend launch from the committed ncu table
    (profiles/attend_dram_traffic.json), if it was taken on the current
    kernel code (matching hash); else None."""
    try:
        with open(TRAFFIC_FILE) as f:
            table = json.load(f)
    except (OSError, ValueError):
        return None
    want = kernel_hash()
    for row in table.get("rows", []):
        if row.get("workload") == workload and row.get("kernel_hash") == want:
            try:
                return float(row["dram_bytes_per_launch"])
            except (KeyError, TypeError, ValueError):
                return None
    return None


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.index)],
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
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for name, val in zip(names, f[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return world, rank, local


def reduce_max(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = torch.device("cuda") if torch.cuda.is_available() and dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------- oracle (CPU)

def oracle_sample(w, inp, seconds: float, min_rows: int = 16):
    """Times the fp64 oracle on node 0, head 0, growing batches of seeded query
    rows until about `seconds` of CPU work; returns (TFLOP/s, rows, secs, cores)."""
    import numpy as np
    import torch
    import oracle
    from paper_2609_22283_gb300 import inputs as I

    oracle.build()
    g = oracle.Geometry(F=w.F, Hp=w.Hp, Wp=w.Wp, H=w.H, d=w.d, pairs=w.pairs, theta=w.theta)
    # node 0's sequence only, as fp32 (bf16 values exactly; the oracle widens
    # each head it reads to fp64)
    seq0 = w.nodes[0][0]
    states = {k: (a.float().numpy(), b.float().numpy())
              for k, (a, b) in I.all_states(w, inp).items() if k[0] == seq0}
    (_, b, _) = w.nodes[0]
    lkv = w.T * (1 + max(0, min(w.W, b - 1)))
    q = inp.q[0].float().numpy()
    rng = np.random.default_rng(5)
    rows_done, spent = 0, 0.0
    batch = min_rows
    while spent < seconds:
        rows = sorted(rng.choice(w.T, size=min(batch, w.T), replace=False).tolist())
        t0 = time.perf_counter()
        oracle.node_forward(g, oracle.POLICY_IDS[w.policy], w.W, w.nodes[0], states, q, [0], rows,
                            1.0 / math.sqrt(w.d))
        spent += time.perf_counter() - t0
        rows_done += len(rows)
        batch = min(w.T, batch * 2)
    flops = 4.0 * rows_done * lkv * w.d
    return flops / spent / 1e12, rows_done, spent, oracle.num_threads()


def run_reference(args, world, rank):
    """The reference arm: the fp64 CPU oracle, as it stands, on the same workload."""
    if rank != 0:
        return 0
    from paper_2609_22283_gb300 import inputs as I
    w = I.WORKLOADS[args.workload]
    inp = I.generate(w)
    per_step = args.reference_seconds
    for _ in range(args.warmup):
        oracle_sample(w, inp, per_step / 4)
    vals, rows_total, secs_total, cores = [], 0, 0.0, 1
    for _ in range(args.steps):
        v, rows, secs, cores = oracle_sample(w, inp, per_step)
        vals.append(v)
        rows_total += rows
        secs_total += secs
    value = 4.0 * rows_total * w.T * (1 + max(0, min(w.W, w.nodes[0][1] - 1))) * w.d / secs_total / 1e12
    sample = (f"node {w.nodes[0]} head 0: {rows_total} seeded query rows over {args.steps} steps "
              f"(fp64 C oracle incl. its RoPE of the node's key states)")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": secs_total / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_of(w, world),
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)
    return 0


def config_of(w, world):
    lkv = [w.T * (1 + max(0, min(w.W, b - 1))) for (_, b, _) in w.nodes]
    return {"workload": w.name, "description": w.description, "nodes": [list(n) for n in w.nodes],
            "policy": w.policy, "heads": w.H, "head_dim": w.d, "tokens_per_chunk": w.T,
            "kv_tokens_per_node": lkv, "window_chunks": w.W, "levels": w.K,
            "within_chunk": w.within,
            "block_sparse": (None if w.sparse is None else
                             {"density": w.sparse, "query_tiles_per_row": w.sparse_rows,
                              "flops": "kept (query tile, key tile) pairs only"}),
            "l2": "flushed between timed steps outside the timed intervals (256 MiB write, then a 256 MiB read that writes the dirty lines back)",
            "parallelism": "single GPU" if world == 1 else f"{world} independent replicas"}


# ---------------------------------------------------------------- GPU arm

def plan_extras(args, world: int, rank: int, workload: str) -> dict:
    """Which measurements run beside the timed step.  The QKV projection and
    the other configurations are timed on a single GPU only (under torchrun
    each rank runs an independent replica of the step and nothing else); the
    oracle's CPU baseline runs on rank 0 of a single-GPU run."""
    single = world == 1
    return {"projection": single and not args.no_projection,
            "per_config": single and not args.no_per_config and workload not in PER_CONFIG,
            "cpu_baseline": single and rank == 0 and not args.no_cpu_baseline}


def run_ours(args, world, rank, local):
    import torch

    import __graft_entry__
    from paper_2609_22283_gb300 import inputs as I
    from paper_2609_22283_gb300.pipeline import Step

    __graft_entry__.build()
    if not torch.cuda.is_available():
        raise RuntimeError("bench.py needs a CUDA GPU (there is no CPU fallback)")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = I.WORKLOADS[args.workload]
    inp = I.generate(w)
    step = Step(w, device=str(dev))
    step.prefill(inp)
    q, k, v = step.device_inputs(inp)
    out, lse = step.outputs()
    stream = torch.cuda.current_stream(dev)
    flush = L2Flush(dev)

    nodes, n = step.node_table()

    def one_step():
        nodes_, _ = step.node_table()            # steps 1-2: selection + Eq. 7 check
        step.cache.rope_kv_write(nodes_, k, v, q, check=False)
        step.attend(nodes_, q, out, lse)             # dense or block-sparse, per workload

    for _ in range(args.warmup):
        one_step()
    status = step.cache.poll()
    if status != 0:
        raise RuntimeError(f"device status {status} after warm-up")

    def timed(K):
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
        torch.cuda.synchronize()
        barrier(world)
        torch.cuda.synchronize()
        for i in range(K):
            flush()
            nodes_, _ = step.node_table()
            ev[i][0].record(stream)
            step.cache.rope_kv_write(nodes_, k, v, q, check=False)
            ev[i][1].record(stream)
            step.attend(nodes_, q, out, lse)
            ev[i][2].record(stream)
        torch.cuda.synchronize()
        barrier(world)
        t_rope = sum(e[0].elapsed_time(e[1]) for e in ev)
        t_attn = sum(e[1].elapsed_time(e[2]) for e in ev)
        return t_rope, t_attn

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    t_rope, t_attn = timed(args.steps)
    clocks = sampler.stop()
    bad = {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}
    remeasured = False
    if clocks and (bad & set(clocks["reasons"])):
        sampler = ClockSampler(local)
        sampler.start()
        time.sleep(0.3)
        t_rope, t_attn = timed(args.steps)
        clocks = sampler.stop()
        remeasured = True
    status = step.cache.poll()
    if status != 0:
        raise RuntimeError(f"device status {status} in the timed region")

    t_step_ms = (t_rope + t_attn) / args.steps
    t_step_ms = reduce_max(t_step_ms, world)
    t_attn_ms = reduce_max(t_attn / args.steps, world)
    t_rope_ms = reduce_max(t_rope / args.steps, world)
    flops = attn_flops(w)
    value = flops * world / (t_step_ms * 1e-3) / 1e12
    nodes_per_s = w.n_nodes * world / (t_step_ms * 1e-3)

    # end to end: host (pinned) inputs -> device, the step, output -> host
    hq = inp.q.pin_memory()
    hk = inp.k_new.pin_memory()
    hv = inp.v_new.pin_memory()
    hout = torch.empty(out.shape, dtype=out.dtype, pin_memory=True)
    e2e_ms = []
    for it in range(args.warmup + min(args.steps, 20)):
        flush()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        q.copy_(hq, non_blocking=True)
        k.copy_(hk, non_blocking=True)
        v.copy_(hv, non_blocking=True)
        one_step()
        hout.copy_(out, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        if it >= args.warmup:
            e2e_ms.append(e0.elapsed_time(e1))
    e2e_serial = reduce_max(sum(e2e_ms) / len(e2e_ms), world)
    h2d = (hq.numel() + hk.numel() + hv.numel()) * 2
    d2h = hout.numel() * 2

    # End to end as a caller streams steps: step i's inputs go up on one
    # stream while step i-1 computes on another and step i-2's output comes
    # back on a third (two device buffer sets, ordered by events).  Every step
    # still copies its inputs from pinned host memory and its output back;
    # the timed region runs from the first copy up to the last copy down.
    # No L2 flush here: a step's working set (the cache it reads plus its
    # inputs and output) exceeds the 129 MB L2.
    s_up, s_cmp, s_down = (torch.cuda.Stream(dev) for _ in range(3))
    bufs = [(q, k, v, out, lse)] + [tuple(torch.empty_like(t) for t in (q, k, v, out, lse))]
    houts = [hout, torch.empty_like(hout, pin_memory=True)]
    up_done = [torch.cuda.Event() for _ in range(2)]
    cmp_done = [torch.cuda.Event() for _ in range(2)]
    down_done = [torch.cuda.Event() for _ in range(2)]

    def streamed(K):
        for i in range(K):
            bi = i % 2
            qb, kb, vb, ob, lb = bufs[bi]
            with torch.cuda.stream(s_up):
                if i >= 2:
                    s_up.wait_event(cmp_done[bi])        # step i-2 has read this buffer set
                qb.copy_(hq, non_blocking=True)
                kb.copy_(hk, non_blocking=True)
                vb.copy_(hv, non_blocking=True)
                up_done[bi].record(s_up)
            with torch.cuda.stream(s_cmp):
                s_cmp.wait_event(up_done[bi])
                if i >= 2:
                    s_cmp.wait_event(down_done[bi])      # step i-2's output has left
                nodes_, _ = step.node_table()
                step.cache.rope_kv_write(nodes_, kb, vb, qb, stream=s_cmp, check=False)
                step.attend(nodes_, qb, ob, lb, stream=s_cmp)
                cmp_done[bi].record(s_cmp)
            with torch.cuda.stream(s_down):
                s_down.wait_event(cmp_done[bi])
                houts[bi].copy_(ob, non_blocking=True)
                down_done[bi].record(s_down)

    streamed(args.warmup + 2)
    torch.cuda.synchronize()
    k_e2e = max(4, min(args.steps, 200))
    e_start = torch.cuda.Event(enable_timing=True)
    e_end = torch.cuda.Event(enable_timing=True)
    barrier(world)
    e_start.record(s_up)
    s_cmp.wait_event(e_start)
    s_down.wait_event(e_start)
    streamed(k_e2e)
    s_down.wait_stream(s_cmp)
    e_end.record(s_down)
    torch.cuda.synchronize()
    barrier(world)
    e2e_step = reduce_max(e_start.elapsed_time(e_end) / k_e2e, world)
    status = step.cache.poll()
    if status != 0:
        raise RuntimeError(f"device status {status} in the end-to-end region")

    peaks, peak_src = load_peaks()
    peak = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    achieved = flops / (t_attn_ms * 1e-3) / 1e12
    traffic = read_traffic(w.name)
    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_step_ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config_of(w, world),
        "nodes_per_s": nodes_per_s,
        "kernels_ms": {"rope_kv_write": t_rope_ms, "attend_nodes": t_attn_ms},
        "rope_gbs": rope_bytes(w) / (t_rope_ms * 1e-3) / 1e9,
        "roofline": {"bound": "tensor", "kernel": "attend_kernel", "achieved": achieved,
                     "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                     "peak_source": f"{peak_src} bf16 dense burst (MEASURED_PEAKS.json)"
                     if peak_src == "measured" else "fallback 1.9 PFLOP/s",
                     "traffic": traffic,
                     "algorithmic_bytes": attn_bytes(w),
                     # context: the cuBLAS loop measured under the power cap
                     "frac_of_sustained": achieved / peaks.get(
                         "bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])},
        "e2e": {"value": flops * world / (e2e_step * 1e-3) / 1e12, "unit": "TFLOP/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_step, "steps": k_e2e,
                "mode": "streamed: copy-up, compute and copy-down of consecutive steps on three "
                        "streams, two device buffer sets",
                "serial_value": flops * world / (e2e_serial * 1e-3) / 1e12,
                "serial_note": "each step alone: copy up, compute, copy down, synchronise"},
        "gpu_launches": 2 * args.steps,
        "clocks": clocks,
    }
    if remeasured:
        line["clocks_note"] = "first timed region saw a slowdown reason; re-measured once"
    extras = plan_extras(args, world, rank, w.name)
    if extras["per_config"]:
        line["per_config"] = {}
    if extras["projection"]:
        line["qkv_project"] = time_projection(step, w, dev, flush, stream, peak, world)
        # the attention layer's three device steps: projection, RoPE + cache
        # write, attention (kernel times summed; the projection is not in `value`)
        line["nodes_per_s_with_projection"] = (
            w.n_nodes * world / ((line["qkv_project"]["ms"] + t_step_ms) * 1e-3))
        # the same layer with the RoPE + cache write fused into the projection
        # (sva_qkv_project_rope, then the attention)
        line["qkv_project_rope"] = time_projection(step, w, dev, flush, stream, peak, world,
                                                   fused=True)
        line["nodes_per_s_fused_layer"] = (
            w.n_nodes * world / ((line["qkv_project_rope"]["ms"] + t_attn_ms) * 1e-3))
    if "per_config" in line:
        step.close()
        step = None
        for name in PER_CONFIG:
            line["per_config"][name] = time_config(I.WORKLOADS[name], dev, flush, stream, peak,
                                                   min(args.steps, 20), args.warmup)
    if extras["cpu_baseline"]:
        tf, rows, secs, cores = oracle_sample(w, inp, args.cpu_seconds)
        line["cpu_baseline"] = {
            "value": tf, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
            "sample": f"node {w.nodes[0]} head 0, {rows} seeded query rows, {secs:.1f} s "
                      f"(fp64 C oracle, OpenMP; incl. its RoPE of the node's key states)"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if step is not None:
        step.close()
    return 0


def time_config(w, dev, flush, stream, peak, K, warmup):
    """Attention and RoPE + cache write of another workload, timed like the
    main step (CUDA events per kernel, L2 flushed between steps)."""
    import torch
    from paper_2609_22283_gb300 import inputs as I
    from paper_2609_22283_gb300.pipeline import Step
    inp = I.generate(w)
    step = Step(w, device=str(dev))
    step.prefill(inp)
    q, k, v = step.device_inputs(inp)
    out, lse = step.outputs()
    for _ in range(warmup):
        nodes_, _ = step.node_table()
        step.cache.rope_kv_write(nodes_, k, v, q, check=False)
        step.attend(nodes_, q, out, lse)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
    torch.cuda.synchronize()
    for i in range(K):
        flush()
        nodes_, _ = step.node_table()
        ev[i][0].record(stream)
        step.cache.rope_kv_write(nodes_, k, v, q, check=False)
        ev[i][1].record(stream)
        step.attend(nodes_, q, out, lse)
        ev[i][2].record(stream)
    torch.cuda.synchronize()
    if step.cache.poll() != 0:
        raise RuntimeError(f"device status after timing {w.name}")
    rope_ms = sum(e[0].elapsed_time(e[1]) for e in ev) / K
    attn_ms = sum(e[1].elapsed_time(e[2]) for e in ev) / K
    step.close()
    flops = attn_flops(w)
    tf = flops / (attn_ms * 1e-3) / 1e12
    return {"attend_ms": attn_ms, "achieved": tf, "unit": "TFLOP/s", "frac": tf / peak,
            "rope_ms": rope_ms, "rope_gbs": rope_bytes(w) / (rope_ms * 1e-3) / 1e9,
            "nodes_per_s": w.n_nodes / ((rope_ms + attn_ms) * 1e-3), "steps": K,
            "kv_tokens_per_node": [w.T * (1 + max(0, min(w.W, b - 1))) for (_, b, _) in w.nodes],
            "nodes": w.n_nodes, "heads": w.H}


def time_projection(step, w, dev, flush, stream, peak, world, fused=False):
    """The input projection in front of the step (sva_qkv_project: [q | k | v] =
    x W^T + b for the step's n*T token rows, hidden size H*d), timed like the
    step: CUDA events per launch, L2 flushed between launches.  Reported
    beside the step, not inside it.  With `fused`, sva_qkv_project_rope: the
    same projection with the RoPE + cache write in its epilogue (it writes the
    nodes' own slots; run after every timed step and check).  Single GPU
    only: replica runs under torchrun never call it."""
    if world != 1:
        raise RuntimeError("the projection is timed on a single GPU only")
    import torch
    from paper_2609_22283_gb300 import inputs as I
    C = w.H * w.d
    x, wt, b = I.projection_inputs(w, C)
    x, wt, b = x.to(dev), wt.to(dev), b.to(dev)
    outs = [torch.empty((w.n_nodes, w.T, w.H, w.d), dtype=torch.bfloat16, device=dev) for _ in range(3)]
    nodes, _ = step.node_table()

    def launch():
        if fused:
            step.cache.qkv_project_rope(nodes, x, wt, b, outs[0], check=False)
        else:
            step.cache.qkv_project(x, wt, b, *outs, check=False)

    for _ in range(3):
        launch()
    K = 20
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    torch.cuda.synchronize()
    for e0, e1 in ev:
        flush()
        e0.record(stream)
        launch()
        e1.record(stream)
    torch.cuda.synchronize()
    if step.cache.poll() != 0:
        raise RuntimeError("device status after the projection")
    ms = reduce_max(sum(a.elapsed_time(c) for a, c in ev) / K, world)
    flops = 2.0 * w.n_nodes * w.T * C * 3 * C
    tf = flops / (ms * 1e-3) / 1e12
    res = {"kernel": "qkv_project_kernel" + (" (fused RoPE + cache write)" if fused else ""),
           "rows": w.n_nodes * w.T, "in_features": C,
           "out_features": 3 * C, "ms": ms, "achieved": tf, "unit": "TFLOP/s",
           "peak": peak, "frac": tf / peak, "launches": K}
    if not fused:
        # context only: the library's bf16 matmul (cuBLAS) of the same shape,
        # without the bias and the split into q, k, v, timed the same way
        x2 = x.reshape(-1, C)
        y = torch.empty((x2.shape[0], 3 * C), dtype=torch.bfloat16, device=dev)
        for _ in range(3):
            torch.matmul(x2, wt.t(), out=y)
        torch.cuda.synchronize()
        for e0, e1 in ev:
            flush()
            e0.record(stream)
            torch.matmul(x2, wt.t(), out=y)
            e1.record(stream)
        torch.cuda.synchronize()
        ms_ref = sum(a.elapsed_time(c) for a, c in ev) / K
        res["cublas_same_shape"] = {"ms": ms_ref, "achieved": flops / (ms_ref * 1e-3) / 1e12,
                                    "unit": "TFLOP/s", "note": "torch.matmul bf16, no bias; context"}
    return res


def compare_schedules(args):
    """Per-chunk attention-layer time of the two executions of Table 3 (Section 5),
    on one GPU: fully serial clean history (Eq. 5; five one-node launches per
    chunk: four denoising updates and the clean refresh, W = 6) against the
    progressive pipeline (one launch of a round's four nodes plus the refresh).
    Each chunk is timed as a whole (CUDA events around it, L2 flushed before
    it) and each launch in it on its own (events around every launch)."""
    import torch

    import __graft_entry__
    from paper_2609_22283_gb300 import inputs as I
    from paper_2609_22283_gb300.pipeline import Step

    __graft_entry__.build()
    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    flush = L2Flush("cuda")
    res, launches, clocks = {}, {}, {}
    for name in ("clean5", "prog4r"):
        w = I.WORKLOADS[name]
        inp = I.generate(w)
        step = Step(w)
        step.prefill(inp)
        q, k, v = step.device_inputs(inp)
        out, lse = step.outputs()
        nodes, n = step.node_table()

        def one_chunk(evs=None):
            def rec():
                if evs is not None:
                    e = torch.cuda.Event(enable_timing=True)
                    e.record(stream)
                    evs.append(e)
            rec()
            if name == "clean5":                        # one launch per node, in order
                for i in range(n):
                    sl = slice(i, i + 1)
                    one = (type(nodes[0]) * 1)(nodes[i])
                    step.cache.rope_kv_write(one, k[sl], v[sl], q[sl], check=False)
                    rec()
                    step.cache.attend_nodes(one, q[sl], out[sl], lse[sl], step.scale, check=False)
                    rec()
            else:
                step.cache.rope_kv_write(nodes, k, v, q, check=False)
                rec()
                step.cache.attend_nodes(nodes, q, out, lse, step.scale, check=False)
                rec()

        for _ in range(args.warmup):
            one_chunk()
        sampler = ClockSampler(0)
        sampler.start()
        time.sleep(0.3)
        total, per = 0.0, None
        for _ in range(args.steps):
            flush()
            evs = []
            one_chunk(evs)
            torch.cuda.synchronize()
            total += evs[0].elapsed_time(evs[-1])
            t = [a.elapsed_time(b) for a, b in zip(evs[:-1], evs[1:])]
            per = t if per is None else [x + y for x, y in zip(per, t)]
        clocks[name] = sampler.stop()
        if step.cache.poll() != 0:
            raise RuntimeError("device status after timing")
        res[name] = total / args.steps
        kinds = ["rope_kv_write", "attend_nodes"] * (n if name == "clean5" else 1)
        launches[name] = [{"kernel": kd, "ms": x / args.steps} for kd, x in zip(kinds, per)]
        step.close()
    line = {"metric": "attention-layer time per chunk (RoPE + cache write + attention), ms",
            "clean_serial_ms": res["clean5"], "progressive_pipeline_ms": res["prog4r"],
            "speedup": res["clean5"] / res["prog4r"], "higher_is_better": False,
            "steps": args.steps, "warmup": args.warmup, "n_gpus": 1, "data": "synthetic",
            "config": {"serial": I.WORKLOADS["clean5"].description,
                       "pipeline": I.WORKLOADS["prog4r"].description},
            "launches": launches, "clocks": clocks,
            "l2": "flushed before each timed chunk (256 MiB write, then a 256 MiB read)",
            "paper_context": "full-DiT steady-state speedup 1.57-2.83x on 4-12 Ascend 910B2C with "
                             "context parallelism (Table 3); not the same measurement"}
    print(json.dumps(line), flush=True)
    return 0


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--reference-seconds", type=float, default=8.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-projection", action="store_true",
                    help="skip timing the QKV projection beside the step")
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip timing the other full-geometry configurations beside the step")
    ap.add_argument("--compare-schedules", action="store_true",
                    help="time clean-serial against progressive-pipeline execution of one chunk")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    return args


def main():
    args = parse_args()
    if args.compare_schedules:
        return compare_schedules(args)
    world, rank, local = dist_setup()
    if args.impl == "reference":
        rc = run_reference(args, world, rank)
    else:
        rc = run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return rc


if __name__ == "__main__":
    sys.exit(main())
