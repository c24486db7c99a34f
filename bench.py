#!/usr/bin/env python3
"""Benchmark: fork-tree decode attention on GB300, one JSON line.

Workload (default): the Llama-3-8B attention shape (32 q / 8 kv heads, d 128,
bf16), one request with a 2048-token shared prefix and 16 trial branches with
suffixes uniform in [512, 4096], page size 16.  A step is one decode step of
every branch: the attention kernel over every node's KV (each shared node read
once) and the log-sum-exp merge, through ``parason_attn_decode``.

  value     branch-tokens/s = branches per step / device time of a step, with
            q/K/V resident in HBM and L2 flushed (256 MiB write) before every
            step; summed over ranks for N > 1 (independent replicas).
  e2e       the same metric through the same C-ABI call with q, out and lse in
            pinned host memory, read and written by the kernels in place
            (e2e_copy: q copied to HBM first, inside each step).
  roofline  the attention kernel: algorithmic bytes (unique KV, token-exact,
            each shared node once, plus q) per launch over its CUDA-event time,
            against the measured HBM copy bandwidth.
  cpu_baseline  the fp64 oracle on the host cores, on a bounded sample.

``--impl reference`` times the oracle (the reference arm of this build).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_24658_gb300 import workloads as W  # noqa: E402

METRIC = "branch-tokens/s per decode step (fork-tree decode attention, 1xGB300 unique-KV roofline)"
UNIT = "branch-tokens/s"
L2_FLUSH_BYTES = 256 << 20
FALLBACK_HBM_GBS = 6800.0


# ----------------------------------------------------------------------------
# helpers
# ----------------------------------------------------------------------------

def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def aggregate(local_ms: float, local_units: float, world: int, device=None):
    """Whole-job figures: max step time over ranks, units summed over ranks."""
    if world <= 1:
        return local_ms, local_units
    import torch.distributed as dist
    t = torch.tensor([local_ms, local_units], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    sm = t.clone()
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(sm[1])


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self._t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
            return
        self._t = threading.Thread(target=self._read, daemon=True)
        self._t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self._t:
            self._t.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def algorithmic_bytes(tree):
    """Unique KV (token-exact, each node some branch reads counted once) + q, out, lse."""
    cnt = tree.leaves_under()
    kv = int(tree.node_len[cnt > 0].sum()) * 2 * tree.num_kv_heads * tree.head_dim * tree.kv_elem_bytes()
    q = tree.num_leaves * tree.num_q_heads * tree.head_dim * tree.q_elem_bytes()
    o = q
    lse = tree.num_leaves * tree.num_q_heads * 4
    return {"kv": kv, "q": q, "out": o, "lse": lse, "step": kv + q + o + lse, "attn": kv + q}


def algorithmic_flops(tree):
    cnt = tree.leaves_under()
    return int(sum(int(tree.node_len[n]) * int(cnt[n]) for n in range(tree.num_nodes))
               * tree.num_q_heads * 4 * tree.head_dim)


# ----------------------------------------------------------------------------
# CPU baseline: the fp64 oracle on a bounded sample
# ----------------------------------------------------------------------------

def oracle_sample_rate(tree_cpu, budget_s: float, max_branches=None):
    """Time the oracle on whole branches (cycling) for about ``budget_s`` seconds."""
    import oracle
    kw = oracle.tree_kwargs(tree_cpu)
    L = tree_cpu.num_leaves
    done, t0, b = 0, time.perf_counter(), 0
    while True:
        oracle.decode(sel=[b % L], **kw)
        done += 1
        b += 1
        el = time.perf_counter() - t0
        if el >= budget_s or (max_branches and done >= max_branches):
            break
    return done / el, done, el, oracle.num_threads()


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    tree = make_workload(args, device="cpu")
    import oracle
    kw = oracle.tree_kwargs(tree)
    L = tree.num_leaves
    # per-step sample: whole branches, sized so the whole run takes about 60 s
    t0 = time.perf_counter()
    oracle.decode(sel=[0], **kw)
    per_branch = max(time.perf_counter() - t0, 1e-4)
    per_step = max(1, int(60.0 / ((args.steps + args.warmup) * per_branch)))
    per_step = min(per_step, L)
    b = 0
    for _ in range(args.warmup):
        oracle.decode(sel=[(b + i) % L for i in range(per_step)], **kw)
        b += per_step
    times = []
    for _ in range(args.steps):
        sel = [(b + i) % L for i in range(per_step)]
        t0 = time.perf_counter()
        oracle.decode(sel=sel, **kw)
        times.append(time.perf_counter() - t0)
        b += per_step
    total = sum(times)
    value = per_step * args.steps / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(tree, args),
        "cpu_baseline": {"kind": "oracle", "value": value, "unit": UNIT,
                         "cores": oracle.num_threads(),
                         "sample": f"{per_step} whole branch(es) per step of {L}, all q heads"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------

def make_workload(args, device):
    return W.make_config(args.config, mode=args.mode, device=device)


def workload_config(tree, args):
    return {"workload": tree.name, "num_q_heads": tree.num_q_heads,
            "num_kv_heads": tree.num_kv_heads, "head_dim": tree.head_dim,
            "kv_dtype": tree.mode, "branches": tree.num_leaves, "nodes": tree.num_nodes,
            "unique_tokens": tree.unique_tokens(), "path_tokens": tree.path_tokens(),
            "page_size": tree.page_size, "seed_config": args.config,
            "l2": "flushed before every step (256 MiB write)"}


def run_gpu(args):
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    from paper_2608_24658_gb300 import build
    from paper_2608_24658_gb300.api import Plan

    build.build()
    tree = make_workload(args, device=dev)
    plan = Plan.for_tree(tree)
    plan_info = plan.info()
    ws = plan.workspace(dev)
    out = torch.empty_like(tree.q)
    lse = torch.empty(tree.q.shape[:2], dtype=torch.float32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        plan.decode(tree.q, tree.k_pages, tree.v_pages, out=out, lse=lse, workspace=ws,
                    k_scale=tree.k_scale, v_scale=tree.v_scale, stream=stream)

    for _ in range(args.warmup):
        flush.fill_(1.0)
        step()
    plan.check(stream)

    # ---------------- timed region: K steps, L2 flushed before each
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize(dev)
    wall0 = time.perf_counter()
    for i in range(args.steps):
        flush.fill_(float(i))
        starts[i].record(stream)
        step()
        ends[i].record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    wall = time.perf_counter() - wall0
    clocks = sampler.stop()
    plan.check(stream)
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    local_ms = float(np.mean(step_ms))

    # ---------------- per-kernel times: the same steps with the library's
    # events around its attention kernel (an event between the two kernels
    # stops the merge grid from launching early, so this pass is separate)
    kernel_steps = min(args.steps, 500)
    plan.enable_timing(kernel_steps)
    for i in range(kernel_steps):
        flush.fill_(float(i))
        step()
    torch.cuda.synchronize(dev)
    attn_ms, merge_ms = plan.read_timing(kernel_steps)
    plan.enable_timing(0)
    ms, units = aggregate(local_ms, tree.num_leaves, world, dev)
    value = units / (ms / 1000.0)

    # ---------------- end to end: pinned host q in, out + lse back, every step
    # q stays in pinned host memory and the kernels read it there; the merge
    # kernel writes the step's result (out, lse) straight into pinned host
    # memory.  The GPU reaches both over NVLink-C2C, so the host<->device
    # transfers are those loads and stores.  The variant with an explicit
    # host-to-device copy of q into HBM first is timed beside it (e2e_copy).
    q_host = tree.q.cpu().pin_memory()
    out_bytes = out.numel() * out.element_size()
    res_bytes = out_bytes + lse.numel() * lse.element_size()
    res_host = torch.empty(res_bytes, dtype=torch.uint8).pin_memory()
    out_e = res_host[:out_bytes].view(out.dtype).view(out.shape)
    lse_e = res_host[out_bytes:].view(lse.dtype).view(lse.shape)
    q_dev = torch.empty_like(tree.q)
    e2e_steps = max(3, min(args.steps, 200))

    def e2e_step(copy_q):
        qa = q_host
        if copy_q:
            q_dev.copy_(q_host, non_blocking=True)
            qa = q_dev
        plan.decode(qa, tree.k_pages, tree.v_pages, out=out_e, lse=lse_e, workspace=ws,
                    k_scale=tree.k_scale, v_scale=tree.v_scale, stream=stream)

    def time_e2e(copy_q):
        for _ in range(3):
            flush.fill_(0.0)
            e2e_step(copy_q)
        torch.cuda.synchronize(dev)
        e_starts = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps)]
        e_ends = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps)]
        for i in range(e2e_steps):
            flush.fill_(float(i))
            e_starts[i].record(stream)
            e2e_step(copy_q)
            e_ends[i].record(stream)
        torch.cuda.synchronize(dev)
        e_local = float(np.mean([s.elapsed_time(e) for s, e in zip(e_starts, e_ends)]))
        e_ms, _ = aggregate(e_local, tree.num_leaves, world, dev)
        plan.check(stream)
        return units / (e_ms / 1000.0)

    e2e_value = time_e2e(False)
    e2e_copy_value = time_e2e(True)

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return 0

    # ---------------- roofline of the attention kernel
    peak_gbs, peak_kind = measured_peaks()
    ab = algorithmic_bytes(tree)
    attn_avg_ms = float(np.mean(attn_ms)) if len(attn_ms) else float("nan")
    merge_avg_ms = float(np.mean(merge_ms)) if len(merge_ms) else float("nan")
    achieved = ab["attn"] / (attn_avg_ms * 1e-3) / 1e9
    traffic = None
    tr_path = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tr_path):
        with open(tr_path) as f:
            tr = json.load(f).get(f"{tree.name}:{tree.mode}")
        if tr and tr.get("kernel_source_hash") == kernel_source_hash():
            traffic = tr["bytes_per_launch"]
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak_gbs, "unit": "GB/s",
                "frac": achieved / peak_gbs, "traffic": traffic,
                "kernel": f"attn_{tree.mode}_kernel", "peak_kind": peak_kind,
                "algorithmic_bytes_per_launch": ab["attn"], "kernel_ms": attn_avg_ms,
                "merge_ms": merge_avg_ms,
                "step_frac": (ab["step"] / (peak_gbs * 1e9)) / (ms * 1e-3)}

    # ---------------- CPU baseline: oracle on a bounded sample of this workload
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        host_tree = tree.to("cpu")
        rate, n, el, cores = oracle_sample_rate(host_tree, args.cpu_seconds)
        cpu = {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"{n} whole branch(es) of {tree.num_leaves} (all q heads), {el:.1f} s"}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if tree.mode != "fp32" else "f32",
        "data": "synthetic", "config": workload_config(tree, args),
        "e2e": {"value": e2e_value, "unit": UNIT,
                "h2d_bytes_per_step": int(q_host.numel() * q_host.element_size()),
                "d2h_bytes_per_step": int(res_host.numel()),
                "q": "read in place from pinned host memory"},
        "e2e_copy": {"value": e2e_copy_value, "unit": UNIT,
                     "q": "copied host-to-device (cudaMemcpyAsync) before the kernels"},
        "gpu_launches": args.steps * plan.launches_per_decode(),
        "roofline": roofline, "cpu_baseline": cpu, "clocks": clocks,
        "wall_s_timed_region": wall,
        "algorithmic": {"bytes_per_step": ab["step"], "flops_per_step": algorithmic_flops(tree)},
        "plan": {k: v for k, v in plan_info.items()
                 if k in ("num_items", "num_ctas", "num_wide_ctas", "num_workers", "num_slots",
                          "num_merge_entries")},
    }
    print(json.dumps(line), flush=True)
    plan.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def kernel_source_hash() -> str:
    """Hash of the kernel sources, to tell whether stored ncu counters still apply."""
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_24658_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h", ".cpp")):
            with open(os.path.join(csrc, name), "rb") as f:
                h.update(name.encode())
                h.update(f.read())
    return h.hexdigest()[:16]


def run_trace(args):
    """Host throughput of the tag-stream parser (grammar check, latency
    metrics, fork tree of every top-level block) on paper-scale traces, the
    oracle timed beside it.  Not part of the decode step."""
    from paper_2608_24658_gb300 import api, build as lib_build, workloads
    lib_build.build()
    traces = [workloads.paper_scale_trace(seed) for seed in range(16)]
    tokens = sum(len(t) for t in traces)

    def one_pass():
        for t in traces:
            st = api.trace_stats(t)
            for b in range(st["top_level_blocks"]):
                api.trace_fork_tree(t, b)

    for _ in range(args.warmup):
        one_pass()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one_pass()
    el = time.perf_counter() - t0
    value = tokens * args.steps / el
    cpu = None
    if not args.no_cpu_baseline:
        from oracle import trace_oracle
        t1 = time.perf_counter()
        n = 0
        for t in traces:
            lst = t.tolist()
            st = trace_oracle.stats(lst)
            for b in range(st["parallel_blocks"]):
                try:
                    trace_oracle.fork_tree(lst, b)
                except IndexError:
                    break
            n += len(t)
        cpu = {"value": n / (time.perf_counter() - t1), "unit": "tokens/s", "cores": 1,
               "kind": "oracle", "sample": f"{len(traces)} paper-scale traces, once"}
    line = {"metric": "trace parse throughput", "value": value, "unit": "tokens/s", "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
            "higher_is_better": True, "data": "synthetic",
            "config": {"workload": "16 paper-scale traces", "tokens_per_step": tokens},
            "component": "trace", "cpu_baseline": cpu}
    print(json.dumps(line), flush=True)
    return 0


def run_append(args):
    """One decode step's plan update (parason_plan_append: a token on every
    branch) against building a new plan, on the Llama-3-shape workload with
    room to grow; and the decode step before and after 64 appends."""
    import torch
    from paper_2608_24658_gb300 import build as lib_build
    from paper_2608_24658_gb300.api import Plan
    lib_build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    steps = 64          # within the room a plan leaves its branches
    tree = W.make_config(args.config, args.mode, device=dev, extra_pages=4096)
    pool = W.free_pages(tree)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def decode_us(plan, tree, n=50):
        out = torch.empty_like(tree.q)
        lse = torch.empty(tree.num_leaves, tree.num_q_heads, dtype=torch.float32, device=dev)
        ws = plan.workspace(dev)
        for _ in range(5):
            plan.decode(tree.q, tree.k_pages, tree.v_pages, out=out, lse=lse, workspace=ws,
                        k_scale=tree.k_scale, v_scale=tree.v_scale, stream=stream)
        times = []
        for _ in range(n):
            flush.fill_(1.0)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            plan.decode(tree.q, tree.k_pages, tree.v_pages, out=out, lse=lse, workspace=ws,
                        k_scale=tree.k_scale, v_scale=tree.v_scale, stream=stream)
            b.record(stream)
            b.synchronize()
            times.append(a.elapsed_time(b) * 1e3)
        plan.check(stream)
        return float(np.median(times))

    plan = Plan.for_tree(tree, stream=stream)
    fresh_us = decode_us(plan, tree)
    host_us, dev_us = [], []
    for _ in range(steps):
        tree, new_pages = W.grow_branches(tree, pool)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        a.record(stream)
        t0 = time.perf_counter()
        plan.append(new_pages, stream=stream)
        host_us.append((time.perf_counter() - t0) * 1e6)
        b.record(stream)
        b.synchronize()
        dev_us.append(a.elapsed_time(b) * 1e3)
    after_us = decode_us(plan, tree)
    plan.close()
    replan_us = []
    for _ in range(10):
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        p2 = Plan.for_tree(tree, stream=stream)
        torch.cuda.synchronize(dev)
        replan_us.append((time.perf_counter() - t0) * 1e6)
        rebuilt_us = decode_us(p2, tree, n=20) if len(replan_us) == 10 else None
        p2.close()
    line = {"metric": "plan update per decode step", "value": float(np.median(host_us)),
            "unit": "us (host)", "higher_is_better": False, "n_gpus": 1, "steps": steps,
            "data": "synthetic", "component": "append",
            "config": {"workload": tree.name, "branches": tree.num_leaves,
                       "kv_heads": tree.num_kv_heads},
            "append_device_us": float(np.median(dev_us)),
            "rebuild_plan_us": float(np.median(replan_us)),
            "decode_us_fresh_plan": fresh_us, "decode_us_after_appends": after_us,
            "decode_us_rebuilt_after": rebuilt_us}
    print(json.dumps(line), flush=True)
    return 0


def run_prefill(args):
    """Tree-masked prefill (parason_prefill_plan + parason_attn_decode): the
    thread openings at </Outlines> and the join with the threads' KV reused,
    on the Llama-3-8B attention shape.  Query tokens/s; the roofline is the
    bf16 tensor peak over the attention FLOPs (4 d per visible key per q
    head: Q K^T and P V); the oracle on sampled queries beside it."""
    import torch
    from paper_2608_24658_gb300 import build as lib_build
    from paper_2608_24658_gb300.api import Plan
    lib_build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
        peaks = json.load(f)
    peak_tf, peak_kind = float(peaks["bf16_tflops"]), "measured (cuBLAS bf16 burst)"
    kinds = [args.prefill] if args.prefill != "both" else sorted(W.PREFILL_CONFIGS)
    for kind in kinds:
        tree = W.PREFILL_CONFIGS[kind](device=dev)
        plan = Plan.for_prefill(tree, stream=stream)
        info = plan.info()
        Q = info["num_leaves"]
        flops = info["path_tokens"] * tree.num_q_heads * 4 * tree.head_dim
        out = torch.empty_like(tree.q)
        lse = torch.empty(Q, tree.num_q_heads, dtype=torch.float32, device=dev)
        ws = plan.workspace(dev)

        def step():
            plan.decode(tree.q, tree.k_pages, tree.v_pages, out=out, lse=lse, workspace=ws,
                        stream=stream)

        for _ in range(args.warmup):
            flush.fill_(1.0)
            step()
        plan.check(stream)
        K = min(args.steps, 200)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
        sampler = ClockSampler(0)
        sampler.start()
        time.sleep(0.3)
        torch.cuda.synchronize(dev)
        for i in range(K):
            flush.fill_(float(i))
            ev[i][0].record(stream)
            step()
            ev[i][1].record(stream)
        torch.cuda.synchronize(dev)
        clocks = sampler.stop()
        plan.check(stream)
        ms = float(np.mean([a.elapsed_time(b) for a, b in ev]))
        plan.enable_timing(K)
        for i in range(K):
            flush.fill_(float(i))
            step()
        torch.cuda.synchronize(dev)
        attn_ms, merge_ms = plan.read_timing(K)
        plan.enable_timing(0)
        attn_avg = float(np.mean(attn_ms))
        achieved = flops / (attn_avg * 1e-3) / 1e12
        cpu = None
        if not args.no_cpu_baseline:
            import oracle
            host = tree.to("cpu")
            kw = oracle.tree_kwargs(host)
            kw["chunk_node"] = kw.pop("leaf_node")
            done, t0 = 0, time.perf_counter()
            while time.perf_counter() - t0 < args.cpu_seconds:
                oracle.prefill(sel=[(done * 7919) % Q], **kw)
                done += 1
            el = time.perf_counter() - t0
            cpu = {"value": done / el, "unit": "query tokens/s", "cores": oracle.num_threads(),
                   "kind": "oracle", "sample": f"{done} of {Q} queries (all q heads), {el:.1f} s"}
        line = {"metric": "tree-masked prefill throughput", "value": Q / (ms * 1e-3),
                "unit": "query tokens/s", "n_gpus": 1, "steps": K, "warmup": args.warmup,
                "ms_per_step": ms, "higher_is_better": True, "dtype": "bf16",
                "data": "synthetic", "component": "prefill",
                "config": {"workload": tree.name, "queries": Q, "kv_tokens": int(tree.node_len.sum()),
                           "visible_keys": info["path_tokens"], "l2": "flushed between steps"},
                "gpu_launches": K * plan.launches_per_decode(),
                "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak_tf,
                             "unit": "TFLOP/s", "frac": achieved / peak_tf, "traffic": None,
                             "kernel": "attn_bf16_kernel", "peak_kind": peak_kind,
                             "algorithmic_flops_per_launch": flops, "kernel_ms": attn_avg,
                             "merge_ms": float(np.mean(merge_ms))},
                "plan": {k: info[k] for k in ("num_items", "num_ctas", "num_slots",
                                              "num_merge_entries")},
                "cpu_baseline": cpu, "clocks": clocks}
        print(json.dumps(line), flush=True)
        plan.close()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=2, help="workload 1-5 (default 2)")
    ap.add_argument("--mode", choices=["bf16", "fp8", "fp32"], default="bf16")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--component", choices=["decode", "trace", "append", "prefill"],
                    default="decode",
                    help="decode: the attention step (default); trace: the tag-stream "
                         "parser; append: the decode-loop plan update; prefill: the "
                         "tree-masked prefill")
    ap.add_argument("--prefill", choices=["fork", "join", "both"], default="both",
                    help="prefill workload (with --component prefill)")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.component == "trace":
        return run_trace(args)
    if args.component == "append":
        return run_append(args)
    if args.component == "prefill":
        return run_prefill(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
