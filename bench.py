#!/usr/bin/env python3
"""Benchmark: fork-tree decode attention on GB300, one JSON line.

Workload of the line (default): batched serving, 32 requests each forking 32
trial branches (1024 branches), Llama-3-8B attention shape (32 q / 8 kv heads,
d 128, bf16), prefixes lognormal (median 2048, clipped to [1024, 8192]),
suffixes uniform in [256, 8192], page size 16, physical pages randomly
permuted: about 4.4 M unique tokens, 18 GB of KV, the largest of the five
workloads and the one that fits one GPU.  A step is one decode step of every
branch: the attention kernel over every node's KV (each shared node read once)
and the log-sum-exp merge, through ``parason_attn_decode``.

  value     branch-tokens/s = branches per step / device time of a step, with
            q/K/V resident in HBM and L2 flushed (256 MiB write) before every
            step.  With N > 1 GPUs the requests are split over the ranks
            (parason_attn_plan_shard; kv heads when there are fewer requests
            than ranks): the whole workload's branches over the slowest rank's
            step, strong scaling, no exchange between ranks.
  e2e       the same metric through the same C-ABI call with q, out and lse in
            pinned host memory, read and written by the kernels in place
            (e2e_copy: q copied to HBM first, inside each step).
  roofline  the attention kernel: algorithmic bytes (unique KV, token-exact,
            each shared node once, plus q) per launch over its CUDA-event time,
            against the measured HBM copy bandwidth.
  cpu_baseline  the fp64 oracle on the host cores, on a bounded sample.
  configs   the other workloads (tiny fork, Llama-3 shape, two-level tree,
            long prefix with bf16 and with e4m3 KV), timed the same way in the
            same process: step, kernels, roofline fractions.

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

def oracle_host_sample(tree, max_branches: int = 64):
    """Host copy of a bounded sample of whole branches (W.host_subset: only
    what they read), taken once, so that a multi-GB pool never goes to the
    host whole and no copy is inside an oracle timing.  The sample is four
    groups of consecutive branches spread over the workload (with several
    requests, four requests' prefixes and suffixes)."""
    L = tree.num_leaves
    n = min(L, max_branches)
    per = max(1, n // 4)
    sel = sorted({(g * L // 4 + i) % L for g in range(4) for i in range(per)})[:n]
    return W.host_subset(tree, sel)


def oracle_branch_seconds(sub, branches):
    """Oracle time (s) of whole branches of a host sample.  Returns (seconds, threads)."""
    import oracle
    kw = oracle.tree_kwargs(sub)
    t0 = time.perf_counter()
    oracle.decode(sel=[int(b) % sub.num_leaves for b in branches], **kw)
    return time.perf_counter() - t0, oracle.num_threads()


def oracle_sample_rate(tree, budget_s: float):
    """Oracle branch-tokens/s on whole branches of a host sample of ``tree``
    (cycling) for about ``budget_s`` seconds of oracle time."""
    sub = oracle_host_sample(tree)
    done, el, cores = 0, 0.0, 1
    while el < budget_s:
        t, cores = oracle_branch_seconds(sub, [done])
        el += t
        done += 1
    return done / el, done, el, cores, sub.num_leaves


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    # the inputs are drawn where the GPU arm draws them (the same seeded
    # values); only the oracle's own calls are timed, on the host cores
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    tree = make_workload(args, device=dev)
    L = tree.num_leaves
    sub = oracle_host_sample(tree)
    del tree.k_pages, tree.v_pages
    per_branch, _ = oracle_branch_seconds(sub, [0])
    per_branch = max(per_branch, 1e-4)
    # whole branches per step, sized so that the whole run takes about 60 s
    per_step = min(L, max(1, int(60.0 / ((args.steps + args.warmup) * per_branch))))
    b = 0
    for _ in range(args.warmup):
        oracle_branch_seconds(sub, range(b, b + per_step))
        b += per_step
    times, cores = [], 1
    for _ in range(args.steps):
        t, cores = oracle_branch_seconds(sub, range(b, b + per_step))
        times.append(t)
        b += per_step
    total = sum(times)
    value = per_step * args.steps / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(tree, args),
        "cpu_baseline": {"kind": "oracle", "value": value, "unit": UNIT, "cores": cores,
                         "sample": f"{per_step} whole branch(es) per step, cycling over "
                                   f"{sub.num_leaves} sampled branches of {L}, all q heads"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------

# the configurations timed beside the headline, in the same process (N = 1)
TABLE = [(1, "bf16"), (2, "bf16"), (3, "bf16"), (4, "bf16"), (5, "bf16"), (5, "fp8")]


def make_workload(args, device, config=None, mode=None):
    if config is None and getattr(args, "workload", None):
        return W.EXTRA[args.workload](mode=mode or args.mode, device=device)
    return W.make_config(config or args.config, mode=mode or args.mode, device=device)


def workload_config(tree, args, shard=None):
    cfg = {"workload": tree.name, "num_q_heads": tree.num_q_heads,
           "num_kv_heads": tree.num_kv_heads, "head_dim": tree.head_dim,
           "kv_dtype": tree.mode, "branches": tree.num_leaves, "nodes": tree.num_nodes,
           "requests": int((tree.parent < 0).sum()),
           "unique_tokens": tree.unique_tokens(), "path_tokens": tree.path_tokens(),
           "page_size": tree.page_size, "page_order": "permuted" if tree.meta.get("permuted")
           else "node-major", "seed_config": args.config,
           "l2": "flushed before every step (256 MiB write)"}
    if shard:
        cfg["parallelism"] = shard
    return cfg


class Rank:
    """One rank's share of a workload: its plan and its q / K / V views."""

    def __init__(self, tree, rank, world, dev):
        from paper_2608_24658_gb300 import _lib
        from paper_2608_24658_gb300.api import Plan
        self.tree, self.kind = tree, None
        self.q, self.k, self.v = tree.q, tree.k_pages, tree.v_pages
        self.k_scale, self.v_scale = tree.k_scale, tree.v_scale
        if world == 1:
            self.plan = Plan.for_tree(tree)
            self.units = tree.num_leaves
            return
        roots = int((tree.parent < 0).sum())
        if roots >= world:
            # requests split over the ranks; the pools are addressed whole
            self.kind = "requests"
            self.plan = Plan.for_tree(tree, shard=(_lib.SHARD_REQUESTS, rank, world))
            br = torch.as_tensor(self.plan.export(_lib.TABLE_SHARD_BRANCHES), dtype=torch.long,
                                 device=dev)
            self.q = tree.q.index_select(0, br).contiguous()
            self.units = self.plan.num_leaves
        elif tree.num_kv_heads % world == 0:
            # kv heads split over the ranks: each rank holds its heads' q and KV
            self.kind = "kv_heads"
            self.plan = Plan.for_tree(tree, shard=(_lib.SHARD_KV_HEADS, rank, world))
            hk = tree.num_kv_heads // world
            g = tree.group
            self.q = tree.q[:, rank * hk * g:(rank + 1) * hk * g].contiguous()
            self.k = tree.k_pages[:, rank * hk:(rank + 1) * hk].contiguous()
            self.v = tree.v_pages[:, rank * hk:(rank + 1) * hk].contiguous()
            if tree.k_scale is not None:
                self.k_scale = tree.k_scale[rank * hk:(rank + 1) * hk].contiguous()
                self.v_scale = tree.v_scale[rank * hk:(rank + 1) * hk].contiguous()
            self.units = tree.num_leaves / world
        else:
            self.kind = "replicas"
            self.plan = Plan.for_tree(tree)
            self.units = tree.num_leaves

    def decode(self, q=None, out=None, lse=None, ws=None, stream=None):
        return self.plan.decode(self.q if q is None else q, self.k, self.v, out=out, lse=lse,
                                workspace=ws, k_scale=self.k_scale, v_scale=self.v_scale,
                                stream=stream)


def time_steps(step, flush, stream, steps, warmup, dev, sampler=None, world=1):
    """Warm-up right before the timed loop, then `steps` steps, each timed
    with CUDA events on the launching stream, L2 flushed (outside the events)
    before every step.  Returns (per-step ms list, wall seconds, clocks)."""
    if sampler is not None:
        sampler.start()
        time.sleep(0.3)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    for _ in range(warmup):
        flush.fill_(1.0)
        step()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    torch.cuda.synchronize(dev)
    wall0 = time.perf_counter()
    for i in range(steps):
        flush.fill_(float(i))
        starts[i].record(stream)
        step()
        ends[i].record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    wall = time.perf_counter() - wall0
    clocks = sampler.stop() if sampler is not None else None
    return [s.elapsed_time(e) for s, e in zip(starts, ends)], wall, clocks


def kernel_times(r, step, flush, dev, steps):
    """Per-kernel times: the same steps with the library's events around its
    attention kernel (an event between the two kernels stops the merge grid
    from launching early, so this pass is separate from the timed one)."""
    r.plan.enable_timing(steps)
    for i in range(steps):
        flush.fill_(float(i))
        step()
    torch.cuda.synchronize(dev)
    attn_ms, merge_ms = r.plan.read_timing(steps)
    r.plan.enable_timing(0)
    return float(np.mean(attn_ms)), float(np.mean(merge_ms))


def traffic_of(tree):
    tr_path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(tr_path):
        return None
    with open(tr_path) as f:
        tr = json.load(f).get(f"{tree.name}:{tree.mode}")
    if tr and tr.get("kernel_source_hash") == kernel_source_hash():
        return tr["bytes_per_launch"]
    return None


def measure_table_entry(idx, mode, args, dev, stream, flush, peak_gbs):
    """One configuration timed in this process: step, kernels, fractions."""
    tree = make_workload(args, dev, config=idx, mode=mode)
    r = Rank(tree, 0, 1, dev)
    ws = r.plan.workspace(dev)
    out = torch.empty_like(tree.q)
    lse = torch.empty(tree.q.shape[:2], dtype=torch.float32, device=dev)
    step = lambda: r.decode(out=out, lse=lse, ws=ws, stream=stream)
    steps = max(10, min(args.steps, args.table_steps))
    ms, _, _ = time_steps(step, flush, stream, steps, args.warmup, dev)
    r.plan.check(stream)
    attn_ms, merge_ms = kernel_times(r, step, flush, dev, steps)
    ab = algorithmic_bytes(tree)
    mean = float(np.mean(ms))
    entry = {"workload": tree.name, "kv_dtype": mode, "branches": tree.num_leaves,
             "steps": steps, "ms_per_step": mean, "ms_per_step_median": float(np.median(ms)),
             "value": tree.num_leaves / (mean * 1e-3), "kernel_ms": attn_ms, "merge_ms": merge_ms,
             "frac": ab["attn"] / (attn_ms * 1e-3) / 1e9 / peak_gbs,
             "step_frac": (ab["step"] / (peak_gbs * 1e9)) / (mean * 1e-3),
             "t_roof_ms": ab["step"] / (peak_gbs * 1e9) * 1e3,
             "algorithmic_bytes_per_step": ab["step"], "traffic": traffic_of(tree)}
    r.plan.close()
    del tree, r, out, lse, ws
    torch.cuda.empty_cache()
    return entry


def run_gpu(args):
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    from paper_2608_24658_gb300 import build

    build.build()
    tree = make_workload(args, device=dev)
    r = Rank(tree, rank, world, dev)
    plan = r.plan
    plan_info = plan.info()
    ws = plan.workspace(dev)
    out = torch.empty_like(r.q)
    lse = torch.empty(r.q.shape[:2], dtype=torch.float32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        r.decode(out=out, lse=lse, ws=ws, stream=stream)

    # compile-time configuration of the kernels and the tensor maps: once,
    # outside the timed region
    step()
    plan.check(stream)

    # ---------------- timed region: warm-up, then K steps, L2 flushed before each
    step_ms, wall, clocks = time_steps(step, flush, stream, args.steps, args.warmup, dev,
                                       sampler=ClockSampler(local), world=world)
    plan.check(stream)
    local_ms = float(np.mean(step_ms))
    attn_ms, merge_ms = kernel_times(r, step, flush, dev, min(args.steps, 500))
    ms, units = aggregate(local_ms, r.units, world, dev)
    med_ms, _ = aggregate(float(np.median(step_ms)), r.units, world, dev)
    value = units / (ms / 1000.0)

    # ---------------- end to end: pinned host q in, out + lse back, every step
    # q stays in pinned host memory and the kernels read it there; the merge
    # kernel writes the step's result (out, lse) straight into pinned host
    # memory.  The GPU reaches both over NVLink-C2C, so the host<->device
    # transfers are those loads and stores.  The variant with an explicit
    # host-to-device copy of q into HBM first is timed beside it (e2e_copy).
    q_host = r.q.cpu().pin_memory()
    out_bytes = out.numel() * out.element_size()
    res_bytes = out_bytes + lse.numel() * lse.element_size()
    res_host = torch.empty(res_bytes, dtype=torch.uint8).pin_memory()
    out_e = res_host[:out_bytes].view(out.dtype).view(out.shape)
    lse_e = res_host[out_bytes:].view(lse.dtype).view(lse.shape)
    q_dev = torch.empty_like(r.q)
    e2e_steps = max(3, min(args.steps, 200))

    def e2e_step(copy_q):
        qa = q_host
        if copy_q:
            q_dev.copy_(q_host, non_blocking=True)
            qa = q_dev
        r.decode(q=qa, out=out_e, lse=lse_e, ws=ws, stream=stream)

    def time_e2e(copy_q):
        e_ms, _, _ = time_steps(lambda: e2e_step(copy_q), flush, stream, e2e_steps, 3, dev,
                                world=world)
        e_ms, _ = aggregate(float(np.mean(e_ms)), r.units, world, dev)
        plan.check(stream)
        return units / (e_ms / 1000.0)

    e2e_value = time_e2e(False)
    e2e_copy_value = time_e2e(True)

    if rank != 0:
        plan.close()
        if world > 1:
            dist.destroy_process_group()
        return 0

    # ---------------- roofline of the attention kernel (this rank's share)
    peak_gbs, peak_kind = measured_peaks()
    ab = algorithmic_bytes(tree) if world == 1 else algorithmic_bytes_of_plan(r)
    achieved = ab["attn"] / (attn_ms * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak_gbs, "unit": "GB/s",
                "frac": achieved / peak_gbs, "traffic": traffic_of(tree) if world == 1 else None,
                "kernel": f"attn_{tree.mode}_kernel", "peak_kind": peak_kind,
                "algorithmic_bytes_per_launch": ab["attn"], "kernel_ms": attn_ms,
                "merge_ms": merge_ms,
                "step_frac": (ab["step"] / (peak_gbs * 1e9)) / (local_ms * 1e-3)}

    # ---------------- CPU baseline: oracle on a bounded sample of this workload
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        rate, n, el, cores, pool = oracle_sample_rate(tree, args.cpu_seconds)
        cpu = {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"{n} whole branch(es), cycling over {pool} sampled branches of "
                         f"{tree.num_leaves} (all q heads), {el:.1f} s of oracle time"}

    shard = None if world == 1 else f"{r.kind} over {world} GPUs"
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "ms_per_step_median": med_ms,
        "higher_is_better": True,
        "scaling": "strong" if r.kind in ("requests", "kv_heads") else "weak",
        "vs_baseline": None, "dtype": "bf16" if tree.mode != "fp32" else "f32",
        "data": "synthetic", "config": workload_config(tree, args, shard),
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
                 if k in ("num_items", "num_ctas", "num_wide_ctas", "num_slots",
                          "num_merge_entries")},
    }
    plan.close()
    del tree, r, out, lse, ws, q_dev
    torch.cuda.empty_cache()

    # ---------------- the other configurations, same process, one GPU
    if world == 1 and args.table:
        table = []
        for idx, mode in TABLE:
            if (idx, mode) == (args.config, args.mode):
                continue
            table.append(measure_table_entry(idx, mode, args, dev, stream, flush, peak_gbs))
        line["configs"] = table
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def algorithmic_bytes_of_plan(r):
    """Algorithmic bytes of one rank's share (unique KV it reads + its q, out, lse)."""
    info = r.plan.info()
    t = r.tree
    hkv = r.plan.num_kv_heads
    kv = info["unique_tokens"] * 2 * hkv * t.head_dim * t.kv_elem_bytes()
    q = r.q.numel() * r.q.element_size()
    lse = r.q.shape[0] * r.q.shape[1] * 4
    return {"kv": kv, "q": q, "out": q, "lse": lse, "step": kv + 2 * q + lse, "attn": kv + q}


def _code_tokens(text: str) -> str:
    """C/C++/CUDA source without comments, whitespace runs collapsed: edits
    to comments or layout leave the hash alone."""
    out, i, n = [], 0, len(text)
    while i < n:
        c = text[i]
        if c in "\"'":                                   # string or char literal
            j = i + 1
            while j < n and text[j] != c:
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        elif text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
        else:
            out.append(c)
            i += 1
    return " ".join("".join(out).split())


def kernel_source_hash() -> str:
    """Hash of the kernel sources' code (comments and whitespace aside), to
    tell whether stored ncu counters still apply."""
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_24658_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h", ".cpp")):
            with open(os.path.join(csrc, name), encoding="utf-8") as f:
                h.update(name.encode())
                h.update(_code_tokens(f.read()).encode())
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
    branch) against building a new plan, on the workload (with room to
    grow); the decode step before and after 64 appends; and a fork of one
    branch into four threads (parason_plan_fork) against building a plan for
    the forked tree, with the decode step after each."""
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
    # a fork: a branch opens four threads (one token each) at </Outlines>;
    # against building a plan for the forked tree
    fork_host, fork_dev, after_fork, fresh_fork = [], [], [], []
    for r in range(10):
        fpool = list(W.free_pages(tree))
        forked, pages = W.fork_branch(tree, r % tree.num_leaves, [1, 1, 1, 1], fpool)
        pf = Plan.for_tree(tree, stream=stream)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        a.record(stream)
        t0 = time.perf_counter()
        pf.fork(r % tree.num_leaves, [1, 1, 1, 1], pages, stream=stream)
        fork_host.append((time.perf_counter() - t0) * 1e6)
        b.record(stream)
        b.synchronize()
        fork_dev.append(a.elapsed_time(b) * 1e3)
        if r == 0:
            after_fork.append(decode_us(pf, forked))
            with Plan.for_tree(forked, stream=stream) as pn:
                fresh_fork.append(decode_us(pn, forked))
        pf.close()
    line = {"metric": "plan update per decode step", "value": float(np.median(host_us)),
            "unit": "us (host)", "higher_is_better": False, "n_gpus": 1, "steps": steps,
            "data": "synthetic", "component": "append",
            "config": {"workload": tree.name, "branches": tree.num_leaves,
                       "kv_heads": tree.num_kv_heads},
            "append_device_us": float(np.median(dev_us)),
            "rebuild_plan_us": float(np.median(replan_us)),
            "decode_us_fresh_plan": fresh_us, "decode_us_after_appends": after_us,
            "decode_us_rebuilt_after": rebuilt_us,
            "fork_4_threads_us_host": float(np.median(fork_host)),
            "fork_4_threads_us_device": float(np.median(fork_dev)),
            "decode_us_after_fork": after_fork[0], "decode_us_fresh_plan_of_forked_tree": fresh_fork[0]}
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

        # the clock sampler starts first, so that the warm-up runs right
        # before the timed loop (the GPU does not idle in between)
        sampler = ClockSampler(0)
        sampler.start()
        time.sleep(0.3)
        for _ in range(args.warmup):
            flush.fill_(1.0)
            step()
        plan.check(stream)
        K = min(args.steps, 200)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
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
    ap.add_argument("--config", type=int, default=4,
                    help="workload 1-5 of the JSON line (default 4: 32 requests x 32 "
                         "branches, permuted pages, the largest that fits one GPU)")
    ap.add_argument("--workload", choices=sorted(W.EXTRA), default=None,
                    help="a measurement workload instead of --config (for profiling: "
                         "batched_4req = the batched workload with 4 requests; "
                         "prefix_only = the 32k prefix under 128 one-token branches)")
    ap.add_argument("--no-table", dest="table", action="store_false",
                    help="skip the other configurations timed after the headline")
    ap.add_argument("--table-steps", type=int, default=300,
                    help="timed steps of each configuration of the table")
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
