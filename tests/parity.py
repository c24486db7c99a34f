"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI
and the fp64 oracle on the same seeded inputs, and compare."""
import numpy as np
import torch

import oracle
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan

# tolerances of the decode path (bf16 KV with fp32 accumulation; fp32 mode)
BF16_MAX_ABS = 2e-2
BF16_MEAN_ABS = 2e-3
BF16_REL_L2 = 1e-2          # stricter gate: near-uniform attention has tiny outputs
FP32_MAX_ABS = 1e-5
LSE_ABS = {"bf16": 2e-3, "fp8": 2e-3, "fp32": 1e-5}


def gpu_decode(tree, plan=None, **kw):
    own = plan is None
    if own:
        plan = Plan.for_tree(tree)
    try:
        out, lse = plan.decode_tree(tree, **kw)
        plan.check()
        return out, lse
    finally:
        if own:
            plan.close()


def oracle_decode(tree, sel=None):
    """Oracle on the host copy of what branches ``sel`` read (all if None)."""
    if sel is None:
        host = tree.to("cpu")
        return oracle.decode(**oracle.tree_kwargs(host))
    sub = W.host_subset(tree, sel)
    return oracle.decode(**oracle.tree_kwargs(sub))


def compare(tree, out, lse, ref_o, ref_l, sel=None, tag=""):
    """Assert the GPU result matches the oracle within the mode's tolerance."""
    o = out.float().cpu().numpy().astype(np.float64)
    l = lse.cpu().numpy().astype(np.float64) if lse is not None else None
    if sel is not None:
        o = o[list(sel)]
        l = l[list(sel)] if l is not None else None
    err = np.abs(o - ref_o)
    assert np.isfinite(o).all(), f"{tag}: non-finite output"
    stats = {"max_abs": float(err.max(initial=0.0)), "mean_abs": float(err.mean()) if err.size else 0.0}
    denom = float(np.linalg.norm(ref_o))
    stats["rel_l2"] = float(np.linalg.norm(o - ref_o) / denom) if denom > 0 else 0.0
    if tree.mode == "fp32":
        assert stats["max_abs"] <= FP32_MAX_ABS, (tag, stats)
    else:
        assert stats["max_abs"] <= BF16_MAX_ABS, (tag, stats)
        assert stats["mean_abs"] <= BF16_MEAN_ABS, (tag, stats)
        assert stats["rel_l2"] <= BF16_REL_L2, (tag, stats)
    if l is not None:
        fin = np.isfinite(ref_l)
        assert np.array_equal(np.isfinite(l), fin), f"{tag}: lse finiteness differs"
        assert np.array_equal(l[~fin], ref_l[~fin])
        if fin.any():
            lerr = float(np.abs(l[fin] - ref_l[fin]).max())
            stats["lse_max_abs"] = lerr
            assert lerr <= LSE_ABS[tree.mode], (tag, stats)
    return stats


def run_and_compare(tree, sel=None, tag=""):
    out, lse = gpu_decode(tree)
    ref_o, ref_l = oracle_decode(tree, sel)
    return compare(tree, out, lse, ref_o, ref_l, sel, tag or tree.name)


def on_gpu(tree):
    return tree.to("cuda")


def nan_fill_unused_pages(tree):
    """Write NaN into every physical page no node owns."""
    owned = np.zeros(tree.num_physical_pages, dtype=bool)
    owned[tree.page_ids] = True
    free = torch.as_tensor(np.nonzero(~owned)[0], device=tree.k_pages.device)
    if free.numel():
        for pages in (tree.k_pages, tree.v_pages):
            if pages.dtype == torch.float8_e4m3fn:
                pages.view(torch.uint8)[free] = 0x7F
            else:
                pages[free] = float("nan")
    return tree
