"""parason_attn_decode_no_alloc (the decode step with the library's fixed
per-device scratch instead of a caller workspace) against parason_attn_decode
with a workspace, on the same plan and inputs, two calls in a row.

Collected last on purpose: it must also pass after every other test has run
kernels, planned and freed memory on the same device.
"""
import numpy as np
import pytest
import torch

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan, ParasonError
from tests import parity as PT


def test_plan_over_scratch_limit_is_rejected_first():
    """No device work: the size check comes before any other."""
    build.build()
    big = W.make_config(5, values=False)                    # 128 branches x 36 K tokens
    with Plan.for_tree(big, host_only=True) as p:
        assert p.workspace_bytes > _lib.NO_ALLOC_SCRATCH_BYTES
        st = _lib.load().parason_attn_decode_no_alloc(p.handle, *([None] * 8))
        assert st == _lib.EUNSUPPORTED
    small = W.figure3_tree(values=False)
    with Plan.for_tree(small, host_only=True) as p:
        assert p.workspace_bytes <= _lib.NO_ALLOC_SCRATCH_BYTES
        st = _lib.load().parason_attn_decode_no_alloc(p.handle, *([None] * 8))
        assert st == _lib.EINVAL                            # host-only plan
    assert _lib.load().parason_attn_decode_no_alloc(None, *([None] * 8)) == _lib.EINVAL


CASES = {
    "llama3_8b_16_trials_bf16": lambda: W.make_config(2, "bf16", device="cuda"),
    "figure3_d128_g8_fp8": lambda: W.figure3_tree(mode="fp8", h_q=16, h_kv=2, d=128, trunk=300,
                                                  subtask=(130, 64, 17), device="cuda"),
    "forest_depth3_fp32": lambda: W.random_tree(5, depth=3, len_range=(0, 300), mode="fp32",
                                                device="cuda"),
}


def _assert_close(mode, got_o, got_l, ref_o, ref_l, tag):
    o = got_o.float().cpu().numpy().astype(np.float64)
    r = ref_o.float().cpu().numpy().astype(np.float64)
    assert np.isfinite(o).all(), tag
    err = float(np.abs(o - r).max(initial=0.0))
    tol = PT.FP32_MAX_ABS if mode == "fp32" else PT.BF16_MAX_ABS
    assert err <= tol, (tag, err)
    gl, rl = got_l.cpu().numpy(), ref_l.cpu().numpy()
    fin = np.isfinite(rl)
    assert np.array_equal(np.isfinite(gl), fin), tag
    assert np.array_equal(gl[~fin], rl[~fin]), tag
    if fin.any():
        assert float(np.abs(gl[fin] - rl[fin]).max()) <= PT.LSE_ABS[mode], tag


@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(CASES))
def test_no_alloc_matches_workspace_decode(name):
    build.build()
    tree = CASES[name]()
    with Plan.for_tree(tree) as plan:
        assert plan.workspace_bytes <= _lib.NO_ALLOC_SCRATCH_BYTES
        ref_o, ref_l = plan.decode_tree(tree)
        plan.check()
        for call in range(2):
            out = torch.full_like(tree.q, float("nan"))
            lse = torch.full((tree.num_leaves, tree.num_q_heads), float("nan"),
                             dtype=torch.float32, device="cuda")
            plan.decode_no_alloc(tree.q, tree.k_pages, tree.v_pages, out, lse,
                                 k_scale=tree.k_scale, v_scale=tree.v_scale)
            plan.check()
            _assert_close(tree.mode, out, lse, ref_o, ref_l, f"{name} call {call}")


@pytest.mark.gpu
def test_no_alloc_rejects_bad_arguments_like_decode():
    build.build()
    tree = W.figure3_tree(device="cuda")
    with Plan.for_tree(tree) as plan:
        out = torch.empty_like(tree.q)
        st = _lib.load().parason_attn_decode_no_alloc(plan.handle, None, None, None, None, None,
                                                      None, None, None)
        assert st == _lib.EINVAL
        with pytest.raises(ValueError):
            plan.decode_no_alloc(tree.q, tree.k_pages, tree.v_pages, out[:1])
        with pytest.raises(ParasonError):
            bad_q = torch.empty(tree.q.numel() * 2 + 8, dtype=tree.q.dtype,
                                device="cuda")[1:1 + tree.q.numel()].view_as(tree.q)
            plan.decode_no_alloc(bad_q, tree.k_pages, tree.v_pages, out)   # misaligned q
