"""parason_attn_decode_no_alloc (the decode step with the library's fixed
per-device scratch instead of a caller workspace) against parason_attn_decode
with a workspace, on the same plan and inputs, two calls in a row.

Collected last on purpose: it must also pass after every other test has run
kernels, planned and freed memory on the same device.
"""
import pytest
import torch

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan, ParasonError


def test_plan_over_scratch_limit_is_rejected_first():
    """No device work: the size check comes before any other."""
    build.build()
    big = W.batched_serving(requests=64, values=False)     # 2048 branches
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


def _assert_same(got_o, got_l, ref_o, ref_l, tag):
    """Bit-identical: the decode is deterministic (each work item runs the
    same code whichever warp pulls it, and the merge order is fixed), so the
    scratch-backed call must reproduce the workspace call exactly; any
    offset or alignment slip in the scratch would show here."""
    assert torch.equal(got_o, ref_o), tag
    assert torch.equal(got_l, ref_l), tag


def _no_alloc(plan, tree):
    out = torch.full_like(tree.q, float("nan"))
    lse = torch.full((tree.num_leaves, tree.num_q_heads), float("nan"), dtype=torch.float32,
                     device="cuda")
    plan.decode_no_alloc(tree.q, tree.k_pages, tree.v_pages, out, lse, k_scale=tree.k_scale,
                         v_scale=tree.v_scale)
    plan.check()
    return out, lse


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
            out, lse = _no_alloc(plan, tree)
            _assert_same(out, lse, ref_o, ref_l, f"{name} call {call}")


@pytest.mark.gpu
def test_no_alloc_larger_then_smaller_plan_share_the_scratch():
    """Two different plans one after the other through the one scratch array:
    the smaller plan's call finds the larger one's partials there and must
    not read them."""
    build.build()
    big = W.make_config(3, "bf16", device="cuda")          # 64 branches, two levels
    small = W.make_config(2, "bf16", device="cuda")        # 16 branches
    with Plan.for_tree(big) as pb, Plan.for_tree(small) as ps:
        assert ps.workspace_bytes < pb.workspace_bytes <= _lib.NO_ALLOC_SCRATCH_BYTES
        ref_b = pb.decode_tree(big)
        ref_s = ps.decode_tree(small)
        pb.check()
        ps.check()
        for tag, plan, tree, ref in (("big", pb, big, ref_b), ("small", ps, small, ref_s),
                                     ("big again", pb, big, ref_b)):
            out, lse = _no_alloc(plan, tree)
            _assert_same(out, lse, ref[0], ref[1], tag)


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
