"""Decode after parason_plan_append, through the C ABI, against the fp64
oracle on the grown tree: every few steps and at every step that opens a
page, for bf16 and e4m3 KV and for branch nodes on the prefix pass."""
import numpy as np
import pytest
import torch

from paper_2608_24658_gb300 import build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan
from tests import parity as PT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()
    torch.cuda.init()


CASES = {
    # branch nodes at lengths around page boundaries, suffix pass
    "bf16": lambda: W.build_tree("grow", [-1, 0, 0, 0, 1, 1], [70, 33, 16, 1, 15, 47], [2, 3, 4, 5],
                                 num_q_heads=8, num_kv_heads=2, head_dim=128, mode="bf16", seed=3,
                                 extra_pages=24, device="cuda"),
    "fp8": lambda: W.build_tree("grow8", [-1, 0, 0, 0], [200, 31, 16, 2], [1, 2, 3],
                                num_q_heads=16, num_kv_heads=2, head_dim=128, mode="fp8", seed=4,
                                extra_pages=24, device="cuda"),
    # 32 rows per branch node: the prefix pass (tcgen05 tile) holds the branches
    "wide_leaves": lambda: W.build_tree("grow-wide", [-1, 0, 0], [300, 31, 64], [1, 2],
                                        num_q_heads=64, num_kv_heads=2, head_dim=128, mode="bf16",
                                        seed=5, extra_pages=16, device="cuda"),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_decode_after_appends_matches_oracle(case):
    tree = CASES[case]()
    pool = W.free_pages(tree)
    checked = 0
    with Plan.for_tree(tree) as plan:
        for step in range(40):
            tree, new_pages = W.grow_branches(tree, pool)
            plan.append(new_pages)
            if step % 7 == 6 or (new_pages >= 0).any():
                out, lse = plan.decode_tree(tree)
                plan.check()
                ref_o, ref_l = PT.oracle_decode(tree)
                PT.compare(tree, out, lse, ref_o, ref_l, tag=f"{case} step {step}")
                checked += 1
        # the appended plan and a plan built for the grown tree agree
        out, lse = plan.decode_tree(tree)
        plan.check()
    with Plan.for_tree(tree) as fresh:
        out2, lse2 = fresh.decode_tree(tree)
        fresh.check()
    assert checked >= 6
    assert float((out.float() - out2.float()).abs().max()) <= PT.BF16_MAX_ABS
    assert float((lse - lse2).abs().max()) <= PT.LSE_ABS[tree.mode]


def test_failed_update_keeps_device_and_host_plans_in_step():
    """A refused device update leaves both copies of the plan as they were:
    the next decode is the old tree's result, and after a successful retry
    the grown tree's (both against the oracle)."""
    from paper_2608_24658_gb300 import _lib
    from paper_2608_24658_gb300.api import ParasonError
    tree = CASES["bf16"]()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree) as plan:
        grown, new_pages = W.grow_branches(tree, list(pool))
        plan.set_debug(_lib.DEBUG_FAIL_UPDATE)
        with pytest.raises(ParasonError) as e:
            plan.append(new_pages)
        assert e.value.status == _lib.ECUDA
        plan.set_debug(0)
        out, lse = plan.decode_tree(tree)
        plan.check()
        ref_o, ref_l = PT.oracle_decode(tree)
        PT.compare(tree, out, lse, ref_o, ref_l, tag="after a failed append")
        plan.append(new_pages)
        out, lse = plan.decode_tree(grown)
        plan.check()
        ref_o, ref_l = PT.oracle_decode(grown)
        PT.compare(grown, out, lse, ref_o, ref_l, tag="after the retried append")
