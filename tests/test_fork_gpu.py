"""Decode after parason_plan_fork (and appends around it), through the C
ABI, against the fp64 oracle on the grown tree; and against a plan built
for that tree."""
import numpy as np
import pytest
import torch

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan, ParasonError
from tests import parity as PT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()
    torch.cuda.init()


CASES = {
    # a trunk shared by 24 branches (tcgen05 prefix tile), g = 4
    "bf16_d128": lambda: W.build_tree("fork-a", [-1, 0, 0] + [1] * 12 + [2] * 12,
                                      [700, 60, 33] + [int(x) for x in np.arange(24) * 9 + 1],
                                      list(range(3, 27)), num_q_heads=16, num_kv_heads=4,
                                      head_dim=128, mode="bf16", seed=21, extra_pages=300,
                                      device="cuda"),
    "fp8_g8": lambda: W.build_tree("fork-b", [-1, 0, 0, 0], [300, 31, 16, 2], [1, 2, 3],
                                   num_q_heads=16, num_kv_heads=2, head_dim=128, mode="fp8",
                                   seed=22, extra_pages=200, device="cuda"),
    "bf16_d64": lambda: W.build_tree("fork-c", [-1, 0, 0, 1], [90, 20, 7, 15], [2, 3],
                                     num_q_heads=8, num_kv_heads=2, head_dim=64, mode="bf16",
                                     seed=23, extra_pages=200, device="cuda"),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_decode_after_forks_matches_oracle(case):
    rng = np.random.default_rng(3)
    tree = CASES[case]()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree) as plan:
        for step in range(12):
            if step in (1, 5, 8):
                b = int(rng.integers(0, tree.num_leaves))
                lens = [int(x) for x in rng.integers(1, 40, size=3)]
                tree, pages = W.fork_branch(tree, b, lens, pool, seed=step)
                plan.fork(b, lens, pages)
            else:
                tree, new_pages = W.grow_branches(tree, pool)
                plan.append(new_pages)
            out, lse = plan.decode_tree(tree)
            plan.check()
            ref_o, ref_l = PT.oracle_decode(tree)
            PT.compare(tree, out, lse, ref_o, ref_l, tag=f"{case} step {step}")
    with Plan.for_tree(tree) as fresh:
        out2, lse2 = fresh.decode_tree(tree)
        fresh.check()
    assert float((out.float() - out2.float()).abs().max()) <= PT.BF16_MAX_ABS
    assert float((lse - lse2).abs().max()) <= PT.LSE_ABS[tree.mode]


def test_failed_fork_keeps_device_and_host_plans_in_step():
    tree = CASES["bf16_d128"]()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree) as plan:
        grown, pages = W.fork_branch(tree, 4, [5, 9, 1], list(pool))
        plan.set_debug(_lib.DEBUG_FAIL_UPDATE)
        with pytest.raises(ParasonError) as e:
            plan.fork(4, [5, 9, 1], pages)
        assert e.value.status == _lib.ECUDA
        plan.set_debug(0)
        out, lse = plan.decode_tree(tree)
        plan.check()
        ref_o, ref_l = PT.oracle_decode(tree)
        PT.compare(tree, out, lse, ref_o, ref_l, tag="after a failed fork")
        plan.fork(4, [5, 9, 1], pages)
        out, lse = plan.decode_tree(grown)
        plan.check()
        ref_o, ref_l = PT.oracle_decode(grown)
        PT.compare(grown, out, lse, ref_o, ref_l, tag="after the retried fork")


def test_fork_of_a_plan_without_work():
    # every node empty: the plan has no attention grid until the fork
    tree = W.build_tree("empty", [-1, 0], [0, 0], [1], num_q_heads=8, num_kv_heads=2,
                        head_dim=128, seed=24, extra_pages=20, device="cuda")
    pool = W.free_pages(tree)
    with Plan.for_tree(tree) as plan:
        tree, pages = W.fork_branch(tree, 0, [20, 3], pool)
        plan.fork(0, [20, 3], pages)
        out, lse = plan.decode_tree(tree)
        plan.check()
        ref_o, ref_l = PT.oracle_decode(tree)
        PT.compare(tree, out, lse, ref_o, ref_l, tag="fork of an empty plan")
