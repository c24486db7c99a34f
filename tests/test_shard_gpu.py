"""Every rank's plan of a sharded decode step (parason_attn_plan_shard), run
one after another on one GPU with the rank's own q / K / V views, against
the fp64 oracle and against the unsharded decode.  The ranks never wait on
one another (the split needs no exchange), so running them in turn on one
GPU exercises exactly what each GPU of a sharded run would compute."""
import numpy as np
import pytest
import torch

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan
from tests import parity as PT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()
    torch.cuda.init()


def forest(mode):
    # 5 requests of different sizes, nested regions, permuted pages; g = 4
    return W.random_tree(31, num_requests=5, depth=2, fanout=(1, 4), len_range=(1, 300), h_q=16,
                         h_kv=4, d=128, mode=mode, device="cuda")


@pytest.mark.parametrize("mode", ["bf16", "fp8"])
@pytest.mark.parametrize("world", [2, 3])
def test_request_shards_decode_like_the_whole(mode, world):
    tree = forest(mode)
    with Plan.for_tree(tree) as full:
        ref_o, ref_l = full.decode_tree(tree)
        full.check()
    got_o = torch.full_like(ref_o, float("nan"))
    got_l = torch.full_like(ref_l, float("nan"))
    for rank in range(world):
        with Plan.for_tree(tree, shard=(_lib.SHARD_REQUESTS, rank, world)) as p:
            br = torch.as_tensor(p.export(_lib.TABLE_SHARD_BRANCHES), dtype=torch.long,
                                 device="cuda")
            if p.num_leaves == 0:
                continue
            q = tree.q.index_select(0, br).contiguous()
            o, l = p.decode(q, tree.k_pages, tree.v_pages, k_scale=tree.k_scale,
                            v_scale=tree.v_scale)
            p.check()
            got_o[br], got_l[br] = o, l
    assert torch.isfinite(got_o.float()).all()
    ref = PT.oracle_decode(tree)
    PT.compare(tree, got_o, got_l, ref[0], ref[1], tag=f"request shards of {world}")
    # the same work item for item, up to the order of the split
    assert float((got_o.float() - ref_o.float()).abs().max()) <= PT.BF16_MAX_ABS


@pytest.mark.parametrize("world", [2, 4])
def test_kv_head_shards_decode_like_the_whole(world):
    tree = forest("bf16")
    ref = PT.oracle_decode(tree)
    got_o = torch.full_like(tree.q, float("nan"))
    got_l = torch.full(tree.q.shape[:2], float("nan"), dtype=torch.float32, device="cuda")
    hk = tree.num_kv_heads // world
    g = tree.group
    for rank in range(world):
        with Plan.for_tree(tree, shard=(_lib.SHARD_KV_HEADS, rank, world)) as p:
            qs = slice(rank * hk * g, (rank + 1) * hk * g)
            ks = slice(rank * hk, (rank + 1) * hk)
            o, l = p.decode(tree.q[:, qs].contiguous(), tree.k_pages[:, ks].contiguous(),
                            tree.v_pages[:, ks].contiguous())
            p.check()
            got_o[:, qs], got_l[:, qs] = o, l
    PT.compare(tree, got_o, got_l, ref[0], ref[1], tag=f"kv-head shards of {world}")
