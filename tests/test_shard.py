"""Sharded plans (parason_attn_plan_shard) on CPU: two gloo ranks each plan
their part of a decode step, and the union of what their branches attend to
is, bit for bit, what the unsharded plan's branches attend to -- every
(branch, kv head) reads the same physical pages with the same valid-token
counts, and no (branch, kv head) is computed by two ranks.  The decode step
needs no exchange between ranks (Sec. 3.4: branches are independent workers,
requests do not share KV; grouped kv heads are independent), so matching
coverage is the whole correctness condition of the split."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan, ParasonError
from tests.plan_cover import coverage, definition

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def shard_tree():
    # 6 requests of different sizes, nested regions, permuted pages
    return W.random_tree(21, num_requests=6, depth=2, fanout=(1, 4), len_range=(0, 120), h_q=16,
                         h_kv=4, d=128, values=False)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    from paper_2608_24658_gb300 import _lib as L
    from paper_2608_24658_gb300.api import Plan as P
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        tree = shard_tree()
        res = {}
        for kind in (L.SHARD_REQUESTS, L.SHARD_KV_HEADS):
            with P.for_tree(tree, host_only=True, shard=(kind, rank, world)) as p:
                head0 = rank * tree.num_kv_heads // world if kind == L.SHARD_KV_HEADS else 0
                res[kind] = coverage(p, head0)
        gathered = [None] * world
        dist.all_gather_object(gathered, res)
        out_q.put((rank, gathered))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_cover_the_unsharded_plan():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    tree = shard_tree()
    with Plan.for_tree(tree, host_only=True) as full:
        want = coverage(full)
    assert want == definition(tree)
    for r in range(2):                            # every rank saw the same gathered result
        assert res[r] == res[0]
    for kind in (_lib.SHARD_REQUESTS, _lib.SHARD_KV_HEADS):
        parts = [res[0][r][kind] for r in range(2)]
        assert parts[0] and parts[1], "both ranks got work"
        assert not set(parts[0]) & set(parts[1]), "a (branch, kv head) on both ranks"
        union = {**parts[0], **parts[1]}
        assert union == want


@pytest.mark.parametrize("world", [1, 2, 3, 4, 8])
def test_request_shards_partition_the_branches(world):
    tree = W.make_config(4, values=False)        # 32 requests x 32 branches
    seen, costs = [], []
    for r in range(world):
        with Plan.for_tree(tree, host_only=True, shard=(_lib.SHARD_REQUESTS, r, world)) as p:
            br = p.export(_lib.TABLE_SHARD_BRANCHES)
            assert (np.diff(br) > 0).all()       # global order kept
            seen.extend(br.tolist())
            costs.append(p.info()["unique_tokens"])
    assert sorted(seen) == list(range(tree.num_leaves))
    # contiguous request groups of about equal cost
    assert max(costs) <= 1.2 * (sum(costs) / world) + 8192


def test_more_ranks_than_requests_gives_empty_plans():
    tree = W.figure3_tree(values=False)          # one request
    with Plan.for_tree(tree, host_only=True, shard=(_lib.SHARD_REQUESTS, 1, 2)) as p:
        assert p.num_leaves == 0 and p.info()["num_items"] == 0
    with Plan.for_tree(tree, host_only=True, shard=(_lib.SHARD_REQUESTS, 0, 2)) as p:
        assert p.num_leaves == tree.num_leaves


def test_shard_arguments_are_checked():
    tree = W.figure3_tree(values=False)          # 2 kv heads
    for shard in [(_lib.SHARD_REQUESTS, 2, 2), (_lib.SHARD_REQUESTS, -1, 2),
                  (_lib.SHARD_REQUESTS, 0, 0), (_lib.SHARD_KV_HEADS, 0, 3), (7, 0, 1)]:
        with pytest.raises(ParasonError) as e:
            Plan.for_tree(tree, host_only=True, shard=shard)
        assert e.value.status == _lib.EINVAL
    bad = W.figure3_tree(values=False)
    bad.parent = bad.parent.copy()
    bad.parent[3] = 5                               # a parent after its child, in another shard
    with pytest.raises(ParasonError) as e:
        Plan.for_tree(bad, host_only=True, shard=(_lib.SHARD_REQUESTS, 0, 1))
    assert e.value.status == _lib.EINVAL
