"""parason_plan_append on host plans (CPU): after every step the plan's work
items, read through the TMA rows the kernels load, cover the grown tree's
pages exactly once per (node, kv head, row tile), with the right last-page
counts; refused appends change nothing."""
import collections

import numpy as np
import pytest

from paper_2608_24658_gb300 import _lib, build
from tests.plan_cover import check_tile_pairs
from paper_2608_24658_gb300.api import Plan, ParasonError
from paper_2608_24658_gb300 import workloads as W


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def verify_rows(tree, plan):
    H = tree.num_kv_heads
    g = tree.group
    items = plan.export(_lib.TABLE_ITEMS)
    irows = plan.export(_lib.TABLE_ITEM_ROWS)
    srows = plan.export(_lib.TABLE_STREAM_ROWS)
    owner, index = {}, {}
    for n in range(tree.num_nodes):
        for k, pg in enumerate(tree.page_ids[tree.node_page_ptr[n]:tree.node_page_ptr[n + 1]]):
            owner[int(pg)], index[int(pg)] = n, k
    cover = collections.defaultdict(list)
    rows_of = collections.defaultdict(set)
    blank = check_tile_pairs(plan)
    for i, it in enumerate(items):
        if i in blank:
            continue
        _, npg, last_valid, _, row0, nrows, kvh, _ = (int(x) for x in it)
        r = srows[irows[i]:irows[i] + npg].astype(np.int64)
        assert (r % 16 == 0).all()
        pages, heads = r // 16 // H, (r // 16) % H
        assert (heads == kvh).all()
        n = owner[int(pages[0])]
        assert all(owner[int(p)] == n for p in pages), "item crosses nodes"
        idx = [index[int(p)] for p in pages]
        assert idx == list(range(idx[0], idx[0] + npg)), "pages not consecutive"
        P = tree.node_page_ptr[n + 1] - tree.node_page_ptr[n]
        want = int(tree.node_len[n]) - 16 * (P - 1) if idx[-1] == P - 1 else 16
        assert last_valid == want
        cover[(n, kvh, row0)].extend(idx)
        rows_of[(n, kvh)].update(range(row0, row0 + nrows))
    read = set(m for b in range(tree.num_leaves) for m in tree.path(b))
    under = tree.leaves_under()
    for n in read:
        if tree.node_len[n] == 0:
            continue
        P = tree.node_page_ptr[n + 1] - tree.node_page_ptr[n]
        for kvh in range(H):
            assert rows_of[(n, kvh)] == set(range(int(under[n]) * g)), (n, kvh)
            tiles = [k for k in cover if k[0] == n and k[1] == kvh]
            for k in tiles:
                assert sorted(cover[k]) == list(range(P)), (n, kvh, k)


def make_tree(mode="bf16", seed=3, **kw):
    # branch nodes at lengths around page boundaries; room to grow
    return W.build_tree("grow", [-1, 0, 0, 0, 1, 1], [70, 33, 16, 1, 15, 47], [2, 3, 4, 5],
                        num_q_heads=8, num_kv_heads=2, head_dim=128, mode=mode, seed=seed,
                        extra_pages=40, values=False, **kw)


@pytest.mark.parametrize("mode", ["bf16", "fp8"])
def test_appends_keep_the_plan_exact(mode):
    tree = make_tree(mode)
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        verify_rows(tree, plan)
        for step in range(40):
            tree, new_pages = W.grow_branches(tree, pool)
            plan.append(new_pages)
            verify_rows(tree, plan)
        info = plan.info()
        assert info["unique_tokens"] == tree.unique_tokens()


def test_appends_on_wide_leaves():
    # 64 q heads over 2 kv heads: a branch node has 32 rows, a prefix-pass run
    tree = W.build_tree("wide-leaves", [-1, 0, 0], [300, 31, 64], [1, 2], num_q_heads=64,
                        num_kv_heads=2, head_dim=128, seed=1, extra_pages=30, values=False)
    pool = W.free_pages(tree)
    plan = Plan.for_tree(tree, host_only=True)
    rebuilds = 0
    for _ in range(70):
        nxt, new_pages = W.grow_branches(tree, list(pool))
        try:
            plan.append(new_pages)
        except ParasonError as e:
            # out of room: the caller builds a plan for the tree as it is
            assert e.status == _lib.ENOSPACE
            plan.close()
            plan = Plan.for_tree(tree, host_only=True)
            rebuilds += 1
            plan.append(new_pages)
        tree = nxt
        used = set(int(x) for x in new_pages)
        pool = [p for p in pool if p not in used]
        verify_rows(tree, plan)
    plan.close()
    assert rebuilds >= 1


def snapshot(plan):
    return [plan.export(t).copy() for t in (_lib.TABLE_ITEMS, _lib.TABLE_ITEM_ROWS,
                                            _lib.TABLE_STREAM_ROWS)]


def test_refused_appends_change_nothing():
    tree = make_tree()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        before = snapshot(plan)
        _, new_pages = W.grow_branches(tree, list(pool))
        bad = new_pages.copy()
        b = int(np.flatnonzero(bad >= 0)[0])
        bad[b] = int(tree.page_ids[0])                      # a page some node owns
        with pytest.raises(ParasonError) as e:
            plan.append(bad)
        assert e.value.status == _lib.EINVAL
        with pytest.raises(ParasonError) as e:
            plan.append(None)                              # a branch needs a page
        assert e.value.status == _lib.EINVAL
        bad[b] = tree.num_physical_pages                    # out of range
        with pytest.raises(ParasonError):
            plan.append(bad)
        for x, y in zip(before, snapshot(plan)):
            assert np.array_equal(x, y)


def test_no_room_after_the_slack():
    tree = W.build_tree("long", [-1, 0], [16, 16], [1], num_q_heads=8, num_kv_heads=2,
                        head_dim=64, seed=2, extra_pages=80, values=False)
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        status = None
        for step in range(16 * 80):
            nxt, new_pages = W.grow_branches(tree, list(pool))
            try:
                plan.append(new_pages)
            except ParasonError as e:
                status = e.status
                break
            tree = nxt
            pool = [p for p in pool if p not in set(int(x) for x in new_pages)]
        assert status == _lib.ENOSPACE
        verify_rows(tree, plan)             # still consistent with the last accepted step


def test_empty_branch_node_needs_a_new_plan():
    tree = W.build_tree("empty-leaf", [-1, 0, 0], [20, 0, 5], [1, 2], num_q_heads=8,
                        num_kv_heads=2, head_dim=64, seed=2, extra_pages=4, values=False)
    with Plan.for_tree(tree, host_only=True) as plan:
        with pytest.raises(ParasonError) as e:
            plan.append(np.array([W.free_pages(tree)[0], -1], dtype=np.int32))
        assert e.value.status == _lib.ENOSPACE


def test_fp32_plans_do_not_append():
    tree = W.build_tree("f", [-1, 0], [20, 5], [1], num_q_heads=8, num_kv_heads=2, head_dim=64,
                        mode="fp32", seed=2, values=False)
    with Plan.for_tree(tree, host_only=True) as plan:
        with pytest.raises(ParasonError) as e:
            plan.append(None)
        assert e.value.status == _lib.EUNSUPPORTED


def test_failed_device_update_changes_nothing():
    """An append whose device step fails (simulated by a debug flag, at the
    point where the device copy would be patched) changes neither the plan's
    tables nor its page accounting: retrying with the same pages succeeds."""
    tree = make_tree()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        for _ in range(3):
            tree, new_pages = W.grow_branches(tree, pool)
            plan.append(new_pages)
        while True:                                          # up to a step that opens a page
            grown, new_pages = W.grow_branches(tree, list(pool))
            if (new_pages >= 0).any():
                break
            tree, _ = W.grow_branches(tree, pool)
            plan.append(None)
        before = snapshot(plan)
        info_before = plan.info()
        plan.set_debug(_lib.DEBUG_FAIL_UPDATE)
        for _ in range(2):
            with pytest.raises(ParasonError) as e:
                plan.append(new_pages)
            assert e.value.status == _lib.ECUDA
            for x, y in zip(before, snapshot(plan)):
                assert np.array_equal(x, y)
            assert plan.info() == info_before
        verify_rows(tree, plan)
        plan.set_debug(0)
        plan.append(new_pages)                               # the pages were not kept
        verify_rows(grown, plan)
