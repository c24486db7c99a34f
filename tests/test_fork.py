"""parason_plan_fork on host plans (CPU): after every fork -- and appends
before and after it -- each (branch, kv head) merges exactly the pages of its
path in the grown tree with the right valid-token counts, partial slots are
written once, and refused forks change nothing."""
import numpy as np
import pytest

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan, ParasonError
from tests.plan_cover import check_tile_pairs, coverage, definition


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def check(tree, plan):
    assert plan.num_leaves == tree.num_leaves
    assert coverage(plan) == definition(tree)
    items = plan.export(_lib.TABLE_ITEMS)
    info = plan.info()
    seen = np.zeros(info["num_slots"], dtype=np.int64)
    for it in items:
        seen[int(it[7]):int(it[7]) + int(it[5])] += 1
    assert (seen == 1).all(), "a partial slot is written by no item or by two"
    assert info["unique_tokens"] == tree.unique_tokens()
    assert info["path_tokens"] == tree.path_tokens()
    nq = plan.export(_lib.TABLE_NARROW_QUEUE)
    wq = plan.export(_lib.TABLE_WIDE_QUEUE)
    assert sorted(wq.tolist() + nq.tolist()) == list(range(len(items)))
    check_tile_pairs(plan)


def base_tree(mode="bf16", **kw):
    # one request: a trunk, two subtask threads, four branches near page edges
    return W.build_tree("fork", [-1, 0, 0, 1, 1, 2, 2], [100, 33, 16, 15, 47, 1, 32],
                        [3, 4, 5, 6], num_q_heads=16, num_kv_heads=4, head_dim=128, mode=mode,
                        seed=5, extra_pages=200, values=False, **kw)


@pytest.mark.parametrize("lens", [[1, 1, 1], [17], [16, 40, 1, 33], [0, 5]])
def test_fork_covers_the_grown_tree(lens):
    tree = base_tree()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        ws0 = plan.workspace_bytes
        grown, pages = W.fork_branch(tree, 2, lens, pool)
        ids = plan.fork(2, lens, pages)
        assert ids == [2] + list(range(tree.num_leaves, tree.num_leaves + len(lens) - 1))
        check(grown, plan)
        assert plan.workspace_bytes > ws0


def test_forks_and_appends_interleaved():
    """Thirty decode steps: a token on every branch each step, forks of
    random branches (new ones and nested ones included) every few steps."""
    rng = np.random.default_rng(7)
    tree = base_tree()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        for step in range(30):
            if step % 4 == 1:
                b = int(rng.integers(0, tree.num_leaves))
                lens = [int(x) for x in rng.integers(1, 20, size=int(rng.integers(1, 4)))]
                tree, pages = W.fork_branch(tree, b, lens, pool)
                plan.fork(b, lens, pages)
            else:
                tree, new_pages = W.grow_branches(tree, pool)
                plan.append(new_pages)
            check(tree, plan)
        assert tree.num_leaves > 4


@pytest.mark.parametrize("idx", [2, 3])
def test_fork_on_the_workloads(idx):
    # the Llama-3 shape (g = 4) and the two-level tree (g = 8): a trial
    # branch opens four threads, then one of them three more
    tree = W.make_config(idx, values=False, extra_pages=256)
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        tree, pages = W.fork_branch(tree, 5, [1, 1, 1, 1], pool)
        plan.fork(5, [1, 1, 1, 1], pages)
        check(tree, plan)
        b = tree.num_leaves - 1
        tree, pages = W.fork_branch(tree, b, [3, 1, 2], pool)
        plan.fork(b, [3, 1, 2], pages)
        check(tree, plan)


def snapshot(plan):
    tabs = [_lib.TABLE_ITEMS, _lib.TABLE_DFS_LEAVES, _lib.TABLE_MERGE_RANGES, _lib.TABLE_MERGE,
            _lib.TABLE_NARROW_QUEUE, _lib.TABLE_ITEM_ROWS, _lib.TABLE_STREAM_ROWS]
    return [plan.export(t).copy() for t in tabs] + [plan.info(), plan.workspace_bytes]


def same(a, b):
    for x, y in zip(a, b):
        if isinstance(x, np.ndarray):
            assert np.array_equal(x, y)
        else:
            assert x == y


def test_refused_forks_change_nothing():
    tree = base_tree()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        before = snapshot(plan)
        owned = int(tree.page_ids[0])
        free = W.free_pages(tree)
        cases = [
            (9, [1], [[free[0]]], _lib.EINVAL),                    # no such branch
            (-1, [1], [[free[0]]], _lib.EINVAL),
            (0, [1, 1], [[owned], [free[0]]], _lib.EINVAL),        # a page some node owns
            (0, [1, 1], [[free[0]], [free[0]]], _lib.EINVAL),      # the same page twice
            (0, [17], [[free[0]]], _lib.EINVAL),                   # 17 tokens need two pages
            (0, [-1], [[]], _lib.EINVAL),
            (0, [1], [[tree.num_physical_pages]], _lib.EINVAL),    # out of range
        ]
        for b, lens, pages, status in cases:
            with pytest.raises(ParasonError) as e:
                plan.fork(b, lens, pages)
            assert e.value.status == status, (b, lens, pages)
            same(before, snapshot(plan))
        with pytest.raises(ParasonError) as e:
            plan.fork(0, [], [])
        assert e.value.status == _lib.EINVAL
        # a failed device step (simulated) leaves everything, page claims included
        grown, pages = W.fork_branch(tree, 1, [3, 3], list(pool))
        plan.set_debug(_lib.DEBUG_FAIL_UPDATE)
        with pytest.raises(ParasonError) as e:
            plan.fork(1, [3, 3], pages)
        assert e.value.status == _lib.ECUDA
        same(before, snapshot(plan))
        plan.set_debug(0)
        plan.fork(1, [3, 3], pages)
        check(grown, plan)


def test_unsupported_forks():
    t32 = base_tree(mode="fp32")
    with Plan.for_tree(t32, host_only=True) as plan:
        with pytest.raises(ParasonError) as e:
            plan.fork(0, [1], [[W.free_pages(t32)[0]]])
        assert e.value.status == _lib.EUNSUPPORTED
    wide = W.build_tree("g32", [-1, 0, 0], [40, 5, 6], [1, 2], num_q_heads=64, num_kv_heads=2,
                        head_dim=128, seed=1, extra_pages=8, values=False)
    with Plan.for_tree(wide, host_only=True) as plan:
        with pytest.raises(ParasonError) as e:
            plan.fork(0, [1], [[W.free_pages(wide)[0]]])
        assert e.value.status == _lib.EUNSUPPORTED      # 32 q heads per kv head
    pre = W.fork_prefill(values=False)
    with Plan.for_prefill(pre, host_only=True) as plan:
        with pytest.raises(ParasonError) as e:
            plan.fork(0, [1], [[0]])
        assert e.value.status == _lib.EUNSUPPORTED


def test_forks_until_no_room():
    """The plan keeps room for forks; past it a fork is refused with
    PARASON_ENOSPACE and the plan stays exact for the tree as it was."""
    tree = W.build_tree("small", [-1, 0], [20, 3], [1], num_q_heads=4, num_kv_heads=2,
                        head_dim=64, seed=3, extra_pages=600, values=False)
    pool = W.free_pages(tree)
    status = None
    with Plan.for_tree(tree, host_only=True) as plan:
        for _ in range(200):
            b = tree.num_leaves - 1
            grown, pages = W.fork_branch(tree, b, [1, 1], list(pool))
            try:
                plan.fork(b, [1, 1], pages)
            except ParasonError as e:
                status = e.status
                break
            tree = grown
            used = {x for p in pages for x in p}
            pool = [p for p in pool if p not in used]
        assert status == _lib.ENOSPACE
        check(tree, plan)


def test_zero_length_child_takes_no_appends():
    tree = base_tree()
    pool = W.free_pages(tree)
    with Plan.for_tree(tree, host_only=True) as plan:
        tree, pages = W.fork_branch(tree, 0, [0, 2], pool)
        plan.fork(0, [0, 2], pages)
        check(tree, plan)
        with pytest.raises(ParasonError) as e:
            plan.append(W.grow_branches(tree, list(pool))[1])
        assert e.value.status == _lib.ENOSPACE
