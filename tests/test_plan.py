"""Planner work lists, checked bit-exactly against the tree (CPU only).

The checks recompute from the tree alone what the work items and merge lists
must cover, and compare exactly:
  * every (node, kv head, node row) of every node some branch reads is
    computed over every page of that node exactly once;
  * every item row maps to a (branch, q head) whose path contains the node;
  * partial slots written by items are unique and fill [0, num_slots);
  * branch b / q head h merges exactly the slots written for its row by the
    items of the nodes on its path;
  * last-page token counts match the node lengths.
"""
import collections

import numpy as np
import pytest

from paper_2608_24658_gb300 import _lib, build
from tests.plan_cover import check_tile_pairs
from paper_2608_24658_gb300.api import Plan
from paper_2608_24658_gb300 import workloads as W


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def node_of_page_pos(tree):
    """node owning each position of page_ids."""
    owner = np.full(int(tree.node_page_ptr[-1]), -1, dtype=np.int64)
    for n in range(tree.num_nodes):
        owner[tree.node_page_ptr[n]:tree.node_page_ptr[n + 1]] = n
    return owner


def verify_plan(tree, plan):
    g = tree.group
    H_kv = tree.num_kv_heads
    info = plan.info()
    items = plan.export(_lib.TABLE_ITEMS)
    dfs = plan.export(_lib.TABLE_DFS_LEAVES)
    mrng = plan.export(_lib.TABLE_MERGE_RANGES)
    ment = plan.export(_lib.TABLE_MERGE)
    assert sorted(dfs.tolist()) == list(range(tree.num_leaves))
    owner = node_of_page_pos(tree)
    paths = [set(tree.path(b)) for b in range(tree.num_leaves)]
    under = collections.defaultdict(set)
    for b, p in enumerate(paths):
        for n in p:
            under[n].add(b)

    # coverage[(node, kv_head, branch, r)] -> list of page positions covered
    coverage = collections.defaultdict(list)
    written = {}                                 # slot -> (node, kvh, branch, r)
    slots_of = collections.defaultdict(list)     # (branch, h) -> slots written for it
    blank = check_tile_pairs(plan)
    for i, it in enumerate(items):
        if i in blank:
            continue
        page_pos, npg, last_valid, leaf_lo, row0, nrows, kvh, slot_base = (int(x) for x in it)
        assert npg >= 1 and 1 <= nrows <= 128 and 0 <= kvh < H_kv
        assert row0 % g == 0, "tiles start at a multiple of g"
        n = int(owner[page_pos])
        assert n >= 0 and owner[page_pos + npg - 1] == n, "chunk crosses a node boundary"
        P = tree.node_page_ptr[n + 1] - tree.node_page_ptr[n]
        ends_node = page_pos + npg == tree.node_page_ptr[n + 1]
        want_last = int(tree.node_len[n]) - 16 * (P - 1) if ends_node else 16
        assert last_valid == want_last
        for row in range(row0, row0 + nrows):
            b = int(dfs[leaf_lo + row // g])
            r = row % g
            assert n in paths[b], "item row belongs to a branch outside the node's subtree"
            coverage[(n, kvh, b, r)].extend(range(page_pos, page_pos + npg))
            slot = slot_base + (row - row0)
            assert slot not in written, "partial slot written twice"
            written[slot] = (n, kvh, b, r)
            slots_of[(b, kvh * g + r)].append(slot)
    assert sorted(written) == list(range(info["num_slots"]))
    # every node some branch reads, every kv head, every row: all pages exactly once
    for n, bs in under.items():
        if tree.node_len[n] == 0:
            continue
        pages = list(range(tree.node_page_ptr[n], tree.node_page_ptr[n + 1]))
        for kvh in range(H_kv):
            for b in bs:
                for r in range(g):
                    assert sorted(coverage[(n, kvh, b, r)]) == pages
    # nothing computed for nodes no branch reads
    assert all(k[0] in under and tree.node_len[k[0]] > 0 for k in coverage)
    # merge lists per (branch, kv head): exactly the slots written for each q head
    # a fresh plan lays the lists out in (branch, kv head) order, end to end
    assert mrng[0, 0] == 0 and mrng[-1, 1] == len(ment) and (mrng[1:, 0] == mrng[:-1, 1]).all()
    for b in range(tree.num_leaves):
        for h in range(tree.num_q_heads):
            j, r = divmod(h, g)
            k = b * H_kv + j
            got = sorted(int(e) + r for e in ment[mrng[k, 0]:mrng[k, 1]])
            assert got == sorted(slots_of[(b, h)]), (b, h)
    assert info["unique_tokens"] == tree.unique_tokens()
    assert info["path_tokens"] == tree.path_tokens()
    # work queues: every item in exactly one queue, longest first; prefix
    # pieces belong to nodes with more than 16 rows
    wq = plan.export(_lib.TABLE_WIDE_QUEUE)
    nq = plan.export(_lib.TABLE_NARROW_QUEUE)
    if tree.mode == "fp32":
        assert len(wq) == 0 and len(nq) == 0
    else:
        assert sorted(wq.tolist() + nq.tolist()) == list(range(len(items)))
        for q in (wq, nq):
            pages = items[q, 1] if len(q) else np.zeros(0)
            assert np.all(np.diff(pages) <= 0), "queue not longest first"
        for i in wq:
            if i not in blank:
                assert len(under[int(owner[items[i][0]])]) * g > 16
        for i in nq:
            assert len(under[int(owner[items[i][0]])]) * g <= 16
        assert info["num_ctas"] <= max(info["num_sms"], 2)
        assert (info["num_wide_ctas"] > 0) == (len(wq) > 0)
    return info


CASES = {
    "figure3": lambda: W.figure3_tree(values=False),
    "tiny_fork": lambda: W.make_config(1, values=False),
    "llama3_trials": lambda: W.make_config(2, values=False),
    "two_level": lambda: W.make_config(3, values=False),
    "random_forest_0": lambda: W.random_tree(0, values=False),
    "random_forest_1": lambda: W.random_tree(1, depth=4, fanout=(0, 3), values=False),
    "random_forest_g1": lambda: W.random_tree(2, h_q=4, h_kv=4, values=False),
    "random_forest_g16": lambda: W.random_tree(3, h_q=32, h_kv=2, values=False),
    "random_forest_g6": lambda: W.random_tree(4, h_q=12, h_kv=2, values=False),
    "chain_with_empty": lambda: W.build_tree("chain", [-1, 0, 1, 2], [17, 0, 33, 5], [3],
                                             num_q_heads=6, num_kv_heads=3, head_dim=64,
                                             values=False),
    "empty_path": lambda: W.build_tree("empty", [-1, 0, 0], [0, 0, 5], [1, 2], num_q_heads=4,
                                       num_kv_heads=2, head_dim=64, values=False),
    "unused_branch_node": lambda: W.build_tree("unused", [-1, 0, 0, 1], [40, 20, 30, 9], [3],
                                               num_q_heads=4, num_kv_heads=2, head_dim=64,
                                               values=False),
    "wide_node": lambda: W.build_tree("wide", [-1] + [0] * 40, [700] + [3] * 40,
                                      list(range(1, 41)), num_q_heads=16, num_kv_heads=2,
                                      head_dim=128, values=False),
}


@pytest.mark.parametrize("name", sorted(CASES))
@pytest.mark.parametrize("mode", ["bf16", "fp32"])
def test_plan_covers_tree_exactly(name, mode):
    tree = CASES[name]()
    tree.mode = mode
    with Plan.for_tree(tree, host_only=True) as plan:
        verify_plan(tree, plan)


def test_tile_pairs_chosen_and_shaped():
    """bf16 at head_dim 128 with most prefix tile-pages in multi-tile pieces:
    pairs (blanks where a piece has an odd tile count); e4m3 and the
    two-level workload (a third of its tile-pages in single-tile pieces):
    single tiles."""
    tree = W.pair_fixture(values=False)
    with Plan.for_tree(tree, host_only=True) as plan:
        assert plan.info()["tile_pairs"] == 1
        assert len(check_tile_pairs(plan)) > 0
        verify_plan(tree, plan)
    for t in (W.pair_fixture(mode="fp8", values=False), W.make_config(3, values=False)):
        with Plan.for_tree(t, host_only=True) as plan:
            assert plan.info()["tile_pairs"] == 0
    with Plan.for_tree(W.make_config(5, values=False), host_only=True) as plan:
        assert plan.info()["tile_pairs"] == 1


@pytest.mark.parametrize("idx", [4, 5])
def test_plan_large_configs(idx):
    tree = W.make_config(idx, values=False)
    with Plan.for_tree(tree, host_only=True) as plan:
        info = plan.info()
        items = plan.export(_lib.TABLE_ITEMS)
        # partial traffic stays a small fraction of the unique KV bytes
        kv_bytes = info["unique_tokens"] * 2 * tree.num_kv_heads * tree.head_dim * 2
        part_bytes = info["num_slots"] * (tree.head_dim * 4 + 8) * 2
        assert part_bytes < 0.05 * kv_bytes, part_bytes / kv_bytes
        assert len(items) >= 152
        # pages of all items of one (kv head, first tile) sum to the unique pages
        one = items[(items[:, 6] == 0) & (items[:, 4] == 0) & (items[:, 5] > 0)]
        assert one[:, 1].sum() == sum(
            tree.node_page_ptr[n + 1] - tree.node_page_ptr[n]
            for n in range(tree.num_nodes) if tree.node_len[n] > 0)
        # suffix pieces are short against a warp's share of the suffix pages
        nq = plan.export(_lib.TABLE_NARROW_QUEUE)
        share = items[nq, 1].sum() / (info["num_sms"] * 8)
        assert items[nq, 1].max() <= max(8, share / 2), (items[nq, 1].max(), share)


def test_plan_deterministic():
    tree = W.make_config(3, values=False)
    with Plan.for_tree(tree, host_only=True) as a, Plan.for_tree(tree, host_only=True) as b:
        for t in range(4):
            assert np.array_equal(a.export(t), b.export(t))


def test_plan_sm_count_changes_split_only():
    tree = W.make_config(2, values=False)
    for sms in (1, 16, 152, 1000):
        with Plan.for_tree(tree, host_only=True, num_sms=sms) as plan:
            assert plan.info()["num_sms"] == sms
            verify_plan(tree, plan)


def test_prefix_ctas_even_out_queue_entries():
    """Decode plans give every prefix CTA the same number of prefix queue
    entries when the runs cut at one CTA's share give up to twice as many
    entries as CTAs: one each up to 3/2 (while half the SMs stay on the
    suffix queue), else two each; more entries keep the cost-model count."""
    cases = {
        (2, "bf16"): 1,      # Llama-3 shape: 24 entries, one per prefix CTA
        (3, "bf16"): 2,      # two-level: 128 entries, two per prefix CTA
    }
    for (idx, mode), per_cta in cases.items():
        tree = W.make_config(idx, mode, values=False)
        with Plan.for_tree(tree, host_only=True, num_sms=152) as plan:
            info = plan.info()
            entries = info["num_wide_items"] // (2 if info["tile_pairs"] else 1)
            assert entries == per_cta * info["num_wide_ctas"], (idx, mode, info)
            assert info["num_ctas"] == 152
            assert info["num_ctas"] - info["num_wide_ctas"] >= 152 // 2
            verify_plan(tree, plan)
    # the two-level tree with e4m3 KV: 128 entries would take 128 of 152
    # SMs one each, so it keeps the cost model's count (more than 64)
    tree = W.make_config(3, "fp8", values=False)
    with Plan.for_tree(tree, host_only=True, num_sms=152) as plan:
        info = plan.info()
        assert 64 < info["num_wide_ctas"] < info["num_wide_items"]
    # the long prefix (3 or more entries per CTA) is left to the cost model
    tree = W.make_config(5, values=False)
    with Plan.for_tree(tree, host_only=True, num_sms=152) as plan:
        info = plan.info()
        entries = info["num_wide_items"] // (2 if info["tile_pairs"] else 1)
        assert entries > 2 * info["num_wide_ctas"]
