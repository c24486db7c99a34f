"""Tree-masked prefill plans (parason_prefill_plan_host), checked against the
tree alone (CPU only): for every query (token t of chunk c) and q head, the
partial slots its merge list names see, between them, every token of every
ancestor of the chunk's node and tokens 0 .. t of the node itself, each
exactly once; no slot is written twice; every key an item's row sees passes
the causal rule; and the unsupported forms are refused."""
import collections

import numpy as np
import pytest

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300 import workloads as W
from tests.plan_cover import check_tile_pairs
from paper_2608_24658_gb300.api import Plan, ParasonError


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def ancestors(tree, n):
    out = []
    n = int(tree.parent[n])
    while n >= 0:
        out.append(n)
        n = int(tree.parent[n])
    return out


def item_keys(tree, it, rows):
    """(node, token) of every stream position of an item (None where a page
    ends a node or the item's last page ends, and in padding), read from its
    page rows: row (page * H_kv + kv head) * 16, plus 16 - valid tokens in the
    low bits of a page that ends a node inside the item; padding pages carry
    the first row past the pool and only follow a page that ends a node, up to
    the next 64-token block."""
    H = tree.num_kv_heads
    npg, last_valid, kvh = int(it[1]), int(it[2]), int(it[6])
    where = {int(pg): i for i, pg in enumerate(tree.page_ids)}
    pad_row = tree.num_physical_pages * H * 16
    keys = []
    for k, row in enumerate(int(x) for x in rows):
        if row == pad_row:
            assert 0 < k < npg - 1 and k % 4 != 0, "padding ends a block, never an item"
            assert keys[16 * k - 1] is None, "padding follows a page that ends a node"
            keys.extend([None] * 16)
            continue
        short, base = row & 15, row >> 4
        assert base % H == kvh
        assert k < npg - 1 or short == 0, "the last page goes by last_valid"
        valid = last_valid if k == npg - 1 else 16 - short
        pos = where[base // H]
        n = int(np.searchsorted(tree.node_page_ptr, pos, side="right")) - 1
        idx = pos - int(tree.node_page_ptr[n])
        P = int(tree.node_page_ptr[n + 1] - tree.node_page_ptr[n])
        node_valid = int(tree.node_len[n]) - 16 * (P - 1) if idx == P - 1 else 16
        assert valid == node_valid, "a page's valid tokens are the node's"
        keys.extend((n, 16 * idx + x) if x < valid else None for x in range(16))
    return keys


def verify_prefill_plan(tree, plan):
    g, H_kv = tree.group, tree.num_kv_heads
    chunks = [int(c) for c in tree.leaf_node]
    lens = [int(tree.node_len[c]) for c in chunks]
    qbase = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    Q = int(qbase[-1])
    info = plan.info()
    assert info["num_leaves"] == Q
    items = plan.export(_lib.TABLE_ITEMS)
    key0 = plan.export(_lib.TABLE_ITEM_KEY0)
    dfs = plan.export(_lib.TABLE_DFS_LEAVES)
    mrng = plan.export(_lib.TABLE_MERGE_RANGES)
    ment = plan.export(_lib.TABLE_MERGE)
    wq = plan.export(_lib.TABLE_WIDE_QUEUE)
    nq = plan.export(_lib.TABLE_NARROW_QUEUE)
    irows = plan.export(_lib.TABLE_ITEM_ROWS)
    srows = plan.export(_lib.TABLE_STREAM_ROWS)
    assert dfs.tolist() == list(range(Q))
    assert len(key0) == len(items)
    assert len(nq) == 0 and wq.tolist() == list(range(len(items)))    # all on the tcgen05 tile

    blank = check_tile_pairs(plan)
    seen = {}                                        # slot -> (query, q head, visible keys)
    for i, (it, k0) in enumerate(zip(items, key0)):
        if i in blank:
            assert int(k0) == -1
            continue
        page_pos, npg, last_valid, leaf_lo, row0, nrows, kvh, slot_base = (int(x) for x in it)
        assert 1 <= nrows <= 128 and row0 % g == 0 and 0 <= kvh < H_kv and npg >= 1
        c = int(np.searchsorted(qbase, leaf_lo, side="right")) - 1
        assert qbase[c] == leaf_lo, "an item's rows start at its chunk's first query"
        keys = item_keys(tree, it, srows[irows[i]:irows[i] + npg])
        path = set(ancestors(tree, chunks[c])) | {chunks[c]}
        assert all(k is None or k[0] in path for k in keys), "a key off the chunk's path"
        for row in range(row0, row0 + nrows):
            t = row // g
            assert t < lens[c]
            vis = [k for p, k in enumerate(keys)
                   if k is not None and (int(k0) == -1 or p <= t - int(k0))]
            # the causal rule: the chunk's own keys up to the row's token only
            assert all(k[0] != chunks[c] or k[1] <= t for k in vis), (i, row)
            slot = slot_base + row - row0
            assert slot not in seen, "partial slot written twice"
            seen[slot] = (int(leaf_lo) + t, kvh * g + row % g, vis)
    assert sorted(seen) == list(range(info["num_slots"]))
    # a fresh plan lays the lists out in (branch, kv head) order, end to end
    assert mrng[0, 0] == 0 and mrng[-1, 1] == len(ment) and (mrng[1:, 0] == mrng[:-1, 1]).all()
    for c, n in enumerate(chunks):
        want_anc = [(a, x) for a in ancestors(tree, n) for x in range(int(tree.node_len[a]))]
        for t in range(lens[c]):
            q = int(qbase[c]) + t
            want = sorted(want_anc + [(n, x) for x in range(t + 1)])
            for h in range(tree.num_q_heads):
                j, r = divmod(h, g)
                k = q * H_kv + j
                got = []
                for e in ment[mrng[k, 0]:mrng[k, 1]]:
                    qq, hh, vis = seen[int(e) + r]
                    assert (qq, hh) == (q, h)
                    assert vis, "a merged slot must see at least one key"
                    got.extend(vis)
                assert sorted(got) == want, (c, t, h)
    # every written slot that sees a key is merged (no wasted tiles beyond the mask)
    merged = {int(e) + r for e in ment for r in range(g)}
    assert all(s in merged for s, (_, _, vis) in seen.items() if vis)
    want_path = sum(lens[c] * sum(int(tree.node_len[a]) for a in ancestors(tree, n)) +
                    lens[c] * (lens[c] + 1) // 2 for c, n in enumerate(chunks))
    assert info["path_tokens"] == want_path
    return info


def prefill(name, parent, node_len, chunks, *, hq=8, hkv=2, **kw):
    return W.build_prefill(name, parent, node_len, chunks, num_q_heads=hq, num_kv_heads=hkv,
                           head_dim=128, values=False, **kw)


CASES = {
    # the join: a prefix, threads under it, the text after </Parallel> as chunks
    "join": lambda: prefill("join", [-1, 0, 0, 0, 1], [300, 70, 33, 64, 41], [2, 3, 4]),
    "root_chunk": lambda: prefill("root", [-1], [200], [0]),
    "page_edges": lambda: prefill("edges", [-1, 0, 0, 0, 0, 0, 0],
                                  [17, 1, 15, 16, 63, 64, 65], [1, 2, 3, 4, 5, 6]),
    "g1": lambda: prefill("g1", [-1, 0, 1], [50, 90, 130], [2], hq=4, hkv=4),
    "g16": lambda: prefill("g16", [-1, 0, 0], [77, 40, 9], [1, 2], hq=32, hkv=2),
    "g6": lambda: prefill("g6", [-1, 0, 1, 1], [33, 21, 70, 5], [2, 3], hq=12, hkv=2),
    "long_chunk": lambda: prefill("long", [-1, 0], [1000, 700], [1]),
    "empty_ancestor": lambda: prefill("emptyanc", [-1, 0, 1], [0, 20, 35], [2]),
    "empty_chunk": lambda: prefill("emptychunk", [-1, 0, 0], [40, 0, 19], [1, 2]),
    "forest": lambda: prefill("forest", [-1, -1, 0, 1], [30, 45, 12, 80], [2, 3]),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_prefill_plan_covers_keys_exactly(name):
    tree = CASES[name]()
    with Plan.for_prefill(tree, host_only=True) as plan:
        verify_prefill_plan(tree, plan)


def test_prefill_plan_sm_counts():
    tree = CASES["join"]()
    for sms in (1, 7, 152, 400):
        with Plan.for_prefill(tree, host_only=True, num_sms=sms) as plan:
            info = verify_prefill_plan(tree, plan)
            assert info["num_ctas"] == info["num_wide_ctas"] == sms


def test_prefill_plan_refusals():
    tree = CASES["join"]()
    for mode, d in (("fp32", 128), ("bf16", 64)):
        t = W.build_prefill("x", tree.parent, tree.node_len, tree.leaf_node, num_q_heads=8,
                            num_kv_heads=2, head_dim=d, mode=mode, values=False)
        with pytest.raises(ParasonError) as e:
            Plan.for_prefill(t, host_only=True)
        assert e.value.status == _lib.EUNSUPPORTED
    # a chunk node with children, or named twice
    for chunks in ([1, 2], [2, 2]):
        t = W.build_tree("y", tree.parent, tree.node_len, [2, 3], num_q_heads=8, num_kv_heads=2,
                         head_dim=128, values=False)
        with pytest.raises(ParasonError) as e:
            Plan(num_q_heads=8, num_kv_heads=2, head_dim=128, mode="bf16", parent=t.parent,
                 node_len=t.node_len, node_page_ptr=t.node_page_ptr, page_ids=t.page_ids,
                 leaf_node=chunks, num_physical_pages=t.num_physical_pages, host_only=True,
                 prefill=True)
        assert e.value.status == _lib.EINVAL
    # appends are for decode plans
    with Plan.for_prefill(tree, host_only=True) as plan:
        with pytest.raises(ParasonError) as e:
            plan.append(None)
        assert e.value.status == _lib.EUNSUPPORTED


def test_prefill_plan_deterministic():
    tree = CASES["page_edges"]()
    tabs = []
    for _ in range(2):
        with Plan.for_prefill(tree, host_only=True) as plan:
            tabs.append([plan.export(t) for t in (_lib.TABLE_ITEMS, _lib.TABLE_ITEM_KEY0,
                                                  _lib.TABLE_MERGE_RANGES, _lib.TABLE_MERGE)])
    for a, b in zip(*tabs):
        assert np.array_equal(a, b)


def test_bf16_pieces_span_the_path():
    """With bf16 KV a piece reads across node boundaries along the chunk's
    path, so a query row has fewer partials than its path has nodes (one each
    on one SM, where every path fits one piece); e4m3 pieces stay within a
    node."""
    tree = CASES["join"]()
    with Plan.for_prefill(tree, host_only=True, num_sms=1) as plan:
        info = verify_prefill_plan(tree, plan)
        mrng = plan.export(_lib.TABLE_MERGE_RANGES)
        assert (mrng[:, 1] - mrng[:, 0] == 1).all()
        srows = plan.export(_lib.TABLE_STREAM_ROWS)
        assert (srows & 15).any(), "a page that ends a node inside a piece"
        assert (srows == tree.num_physical_pages * tree.num_kv_heads * 16).any(), "padding"
    t8 = W.build_prefill("j8", tree.parent, tree.node_len, tree.leaf_node, num_q_heads=8,
                         num_kv_heads=2, head_dim=128, mode="fp8", values=False)
    with Plan.for_prefill(t8, host_only=True, num_sms=1) as plan:
        verify_prefill_plan(t8, plan)
        assert not (plan.export(_lib.TABLE_STREAM_ROWS) & 15).any()
        mrng = plan.export(_lib.TABLE_MERGE_RANGES)
        assert (mrng[:, 1] - mrng[:, 0] > 1).any()
