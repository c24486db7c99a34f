"""What a plan's branches attend to, read back from the plan's exported
tables (merge ranges, items, page streams), and what the tree says they must
attend to -- for checks that hold however the plan is cut into work."""
import numpy as np

from paper_2608_24658_gb300 import _lib


def coverage(plan, head0=0):
    """{(global branch, global kv head): sorted ((physical page, valid tokens), ...)}
    read from the plan's merge lists, items and page streams."""
    H = plan.num_kv_heads
    items = plan.export(_lib.TABLE_ITEMS)
    irows = plan.export(_lib.TABLE_ITEM_ROWS)
    srows = plan.export(_lib.TABLE_STREAM_ROWS)
    mrng = plan.export(_lib.TABLE_MERGE_RANGES)
    ment = plan.export(_lib.TABLE_MERGE)
    glob = plan.export(_lib.TABLE_SHARD_BRANCHES)
    owner = {}
    for i, it in enumerate(items):
        for s in range(int(it[7]), int(it[7]) + int(it[5])):
            owner[s] = i
    out = {}
    for b in range(plan.num_leaves):
        for j in range(H):
            cov = []
            for e in ment[mrng[b * H + j, 0]:mrng[b * H + j, 1]]:
                i = owner[int(e)]
                npg, last_valid = int(items[i][1]), int(items[i][2])
                r = srows[irows[i]:irows[i] + npg].astype(np.int64) // 16
                assert ((r % H) == j).all()
                for k, pg in enumerate(r // H):
                    cov.append((int(pg), last_valid if k == npg - 1 else 16))
            out[(int(glob[b]), head0 + j)] = tuple(sorted(cov))
    return out


def definition(tree):
    """What each (branch, kv head) must attend to: every page of every node on
    its path with its valid tokens (empty nodes hold no page)."""
    out = {}
    for b in range(tree.num_leaves):
        cov = []
        for n in tree.path(b):
            ln = int(tree.node_len[n])
            pages = tree.page_ids[tree.node_page_ptr[n]:tree.node_page_ptr[n + 1]]
            for k, pg in enumerate(pages):
                cov.append((int(pg), ln - 16 * k if k == len(pages) - 1 else 16))
        for j in range(tree.num_kv_heads):
            out[(b, j)] = tuple(sorted(cov))
    return out


def check_tile_pairs(plan):
    """The prefix queue in pair mode: entries 2k and 2k + 1 are two row tiles
    of one piece (the same pages and kv head, the second's rows right after
    the first's) or a tile and a blank (no rows, never merged).  Returns the
    blank items; outside pair mode there are none and every item has rows."""
    info = plan.info()
    items = plan.export(_lib.TABLE_ITEMS)
    wq = plan.export(_lib.TABLE_WIDE_QUEUE)
    blank = {i for i, it in enumerate(items) if int(it[5]) == 0}
    if not info["tile_pairs"]:
        assert not blank, "an item without rows outside pair mode"
        return blank
    assert len(wq) % 2 == 0
    seconds = set()
    for k in range(0, len(wq), 2):
        a, b = items[wq[k]], items[wq[k + 1]]
        assert int(a[5]) >= 1, "a pair's first tile has rows"
        seconds.add(int(wq[k + 1]))
        if int(b[5]) == 0:
            continue
        assert a[0] == b[0] and a[1] == b[1] and a[2] == b[2], "a pair reads one page range"
        assert a[6] == b[6] and a[3] == b[3], "a pair is one kv head of one node"
        assert b[4] == a[4] + a[5], "a pair's tiles are consecutive row tiles"
    assert blank <= seconds, "a blank item outside a pair's second place"
    return blank
