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
