"""Pins of the tree-masked prefill oracle: query t of a chunk equals the
(separately pinned) decode oracle on the tree with the chunk cut to t + 1
tokens, bit for bit; and a library cross-check (fp64 softmax with an explicit
causal mask) on KV gathered contiguously."""
from dataclasses import replace

import numpy as np
import pytest
import torch

import oracle
from paper_2608_24658_gb300 import workloads as W


def prefill_kw(tree, **extra):
    kw = oracle.tree_kwargs(tree)
    kw["chunk_node"] = kw.pop("leaf_node")
    kw.update(extra)
    return kw


def truncated(tree, chunk, t):
    """The tree with chunk node `chunk` cut to t + 1 tokens, as a decode tree
    whose only branch is that node, with query q."""
    node_len = tree.node_len.copy()
    node_len[chunk] = t + 1
    return node_len


def make(mode="bf16", seed=0):
    # root 37 -> A 20 -> chunk 23;  root -> chunk 18;  A -> chunk 1
    return W.build_prefill("pf", [-1, 0, 1, 0, 1], [37, 20, 23, 18, 1], [2, 3, 4],
                           num_q_heads=6, num_kv_heads=2, head_dim=64, mode=mode, seed=seed)


@pytest.mark.parametrize("mode", ["bf16", "fp8", "fp32"])
def test_query_equals_decode_on_the_cut_tree(mode):
    tree = make(mode)
    out, lse = oracle.prefill(**prefill_kw(tree))
    k = 0
    for c in tree.leaf_node:
        for t in range(int(tree.node_len[c])):
            node_len = truncated(tree, int(c), t)
            kw = oracle.tree_kwargs(tree)
            ptr = kw["node_page_ptr"]
            # the cut node keeps its pages; drop the ones past t
            need = [(int(n), (int(node_len[n]) + 15) // 16) for n in range(tree.num_nodes)]
            pages, newptr = [], [0]
            for n, np_ in need:
                pages.extend(kw["page_ids"][ptr[n]:ptr[n] + np_])
                newptr.append(len(pages))
            kw.update(node_len=node_len, node_page_ptr=np.asarray(newptr, np.int32),
                      page_ids=np.asarray(pages, np.int32), leaf_node=np.asarray([c], np.int32),
                      q=tree.q[k:k + 1])
            o_ref, l_ref = oracle.decode(**kw)
            assert np.array_equal(out[k], o_ref[0]), (c, t)
            assert np.array_equal(lse[k], l_ref[0]), (c, t)
            k += 1
    assert k == out.shape[0]


def test_library_cross_check_with_causal_mask():
    tree = make("fp32", seed=3)
    out, lse = oracle.prefill(**prefill_kw(tree))
    g = tree.num_q_heads // tree.num_kv_heads
    scale = 1.0 / np.sqrt(tree.head_dim)
    kp = tree.k_pages.double()
    vp = tree.v_pages.double()
    k = 0
    for c in tree.leaf_node:
        c = int(c)
        nodes = []
        n = c
        while n >= 0:
            nodes.append(n)
            n = int(tree.parent[n])
        nodes.reverse()
        keys = []               # (page, slot) root first
        own_start = 0
        for n in nodes:
            if n == c:
                own_start = len(keys)
            for t in range(int(tree.node_len[n])):
                keys.append((int(tree.page_ids[tree.node_page_ptr[n] + t // 16]), t % 16))
        C = int(tree.node_len[c])
        for t in range(C):
            vis = own_start + t + 1
            for h in range(tree.num_q_heads):
                kvh = h // g
                K = torch.stack([kp[p, kvh, s] for p, s in keys[:vis]])
                V = torch.stack([vp[p, kvh, s] for p, s in keys[:vis]])
                qv = tree.q[k + t, h].double()
                s_ = (K @ qv) * scale
                o_ref = torch.softmax(s_, 0) @ V
                l_ref = torch.logsumexp(s_, 0)
                assert np.abs(out[k + t, h] - o_ref.numpy()).max() < 1e-12
                assert abs(lse[k + t, h] - float(l_ref)) < 1e-12
        k += C


def test_selected_queries():
    tree = make("bf16", seed=5)
    out, lse = oracle.prefill(**prefill_kw(tree))
    sel = [0, 5, 22, 23, 41]
    o2, l2 = oracle.prefill(**prefill_kw(tree, sel=sel))
    assert np.array_equal(o2, out[sel]) and np.array_equal(l2, lse[sel])
