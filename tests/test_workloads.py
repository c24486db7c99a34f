"""Seeded workload generators: shapes, draw recipe, determinism (CPU only)."""
import os

import numpy as np
import torch

from paper_2608_24658_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_shape(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                n, p, kind = line.split()
                rows.append((int(n), int(p), kind))
    return rows


def test_figure3_shape_matches_golden():
    rows = _golden_shape("figure3_tree_shape.txt")
    tree = W.figure3_tree()
    assert list(tree.parent) == [p for _, p, _ in rows]
    leaves = sorted(n for n, _, kind in rows if kind == "trial")
    assert sorted(tree.leaf_node.tolist()) == leaves
    # trials per subtask: 4, 1, 3
    per = [sum(1 for b in tree.leaf_node if tree.parent[b] == s) for s in (1, 2, 3)]
    assert per == [4, 1, 3]


def _check_pages(tree):
    ptr, ids = tree.node_page_ptr, tree.page_ids
    for n in range(tree.num_nodes):
        assert ptr[n + 1] - ptr[n] == (tree.node_len[n] + 15) // 16
    assert len(set(ids.tolist())) == len(ids)
    assert ids.min(initial=0) >= 0 and ids.max(initial=-1) < tree.num_physical_pages
    assert all(tree.parent[i] < i for i in range(tree.num_nodes))


def test_config_shapes_small():
    t = W.make_config(1)
    assert (t.num_q_heads, t.num_kv_heads, t.head_dim) == (8, 2, 64)
    assert list(t.node_len) == [256, 32, 40, 48, 64]
    assert t.q.dtype == torch.bfloat16 and t.k_pages.shape[1:] == (2, 16, 64)
    _check_pages(t)


def test_config_lengths_follow_recipe():
    # lengths only (no value draw) by reproducing the draw order on a fresh rng
    rng = np.random.default_rng(1)
    lens = [int(rng.integers(512, 4097)) for _ in range(16)]
    t = W.llama3_trials(device="cpu")
    assert list(t.node_len[1:]) == lens and t.node_len[0] == 2048
    assert all(512 <= x <= 4096 for x in lens)
    q = t.q.float()
    assert abs(q.std().item() - 1 / np.sqrt(128)) < 0.01


def test_determinism_and_fp8_recipe():
    a = W.figure3_tree(mode="fp8", seed=3)
    b = W.figure3_tree(mode="fp8", seed=3)
    assert torch.equal(a.k_pages.view(torch.uint8), b.k_pages.view(torch.uint8))
    assert a.k_scale.shape == (a.num_kv_heads,)
    deq = a.k_pages.float().abs().amax(dim=(0, 2, 3))
    assert torch.all(deq <= 448.0)
    _check_pages(a)


def test_random_forest_valid():
    for s in range(5):
        t = W.random_tree(s)
        _check_pages(t)
        assert len(set(t.leaf_node.tolist())) == t.num_leaves


def test_tail_fill():
    t = W.build_tree("x", [-1, 0], [20, 7], [1], num_q_heads=2, num_kv_heads=1, head_dim=64,
                     tail_value=float("nan"))
    p_last = t.page_ids[t.node_page_ptr[1]]
    assert torch.isnan(t.k_pages[p_last, :, 7:].float()).all()
    assert not torch.isnan(t.k_pages[p_last, :, :7].float()).any()


def test_host_subset_preserves_paths():
    t = W.random_tree(7)
    sel = [t.num_leaves - 1, 0]
    s = W.host_subset(t, sel)
    for i, b in enumerate(sel):
        assert [int(t.node_len[n]) for n in t.path(b)] == [int(s.node_len[n]) for n in s.path(i)]
    assert torch.equal(s.q[0], t.q[sel[0]])
