"""Tree-masked prefill through the C ABI (parason_prefill_plan +
parason_attn_decode) against the fp64 prefill oracle: every query of small
trees spanning page edges, several tiles and ragged tails, GQA groups 1 to
16, and sampled queries of the thread-opening and join workloads at full
size."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_24658_gb300 import build
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan
from tests import parity as PT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()
    torch.cuda.init()


def oracle_prefill(tree, sel=None):
    """fp64 oracle on the host copy (e4m3 KV read with the tree's per-kv-head scales)."""
    host = tree.to("cpu")
    kw = oracle.tree_kwargs(host)
    kw["chunk_node"] = kw.pop("leaf_node")
    return oracle.prefill(sel=sel, **kw)


def run(tree, sel=None, tag=""):
    with Plan.for_prefill(tree) as plan:
        out, lse = plan.decode_tree(tree)
        plan.check()
    ref_o, ref_l = oracle_prefill(tree, sel)
    return PT.compare(tree, out, lse, ref_o, ref_l, sel, tag or tree.name)


def small(name, parent, node_len, chunks, *, hq=8, hkv=2, mode="bf16", **kw):
    return W.build_prefill(name, parent, node_len, chunks, num_q_heads=hq, num_kv_heads=hkv,
                           head_dim=128, mode=mode, device="cuda",
                           q_std=1.0 / np.sqrt(128.0) * 4, **kw)


CASES = {
    "join": lambda: small("join", [-1, 0, 0, 0, 1], [300, 70, 33, 64, 41], [2, 3, 4], seed=1),
    "root_chunk": lambda: small("root", [-1], [200], [0], seed=2),
    "page_edges": lambda: small("edges", [-1, 0, 0, 0, 0, 0, 0], [17, 1, 15, 16, 63, 64, 65],
                                [1, 2, 3, 4, 5, 6], seed=3),
    "g1": lambda: small("g1", [-1, 0, 1], [50, 90, 130], [2], hq=4, hkv=4, seed=4),
    "g16": lambda: small("g16", [-1, 0, 0], [77, 40, 9], [1, 2], hq=32, hkv=2, seed=5),
    "g6": lambda: small("g6", [-1, 0, 1, 1], [33, 21, 70, 5], [2, 3], hq=12, hkv=2, seed=6),
    "long_chunk": lambda: small("long", [-1, 0], [1000, 700], [1], hq=32, hkv=8, seed=7),
    "empty_nodes": lambda: small("empty", [-1, 0, 1, 0], [0, 20, 35, 0], [2, 3], seed=8),
    # V past each node's last token is NaN: the tile must not let it through
    "nan_tails": lambda: small("nantail", [-1, 0, 0], [45, 29, 50], [1, 2], seed=9,
                               tail_value=float("nan"), permute_pages=True, extra_pages=8),
    # e4m3 KV (converted to f16 in the tile)
    "fp8_join": lambda: small("join8", [-1, 0, 0, 0, 1], [300, 70, 33, 64, 41], [2, 3, 4], seed=10,
                              mode="fp8"),
    "fp8_g16": lambda: small("g16_8", [-1, 0, 0], [77, 40, 9], [1, 2], hq=32, hkv=2, seed=11,
                             mode="fp8"),
}


@pytest.mark.parametrize("case", sorted(CASES))
def test_prefill_matches_oracle(case):
    tree = CASES[case]()
    if case == "nan_tails":
        PT.nan_fill_unused_pages(tree)
    run(tree, tag=case)


@pytest.mark.parametrize("kind", sorted(W.PREFILL_CONFIGS))
def test_prefill_workloads_sampled(kind):
    tree = W.PREFILL_CONFIGS[kind](device="cuda")
    Q = tree.q.shape[0]
    rng = np.random.default_rng(0)
    # both ends of every chunk and tile edges, plus random queries
    sel = sorted(set([0, 1, 31, 32, 63, 64, Q - 1] + rng.integers(0, Q, 24).tolist()))
    sel = [s for s in sel if s < Q]
    run(tree, sel=sel, tag=kind)


def test_prefill_repeatable():
    # the dynamic work queue changes the order partials are produced, not
    # the merge: two runs give the same bits
    tree = CASES["join"]()
    with Plan.for_prefill(tree) as plan:
        o1, l1 = plan.decode_tree(tree)
        o2, l2 = plan.decode_tree(tree)
        plan.check()
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
