"""GPU decode through the C ABI vs the fp64 oracle, element by element.

Small fixtures span several tiles, chunks and ragged last pages; the five
workloads run at full size, every branch compared (the two largest with the
oracle run a request or a group of branches at a time on host copies of only
what those branches read).
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_24658_gb300 import _lib
from paper_2608_24658_gb300 import workloads as W
from paper_2608_24658_gb300.api import Plan, ParasonError, lse_merge
from tests import parity as PT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_24658_gb300 import build
    build.build()
    torch.cuda.init()


FIXTURES = {
    "figure3_d64": lambda m: W.figure3_tree(mode=m, device="cuda"),
    "figure3_d128_g8": lambda m: W.figure3_tree(mode=m, h_q=16, h_kv=2, d=128, trunk=300,
                                                subtask=(130, 64, 17), device="cuda"),
    "forest_depth3": lambda m: W.random_tree(5, depth=3, len_range=(0, 300), mode=m,
                                             device="cuda", tail_value=float("nan")),
    "forest_g1_d128": lambda m: W.random_tree(6, h_q=4, h_kv=4, d=128, len_range=(1, 200),
                                              mode=m, device="cuda"),
    "forest_g16": lambda m: W.random_tree(7, h_q=32, h_kv=2, d=64, depth=2, len_range=(0, 90),
                                          mode=m, device="cuda"),
    "forest_g6": lambda m: W.random_tree(8, h_q=12, h_kv=2, d=128, depth=2, mode=m,
                                         device="cuda"),
    "wide_root_40_branches": lambda m: W.build_tree(
        "wide", [-1] + [0] * 40, [1500] + [int(x) for x in np.arange(40) * 7 + 1],
        list(range(1, 41)), num_q_heads=16, num_kv_heads=2, head_dim=128, mode=m, seed=3,
        device="cuda", tail_value=float("nan")),
    "chain_with_empty_nodes": lambda m: W.build_tree(
        "chain", [-1, 0, 1, 2], [17, 0, 33, 5], [3], num_q_heads=6, num_kv_heads=3,
        head_dim=64, mode=m, seed=9, device="cuda", tail_value=float("nan")),
    "exact_page_multiples": lambda m: W.build_tree(
        "pages16", [-1, 0, 0], [64, 16, 32], [1, 2], num_q_heads=8, num_kv_heads=2,
        head_dim=128, mode=m, seed=4, device="cuda"),
    "single_token_branches": lambda m: W.build_tree(
        "ones", [-1, 0, 0, 0], [1, 1, 1, 1], [1, 2, 3], num_q_heads=8, num_kv_heads=1,
        head_dim=64, mode=m, seed=5, device="cuda"),
    "custom_scale": lambda m: W.figure3_tree(mode=m, sm_scale=0.21, device="cuda"),
    # bf16 runs the prefix tile in pairs of row tiles here: 320 root rows (a
    # pair and a tile without a partner), 136 and 184 rows under the two
    # inner nodes (pairs whose second tile has 8 and 56 rows)
    "tile_pairs_odd": lambda m: W.pair_fixture(mode=m, device="cuda", tail_value=float("nan")),
}


@pytest.mark.parametrize("mode", ["bf16", "fp32", "fp8"])
@pytest.mark.parametrize("name", sorted(FIXTURES))
def test_fixture_parity(name, mode):
    tree = FIXTURES[name](mode)
    if mode == "fp8" and tree.head_dim != 128:
        pytest.skip("e4m3 KV has a kernel for head_dim 128 only")
    tree = PT.nan_fill_unused_pages(tree)
    PT.run_and_compare(tree, tag=f"{name}/{mode}")


@pytest.mark.parametrize("d", [64, 128])
def test_many_branches_grouped_merge(d):
    # 2048 branches x 2 kv heads: 4096 (branch, kv head) pairs with g = 2 take
    # the merge kernel that serves every q head of a pair from one warp
    rng = np.random.default_rng(12)
    lens = [300] + [int(x) for x in rng.integers(1, 40, 2048)]
    tree = W.build_tree("many", [-1] + [0] * 2048, lens, list(range(1, 2049)), num_q_heads=4,
                        num_kv_heads=2, head_dim=d, mode="bf16", seed=12, device="cuda",
                        tail_value=float("nan"))
    PT.run_and_compare(PT.nan_fill_unused_pages(tree), tag=f"many_branches_d{d}")


@pytest.mark.parametrize("mode", ["bf16", "fp8"])
def test_host_memory_q_and_result(mode):
    # q, out and lse in page-locked host memory: the kernels read and store
    # there directly; bit-identical to device buffers
    tree = W.make_config(2, mode=mode, device="cuda")
    with Plan.for_tree(tree) as plan:
        ref_o, ref_l = plan.decode_tree(tree)
        out_h = torch.empty(tuple(ref_o.shape), dtype=ref_o.dtype).pin_memory()
        lse_h = torch.empty(tuple(ref_l.shape), dtype=ref_l.dtype).pin_memory()
        plan.decode_tree(tree, out=out_h, lse=lse_h)
        plan.check()
        assert torch.equal(out_h, ref_o.cpu()) and torch.equal(lse_h, ref_l.cpu())
        q_h = tree.q.cpu().pin_memory()
        o2, l2 = plan.decode(q_h, tree.k_pages, tree.v_pages, k_scale=tree.k_scale,
                             v_scale=tree.v_scale)
        plan.check()
        assert o2.is_pinned() and torch.equal(o2, ref_o.cpu()) and torch.equal(l2, ref_l.cpu())


def test_empty_path_gives_zero_and_neg_inf():
    tree = W.build_tree("empty", [-1, 0, 0], [0, 0, 5], [1, 2], num_q_heads=4, num_kv_heads=2,
                        head_dim=64, seed=2, device="cuda")
    out, lse = PT.gpu_decode(tree)
    assert torch.all(out[0] == 0) and torch.all(torch.isneginf(lse[0]))
    PT.run_and_compare(tree)


def test_permuted_variants_of_small_workloads():
    for idx in (1, 2):
        tree = W.make_config(idx, device="cuda", permute_pages=True, extra_pages=5)
        PT.run_and_compare(PT.nan_fill_unused_pages(tree), tag=f"config{idx}-permuted")


@pytest.mark.parametrize("idx,mode", [(1, "bf16"), (2, "bf16"), (3, "bf16"), (2, "fp8"),
                                      (3, "fp8"), (1, "fp32"), (2, "fp32")])
def test_workload_full_parity(idx, mode):
    if mode == "fp8" and idx == 1:
        pytest.skip("head_dim 64")
    tree = W.make_config(idx, mode=mode, device="cuda")
    stats = PT.run_and_compare(tree, tag=tree.name)
    print(tree.name, stats)


@pytest.mark.parametrize("idx,mode,group", [(4, "bf16", 32), (5, "bf16", 16), (5, "fp8", 16)])
def test_workload_every_branch_parity(idx, mode, group):
    """The two largest workloads at full size, every branch and q head
    against the oracle.  Branch outputs are all needed (they are concatenated
    into later context, Fig. 1 caption and Sec. 3.1), so none is sampled
    away.  The oracle runs on `group` branches at a time on a host copy of
    only what they read (one request of the batched workload at a time), so
    the multi-GB pool never goes to the host whole."""
    tree = W.make_config(idx, mode=mode, device="cuda")
    out, lse = PT.gpu_decode(tree)
    L = tree.num_leaves
    ref_o = np.empty((L, tree.num_q_heads, tree.head_dim), dtype=np.float64)
    ref_l = np.empty((L, tree.num_q_heads), dtype=np.float64)
    for s0 in range(0, L, group):
        sel = list(range(s0, min(L, s0 + group)))
        ro, rl = PT.oracle_decode(tree, sel)
        ref_o[sel], ref_l[sel] = ro, rl
    stats = PT.compare(tree, out, lse, ref_o, ref_l, tag=f"{tree.name}/{mode}")
    print(tree.name, mode, stats)
    del tree
    torch.cuda.empty_cache()


def test_repeat_calls_bit_identical_and_plan_reuse():
    tree = W.make_config(3, device="cuda")
    with Plan.for_tree(tree) as plan:
        o1, l1 = plan.decode_tree(tree)
        o2, l2 = plan.decode_tree(tree)
        plan.check()
        assert torch.equal(o1, o2) and torch.equal(l1, l2)


def test_cuda_graph_capture_replay():
    tree = W.make_config(2, device="cuda")
    with Plan.for_tree(tree) as plan:
        ws = plan.workspace()
        out = torch.empty_like(tree.q)
        lse = torch.empty(tree.q.shape[:2], dtype=torch.float32, device="cuda")
        plan.decode_tree(tree, out=out, lse=lse, workspace=ws)      # warm-up (configures)
        torch.cuda.synchronize()
        eager = out.clone()
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                plan.decode_tree(tree, out=out, lse=lse, workspace=ws, stream=s)
        out.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(out, eager)


def test_timeout_path_reports_and_recovers():
    """A wait that can never complete returns ETIMEOUT; the context stays usable."""
    tree = W.figure3_tree(device="cuda", trunk=200)
    with Plan.for_tree(tree) as plan:
        plan.set_debug(_lib.DEBUG_SKIP_FIRST_LOAD, wait_limit_ns=2_000_000)
        plan.decode_tree(tree)
        with pytest.raises(ParasonError) as e:
            plan.check()
        assert e.value.status == _lib.ETIMEOUT
        plan.set_debug(0, wait_limit_ns=2_000_000_000)
        out, lse = plan.decode_tree(tree)
        plan.check()
        ref_o, ref_l = PT.oracle_decode(tree)
        PT.compare(tree, out, lse, ref_o, ref_l)


def test_decode_rejects_bad_arguments():
    tree = W.figure3_tree(device="cuda")
    with Plan.for_tree(tree) as plan:
        lib = _lib.load()
        p = lambda t: None if t is None else t.data_ptr()
        out = torch.empty_like(tree.q)
        ws = plan.workspace()
        base = [plan.handle, p(tree.q), p(tree.k_pages), p(tree.v_pages), None, None, p(out),
                None, p(ws), ws.numel()]
        s = torch.cuda.current_stream().cuda_stream
        assert lib.parason_attn_decode(*base, s) == _lib.OK
        short = list(base)
        short[9] = plan.workspace_bytes - 1
        assert lib.parason_attn_decode(*short, s) == _lib.EINVAL
        nokv = list(base)
        nokv[2] = None
        assert lib.parason_attn_decode(*nokv, s) == _lib.EINVAL
        mis = list(base)
        mis[8] = p(ws) + 16
        assert lib.parason_attn_decode(*mis, s) == _lib.EINVAL
        plan.check()


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("d", [64, 128])
def test_lse_merge_matches_oracle(dtype, d):
    g = torch.Generator(device="cuda").manual_seed(11)
    rows = 1000
    o_a = torch.randn((rows, d), generator=g, device="cuda").to(dtype)
    o_b = torch.randn((rows, d), generator=g, device="cuda").to(dtype)
    la = torch.randn(rows, generator=g, device="cuda") * 5
    lb = torch.randn(rows, generator=g, device="cuda") * 5
    la[::7] = -math.inf
    lb[::11] = -math.inf
    o, l = lse_merge(o_a, la, o_b, lb)
    ref_o, ref_l = oracle.lse_merge(o_a.double().cpu().numpy(), la.double().cpu().numpy(),
                                    o_b.double().cpu().numpy(), lb.double().cpu().numpy())
    tol = 1e-5 if dtype == torch.float32 else 1e-2
    assert np.abs(o.double().cpu().numpy() - ref_o).max() <= tol
    lc = l.cpu().numpy()
    fin = np.isfinite(ref_l)
    assert np.array_equal(np.isfinite(lc), fin)
    assert np.abs(lc[fin] - ref_l[fin]).max() <= 1e-5


def test_lse_merge_of_two_decodes_equals_whole():
    """Decode two KV halves separately and merge: equals decoding the whole."""
    tree = W.build_tree("halves", [-1, 0], [300, 200], [1], num_q_heads=8, num_kv_heads=2,
                        head_dim=128, seed=12, device="cuda")
    # the same branch as two single-node trees: the root alone, the suffix alone
    ptr = tree.node_page_ptr
    a = W.ForkTree(**{**tree.__dict__, "parent": np.array([-1], np.int32),
                      "node_len": tree.node_len[:1].copy(),
                      "node_page_ptr": ptr[:2].copy(), "page_ids": tree.page_ids[:ptr[1]].copy(),
                      "leaf_node": np.array([0], np.int32)})
    b = W.ForkTree(**{**tree.__dict__, "parent": np.array([-1], np.int32),
                      "node_len": tree.node_len[1:].copy(),
                      "node_page_ptr": (ptr[1:] - ptr[1]).astype(np.int32),
                      "page_ids": tree.page_ids[ptr[1]:].copy(),
                      "leaf_node": np.array([0], np.int32)})
    oa, la = PT.gpu_decode(a)
    ob, lb = PT.gpu_decode(b)
    o, l = lse_merge(oa, la, ob, lb)
    ref_o, ref_l = PT.oracle_decode(tree)
    PT.compare(tree, o, l, ref_o, ref_l, tag="halves merged")


@pytest.mark.parametrize("where", ["suffix_16row", "suffix_transposed", "prefix_tile"])
def test_e4m3_q_beyond_f16_is_reported(where):
    """With e4m3 KV the kernels narrow q to f16.  Large q within f16's range
    still matches the oracle; a q element of magnitude 1e5 (beyond 65504)
    makes the next check return PARASON_ERANGE instead of a silently wrong
    result, and the plan works again afterwards.  `where` picks the path that
    loads the row: suffix warps with the 16-row step (2 branches, g = 2: every
    tile has at most 4 rows), the transposed step (2 branches, g = 8), or the
    tcgen05 prefix tile (a trunk shared by 40 branches, 320 rows)."""
    if where == "suffix_16row":
        tree = W.build_tree("two", [-1, 0, 0], [100, 50, 20], [1, 2], num_q_heads=4,
                            num_kv_heads=2, head_dim=128, mode="fp8", seed=31, device="cuda")
    elif where == "suffix_transposed":
        tree = W.build_tree("two8", [-1, 0, 0], [100, 50, 20], [1, 2], num_q_heads=16,
                            num_kv_heads=2, head_dim=128, mode="fp8", seed=32, device="cuda")
    else:
        tree = FIXTURES["wide_root_40_branches"]("fp8")
    with Plan.for_tree(tree) as plan:
        big = tree.q.clone()
        big[1] = (big[1].float() * 100.0).to(big.dtype)          # |q| up to a few hundred
        tree.q = big
        out, lse = plan.decode_tree(tree)
        plan.check()
        ref_o, ref_l = PT.oracle_decode(tree)
        PT.compare(tree, out, lse, ref_o, ref_l, tag=f"large q in f16 range ({where})")
        bad = big.clone()
        bad[1, 3, 7] = 1.0e5
        plan.decode(bad, tree.k_pages, tree.v_pages, k_scale=tree.k_scale, v_scale=tree.v_scale)
        with pytest.raises(ParasonError) as e:
            plan.check()
        assert e.value.status == _lib.ERANGE
        out, lse = plan.decode_tree(tree)
        plan.check()
        PT.compare(tree, out, lse, ref_o, ref_l, tag=f"after the range error ({where})")
