"""Seeded synthetic fork-tree decode workloads.

This module only draws inputs: tree shapes, node lengths, page tables and
q/K/V values.  It holds none of the attention arithmetic, imports neither the
CUDA binding nor the oracle, and is the one piece of code both sides share.

A workload is one decode step of every live branch of a parallel-reasoning
fork tree.  The paper's runtime dispatches each <Subtask>/<Trial> entry of a
<Parallel> region as an independent worker (Sec. 3.4); threads may nest further
<Parallel> regions (Fig. 4, rule W -> <Thread> B </Thread>), so the tree can
be deeper than one level, as in the 24-puzzle example of Fig. 3 (three subtasks
with four, one and three trials).

Tree encoding (what ``parason_attn_plan`` takes):
  parent[i]        parent node of node i, -1 for a root; parent[i] < i
  node_len[i]      tokens held by node i (a leaf's count includes the token
                   decoded this step)
  node_page_ptr    CSR offsets [num_nodes + 1] into page_ids
  page_ids         physical page of each node's j-th logical page; node i owns
                   exactly ceil(node_len[i] / page_size) pages and no page is
                   shared between nodes
  leaf_node[b]     node holding branch b's private suffix; branch b's query is
                   row b of q

Value recipe: q, K, V ~ N(0, 1) rounded to the KV dtype (q scaled by 1/sqrt(d)
in the 16-branch Llama-3-8B-shape workload); fp8 KV is the bf16 draw divided
by a per-kv-head scale amax/448 and rounded to e4m3.  Draw order per seed:
node lengths in node order, the page permutation, q, K, V.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace
from typing import Optional, Sequence

import numpy as np
import torch

PAGE_SIZE = 16
E4M3_MAX = 448.0


@dataclass
class ForkTree:
    name: str
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    mode: str                      # "bf16" | "fp32" | "fp8"
    parent: np.ndarray
    node_len: np.ndarray
    node_page_ptr: np.ndarray
    page_ids: np.ndarray
    leaf_node: np.ndarray
    num_physical_pages: int
    q: torch.Tensor                # [L, H_q, d]
    k_pages: torch.Tensor          # [P, H_kv, page_size, d]
    v_pages: torch.Tensor
    k_scale: Optional[torch.Tensor] = None   # [H_kv] fp32, fp8 mode
    v_scale: Optional[torch.Tensor] = None
    sm_scale: float = 0.0          # 0 => 1/sqrt(head_dim)
    page_size: int = PAGE_SIZE
    meta: dict = field(default_factory=dict)

    @property
    def num_nodes(self) -> int:
        return len(self.parent)

    @property
    def num_leaves(self) -> int:
        return len(self.leaf_node)

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    def path(self, b: int) -> list:
        """Nodes on the path root -> leaf of branch b, root first."""
        out, n = [], int(self.leaf_node[b])
        while n >= 0:
            out.append(n)
            n = int(self.parent[n])
        return out[::-1]

    def leaves_under(self) -> np.ndarray:
        """Number of branches whose path contains each node."""
        cnt = np.zeros(self.num_nodes, dtype=np.int64)
        for b in range(self.num_leaves):
            for n in self.path(b):
                cnt[n] += 1
        return cnt

    def unique_tokens(self) -> int:
        """Tokens of every node on some branch's path, each node counted once."""
        cnt = self.leaves_under()
        return int(self.node_len[cnt > 0].sum())

    def path_tokens(self) -> int:
        """Tokens summed over branches with no sharing (every branch's full path)."""
        return int(sum(int(self.node_len[self.path(b)].sum()) for b in range(self.num_leaves)))

    def kv_elem_bytes(self) -> int:
        return {"bf16": 2, "fp32": 4, "fp8": 1}[self.mode]

    def q_elem_bytes(self) -> int:
        return 4 if self.mode == "fp32" else 2

    def to(self, device) -> "ForkTree":
        mv = lambda t: None if t is None else t.to(device)
        return replace(self, q=mv(self.q), k_pages=mv(self.k_pages),
                       v_pages=mv(self.v_pages), k_scale=mv(self.k_scale),
                       v_scale=mv(self.v_scale))


# ----------------------------------------------------------------------------
# page tables
# ----------------------------------------------------------------------------

def assign_pages(node_len: Sequence[int], rng: Optional[np.random.Generator] = None,
                 permute: bool = False, page_size: int = PAGE_SIZE,
                 extra_pages: int = 0):
    """Give every node ceil(len/page_size) fresh pages, node-major.

    With ``permute`` the logical->physical map is a random permutation drawn
    from ``rng`` (this is the draw that follows the node lengths).  Returns
    (node_page_ptr, page_ids, num_physical_pages).
    """
    counts = np.array([(int(n) + page_size - 1) // page_size for n in node_len], dtype=np.int64)
    ptr = np.zeros(len(counts) + 1, dtype=np.int64)
    np.cumsum(counts, out=ptr[1:])
    total = int(ptr[-1])
    num_phys = total + int(extra_pages)
    if permute:
        assert rng is not None
        perm = rng.permutation(num_phys)[:total]
    else:
        perm = np.arange(total)
    return ptr.astype(np.int32), perm.astype(np.int32), num_phys


# ----------------------------------------------------------------------------
# value draws
# ----------------------------------------------------------------------------

def _randn(shape, gen, device, dtype, chunk_rows: int = 1 << 14):
    """N(0,1) draw of ``shape`` in float32, rounded to ``dtype``.

    Drawn in slices along dim 0 so that multi-GB KV pools never need an fp32
    copy of the whole pool; the slice size is fixed, so the values depend only
    on the seed.
    """
    out = torch.empty(shape, dtype=dtype, device=device)
    for s in range(0, shape[0], chunk_rows):
        e = min(shape[0], s + chunk_rows)
        out[s:e] = torch.randn((e - s,) + tuple(shape[1:]), generator=gen,
                               device=device, dtype=torch.float32).to(dtype)
    return out


def _quantize_e4m3(pages_bf16: torch.Tensor, chunk_rows: int = 1 << 14):
    """Per-kv-head scale amax/448 and the e4m3 rounding of pages/scale."""
    hkv = pages_bf16.shape[1]
    amax = torch.zeros(hkv, dtype=torch.float32, device=pages_bf16.device)
    for s in range(0, pages_bf16.shape[0], chunk_rows):
        blk = pages_bf16[s:s + chunk_rows].float().abs()
        amax = torch.maximum(amax, blk.amax(dim=(0, 2, 3)))
    scale = torch.where(amax > 0, amax / E4M3_MAX, torch.ones_like(amax))
    out = torch.empty(pages_bf16.shape, dtype=torch.float8_e4m3fn, device=pages_bf16.device)
    for s in range(0, pages_bf16.shape[0], chunk_rows):
        blk = pages_bf16[s:s + chunk_rows].float() / scale.view(1, -1, 1, 1)
        out[s:s + chunk_rows] = blk.to(torch.float8_e4m3fn)
    return out, scale


def _fill_tail_slots(tree: ForkTree, value: float):
    """Write ``value`` into the unused slots of every node's last page."""
    ps = tree.page_size
    for n in range(tree.num_nodes):
        ln = int(tree.node_len[n])
        if ln % ps == 0:
            continue
        page = int(tree.page_ids[int(tree.node_page_ptr[n + 1]) - 1])
        for pages in (tree.k_pages, tree.v_pages):
            if pages.dtype == torch.float8_e4m3fn:
                pages.view(torch.uint8)[page, :, ln % ps:, :] = 0x7F if math.isnan(value) else 0
            else:
                pages[page, :, ln % ps:, :] = value


def build_tree(name: str, parent, node_len, leaf_node, *, num_q_heads: int,
               num_kv_heads: int, head_dim: int, mode: str = "bf16", seed: int = 0,
               rng: Optional[np.random.Generator] = None, permute_pages: bool = False,
               extra_pages: int = 0, q_std: float = 1.0, device="cpu",
               tail_value: Optional[float] = None, sm_scale: float = 0.0,
               meta: Optional[dict] = None, values: bool = True) -> ForkTree:
    """Assemble a workload from a tree shape; draws pages, then q, K, V.

    ``values=False`` stops after the page table (tensors are left empty): the
    tree shape of a multi-GB workload without its q/K/V.
    """
    if rng is None:
        rng = np.random.default_rng(seed)
    meta = dict(meta or {})
    meta.setdefault("permuted", bool(permute_pages))
    meta.setdefault("q_std", float(q_std))
    parent = np.asarray(parent, dtype=np.int32)
    node_len = np.asarray(node_len, dtype=np.int32)
    leaf_node = np.asarray(leaf_node, dtype=np.int32)
    ptr, pages, nphys = assign_pages(node_len, rng, permute_pages, PAGE_SIZE, extra_pages)
    if not values:
        empty = torch.empty(0)
        return ForkTree(name=name, num_q_heads=num_q_heads, num_kv_heads=num_kv_heads,
                        head_dim=head_dim, mode=mode, parent=parent, node_len=node_len,
                        node_page_ptr=ptr, page_ids=pages, leaf_node=leaf_node,
                        num_physical_pages=nphys, q=empty, k_pages=empty, v_pages=empty,
                        sm_scale=sm_scale, meta=dict(meta or {}))
    gen = torch.Generator(device=device)
    gen.manual_seed(int(rng.integers(0, 2**62)))
    L = len(leaf_node)
    q_dtype = torch.float32 if mode == "fp32" else torch.bfloat16
    kv_draw_dtype = torch.float32 if mode == "fp32" else torch.bfloat16
    q = torch.randn((L, num_q_heads, head_dim), generator=gen, device=device,
                    dtype=torch.float32)
    if q_std != 1.0:
        q = q * q_std
    q = q.to(q_dtype)
    shape = (max(nphys, 1), num_kv_heads, PAGE_SIZE, head_dim)
    k = _randn(shape, gen, device, kv_draw_dtype)
    v = _randn(shape, gen, device, kv_draw_dtype)
    k_scale = v_scale = None
    if mode == "fp8":
        k, k_scale = _quantize_e4m3(k)
        v, v_scale = _quantize_e4m3(v)
    tree = ForkTree(name=name, num_q_heads=num_q_heads, num_kv_heads=num_kv_heads,
                    head_dim=head_dim, mode=mode, parent=parent, node_len=node_len,
                    node_page_ptr=ptr, page_ids=pages, leaf_node=leaf_node,
                    num_physical_pages=nphys, q=q, k_pages=k, v_pages=v,
                    k_scale=k_scale, v_scale=v_scale, sm_scale=sm_scale,
                    meta=dict(meta or {}))
    if tail_value is not None:
        _fill_tail_slots(tree, tail_value)
    return tree


# ----------------------------------------------------------------------------
# the five workloads
# ----------------------------------------------------------------------------

def _uniform(rng, lo, hi):
    return int(rng.integers(lo, hi + 1))      # inclusive bounds


def tiny_fork(mode="bf16", device="cpu", **kw) -> ForkTree:
    """1 request, 4 branches, 8 q / 2 kv heads, d 64, prefix 256, suffixes 32/40/48/64."""
    rng = np.random.default_rng(0)
    parent = [-1, 0, 0, 0, 0]
    node_len = [256, 32, 40, 48, 64]
    return build_tree("tiny_fork_h8_2_d64", parent, node_len, [1, 2, 3, 4], num_q_heads=8,
                      num_kv_heads=2, head_dim=64, mode=mode, rng=rng, device=device, **kw)


def llama3_trials(mode="bf16", device="cpu", **kw) -> ForkTree:
    """Llama-3-8B attention shape (32 q / 8 kv, d 128), prefix 2048, 16 trials U[512,4096]."""
    rng = np.random.default_rng(1)
    lens = [2048] + [_uniform(rng, 512, 4096) for _ in range(16)]
    parent = [-1] + [0] * 16
    return build_tree("llama3_8b_prefix2048_16trials", parent, lens, list(range(1, 17)),
                      num_q_heads=32, num_kv_heads=8, head_dim=128, mode=mode, rng=rng,
                      q_std=1.0 / math.sqrt(128.0), device=device, **kw)


def subtask_trial_tree(mode="bf16", device="cpu", **kw) -> ForkTree:
    """Two-level tree: root 4096, 8 subtasks x 1024, 8 trials each U[256,2048]; 64/8/128."""
    rng = np.random.default_rng(2)
    parent, lens, leaves = [-1], [4096], []
    for s in range(8):
        parent.append(0)
        lens.append(1024)
    for s in range(8):
        for t in range(8):
            parent.append(1 + s)
            lens.append(_uniform(rng, 256, 2048))
            leaves.append(len(parent) - 1)
    return build_tree("two_level_root4096_8x1024_64trials", parent, lens, leaves,
                      num_q_heads=64, num_kv_heads=8, head_dim=128, mode=mode, rng=rng,
                      device=device, **kw)


def lognormal_prefix(rng, median=2048, sigma=0.5, lo=1024, hi=8192) -> int:
    x = math.exp(math.log(median) + sigma * float(rng.standard_normal()))
    return int(min(hi, max(lo, int(round(x)))))


def batched_serving(mode="bf16", device="cpu", requests=32, branches=32, **kw) -> ForkTree:
    """32 requests x 32 trials (1024 branches), lognormal prefixes, U[256,8192], permuted pages."""
    rng = np.random.default_rng(3)
    parent, lens, leaves = [], [], []
    for r in range(requests):
        root = len(parent)
        parent.append(-1)
        lens.append(lognormal_prefix(rng))
        for b in range(branches):
            parent.append(root)
            lens.append(_uniform(rng, 256, 8192))
            leaves.append(len(parent) - 1)
    return build_tree(f"batched_{requests}req_x{branches}_permuted", parent, lens, leaves,
                      num_q_heads=32, num_kv_heads=8, head_dim=128, mode=mode, rng=rng,
                      permute_pages=True, device=device, **kw)


def long_reasoning(mode="bf16", device="cpu", branches=128, **kw) -> ForkTree:
    """Prefix 32768, 128 branches U[4096,16384], 64/8/128; bf16 or fp8 e4m3 KV."""
    rng = np.random.default_rng(4)
    lens = [32768] + [_uniform(rng, 4096, 16384) for _ in range(branches)]
    parent = [-1] + [0] * branches
    return build_tree(f"long_prefix32768_{branches}x4k_16k", parent, lens,
                      list(range(1, branches + 1)), num_q_heads=64, num_kv_heads=8,
                      head_dim=128, mode=mode, rng=rng, device=device, **kw)


def long_prefix_only(mode="bf16", device="cpu", branches=128, **kw) -> ForkTree:
    """The long-reasoning prefix (32768 tokens, 64 q / 8 kv heads, d 128)
    under `branches` branches of one token each: nearly all of the step is
    the stacked prefix tile (1024 rows per kv head), for measuring it alone."""
    rng = np.random.default_rng(4)
    lens = [32768] + [1] * branches
    parent = [-1] + [0] * branches
    return build_tree(f"prefix_only_32768_{branches}x1", parent, lens,
                      list(range(1, branches + 1)), num_q_heads=64, num_kv_heads=8,
                      head_dim=128, mode=mode, rng=rng, device=device, **kw)


def pair_fixture(mode="bf16", device="cpu", **kw) -> ForkTree:
    """A small tree whose prefix tiles come in pairs with bf16 KV (16 q / 2
    kv heads, d 128, g 8): a 700-token root under 40 branches (320 rows: a
    pair and an odd tile), inner nodes of 90 and 35 tokens under 17 and 23
    branches (136 and 184 rows: pairs with 8- and 56-row second tiles), and
    one-token to 40-token branch nodes."""
    parent = [-1, 0, 0] + [1] * 17 + [2] * 23
    lens = [700, 90, 35] + [1 + k for k in range(40)]
    return build_tree("tile_pairs_odd", parent, lens, list(range(3, 43)), num_q_heads=16,
                      num_kv_heads=2, head_dim=128, mode=mode, seed=12, device=device, **kw)


CONFIGS = {1: tiny_fork, 2: llama3_trials, 3: subtask_trial_tree, 4: batched_serving,
           5: long_reasoning}

# measurement workloads beside the five: a scaled-down batched workload (for
# counter captures that must stay small) and the prefix tile alone
EXTRA = {"batched_4req": lambda mode="bf16", device="cpu", **kw: batched_serving(
             mode=mode, device=device, requests=4, **kw),
         "prefix_only": long_prefix_only}


def make_config(idx: int, mode: Optional[str] = None, device="cpu", **kw) -> ForkTree:
    fn = CONFIGS[idx]
    return fn(mode=mode or "bf16", device=device, **kw)


# ----------------------------------------------------------------------------
# small fixtures
# ----------------------------------------------------------------------------

def figure3_tree(mode="bf16", device="cpu", seed=11, h_q=8, h_kv=2, d=64,
                 trunk=40, subtask=(24, 17, 33), trial_len=None, **kw) -> ForkTree:
    """Shape of the 24-puzzle example: 3 subtask threads with 4, 1 and 3 trials."""
    rng = np.random.default_rng(seed)
    parent, lens, leaves = [-1], [trunk], []
    for s, n_trials in enumerate((4, 1, 3)):
        parent.append(0)
        lens.append(subtask[s])
    for s, n_trials in enumerate((4, 1, 3)):
        for t in range(n_trials):
            parent.append(1 + s)
            lens.append(int(rng.integers(1, 70)) if trial_len is None else trial_len)
            leaves.append(len(parent) - 1)
    return build_tree("figure3_3subtasks_4_1_3_trials", parent, lens, leaves, num_q_heads=h_q,
                      num_kv_heads=h_kv, head_dim=d, mode=mode, rng=rng, device=device, **kw)


def random_tree(seed: int, *, num_requests=2, depth=3, fanout=(1, 4), len_range=(0, 80),
                h_q=8, h_kv=2, d=64, mode="bf16", device="cpu", permute_pages=True,
                extra_pages=3, leaf_min_len=1, **kw) -> ForkTree:
    """Random forest of nested parallel regions (depth levels below each root)."""
    rng = np.random.default_rng(seed)
    parent, lens, leaves = [], [], []

    def grow(node, level):
        if level == depth:
            leaves.append(node)
            return
        k = int(rng.integers(fanout[0], fanout[1] + 1))
        for _ in range(k):
            parent.append(node)
            lens.append(0)
            grow(len(parent) - 1, level + 1)

    for _ in range(num_requests):
        parent.append(-1)
        lens.append(0)
        grow(len(parent) - 1, 0)
    leafset = set(leaves)
    for n in range(len(parent)):
        lo = max(len_range[0], leaf_min_len) if n in leafset else len_range[0]
        lens[n] = int(rng.integers(lo, len_range[1] + 1))
    return build_tree(f"random_forest_seed{seed}", parent, lens, leaves, num_q_heads=h_q,
                      num_kv_heads=h_kv, head_dim=d, mode=mode, rng=rng,
                      permute_pages=permute_pages, extra_pages=extra_pages, device=device, **kw)


def host_subset(tree: ForkTree, sel: Sequence[int]) -> ForkTree:
    """Host copy of only what branches ``sel`` read, with a compact page table.

    Lets a CPU check of a multi-GB workload copy a few MB: the selected
    branches keep their order (branch i of the result is sel[i]), their path
    nodes keep their lengths, and their pages are copied to the host.
    """
    nodes = sorted({n for b in sel for n in tree.path(int(b))})
    remap = {n: i for i, n in enumerate(nodes)}
    parent = [remap[int(tree.parent[n])] if tree.parent[n] >= 0 else -1 for n in nodes]
    node_len = [int(tree.node_len[n]) for n in nodes]
    phys = []
    ptr = [0]
    for n in nodes:
        phys.extend(int(p) for p in tree.page_ids[tree.node_page_ptr[n]:tree.node_page_ptr[n + 1]])
        ptr.append(len(phys))
    idx = torch.as_tensor(phys if phys else [0], dtype=torch.long, device=tree.k_pages.device)
    k = tree.k_pages.index_select(0, idx).cpu()
    v = tree.v_pages.index_select(0, idx).cpu()
    sel_t = torch.as_tensor(list(sel), dtype=torch.long, device=tree.q.device)
    q = tree.q.index_select(0, sel_t).cpu()
    return replace(tree, name=tree.name + "_subset", parent=np.array(parent, np.int32),
                   node_len=np.array(node_len, np.int32), node_page_ptr=np.array(ptr, np.int32),
                   page_ids=np.arange(len(phys), dtype=np.int32),
                   leaf_node=np.array([remap[int(tree.leaf_node[b])] for b in sel], np.int32),
                   num_physical_pages=len(phys), q=q, k_pages=k, v_pages=v,
                   k_scale=None if tree.k_scale is None else tree.k_scale.cpu(),
                   v_scale=None if tree.v_scale is None else tree.v_scale.cpu())


# ----------------------------------------------------------------------------
# reasoning traces (tag streams of the parallel-reasoning grammar, Fig. 4)
# ----------------------------------------------------------------------------

# tag codes of a trace symbol stream (text tokens are ids >= 0)
TAG_THINK, TAG_THINK_END = -1, -2
TAG_PARALLEL, TAG_PARALLEL_END = -3, -4
TAG_OUTLINES, TAG_OUTLINES_END = -5, -6
TAG_SUBTASK, TAG_SUBTASK_END = -7, -8
TAG_TRIAL, TAG_TRIAL_END = -9, -10
TAG_THREAD, TAG_THREAD_END = -11, -12


def random_trace(seed: int, *, max_depth: int = 2, p_parallel: float = 0.5,
                 text_len=(1, 24), entry_len=(1, 6), entries=(1, 4), body_items=(1, 3),
                 p_mismatch: float = 0.1, p_empty_thread: float = 0.05) -> np.ndarray:
    """A random trace in the grammar: bodies of text runs and parallel blocks
    nested up to `max_depth`, outlines of 1..4 Subtask/Trial entries, usually
    one thread per entry (sometimes one more or one fewer), occasionally an
    empty thread body.  Text token ids are random non-negative ints."""
    rng = np.random.default_rng(seed)
    out = [TAG_THINK]

    def text(lo_hi):
        n = int(rng.integers(lo_hi[0], lo_hi[1] + 1))
        out.extend(int(x) for x in rng.integers(0, 1 << 17, size=n))

    def body(level, allow_empty):
        if allow_empty and rng.random() < p_empty_thread:
            return
        for _ in range(int(rng.integers(body_items[0], body_items[1] + 1))):
            if level < max_depth and rng.random() < p_parallel:
                region(level)
            else:
                text(text_len)

    def region(level):
        out.extend([TAG_PARALLEL, TAG_OUTLINES])
        k = int(rng.integers(entries[0], entries[1] + 1))
        for _ in range(k):
            sub = rng.random() < 0.5
            out.append(TAG_SUBTASK if sub else TAG_TRIAL)
            text(entry_len)
            out.append(TAG_SUBTASK_END if sub else TAG_TRIAL_END)
        out.append(TAG_OUTLINES_END)
        nthreads = k
        if rng.random() < p_mismatch:
            nthreads = max(1, k + int(rng.choice([-1, 1])))
        for _ in range(nthreads):
            out.append(TAG_THREAD)
            body(level + 1, True)
            out.append(TAG_THREAD_END)
        out.append(TAG_PARALLEL_END)

    body(0, False)
    out.append(TAG_THINK_END)
    return np.asarray(out, dtype=np.int32)


def paper_scale_trace(seed: int) -> np.ndarray:
    """A trace of about the size the paper reports (tens of thousands of
    generated tokens, token-level acceleration near 1.7-1.9; Tab. 4, Tab. 5):
    one level of parallel blocks with 2-3 threads each."""
    return random_trace(seed, max_depth=1, p_parallel=0.4, text_len=(250, 1200),
                        entry_len=(10, 60), entries=(2, 3), body_items=(5, 10), p_mismatch=0.0,
                        p_empty_thread=0.0)


def free_pages(tree: ForkTree) -> list:
    """Physical pages no node owns, in index order."""
    used = set(int(x) for x in tree.page_ids)
    return [p for p in range(tree.num_physical_pages) if p not in used]


def grow_branches(tree: ForkTree, pool: list):
    """The tree after one generated token per branch: every branch node gains
    one token; a branch whose node length is a multiple of 16 takes the next
    page of `pool` (consumed in place).  Returns (tree, new_pages) with
    new_pages[b] the page branch b took, or -1.  The token's K and V are the
    values already in that slot of the pool."""
    node_len = tree.node_len.copy()
    pages = [list(tree.page_ids[tree.node_page_ptr[n]:tree.node_page_ptr[n + 1]])
             for n in range(tree.num_nodes)]
    new_pages = np.full(tree.num_leaves, -1, dtype=np.int32)
    for b, n in enumerate(tree.leaf_node):
        if node_len[n] % PAGE_SIZE == 0:
            pg = pool.pop(0)
            new_pages[b] = pg
            pages[n].append(pg)
        node_len[n] += 1
    ptr = np.zeros(tree.num_nodes + 1, dtype=np.int32)
    ptr[1:] = np.cumsum([len(p) for p in pages])
    ids = np.asarray([x for p in pages for x in p], dtype=np.int32)
    return replace(tree, node_len=node_len, node_page_ptr=ptr, page_ids=ids), new_pages


def fork_branch(tree: ForkTree, b: int, child_lens: Sequence[int], pool: list, seed: int = 0):
    """The tree after branch b forks into len(child_lens) threads (its node
    gets one child node per thread, appended in order).  Child 0 is branch
    b; child c >= 1 is the new branch num_leaves + c - 1, with a fresh query
    row drawn from ``seed``.  Each child takes ceil(len / 16) pages of `pool`
    (consumed in place); their K and V are the values already in the pool.
    Returns (tree, child_pages) with child_pages[c] the pages of child c."""
    k = len(child_lens)
    nb = int(tree.leaf_node[b])
    n0 = tree.num_nodes
    child_pages = []
    for ln in child_lens:
        child_pages.append([pool.pop(0) for _ in range((int(ln) + PAGE_SIZE - 1) // PAGE_SIZE)])
    parent = np.concatenate([tree.parent, np.full(k, nb, dtype=np.int32)]).astype(np.int32)
    node_len = np.concatenate([tree.node_len, np.asarray(child_lens, dtype=np.int32)]).astype(np.int32)
    counts = [len(p) for p in child_pages]
    ptr = np.concatenate([tree.node_page_ptr,
                          tree.node_page_ptr[-1] + np.cumsum(counts, dtype=np.int64)]).astype(np.int32)
    page_ids = np.concatenate([tree.page_ids,
                               np.asarray([x for p in child_pages for x in p], dtype=np.int32)])
    leaf_node = tree.leaf_node.copy()
    leaf_node[b] = n0
    leaf_node = np.concatenate([leaf_node, np.arange(n0 + 1, n0 + k, dtype=np.int32)])
    q = tree.q
    if k > 1 and q.numel():
        gen = torch.Generator(device=q.device)
        gen.manual_seed(int(seed) + 104729)
        extra = torch.randn((k - 1,) + tuple(q.shape[1:]), generator=gen, device=q.device,
                            dtype=torch.float32) * float(tree.meta.get("q_std", 1.0))
        q = torch.cat([q, extra.to(q.dtype)], dim=0)
    return replace(tree, parent=parent, node_len=node_len, node_page_ptr=ptr,
                   page_ids=page_ids.astype(np.int32), leaf_node=leaf_node.astype(np.int32),
                   q=q), child_pages


def build_prefill(name: str, parent, node_len, chunk_node, *, num_q_heads: int,
                  num_kv_heads: int, head_dim: int, mode: str = "bf16", seed: int = 0,
                  device="cpu", q_std: float = 1.0, **kw) -> ForkTree:
    """A tree-masked prefill workload: the tree and KV of build_tree, with
    every token of each chunk node (childless) a query.  leaf_node holds the
    chunk nodes; q is [sum of chunk lengths, H_q, d], chunk by chunk."""
    tree = build_tree(name, parent, node_len, chunk_node, num_q_heads=num_q_heads,
                      num_kv_heads=num_kv_heads, head_dim=head_dim, mode=mode, seed=seed,
                      device=device, q_std=q_std, **kw)
    nq = int(sum(int(tree.node_len[c]) for c in tree.leaf_node))
    gen = torch.Generator(device=device)
    gen.manual_seed(seed + 7919)
    q = torch.randn((nq, num_q_heads, head_dim), generator=gen, device=device,
                    dtype=torch.float32) * q_std
    q = q.to(torch.float32 if mode == "fp32" else torch.bfloat16)
    meta = dict(tree.meta)
    meta["prefill"] = True
    return replace(tree, q=q, meta=meta)


def fork_prefill(mode="bf16", device="cpu", chunk=64, threads=16, **kw) -> ForkTree:
    """Thread openings at </Outlines> on the Llama-3-8B shape (32 q / 8 kv, d
    128): prefix 2048 and `threads` chunks of `chunk` tokens under it, each a
    thread's first tokens prefilled against the shared prefix."""
    rng = np.random.default_rng(6)
    parent = [-1] + [0] * threads
    lens = [2048] + [chunk] * threads
    return build_prefill(f"fork_prefill_2048_{threads}x{chunk}", parent, lens,
                         list(range(1, threads + 1)), num_q_heads=32, num_kv_heads=8,
                         head_dim=128, mode=mode, rng=rng, q_std=1.0 / math.sqrt(128.0),
                         device=device, **kw)


def join_prefill(mode="bf16", device="cpu", chunk=1024, threads=16, **kw) -> ForkTree:
    """The join with the threads' KV reused in place, on the Llama-3-8B shape:
    a chain prefix 2048 -> `threads` thread nodes of U[512, 4096] tokens (the
    trials of llama3_trials, concatenated in order) -> a `chunk`-token node
    prefilled against all of it."""
    rng = np.random.default_rng(1)
    lens = [2048] + [_uniform(rng, 512, 4096) for _ in range(threads)] + [chunk]
    parent = [-1] + list(range(len(lens) - 1))
    return build_prefill(f"join_prefill_2048_{threads}threads_{chunk}", parent, lens,
                         [len(lens) - 1], num_q_heads=32, num_kv_heads=8, head_dim=128,
                         mode=mode, rng=rng, q_std=1.0 / math.sqrt(128.0), device=device, **kw)


PREFILL_CONFIGS = {"fork": fork_prefill, "join": join_prefill}
