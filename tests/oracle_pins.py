"""Checks that pin the fp64 oracle to things other than itself.

Each ``check_*`` takes an ``oracle.Oracle`` and raises AssertionError when the
oracle disagrees with what the definition and mathematics fix:

* the bf16 / e4m3 decoders against torch's own dtype conversions;
* decode against torch's softmax / logsumexp / matmul (library routines) on a
  contiguous K/V that this file gathers from the page table itself;
* the split invariant: attention over a KV range split in two and merged by
  log-sum-exp equals attention over the whole range;
* symmetries: GQA equals repeat-interleaved MHA, page permutation and
  identical suffixes give bit-identical outputs;
* closed forms: constant V, constant K, a dominant key, a zero query, an
  empty path.

The same checks run against copies of the oracle with a planted mistake
(tests/test_oracle_mutations.py) to show that each mistake is caught.
"""
import math

import numpy as np
import torch

from paper_2608_24658_gb300 import workloads as W

TOL = 1e-12


# ----------------------------------------------------------------------------
# helpers written independently of the oracle
# ----------------------------------------------------------------------------

def _to_f64(t: torch.Tensor, scale=None) -> torch.Tensor:
    x = t.to(torch.float64)
    if scale is not None:
        x = x * scale.to(torch.float64).view(1, -1, 1, 1)
    return x


def gather_path(tree: W.ForkTree, b: int):
    """Contiguous K, V [T, H_kv, d] float64 for branch b, root first."""
    ks, vs = [], []
    kp = _to_f64(tree.k_pages.cpu(), tree.k_scale.cpu() if tree.k_scale is not None else None)
    vp = _to_f64(tree.v_pages.cpu(), tree.v_scale.cpu() if tree.v_scale is not None else None)
    for n in tree.path(b):
        ln = int(tree.node_len[n])
        pages = tree.page_ids[tree.node_page_ptr[n]:tree.node_page_ptr[n + 1]]
        if ln == 0:
            continue
        idx = torch.as_tensor(pages.astype(np.int64))
        k = kp.index_select(0, idx).permute(0, 2, 1, 3).reshape(-1, tree.num_kv_heads, tree.head_dim)
        v = vp.index_select(0, idx).permute(0, 2, 1, 3).reshape(-1, tree.num_kv_heads, tree.head_dim)
        ks.append(k[:ln])
        vs.append(v[:ln])
    if not ks:
        z = torch.zeros((0, tree.num_kv_heads, tree.head_dim), dtype=torch.float64)
        return z, z.clone()
    return torch.cat(ks), torch.cat(vs)


def torch_attention(q, k, v, scale):
    """q [d], k/v [T, d] float64 -> (o [d], lse) via library softmax/logsumexp."""
    s = (k @ q) * scale
    p = torch.softmax(s, dim=0)
    return p @ v, torch.logsumexp(s, dim=0)


def reference_decode(tree: W.ForkTree):
    scale = tree.sm_scale if tree.sm_scale > 0 else 1.0 / math.sqrt(tree.head_dim)
    g = tree.group
    q = tree.q.cpu().to(torch.float64)
    out = np.zeros((tree.num_leaves, tree.num_q_heads, tree.head_dim))
    lse = np.zeros((tree.num_leaves, tree.num_q_heads))
    for b in range(tree.num_leaves):
        k, v = gather_path(tree, b)
        for h in range(tree.num_q_heads):
            if k.shape[0] == 0:
                out[b, h] = 0.0
                lse[b, h] = -math.inf
                continue
            o, l = torch_attention(q[b, h], k[:, h // g], v[:, h // g], scale)
            out[b, h] = o.numpy()
            lse[b, h] = float(l)
    return out, lse


def run(orc, tree, **kw):
    return orc.decode(num_q_heads=tree.num_q_heads, num_kv_heads=tree.num_kv_heads,
                      head_dim=tree.head_dim, mode=tree.mode, parent=tree.parent,
                      node_len=tree.node_len, node_page_ptr=tree.node_page_ptr,
                      page_ids=tree.page_ids, leaf_node=tree.leaf_node, q=tree.q,
                      k_pages=tree.k_pages, v_pages=tree.v_pages, k_scale=tree.k_scale,
                      v_scale=tree.v_scale, sm_scale=tree.sm_scale, **kw)


def single_node_tree(k, v, q, mode="bf16", permute_seed=None):
    """One-node tree over contiguous K/V [T, H_kv, d] (already in the KV dtype)."""
    T, hkv, d = k.shape
    npages = (T + 15) // 16
    shape = (max(npages, 1), hkv, 16, d)
    kp = torch.zeros(shape, dtype=k.dtype)
    vp = torch.zeros(shape, dtype=v.dtype)
    for t in range(T):
        kp[t // 16, :, t % 16] = k[t]
        vp[t // 16, :, t % 16] = v[t]
    ids = np.arange(npages, dtype=np.int32)
    if permute_seed is not None and npages > 1:
        perm = np.random.default_rng(permute_seed).permutation(npages)
        kp2, vp2 = kp.clone(), vp.clone()
        kp2[perm] = kp[:npages]
        vp2[perm] = vp[:npages]
        kp, vp, ids = kp2, vp2, perm.astype(np.int32)
    return W.ForkTree(name="single", num_q_heads=q.shape[1], num_kv_heads=hkv, head_dim=d,
                      mode=mode, parent=np.array([-1], np.int32), node_len=np.array([T], np.int32),
                      node_page_ptr=np.array([0, npages], np.int32), page_ids=ids,
                      leaf_node=np.array([0], np.int32), num_physical_pages=shape[0],
                      q=q, k_pages=kp, v_pages=vp)


def _close(a, b, tol=TOL, what=""):
    a, b = np.asarray(a), np.asarray(b)
    assert a.shape == b.shape, (what, a.shape, b.shape)
    fin = np.isfinite(b)
    assert np.array_equal(np.isfinite(a), fin), f"{what}: finiteness differs"
    assert np.array_equal(a[~fin], b[~fin], equal_nan=True), f"{what}: non-finite values differ"
    if fin.any():
        err = float(np.max(np.abs(a[fin] - b[fin])))
        assert err <= tol, f"{what}: max abs err {err:.3e} > {tol:.1e}"


# ----------------------------------------------------------------------------
# pins
# ----------------------------------------------------------------------------

def check_bf16_decoder(orc):
    bits = np.arange(1 << 16, dtype=np.uint16)
    ref = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    got = np.array([orc.bf16_to_double(int(x)) for x in bits])
    _close(got, ref, 0.0, "bf16 decode")


def check_e4m3_decoder(orc):
    bits = np.arange(256, dtype=np.uint8)
    ref = torch.from_numpy(bits).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    got = np.array([orc.e4m3_to_double(int(x)) for x in bits])
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan), "e4m3 NaN codes differ"
    _close(got[~nan], ref[~nan], 0.0, "e4m3 decode")


def _plain_cases():
    yield W.figure3_tree(seed=5)
    yield W.random_tree(21, h_q=8, h_kv=2, d=64, len_range=(0, 70))
    yield W.random_tree(22, h_q=4, h_kv=4, d=128, depth=2, len_range=(0, 40))
    yield W.random_tree(23, h_q=16, h_kv=2, d=64, depth=1, num_requests=3, mode="fp32")
    yield W.random_tree(24, h_q=8, h_kv=2, d=64, depth=2, mode="fp8")
    yield W.figure3_tree(seed=6, sm_scale=0.37)
    yield W.build_tree("chain", [-1, 0, 1, 2], [17, 0, 33, 5], [3], num_q_heads=6,
                       num_kv_heads=3, head_dim=64, seed=9, tail_value=float("nan"))


def check_plain_attention(orc):
    """Every branch and head equals library softmax attention over its gathered path."""
    for tree in _plain_cases():
        out, lse = run(orc, tree)
        ref_o, ref_l = reference_decode(tree)
        _close(out, ref_o, TOL, f"{tree.name} out")
        _close(lse, ref_l, TOL, f"{tree.name} lse")


def check_selection(orc):
    tree = W.figure3_tree(seed=7)
    full_o, full_l = run(orc, tree)
    sel = [5, 0, 3]
    o, l = run(orc, tree, sel=sel)
    assert np.array_equal(o, full_o[sel]) and np.array_equal(l, full_l[sel])


def check_split_merge(orc):
    """Attention over [0,T) equals the LSE merge of [0,s) and [s,T), s in {0..T}."""
    g = torch.Generator().manual_seed(3)
    T, hkv, hq, d = 75, 2, 4, 64
    k = torch.randn((T, hkv, d), generator=g).to(torch.bfloat16)
    v = torch.randn((T, hkv, d), generator=g).to(torch.bfloat16)
    q = torch.randn((1, hq, d), generator=g).to(torch.bfloat16)
    whole_o, whole_l = run(orc, single_node_tree(k, v, q))
    for s in (0, 1, 16, 31, 40, 74, 75):
        oa, la = run(orc, single_node_tree(k[:s], v[:s], q))
        ob, lb = run(orc, single_node_tree(k[s:], v[s:], q, permute_seed=s))
        o, l = orc.lse_merge(oa, la, ob, lb)
        _close(o, whole_o, TOL, f"split {s} out")
        _close(l, whole_l, TOL, f"split {s} lse")


def check_lse_merge_identities(orc):
    rng = np.random.default_rng(0)
    o = rng.standard_normal((3, 8))
    lse = rng.standard_normal(3)
    ninf = np.full(3, -np.inf)
    zero = np.zeros((3, 8))
    m, l = orc.lse_merge(o, lse, zero, ninf)
    _close(m, o, 0.0, "merge with empty (right)")
    _close(l, lse, 0.0, "merge lse with empty (right)")
    m, l = orc.lse_merge(zero, ninf, o, lse)
    _close(m, o, 0.0, "merge with empty (left)")
    m, l = orc.lse_merge(zero, ninf, zero, ninf)
    _close(m, zero, 0.0, "merge empty/empty")
    assert np.all(l == -np.inf)
    m, l = orc.lse_merge(o, lse, o, lse)      # equal halves: same o, lse + ln 2
    _close(m, o, 1e-15, "merge equal halves")
    _close(l, lse + math.log(2.0), 1e-15, "merge equal halves lse")


def check_identical_suffixes(orc):
    tree = W.build_tree("twins", [-1, 0, 0], [50, 29, 29], [1, 2], num_q_heads=8,
                        num_kv_heads=2, head_dim=64, seed=4)
    p1 = tree.page_ids[tree.node_page_ptr[1]:tree.node_page_ptr[2]]
    p2 = tree.page_ids[tree.node_page_ptr[2]:tree.node_page_ptr[3]]
    for pages in (tree.k_pages, tree.v_pages):
        pages[torch.as_tensor(p2.astype(np.int64))] = pages[torch.as_tensor(p1.astype(np.int64))]
    tree.q[1] = tree.q[0]
    out, lse = run(orc, tree)
    assert np.array_equal(out[0], out[1]) and np.array_equal(lse[0], lse[1])
    # and the two suffixes really are distinct from the other branches' data
    ref_o, _ = reference_decode(tree)
    _close(out, ref_o, TOL, "twins")


def check_gqa_equals_mha(orc):
    tree = W.random_tree(31, h_q=8, h_kv=2, d=64, depth=2, len_range=(1, 50))
    out, lse = run(orc, tree)
    g = tree.group
    mha = W.ForkTree(**{**tree.__dict__, "num_kv_heads": tree.num_q_heads,
                        "k_pages": tree.k_pages.repeat_interleave(g, dim=1),
                        "v_pages": tree.v_pages.repeat_interleave(g, dim=1)})
    out2, lse2 = run(orc, mha)
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2), "GQA != repeat-interleaved MHA"


def check_page_permutation(orc):
    tree = W.random_tree(41, h_q=4, h_kv=2, d=64, depth=2, permute_pages=False, extra_pages=0)
    out, lse = run(orc, tree)
    P = tree.num_physical_pages
    perm = np.random.default_rng(1).permutation(P)
    kp = torch.empty_like(tree.k_pages)
    vp = torch.empty_like(tree.v_pages)
    kp[torch.as_tensor(perm)] = tree.k_pages
    vp[torch.as_tensor(perm)] = tree.v_pages
    moved = W.ForkTree(**{**tree.__dict__, "k_pages": kp, "v_pages": vp,
                          "page_ids": perm[tree.page_ids].astype(np.int32)})
    out2, lse2 = run(orc, moved)
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2), "page permutation changed output"


def check_closed_forms(orc):
    g = torch.Generator().manual_seed(5)
    T, hkv, hq, d = 53, 2, 4, 64
    q = torch.randn((1, hq, d), generator=g).to(torch.float32)
    k = torch.randn((T, hkv, d), generator=g).to(torch.float32)
    v = torch.randn((T, hkv, d), generator=g).to(torch.float32)
    scale = 1.0 / math.sqrt(d)
    # V constant per head => o equals that constant
    vc = torch.zeros_like(v)
    vc[:, 0] = 0.75
    vc[:, 1] = -2.5
    o, _ = run(orc, single_node_tree(k, vc, q, mode="fp32"))
    for h in range(hq):
        _close(o[0, h], np.full(d, 0.75 if h // 2 == 0 else -2.5), 1e-14, "V const")
    # K constant => uniform weights: o = mean V, lse = s + ln T
    kc = k[:1].expand(T, hkv, d).contiguous()
    o, l = run(orc, single_node_tree(kc, v, q, mode="fp32"))
    for h in range(hq):
        s = float((q[0, h].double() * kc[0, h // 2].double()).sum()) * scale
        _close(o[0, h], v[:, h // 2].double().mean(0).numpy(), 1e-14, "K const")
        _close(l[0, h], s + math.log(T), 1e-13, "K const lse")
    # q = 0 => o = mean V, lse = ln T
    qz = torch.zeros_like(q)
    o, l = run(orc, single_node_tree(k, v, qz, mode="fp32"))
    for h in range(hq):
        _close(o[0, h], v[:, h // 2].double().mean(0).numpy(), 1e-14, "q zero")
        _close(l[0, h], math.log(T), 1e-14, "q zero lse")
    # one key aligned with q at a huge score => o equals that key's value
    kd = k.clone()
    j = 17
    for h in range(hkv):
        kd[j, h] = q[0, 2 * h] * 400.0
    o, _ = run(orc, single_node_tree(kd, v, q, mode="fp32"))
    for h in range(0, hq, 2):
        _close(o[0, h], v[j, h // 2].double().numpy(), 1e-12, "dominant key")


def check_empty_path(orc):
    tree = W.build_tree("empty", [-1, 0, 0], [0, 0, 5], [1, 2], num_q_heads=4,
                        num_kv_heads=2, head_dim=64, seed=2)
    out, lse = run(orc, tree)
    assert np.all(out[0] == 0.0) and np.all(lse[0] == -np.inf)
    ref_o, ref_l = reference_decode(tree)
    _close(out, ref_o, TOL, "empty path")
    _close(lse, ref_l, TOL, "empty path lse")


ALL_CHECKS = [check_bf16_decoder, check_e4m3_decoder, check_plain_attention, check_selection,
              check_split_merge, check_lse_merge_identities, check_identical_suffixes,
              check_gqa_equals_mha, check_page_permutation, check_closed_forms,
              check_empty_path]
