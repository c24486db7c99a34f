"""fp64 CPU oracle for fork-tree decode attention -- TEST INFRASTRUCTURE.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this package.  The product path (``paper_2608_24658_gb300``)
never imports it and shares no code with it.

The arithmetic lives in ``parason_oracle.c`` (plain C, fp64); this module
only marshals buffers.  ``decode`` evaluates, for each selected branch, plain
softmax attention over the branch's full root-to-leaf KV (Sec. 3.4: branches
are independent workers; Fig. 1 / Sec. 3.1: branch outputs are concatenated
into later context, so every branch's attention output is needed).
``lse_merge`` is the log-sum-exp combination of two attention results over
disjoint key sets.
"""
import ctypes

import numpy as np
import torch

from . import build as _build

MODES = {"bf16": 0, "fp32": 1, "fp8": 2}


def _i32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _cpu(t):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        t = torch.as_tensor(t)
    return t.detach().to("cpu").contiguous()


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        return x.ctypes.data_as(ctypes.c_void_p)
    return ctypes.c_void_p(x.data_ptr())


class Oracle:
    """ctypes front end of one build of ``parason_oracle.c``."""

    def __init__(self, lib_path: str):
        lib = ctypes.CDLL(lib_path)
        p = ctypes.c_void_p
        i32 = ctypes.c_int32
        lib.parason_oracle_decode.restype = ctypes.c_int
        lib.parason_oracle_decode.argtypes = [
            i32, i32, i32, i32, i32, ctypes.c_double,
            i32, p, p, p, p, i32, p, p, p, p, p, p,
            i32, p, p, p, i32]
        lib.parason_oracle_prefill.restype = ctypes.c_int
        lib.parason_oracle_prefill.argtypes = [
            i32, i32, i32, i32, i32, ctypes.c_double,
            i32, p, p, p, p, i32, p, p, p, p, p, p,
            i32, p, p, p, i32]
        lib.parason_oracle_lse_merge.restype = None
        lib.parason_oracle_lse_merge.argtypes = [p, p, p, p, p, p, ctypes.c_int64, i32]
        lib.parason_oracle_bf16_to_double.restype = ctypes.c_double
        lib.parason_oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.parason_oracle_e4m3_to_double.restype = ctypes.c_double
        lib.parason_oracle_e4m3_to_double.argtypes = [ctypes.c_uint8]
        lib.parason_oracle_num_threads.restype = ctypes.c_int
        self.lib = lib
        self.path = lib_path

    def num_threads(self) -> int:
        return self.lib.parason_oracle_num_threads()

    def decode(self, *, num_q_heads, num_kv_heads, head_dim, mode, parent, node_len,
               node_page_ptr, page_ids, leaf_node, q, k_pages, v_pages,
               k_scale=None, v_scale=None, sm_scale=0.0, page_size=16, sel=None,
               threads=0):
        """Return (out [S, H_q, d] float64, lse [S, H_q] float64) for branches ``sel``.

        ``q``/``k_pages``/``v_pages`` are tensors holding the raw values the GPU
        path reads (bf16, fp32, or e4m3 bytes for KV in fp8 mode); they are
        passed as bytes and widened to fp64 inside the C code.
        """
        parent, node_len = _i32(parent), _i32(node_len)
        node_page_ptr, page_ids, leaf_node = _i32(node_page_ptr), _i32(page_ids), _i32(leaf_node)
        q, k_pages, v_pages = _cpu(q), _cpu(k_pages), _cpu(v_pages)
        k_scale = None if k_scale is None else _cpu(k_scale).to(torch.float32)
        v_scale = None if v_scale is None else _cpu(v_scale).to(torch.float32)
        sel_arr = None if sel is None else _i32(sel)
        n_sel = len(leaf_node) if sel is None else len(sel_arr)
        out = np.zeros((n_sel, num_q_heads, head_dim), dtype=np.float64)
        lse = np.zeros((n_sel, num_q_heads), dtype=np.float64)
        st = self.lib.parason_oracle_decode(
            num_q_heads, num_kv_heads, head_dim, page_size, MODES[mode], float(sm_scale),
            len(parent), _ptr(parent), _ptr(node_len), _ptr(node_page_ptr), _ptr(page_ids),
            len(leaf_node), _ptr(leaf_node), _ptr(q), _ptr(k_pages), _ptr(v_pages),
            _ptr(k_scale), _ptr(v_scale), n_sel, _ptr(sel_arr), _ptr(out), _ptr(lse),
            int(threads))
        if st != 0:
            raise ValueError(f"oracle decode failed with status {st}")
        return out, lse

    def prefill(self, *, num_q_heads, num_kv_heads, head_dim, mode, parent, node_len,
                node_page_ptr, page_ids, chunk_node, q, k_pages, v_pages, k_scale=None,
                v_scale=None, sm_scale=0.0, page_size=16, sel=None, threads=0, **_):
        """Tree-masked prefill: (out [S, H_q, d], lse [S, H_q]) fp64 for queries ``sel``
        (every token of every chunk node, chunk by chunk; all if None)."""
        parent, node_len = _i32(parent), _i32(node_len)
        node_page_ptr, page_ids, chunk_node = _i32(node_page_ptr), _i32(page_ids), _i32(chunk_node)
        q, k_pages, v_pages = _cpu(q), _cpu(k_pages), _cpu(v_pages)
        k_scale = None if k_scale is None else _cpu(k_scale).float().contiguous()
        v_scale = None if v_scale is None else _cpu(v_scale).float().contiguous()
        total = int(sum(int(node_len[c]) for c in chunk_node))
        sel_arr = None if sel is None else _i32(sel)
        n_sel = total if sel is None else len(sel_arr)
        out = np.zeros((n_sel, num_q_heads, head_dim), dtype=np.float64)
        lse = np.zeros((n_sel, num_q_heads), dtype=np.float64)
        st = self.lib.parason_oracle_prefill(
            num_q_heads, num_kv_heads, head_dim, page_size, MODES[mode], float(sm_scale),
            len(parent), _ptr(parent), _ptr(node_len), _ptr(node_page_ptr), _ptr(page_ids),
            len(chunk_node), _ptr(chunk_node), _ptr(q), _ptr(k_pages), _ptr(v_pages),
            _ptr(k_scale), _ptr(v_scale), n_sel, _ptr(sel_arr), _ptr(out), _ptr(lse),
            int(threads))
        if st != 0:
            raise ValueError(f"oracle prefill failed with status {st}")
        return out, lse

    def lse_merge(self, o_a, lse_a, o_b, lse_b):
        """Merge two attention results over disjoint key sets (fp64 in, fp64 out)."""
        o_a = np.ascontiguousarray(o_a, dtype=np.float64)
        o_b = np.ascontiguousarray(o_b, dtype=np.float64)
        lse_a = np.ascontiguousarray(lse_a, dtype=np.float64)
        lse_b = np.ascontiguousarray(lse_b, dtype=np.float64)
        d = o_a.shape[-1]
        rows = o_a.size // d
        o = np.zeros_like(o_a)
        lse = np.zeros_like(lse_a)
        self.lib.parason_oracle_lse_merge(_ptr(o_a), _ptr(lse_a), _ptr(o_b), _ptr(lse_b),
                                          _ptr(o), _ptr(lse), rows, d)
        return o, lse

    def bf16_to_double(self, bits: int) -> float:
        return self.lib.parason_oracle_bf16_to_double(bits)

    def e4m3_to_double(self, bits: int) -> float:
        return self.lib.parason_oracle_e4m3_to_double(bits)


_default = None


def default() -> Oracle:
    global _default
    if _default is None:
        _default = Oracle(_build.build())
    return _default


def num_threads() -> int:
    return default().num_threads()


def decode(**kw):
    return default().decode(**kw)


def lse_merge(o_a, lse_a, o_b, lse_b):
    return default().lse_merge(o_a, lse_a, o_b, lse_b)


def prefill(**kw):
    return default().prefill(**kw)


def bf16_to_double(bits: int) -> float:
    return default().bf16_to_double(bits)


def e4m3_to_double(bits: int) -> float:
    return default().e4m3_to_double(bits)


def tree_kwargs(tree):
    """The oracle's keyword arguments for a fork-tree workload object.

    Reads only plain fields (shapes, integer arrays, input tensors), so the
    oracle stays independent of how the workload was generated.
    """
    return dict(num_q_heads=tree.num_q_heads, num_kv_heads=tree.num_kv_heads,
                head_dim=tree.head_dim, mode=tree.mode, parent=tree.parent,
                node_len=tree.node_len, node_page_ptr=tree.node_page_ptr,
                page_ids=tree.page_ids, leaf_node=tree.leaf_node, q=tree.q,
                k_pages=tree.k_pages, v_pages=tree.v_pages,
                k_scale=tree.k_scale, v_scale=tree.v_scale,
                sm_scale=tree.sm_scale, page_size=tree.page_size)


__all__ = ["Oracle", "default", "decode", "lse_merge", "bf16_to_double",
           "e4m3_to_double", "num_threads", "tree_kwargs", "MODES"]
