"""Python binding of libparason: argument marshalling only.

Every step of the decode path runs in the library's CUDA kernels; this module
checks shapes/dtypes/devices of torch tensors, passes raw pointers through the
C ABI (include/parason.h) and turns statuses into exceptions.  PyTorch provides
device memory and streams, nothing else.
"""
from __future__ import annotations

import ctypes
from typing import Optional

import numpy as np
import torch

from . import _lib
from ._lib import ParasonError, check

_KV_DTYPES = {"bf16": torch.bfloat16, "fp32": torch.float32, "fp8": torch.float8_e4m3fn}
_Q_DTYPES = {"bf16": torch.bfloat16, "fp32": torch.float32, "fp8": torch.bfloat16}


def _stream_handle(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ptr(x) -> Optional[ctypes.c_void_p]:
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        return x.ctypes.data_as(ctypes.c_void_p)
    return ctypes.c_void_p(x.data_ptr())


class Plan:
    """Decode plan of one fork tree (C type ``parason_plan``).

    ``host_only=True`` builds the same work decomposition without touching
    CUDA (for inspection on machines without a GPU).  ``prefill=True`` plans a
    tree-masked prefill instead (parason_prefill_plan): ``leaf_node`` then
    lists the chunk nodes, and every token of every chunk is a query row of
    ``q`` (chunk by chunk) in ``decode``.
    """

    def __init__(self, *, num_q_heads: int, num_kv_heads: int, head_dim: int, mode: str,
                 parent, node_len, node_page_ptr, page_ids, leaf_node,
                 num_physical_pages: int, sm_scale: float = 0.0, page_size: int = 16,
                 stream=None, host_only: bool = False, num_sms: int = 152,
                 prefill: bool = False, shard=None):
        lib = _lib.load()
        self.mode = mode
        self.num_q_heads, self.num_kv_heads, self.head_dim = num_q_heads, num_kv_heads, head_dim
        self.num_leaves = len(leaf_node)
        self.num_physical_pages = int(num_physical_pages)
        self._cfg = _lib.AttnConfig(num_q_heads, num_kv_heads, head_dim, page_size,
                                    _lib.MODES[mode], float(sm_scale))
        parent, node_len = _i32(parent), _i32(node_len)
        node_page_ptr, page_ids, leaf_node = _i32(node_page_ptr), _i32(page_ids), _i32(leaf_node)
        out = ctypes.c_void_p()
        kind = "prefill" if prefill else "attn"
        self.shard = shard
        if shard is not None:
            # (kind, rank, world): one rank's plan (parason_attn_plan_shard)
            skind, rank, world = (int(x) for x in shard)
            if prefill:
                raise ValueError("prefill plans are not sharded")
            args = (ctypes.byref(self._cfg), len(parent), _ptr(parent), _ptr(node_len),
                    _ptr(node_page_ptr), _ptr(page_ids), len(leaf_node), _ptr(leaf_node),
                    self.num_physical_pages, skind, rank, world)
            if host_only:
                st = lib.parason_attn_plan_shard_host(*args, num_sms, ctypes.byref(out))
            else:
                st = lib.parason_attn_plan_shard(*args, _stream_handle(stream), ctypes.byref(out))
            check(st, "parason_attn_plan_shard")
            self._h = out
            self._ws = None
            self.host_only = host_only
            self.prefill = False
            info = self.info()
            self.num_leaves = int(info["num_leaves"])
            if skind == _lib.SHARD_KV_HEADS:
                self.num_q_heads //= world
                self.num_kv_heads //= world
            return
        if host_only:
            fn = getattr(lib, f"parason_{kind}_plan_host")
            st = fn(ctypes.byref(self._cfg), len(parent), _ptr(parent), _ptr(node_len),
                    _ptr(node_page_ptr), _ptr(page_ids), len(leaf_node), _ptr(leaf_node),
                    self.num_physical_pages, num_sms, ctypes.byref(out))
        else:
            fn = getattr(lib, f"parason_{kind}_plan")
            st = fn(ctypes.byref(self._cfg), len(parent), _ptr(parent), _ptr(node_len),
                    _ptr(node_page_ptr), _ptr(page_ids), len(leaf_node), _ptr(leaf_node),
                    self.num_physical_pages, _stream_handle(stream), ctypes.byref(out))
        check(st, f"parason_{kind}_plan")
        self._h = out
        self._ws = None
        self.host_only = host_only
        self.prefill = prefill
        if prefill:
            self.num_leaves = int(self.info()["num_leaves"])     # queries

    @classmethod
    def for_tree(cls, tree, **kw) -> "Plan":
        """Plan of a ``workloads.ForkTree`` (or any object with the same fields)."""
        return cls(num_q_heads=tree.num_q_heads, num_kv_heads=tree.num_kv_heads,
                   head_dim=tree.head_dim, mode=tree.mode, parent=tree.parent,
                   node_len=tree.node_len, node_page_ptr=tree.node_page_ptr,
                   page_ids=tree.page_ids, leaf_node=tree.leaf_node,
                   num_physical_pages=tree.num_physical_pages, sm_scale=tree.sm_scale,
                   page_size=tree.page_size, **kw)

    @classmethod
    def for_prefill(cls, tree, **kw) -> "Plan":
        """Prefill plan of a ``workloads.build_prefill`` workload (chunk nodes
        in ``leaf_node``)."""
        return cls.for_tree(tree, prefill=True, **kw)

    # ---------------------------------------------------------------- lifetime
    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            _lib.load().parason_plan_destroy(self._h)
        self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # ---------------------------------------------------------------- queries
    @property
    def handle(self) -> ctypes.c_void_p:
        if self._h is None:
            raise ValueError("plan is closed")
        return self._h

    @property
    def workspace_bytes(self) -> int:
        return int(_lib.load().parason_plan_workspace_bytes(self.handle))

    def info(self) -> dict:
        inf = _lib.PlanInfo()
        check(_lib.load().parason_plan_get_info(self.handle, ctypes.byref(inf)), "plan_get_info")
        return {name: getattr(inf, name) for name, _ in _lib.PlanInfo._fields_}

    def export(self, table: int) -> np.ndarray:
        inf = self.info()
        shape = {_lib.TABLE_ITEMS: (inf["num_items"], 8),
                 _lib.TABLE_DFS_LEAVES: (inf["num_leaves"],),
                 _lib.TABLE_MERGE_RANGES: (inf["num_leaves"] * self.num_kv_heads, 2),
                 _lib.TABLE_MERGE: (inf["num_merge_entries"],),
                 _lib.TABLE_WIDE_QUEUE: (inf["num_wide_items"],),
                 _lib.TABLE_NARROW_QUEUE: (inf["num_narrow_items"],),
                 _lib.TABLE_ITEM_ROWS: (inf["num_items"] + 1,),
                 _lib.TABLE_STREAM_ROWS: (inf["num_stream_rows"],),
                 _lib.TABLE_ITEM_KEY0: (inf["num_items"] if self.prefill else 0,),
                 _lib.TABLE_SHARD_BRANCHES: (inf["num_leaves"],)}[table]
        buf = np.zeros(shape, dtype=np.int32)
        check(_lib.load().parason_plan_export(self.handle, table, _ptr(buf), buf.nbytes),
              "plan_export")
        return buf

    def launches_per_decode(self) -> int:
        return int(_lib.load().parason_plan_launches_per_decode(self.handle))

    # ---------------------------------------------------------------- decode
    def workspace(self, device="cuda") -> torch.Tensor:
        """A cached device workspace of the size the plan needs."""
        n = max(self.workspace_bytes, 256)
        if self._ws is None or self._ws.numel() < n or self._ws.device != torch.device(device):
            self._ws = torch.empty(n, dtype=torch.uint8, device=device)
        return self._ws

    def decode(self, q: torch.Tensor, k_pages: torch.Tensor, v_pages: torch.Tensor,
               out: Optional[torch.Tensor] = None, lse: Optional[torch.Tensor] = None,
               workspace: Optional[torch.Tensor] = None, k_scale=None, v_scale=None,
               stream=None, want_lse: bool = True):
        """One decode step; returns (out, lse).  Asynchronous on ``stream``.
        ``q``, ``out`` and ``lse`` may be pinned host tensors: the kernels
        then read q from, and write the result to, host memory directly."""
        L, Hq, Hkv, d = self.num_leaves, self.num_q_heads, self.num_kv_heads, self.head_dim
        qd, kvd = _Q_DTYPES[self.mode], _KV_DTYPES[self.mode]
        if (q.dtype != qd or tuple(q.shape) != (L, Hq, d) or not q.is_contiguous()
                or not (q.is_cuda or q.is_pinned())):
            raise ValueError(f"q must be a contiguous cuda (or pinned host) {qd} tensor of "
                             f"shape {(L, Hq, d)}")
        dev = k_pages.device
        for name, t in (("k_pages", k_pages), ("v_pages", v_pages)):
            if (t.dtype != kvd or t.dim() != 4 or tuple(t.shape[1:]) != (Hkv, 16, d)
                    or t.shape[0] < self.num_physical_pages or not t.is_contiguous()
                    or not t.is_cuda or t.device != dev):
                raise ValueError(f"{name} must be a contiguous cuda {kvd} tensor "
                                 f"[>= {self.num_physical_pages}, {Hkv}, 16, {d}] on one device")
        if q.is_cuda and q.device != dev:
            raise ValueError(f"q must be on {dev}")
        if out is None:
            out = torch.empty_like(q) if q.is_cuda else torch.empty(q.shape, dtype=q.dtype).pin_memory()
        if lse is None and want_lse:
            lse = (torch.empty((L, Hq), dtype=torch.float32, device=dev) if q.is_cuda else
                   torch.empty((L, Hq), dtype=torch.float32).pin_memory())
        if workspace is None:
            workspace = self.workspace(dev)
        if self.mode == "fp8":
            if k_scale is None or v_scale is None:
                raise ValueError("fp8 mode needs k_scale and v_scale")
            for s in (k_scale, v_scale):
                if s.dtype != torch.float32 or s.numel() != Hkv or not s.is_cuda:
                    raise ValueError(f"scales must be cuda float32 [{Hkv}]")
        st = _lib.load().parason_attn_decode(
            self.handle, _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(k_scale), _ptr(v_scale),
            _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel() * workspace.element_size(),
            _stream_handle(stream))
        check(st, "parason_attn_decode")
        return out, lse

    def decode_no_alloc(self, q: torch.Tensor, k_pages: torch.Tensor, v_pages: torch.Tensor,
                        out: torch.Tensor, lse: Optional[torch.Tensor] = None, k_scale=None,
                        v_scale=None, stream=None):
        """``decode`` into caller-given ``out`` / ``lse`` with the library's fixed
        per-device scratch instead of a workspace; returns (out, lse).  Calls on
        one device must not overlap in time (they share the scratch)."""
        L, Hq, Hkv, d = self.num_leaves, self.num_q_heads, self.num_kv_heads, self.head_dim
        qd, kvd = _Q_DTYPES[self.mode], _KV_DTYPES[self.mode]
        for name, t in (("q", q), ("out", out)):
            if t.dtype != qd or tuple(t.shape) != (L, Hq, d) or not t.is_cuda or not t.is_contiguous():
                raise ValueError(f"{name} must be a contiguous cuda {qd} tensor of shape {(L, Hq, d)}")
        for name, t in (("k_pages", k_pages), ("v_pages", v_pages)):
            if (t.dtype != kvd or t.dim() != 4 or tuple(t.shape[1:]) != (Hkv, 16, d)
                    or t.shape[0] < self.num_physical_pages or not t.is_contiguous()
                    or t.device != q.device):
                raise ValueError(f"{name} must be a contiguous {kvd} tensor "
                                 f"[>= {self.num_physical_pages}, {Hkv}, 16, {d}] on {q.device}")
        if lse is not None and (lse.dtype != torch.float32 or tuple(lse.shape) != (L, Hq)
                                or not lse.is_cuda or not lse.is_contiguous()):
            raise ValueError(f"lse must be a contiguous cuda float32 tensor of shape {(L, Hq)}")
        if self.mode == "fp8":
            if k_scale is None or v_scale is None:
                raise ValueError("fp8 mode needs k_scale and v_scale")
            for s in (k_scale, v_scale):
                if s.dtype != torch.float32 or s.numel() != Hkv or not s.is_cuda:
                    raise ValueError(f"scales must be cuda float32 [{Hkv}]")
        st = _lib.load().parason_attn_decode_no_alloc(
            self.handle, _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(k_scale), _ptr(v_scale),
            _ptr(out), _ptr(lse), _stream_handle(stream))
        check(st, "parason_attn_decode_no_alloc")
        return out, lse

    def append(self, new_pages=None, stream=None) -> None:
        """One token appended to every branch's node (parason_plan_append).
        ``new_pages``: int32 [num_leaves], the page for each branch whose
        token opens one (-1 elsewhere), or None when no branch opens a page."""
        a = None
        if new_pages is not None:
            a = np.ascontiguousarray(np.asarray(new_pages, dtype=np.int32))
            if a.shape != (self.num_leaves,):
                raise ValueError(f"new_pages must have shape ({self.num_leaves},)")
        sh = None if self.host_only else _stream_handle(stream)
        check(_lib.load().parason_plan_append(self.handle, _ptr(a), sh), "parason_plan_append")

    def fork(self, branch: int, child_len, child_pages, stream=None) -> list:
        """Branch ``branch`` forks into len(child_len) threads
        (parason_plan_fork).  ``child_pages``: one list of fresh physical
        pages per child, ceil(len / 16) each.  Returns the branch index of
        every child: child 0 keeps ``branch``, the others are appended."""
        lens = np.ascontiguousarray(np.asarray(child_len, dtype=np.int32))
        ptr = np.zeros(len(lens) + 1, dtype=np.int32)
        ptr[1:] = np.cumsum([len(pg) for pg in child_pages]) if len(child_pages) else []
        flat = np.ascontiguousarray(np.asarray([x for pg in child_pages for x in pg] or [0],
                                               dtype=np.int32))
        sh = None if self.host_only else _stream_handle(stream)
        L = self.num_leaves
        check(_lib.load().parason_plan_fork(self.handle, int(branch), len(lens), _ptr(lens),
                                            _ptr(ptr), _ptr(flat), sh), "parason_plan_fork")
        self.num_leaves = int(self.info()["num_leaves"])
        return [int(branch)] + list(range(L, L + len(lens) - 1))

    def decode_tree(self, tree, **kw):
        """``decode`` with the tensors of a ``workloads.ForkTree``."""
        return self.decode(tree.q, tree.k_pages, tree.v_pages, k_scale=tree.k_scale,
                           v_scale=tree.v_scale, **kw)

    def check(self, stream=None) -> None:
        """Synchronise ``stream`` and raise if a kernel reported a failure."""
        check(_lib.load().parason_plan_check(self.handle, _stream_handle(stream)), "plan_check")

    def set_debug(self, flags: int = 0, wait_limit_ns: int = 0) -> None:
        check(_lib.load().parason_plan_set_debug(self.handle, flags, wait_limit_ns), "set_debug")

    def enable_timing(self, max_calls: int) -> None:
        check(_lib.load().parason_plan_enable_timing(self.handle, max_calls), "enable_timing")

    def read_timing(self, capacity: int = 4096):
        """(attention-kernel ms, merge-kernel ms) per recorded decode call."""
        a = np.zeros(capacity, dtype=np.float32)
        m = np.zeros(capacity, dtype=np.float32)
        n = ctypes.c_int32()
        check(_lib.load().parason_plan_read_timing(self.handle, _ptr(a), _ptr(m), capacity,
                                                   ctypes.byref(n)), "read_timing")
        return a[:n.value].copy(), m[:n.value].copy()


def lse_merge(o_a: torch.Tensor, lse_a: torch.Tensor, o_b: torch.Tensor, lse_b: torch.Tensor,
              o_out: Optional[torch.Tensor] = None, lse_out: Optional[torch.Tensor] = None,
              stream=None):
    """Merge two attention results over disjoint key sets (``parason_lse_merge``)."""
    if o_a.shape != o_b.shape or o_a.dtype != o_b.dtype:
        raise ValueError("o_a and o_b must match in shape and dtype")
    if o_a.dtype not in (torch.bfloat16, torch.float32):
        raise ValueError("o must be bf16 or fp32")
    d = o_a.shape[-1]
    rows = o_a.numel() // d
    for t in (o_a, o_b, lse_a, lse_b):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("inputs must be contiguous cuda tensors")
    if lse_a.dtype != torch.float32 or lse_a.numel() != rows or lse_b.numel() != rows:
        raise ValueError("lse must be float32 with one value per row")
    o_out = torch.empty_like(o_a) if o_out is None else o_out
    lse_out = torch.empty_like(lse_a) if lse_out is None else lse_out
    mode = _lib.MODES["fp32" if o_a.dtype == torch.float32 else "bf16"]
    st = _lib.load().parason_lse_merge(_ptr(o_a), _ptr(lse_a), _ptr(o_b), _ptr(lse_b),
                                       _ptr(o_out), _ptr(lse_out), rows, d, mode,
                                       _stream_handle(stream))
    check(st, "parason_lse_merge")
    return o_out, lse_out


def version() -> str:
    return _lib.load().parason_version().decode()


__all__ = ["Plan", "lse_merge", "version", "ParasonError"]


# ---------------------------------------------------------------------------
# reasoning traces (tag streams of the parallel-reasoning grammar)
# ---------------------------------------------------------------------------

class TraceError(ParasonError):
    """A trace outside the grammar; ``pos`` is the first symbol no derivation accepts."""

    def __init__(self, pos: int):
        super().__init__(_lib.EINVAL, f"trace outside the grammar at symbol {pos}")
        self.pos = pos


def _symbols(symbols) -> np.ndarray:
    a = np.ascontiguousarray(np.asarray(symbols, dtype=np.int32))
    if a.ndim != 1:
        raise ValueError("a trace is a 1-D array of int32 symbols")
    return a


def trace_stats(symbols) -> dict:
    """Token metrics of one trace (see parason_trace_analyze)."""
    a = _symbols(symbols)
    st = _lib.TraceStats()
    err = ctypes.c_int64(-1)
    rc = _lib.load().parason_trace_analyze(_ptr(a), a.size, ctypes.byref(st), ctypes.byref(err))
    if rc == _lib.EINVAL and err.value >= 0:
        raise TraceError(err.value)
    check(rc, "parason_trace_analyze")
    return {name: getattr(st, name) for name, _ in _lib.TraceStats._fields_}


def trace_fork_tree(symbols, block: int = 0):
    """(parent, node_len, leaf_node) of top-level block `block` (int32 arrays)."""
    a = _symbols(symbols)
    nn, nl = ctypes.c_int32(0), ctypes.c_int32(0)
    lib = _lib.load()
    cap = 64
    while True:
        parent = np.zeros(cap, np.int32)
        node_len = np.zeros(cap, np.int32)
        leaf = np.zeros(cap, np.int32)
        rc = lib.parason_trace_fork_tree(_ptr(a), a.size, block, cap, _ptr(parent), _ptr(node_len),
                                         _ptr(leaf), ctypes.byref(nn), ctypes.byref(nl))
        if rc == _lib.EINVAL and nn.value > cap:
            cap = nn.value
            continue
        check(rc, "parason_trace_fork_tree")
        return parent[:nn.value].copy(), node_len[:nn.value].copy(), leaf[:nl.value].copy()
