"""C ABI: the library loads, exports every declared symbol, and validates on
the host (CPU only; no compute call needs a GPU here)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_24658_gb300 import _lib, build
from paper_2608_24658_gb300.api import Plan, ParasonError
from paper_2608_24658_gb300 import workloads as W

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "parason.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return _lib.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"\b(parason_[a-z0-9_]+)\s*\(", text)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert "parason_attn_plan" in names and "parason_attn_decode" in names
    assert "parason_lse_merge" in names
    for n in names:
        assert hasattr(lib, n), f"{n} declared in parason.h but not exported"
    assert set(names) == set(_lib.SIGNATURES), "binding and header disagree"


def test_status_strings_and_version(lib):
    assert lib.parason_status_string(0) == b"ok"
    assert lib.parason_status_string(4) == b"device wait timed out"
    assert re.fullmatch(rb"\d+\.\d+\.\d+", lib.parason_version())


def _host_plan(tree, **kw):
    return Plan.for_tree(tree, host_only=True, **kw)


def _fields(tree):
    return dict(num_q_heads=tree.num_q_heads, num_kv_heads=tree.num_kv_heads,
                head_dim=tree.head_dim, mode=tree.mode, parent=tree.parent.copy(),
                node_len=tree.node_len.copy(), node_page_ptr=tree.node_page_ptr.copy(),
                page_ids=tree.page_ids.copy(), leaf_node=tree.leaf_node.copy(),
                num_physical_pages=tree.num_physical_pages)


def _expect_einval(**f):
    with pytest.raises(ParasonError) as e:
        Plan(host_only=True, **f)
    assert e.value.status == _lib.EINVAL, str(e.value)


def test_validation_rejects_malformed_trees(lib):
    tree = W.figure3_tree(values=False)
    good = _fields(tree)
    Plan(host_only=True, **good).close()
    bad = dict(good, parent=good["parent"].copy())
    bad["parent"][3] = 5                       # parent not smaller than child
    _expect_einval(**bad)
    bad = dict(good, parent=good["parent"].copy())
    bad["parent"][2] = -2
    _expect_einval(**bad)
    bad = dict(good, node_len=good["node_len"].copy())
    bad["node_len"][1] += 16                   # page count no longer ceil(len/16)
    _expect_einval(**bad)
    bad = dict(good, node_len=good["node_len"].copy())
    bad["node_len"][0] = -1
    _expect_einval(**bad)
    bad = dict(good, page_ids=good["page_ids"].copy())
    bad["page_ids"][0] = tree.num_physical_pages   # out of range
    _expect_einval(**bad)
    bad = dict(good, page_ids=good["page_ids"].copy())
    bad["page_ids"][1] = bad["page_ids"][0]        # page owned twice
    _expect_einval(**bad)
    bad = dict(good, leaf_node=good["leaf_node"].copy())
    bad["leaf_node"][0] = 1                        # a node with children
    _expect_einval(**bad)
    bad = dict(good, leaf_node=good["leaf_node"].copy())
    bad["leaf_node"][1] = bad["leaf_node"][0]      # repeated branch node
    _expect_einval(**bad)
    bad = dict(good, leaf_node=good["leaf_node"].copy())
    bad["leaf_node"][0] = tree.num_nodes
    _expect_einval(**bad)
    _expect_einval(**dict(good, num_kv_heads=3))   # H_q % H_kv != 0
    _expect_einval(**dict(good, head_dim=96))
    _expect_einval(**dict(good, page_size=32))
    with pytest.raises(ParasonError):
        Plan(host_only=True, sm_scale=-1.0, **good)


def test_null_pointers_rejected(lib):
    cfg = _lib.AttnConfig(8, 2, 64, 16, 0, 0.0)
    out = ctypes.c_void_p()
    st = lib.parason_attn_plan_host(ctypes.byref(cfg), 3, None, None, None, None, 1, None, 10,
                                    152, ctypes.byref(out))
    assert st == _lib.EINVAL
    assert lib.parason_attn_plan_host(None, 0, None, None, None, None, 0, None, 0, 152,
                                      ctypes.byref(out)) == _lib.EINVAL


def test_decode_on_host_plan_is_einval(lib):
    tree = W.figure3_tree(values=False)
    with _host_plan(tree) as p:
        st = lib.parason_attn_decode(p.handle, None, None, None, None, None, None, None, None, 0,
                                     None)
        assert st == _lib.EINVAL
        assert lib.parason_plan_check(p.handle, None) == _lib.EINVAL


def test_device_plan_without_gpu_reports_einval_first(lib):
    """Malformed input is EINVAL even where no CUDA device exists."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("checks the no-GPU path")
    tree = W.figure3_tree(values=False)
    f = _fields(tree)
    f["parent"][3] = 7
    cfg = _lib.AttnConfig(8, 2, 64, 16, 0, 0.0)
    out = ctypes.c_void_p()
    a = lambda x: np.ascontiguousarray(x, dtype=np.int32).ctypes.data_as(ctypes.c_void_p)
    st = lib.parason_attn_plan(ctypes.byref(cfg), len(f["parent"]), a(f["parent"]),
                               a(f["node_len"]), a(f["node_page_ptr"]), a(f["page_ids"]),
                               len(f["leaf_node"]), a(f["leaf_node"]), f["num_physical_pages"],
                               None, ctypes.byref(out))
    assert st == _lib.EINVAL
    f = _fields(tree)
    st = lib.parason_attn_plan(ctypes.byref(cfg), len(f["parent"]), a(f["parent"]),
                               a(f["node_len"]), a(f["node_page_ptr"]), a(f["page_ids"]),
                               len(f["leaf_node"]), a(f["leaf_node"]), f["num_physical_pages"],
                               None, ctypes.byref(out))
    assert st == _lib.ECUDA


def test_lse_merge_argument_checks(lib):
    assert lib.parason_lse_merge(None, None, None, None, None, None, 0, 128, 0, None) == _lib.OK
    assert lib.parason_lse_merge(None, None, None, None, None, None, 4, 128, 0, None) == _lib.EINVAL
    assert lib.parason_lse_merge(None, None, None, None, None, None, 4, 96, 0, None) == _lib.EINVAL
    assert lib.parason_lse_merge(None, None, None, None, None, None, 4, 128, 7, None) == _lib.EINVAL


def test_fp8_head_dim_64_unsupported(lib):
    tree = W.figure3_tree(values=False)          # head_dim 64
    f = _fields(tree)
    f["mode"] = "fp8"
    with pytest.raises(ParasonError) as e:
        Plan(host_only=True, **f)
    assert e.value.status == _lib.EUNSUPPORTED
