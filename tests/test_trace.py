"""The library's trace parser (parason_trace_analyze / parason_trace_fork_tree)
against the trace oracle: same metrics, same fork trees, same error
positions, on random traces of the grammar and on corrupted ones (CPU)."""
import numpy as np
import pytest

from oracle import trace_oracle as T
from paper_2608_24658_gb300 import api, build
from paper_2608_24658_gb300 import workloads as W

INT_KEYS = ("total_tokens", "latency_tokens", "subtask_tokens", "trial_tokens", "parallel_blocks",
            "threads", "max_depth")


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def assert_same(s):
    ref = T.stats(s)
    got = api.trace_stats(s)
    for k in INT_KEYS:
        assert got[k] == ref[k], (k, got[k], ref[k])
    assert got["acceleration"] == pytest.approx(ref["acceleration"], rel=1e-15)
    assert got["eta"] == pytest.approx(ref["eta"], rel=1e-12, abs=1e-15)
    items = T.parse(list(s))
    assert got["top_level_blocks"] == len(T.top_level_regions(items))
    for b in range(got["top_level_blocks"]):
        rp, rl, rf = T.fork_tree(list(s), b)
        gp, gl, gf = api.trace_fork_tree(s, b)
        assert gp.tolist() == rp and gl.tolist() == rl and gf.tolist() == rf


@pytest.mark.parametrize("seed", range(200))
def test_random_traces_match_oracle(seed):
    assert_same(W.random_trace(seed))


@pytest.mark.parametrize("seed", range(200, 400))
def test_deep_random_traces_match_oracle(seed):
    assert_same(W.random_trace(seed, max_depth=4, p_parallel=0.6, text_len=(1, 4)))


def test_paper_scale_traces_match_oracle():
    for seed in range(4):
        assert_same(W.paper_scale_trace(seed))


def _corrupt(s, rng):
    s = list(s)
    op = rng.integers(3)
    i = int(rng.integers(len(s)))
    tag = int(rng.integers(-13, 1)) if rng.random() < 0.8 else int(rng.integers(0, 100))
    if op == 0:
        del s[i]
    elif op == 1:
        s[i] = tag
    else:
        s.insert(i, tag)
    return s


def test_corrupted_traces_same_error_position():
    rng = np.random.default_rng(0)
    checked = 0
    for seed in range(600):
        s = _corrupt(W.random_trace(seed, max_depth=3), rng)
        try:
            T.stats(s)
            ref_pos = None
        except T.TraceError as e:
            ref_pos = e.pos
        if ref_pos is None:
            assert_same(s)
            continue
        with pytest.raises(api.TraceError) as e:
            api.trace_stats(s)
        assert e.value.pos == ref_pos, (seed, e.value.pos, ref_pos)
        checked += 1
    assert checked > 300


def test_edge_cases():
    assert api.trace_stats([T.THINK, T.THINK_END])["latency_tokens"] == 2
    for s, pos in (([], 0), ([T.THINK], 1), ([T.THINK_END], 0), ([5], 0)):
        with pytest.raises(api.TraceError) as e:
            api.trace_stats(s)
        assert e.value.pos == pos
    with pytest.raises(api.ParasonError):
        api.trace_fork_tree([T.THINK, 3, T.THINK_END], 0)    # no block


def test_fork_tree_grows_its_buffers():
    # a block with 200 threads needs more than the binding's first guess
    s = [T.THINK, T.PARALLEL, T.OUTLINES, T.TRIAL, 1, T.TRIAL_END, T.OUTLINES_END]
    for k in range(200):
        s += [T.THREAD, k, T.THREAD_END]
    s += [T.PARALLEL_END, T.THINK_END]
    p, l, f = api.trace_fork_tree(s, 0)
    assert len(p) == 201 and len(f) == 200 and (l[1:] == 3).all() and l[0] == 7
