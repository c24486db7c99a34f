"""Pins of the trace oracle (grammar of Fig. 4, latency of Sec. 4, ratios of
Tab. 4 / Sec. 3.5) against hand-derived values, an independent schedule
computation of the latency, and grammar errors at known positions."""
import numpy as np
import pytest

from oracle import trace_oracle as T
from paper_2608_24658_gb300 import workloads as W

TH, THE = T.THINK, T.THINK_END
PA, PAE = T.PARALLEL, T.PARALLEL_END
OU, OUE = T.OUTLINES, T.OUTLINES_END
SU, SUE = T.SUBTASK, T.SUBTASK_END
TR, TRE = T.TRIAL, T.TRIAL_END
TD, TDE = T.THREAD, T.THREAD_END


def txt(n, v=7):
    return [v] * n


def example_one_region():
    # <think> a3 <Parallel><Outlines><Subtask>x2</Subtask><Trial>y1</Trial></Outlines>
    #   <Thread>b4</Thread><Thread>c7</Thread></Parallel> d2 </think>
    return ([TH] + txt(3) + [PA, OU, SU] + txt(2) + [SUE, TR] + txt(1) + [TRE, OUE] +
            [TD] + txt(4) + [TDE, TD] + txt(7) + [TDE, PAE] + txt(2) + [THE])


def example_nested():
    # Fig. 3's shape: two Subtask threads, the first holding a Trial block
    return ([TH] + txt(5) + [PA, OU, SU] + txt(1) + [SUE, SU] + txt(1) + [SUE, OUE] +
            [TD] + txt(2) + [PA, OU, TR] + txt(1) + [TRE, TR] + txt(1) + [TRE, OUE] +
            [TD] + txt(3) + [TDE, TD] + txt(5) + [TDE, PAE] + txt(1) + [TDE] +
            [TD] + txt(4) + [TDE, PAE, THE])


def schedule_latency(s):
    """Latency as the finish time of the last token when every token takes one
    step, tokens of a strand run in order, a thread starts after its block's
    outlines and </Parallel> waits for every thread of its block."""
    stack = [{"kind": "strand", "t": 0}]
    t = 0
    for x in s:
        top = stack[-1]
        if x == TD:
            region = top
            t = region["outl"] + 1
            stack.append({"kind": "strand", "t": t})
        elif x == TDE:
            t = top["t"] + 1
            stack.pop()
            stack[-1]["ends"].append(t)
        elif x == PA:
            t = top["t"] + 1
            top["t"] = t
            stack.append({"kind": "region", "t": t, "outl": None, "ends": []})
        elif x == OUE:
            t = top["t"] + 1
            top["t"] = t
            top["outl"] = t
        elif x == PAE:
            t = max(top["ends"]) + 1
            stack.pop()
            stack[-1]["t"] = t
        else:
            t = top["t"] + 1
            top["t"] = t
    return t


def test_no_parallel_block():
    st = T.stats([TH, 5, 6, 7, THE])
    assert st["total_tokens"] == 5 and st["latency_tokens"] == 5
    assert st["acceleration"] == 1.0 and st["eta"] == 0.0
    assert st["parallel_blocks"] == 0 and st["subtask_tokens"] == 0 and st["trial_tokens"] == 0


def test_one_region_by_hand():
    s = example_one_region()
    st = T.stats(s)
    # total: 1 + 3 + 1 + (1 + 4 + 3 + 1) + 6 + 9 + 1 + 2 + 1
    assert st["total_tokens"] == len(s) == 33
    # latency: 1 + 3 + (1 + 9 + max(6, 9) + 1) + 2 + 1
    assert st["latency_tokens"] == 27
    assert st["subtask_tokens"] == 6 and st["trial_tokens"] == 9
    assert st["acceleration"] == pytest.approx(33 / 27)
    assert st["eta"] == pytest.approx(6 / 33)
    assert (st["parallel_blocks"], st["threads"], st["max_depth"]) == (1, 2, 1)
    parent, node_len, leaves = T.fork_tree(s, 0)
    assert parent == [-1, 0, 0] and node_len == [14, 6, 9] and leaves == [1, 2]


def test_nested_region_by_hand():
    s = example_nested()
    st = T.stats(s)
    assert st["total_tokens"] == len(s) == 50
    # inner block 1 + 8 + max(5, 7) + 1 = 17; thread A 1 + 2 + 17 + 1 + 1 = 22;
    # outer block 1 + 8 + max(22, 6) + 1 = 32; trace 1 + 5 + 32 + 1 = 39
    assert st["latency_tokens"] == 39
    # Subtask: thread A's own 15 tokens + thread B's 6; Trial: the inner threads 5 + 7
    assert st["subtask_tokens"] == 21 and st["trial_tokens"] == 12
    assert (st["parallel_blocks"], st["threads"], st["max_depth"]) == (2, 4, 2)
    parent, node_len, leaves = T.fork_tree(s, 0)
    assert parent == [-1, 0, 1, 1, 0]
    assert node_len == [15, 12, 5, 7, 6]
    assert leaves == [2, 3, 4]


def test_latency_equals_independent_schedule():
    for s in (example_one_region(), example_nested()):
        assert T.stats(s)["latency_tokens"] == schedule_latency(s)
    for seed in range(300):
        s = W.random_trace(seed).tolist()
        st = T.stats(s)
        assert st["latency_tokens"] == schedule_latency(s), seed


def test_properties_on_random_traces():
    for seed in range(300):
        s = W.random_trace(seed, max_depth=3)
        st = T.stats(s)
        assert st["latency_tokens"] <= st["total_tokens"]
        if st["parallel_blocks"] == 0:                    # (a one-thread block saves nothing)
            assert st["latency_tokens"] == st["total_tokens"]
        if st["latency_tokens"] < st["total_tokens"]:
            assert st["threads"] > st["parallel_blocks"]
        assert st["subtask_tokens"] + st["trial_tokens"] <= st["total_tokens"]
        for r in range(st["parallel_blocks"]):
            try:
                parent, node_len, leaves = T.fork_tree(s, r)
            except IndexError:
                break                  # fewer top-level regions than blocks (nesting)
            assert parent[0] == -1 and all(0 <= parent[i] < i for i in range(1, len(parent)))
            assert all(parent[i] != leaf for leaf in leaves for i in range(len(parent)))
            assert all(n > 0 for n in node_len)


def test_trigger_ratio():
    plain = [TH, 1, THE]
    assert T.trigger_ratio([plain, example_one_region(), example_nested(), plain]) == 0.5


@pytest.mark.parametrize("s,pos", [
    ([TH, 1, PA, OU, OUE, TD, TDE, PAE, THE], 4),          # outlines without entries
    ([TH, PA, OU, SU, SUE, OUE, TD, TDE, PAE, THE], 4),     # entry without text
    ([TH, 1, 2], 3),                                        # missing </think>
    ([TH, 1, THE, 5], 3),                                   # symbols after </think>
    ([TH, PA, TD, 1, TDE, PAE, THE], 2),                    # thread before outlines
    ([TH, 1, -99, THE], 2),                                 # unknown tag code
    ([TH, PA, OU, TR, 1, TRE, OUE, PAE, THE], 7),           # block without threads
    ([TH, 1, TDE, THE], 2),                                 # stray closing tag
    ([1, TH, THE], 0),                                      # text before <think>
])
def test_grammar_errors(s, pos):
    with pytest.raises(T.TraceError) as e:
        T.stats(s)
    assert e.value.pos == pos
