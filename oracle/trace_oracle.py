"""Reasoning-trace grammar and token-latency metrics -- TEST INFRASTRUCTURE.

A plain recursive-descent parser of the context-free grammar of parallel
reasoning (Fig. 4): one function per production, in the grammar's order,
written for a reader to check against the figure.  It is slow and obviously
correct; the library's parser (``csrc/trace.cpp``) is tested against it and
shares no code with it.  Only the tests and the benchmark's CPU-baseline
leg use this module.

Symbols: a text token is any id >= 0; the twelve tags are the negative codes
below (each tag is one generated token).

Metrics (Sec. 4, "Evaluation"; Tab. 4 and Tab. 5 captions; Sec. 3.5):
  * total tokens: every symbol of the trace;
  * latency tokens (token length of the longest generation path): sequential
    tokens count one each, a <Parallel> block counts its tags and its
    outlines block plus the largest latency among its threads;
  * acceleration ratio: total / latency;
  * eta = 1 - latency / total;
  * Subtask / Trial tokens: tokens inside a thread whose outline entry (same
    position in the block) is a Subtask / Trial, each token counted for its
    innermost enclosing thread; threads beyond the entry count are untyped;
  * trigger ratio (over a batch): share of traces with >= 1 <Parallel> block.

Fork tree of a top-level parallel region (the decode state in which every
innermost thread of the region is running, each at its full length):
  node 0 holds every token before the region's first <Thread> (earlier
  regions are joined, so all of it is context); a thread is a node holding
  its tokens up to the end of its first nested outlines block, whose threads
  become its children, or all its tokens if it has no nested region; the
  branches (leaves) are the threads with no nested region, in tree order.
"""
from dataclasses import dataclass, field
from typing import List, Optional

THINK, THINK_END = -1, -2
PARALLEL, PARALLEL_END = -3, -4
OUTLINES, OUTLINES_END = -5, -6
SUBTASK, SUBTASK_END = -7, -8
TRIAL, TRIAL_END = -9, -10
THREAD, THREAD_END = -11, -12
TAGS = {THINK, THINK_END, PARALLEL, PARALLEL_END, OUTLINES, OUTLINES_END, SUBTASK, SUBTASK_END,
        TRIAL, TRIAL_END, THREAD, THREAD_END}

UNTYPED, SUBTASK_T, TRIAL_T = 0, 1, 2


class TraceError(ValueError):
    def __init__(self, pos: int, msg: str):
        super().__init__(f"position {pos}: {msg}")
        self.pos = pos


@dataclass
class Thread:
    start: int = 0            # index of <Thread>
    end: int = 0              # one past </Thread>
    kind: int = UNTYPED
    body: list = field(default_factory=list)   # items of B: ("text", a, b) | ("par", Region)


@dataclass
class Region:
    start: int = 0            # index of <Parallel>
    outlines_end: int = 0     # one past </Outlines>
    end: int = 0              # one past </Parallel>
    entries: List[int] = field(default_factory=list)
    threads: List[Thread] = field(default_factory=list)


class _Parser:
    def __init__(self, symbols):
        self.s = [int(x) for x in symbols]
        self.i = 0

    def peek(self) -> Optional[int]:
        return self.s[self.i] if self.i < len(self.s) else None

    def expect(self, tag: int, what: str):
        if self.peek() != tag:
            raise TraceError(self.i, f"expected {what}")
        self.i += 1

    def is_text(self) -> bool:
        x = self.peek()
        return x is not None and x >= 0

    # S -> <think> B </think>
    def S(self):
        self.expect(THINK, "<think>")
        body = self.B()
        self.expect(THINK_END, "</think>")
        if self.i != len(self.s):
            raise TraceError(self.i, "symbols after </think>")
        return body

    # B -> T B | P B | eps
    def B(self):
        items = []
        while True:
            x = self.peek()
            if x is not None and x < 0 and x not in TAGS:
                raise TraceError(self.i, "unknown tag code")
            if self.is_text():
                a = self.i
                self.T()
                items.append(("text", a, self.i))
            elif x == PARALLEL:
                items.append(("par", self.P()))
            else:
                return items

    # P -> <Parallel> O H </Parallel>
    def P(self):
        r = Region(start=self.i)
        self.expect(PARALLEL, "<Parallel>")
        r.entries = self.O()
        r.outlines_end = self.i
        r.threads = self.H()
        self.expect(PARALLEL_END, "</Parallel>")
        r.end = self.i
        for k, t in enumerate(r.threads):
            t.kind = r.entries[k] if k < len(r.entries) else UNTYPED
        return r

    # O -> <Outlines> G </Outlines>
    def O(self):
        self.expect(OUTLINES, "<Outlines>")
        entries = self.G()
        self.expect(OUTLINES_END, "</Outlines>")
        return entries

    # G -> E G | E
    def G(self):
        entries = [self.E()]
        while self.peek() in (SUBTASK, TRIAL):
            entries.append(self.E())
        return entries

    # E -> <Subtask> T </Subtask> | <Trial> T </Trial>
    def E(self):
        if self.peek() == SUBTASK:
            self.i += 1
            self.T()
            self.expect(SUBTASK_END, "</Subtask>")
            return SUBTASK_T
        if self.peek() == TRIAL:
            self.i += 1
            self.T()
            self.expect(TRIAL_END, "</Trial>")
            return TRIAL_T
        raise TraceError(self.i, "expected <Subtask> or <Trial>")

    # H -> W H | W
    def H(self):
        threads = [self.W()]
        while self.peek() == THREAD:
            threads.append(self.W())
        return threads

    # W -> <Thread> B </Thread>
    def W(self):
        t = Thread(start=self.i)
        self.expect(THREAD, "<Thread>")
        t.body = self.B()
        self.expect(THREAD_END, "</Thread>")
        t.end = self.i
        return t

    # T -> nonempty free-form text (text tokens only)
    def T(self):
        if not self.is_text():
            raise TraceError(self.i, "expected text")
        while self.is_text():
            self.i += 1


def parse(symbols):
    """Parse a trace; return the list of items of its top-level body."""
    return _Parser(symbols).S()


def _body_latency(items) -> int:
    lat = 0
    for it in items:
        if it[0] == "text":
            lat += it[2] - it[1]
        else:
            lat += _region_latency(it[1])
    return lat


def _region_latency(r: Region) -> int:
    # tags of the block + the whole outlines block, then the slowest thread
    outlines = r.outlines_end - r.start - 1
    return 1 + outlines + max(1 + _body_latency(t.body) + 1 for t in r.threads) + 1


def _typed_tokens(items, kind, acc):
    """Add to acc[kind] the tokens of these body items, nested threads by their own kind."""
    for it in items:
        if it[0] == "text":
            acc[kind] += it[2] - it[1]
        else:
            r = it[1]
            acc[kind] += (r.outlines_end - r.start) + 1        # <Parallel>, outlines, </Parallel>
            for t in r.threads:
                acc[t.kind] += 2                                # <Thread>, </Thread>
                _typed_tokens(t.body, t.kind, acc)


def stats(symbols) -> dict:
    """Token metrics of one trace (raises TraceError if it is not in the grammar)."""
    items = parse(symbols)
    total = len(symbols)
    latency = 1 + _body_latency(items) + 1
    acc = {UNTYPED: 0, SUBTASK_T: 0, TRIAL_T: 0}
    acc[UNTYPED] += 2
    _typed_tokens(items, UNTYPED, acc)
    assert sum(acc.values()) == total
    regions, threads, depth = _count(items, 0)
    return {"total_tokens": total, "latency_tokens": latency,
            "subtask_tokens": acc[SUBTASK_T], "trial_tokens": acc[TRIAL_T],
            "parallel_blocks": regions, "threads": threads, "max_depth": depth,
            "acceleration": total / latency, "eta": 1.0 - latency / total}


def _count(items, depth):
    regions = threads = 0
    best = depth
    for it in items:
        if it[0] == "par":
            regions += 1
            for t in it[1].threads:
                threads += 1
                r2, t2, d2 = _count(t.body, depth + 1)
                regions += r2
                threads += t2
                best = max(best, d2)
            best = max(best, depth + 1)
    return regions, threads, best


def trigger_ratio(traces) -> float:
    """Share of traces with at least one <Parallel> block (Tab. 4 caption)."""
    return sum(1 for s in traces if stats(s)["parallel_blocks"] > 0) / len(traces)


def top_level_regions(items):
    return [it[1] for it in items if it[0] == "par"]


def fork_tree(symbols, region: int):
    """(parent, node_len, leaf_node) of top-level region `region` (see the header)."""
    items = parse(symbols)
    regions = top_level_regions(items)
    if not 0 <= region < len(regions):
        raise IndexError("no such top-level region")
    r = regions[region]
    parent, node_len, leaves = [-1], [r.threads[0].start], []

    def add_threads(reg, par):
        for t in reg.threads:
            nested = next((it[1] for it in t.body if it[0] == "par"), None)
            me = len(parent)
            parent.append(par)
            if nested is None:
                node_len.append(t.end - t.start)
                leaves.append(me)
            else:
                node_len.append(nested.outlines_end - t.start)
                add_threads(nested, me)

    add_threads(r, 0)
    return parent, node_len, leaves
