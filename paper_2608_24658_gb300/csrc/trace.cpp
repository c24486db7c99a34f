// trace.cpp -- the tag stream of a parallel-reasoning trace: grammar check,
// token-latency metrics and the decode-time fork tree of a parallel block.
//
// Grammar (Fig. 4):  S -> <think> B </think>;  B -> T B | P B | eps;
//   P -> <Parallel> O H </Parallel>;  O -> <Outlines> G </Outlines>;
//   G -> E G | E;  E -> <Subtask> T </Subtask> | <Trial> T </Trial>;
//   H -> W H | W;  W -> <Thread> B </Thread>;  T -> one or more text tokens.
// The grammar is LL(1), so the first symbol no derivation can accept is
// well defined; it is what an error reports.
//
// One left-to-right pass of a pushdown automaton (an explicit stack, no
// recursion, so nesting depth is bounded only by memory) checks the stream
// and accumulates:
//   * latency (Sec. 4, "Evaluation"): sequential tokens count one each; a
//     <Parallel> block counts its two tags and its outlines block plus the
//     largest latency of its threads;
//   * Subtask / Trial tokens (Sec. 3.5): thread k of a block has the type of
//     outline entry k (untyped past the last entry); every token counts for
//     the type of its innermost enclosing thread;
//   * acceleration = total / latency (Tab. 4), eta = 1 - latency / total.
#include <cstdint>
#include <utility>
#include <vector>

#include "parason.h"

namespace {

enum : int32_t {
    kUntyped = 0,
    kSubtask = 1,
    kTrial = 2,
};

// frames of the automaton
enum FrameKind : int32_t {
    kRootBody,     // B inside <think> ... </think>
    kThreadBody,   // B inside <Thread> ... </Thread>
    kBlock,        // P after <Parallel>
    kEntry,        // E after <Subtask> / <Trial>
};

// phases of a kBlock frame
enum BlockPhase : int32_t {
    kWantOutlines,    // after <Parallel>
    kWantFirstEntry,  // after <Outlines>
    kEntryOrEnd,      // after an entry: another entry or </Outlines>
    kWantFirstThread, // after </Outlines>
    kThreadOrEnd,     // after a thread: another thread or </Parallel>
};

struct Frame {
    FrameKind kind;
    int32_t phase = 0;            // kBlock: BlockPhase; kEntry: text tokens seen
    int64_t latency = 0;          // body: latency so far; block: max thread latency
    int32_t type = kUntyped;      // thread body / entry: its type
    int32_t block = -1;           // thread body: index of its block; block: its record
    int32_t thread = -1;          // thread body: its record
};

struct BlockRec {
    int64_t start, outlines_end = -1, end = -1;
    int32_t parent_thread;        // -1: top level
    std::vector<int32_t> threads;
    std::vector<int32_t> entries;
};

struct ThreadRec {
    int64_t start, end = -1;
    int32_t block;
    int32_t first_nested = -1;    // first block directly in its body
};

struct Parsed {
    parason_trace_stats st{};
    std::vector<BlockRec> blocks;
    std::vector<ThreadRec> threads;
    std::vector<int32_t> top_blocks;
};

bool is_text(int32_t x) { return x >= 0; }

// Parse; on a grammar error return false with *err = the offending position.
bool parse(const int32_t *s, int64_t n, Parsed *out, int64_t *err) {
    std::vector<Frame> stack;
    int64_t tokens[3] = {0, 0, 0};
    int32_t depth = 0, max_depth = 0;
    auto fail = [&](int64_t pos) {
        *err = pos;
        return false;
    };
    auto cur_type = [&]() {
        for (size_t k = stack.size(); k-- > 0;)
            if (stack[k].kind == kThreadBody) return stack[k].type;
        return static_cast<int32_t>(kUntyped);
    };
    if (n < 1 || s[0] != PARASON_TAG_THINK) return fail(0);
    stack.push_back(Frame{kRootBody});
    tokens[kUntyped] += 1;
    int64_t i = 1;
    for (; i < n && !stack.empty(); ++i) {
        const int32_t x = s[i];
        Frame &f = stack.back();
        switch (f.kind) {
        case kRootBody:
        case kThreadBody:
            if (is_text(x)) {
                f.latency += 1;
                tokens[cur_type()] += 1;
            } else if (x == PARASON_TAG_PARALLEL) {
                tokens[cur_type()] += 1;
                BlockRec b;
                b.start = i;
                b.parent_thread = f.kind == kThreadBody ? f.thread : -1;
                const int32_t bi = static_cast<int32_t>(out->blocks.size());
                if (f.kind == kThreadBody && out->threads[f.thread].first_nested < 0)
                    out->threads[f.thread].first_nested = bi;
                if (f.kind == kRootBody) out->top_blocks.push_back(bi);
                out->blocks.push_back(std::move(b));
                Frame nf{kBlock};
                nf.phase = kWantOutlines;
                nf.block = bi;
                stack.push_back(nf);
                ++depth;
                if (depth > max_depth) max_depth = depth;
            } else if (f.kind == kRootBody && x == PARASON_TAG_THINK_END) {
                tokens[kUntyped] += 1;
                out->st.latency_tokens = 1 + f.latency + 1;
                stack.pop_back();
            } else if (f.kind == kThreadBody && x == PARASON_TAG_THREAD_END) {
                tokens[f.type] += 1;
                const int64_t lat = 1 + f.latency + 1;
                out->threads[f.thread].end = i + 1;
                stack.pop_back();
                Frame &blk = stack.back();
                if (lat > blk.latency) blk.latency = lat;
                blk.phase = kThreadOrEnd;
            } else {
                return fail(i);
            }
            break;
        case kBlock: {
            BlockRec &b = out->blocks[f.block];
            switch (f.phase) {
            case kWantOutlines:
                if (x != PARASON_TAG_OUTLINES) return fail(i);
                tokens[cur_type()] += 1;
                f.phase = kWantFirstEntry;
                break;
            case kWantFirstEntry:
            case kEntryOrEnd:
                if (x == PARASON_TAG_SUBTASK || x == PARASON_TAG_TRIAL) {
                    tokens[cur_type()] += 1;
                    Frame nf{kEntry};
                    nf.type = x == PARASON_TAG_SUBTASK ? kSubtask : kTrial;
                    nf.block = f.block;
                    stack.push_back(nf);
                } else if (f.phase == kEntryOrEnd && x == PARASON_TAG_OUTLINES_END) {
                    tokens[cur_type()] += 1;
                    b.outlines_end = i + 1;
                    f.phase = kWantFirstThread;
                } else {
                    return fail(i);
                }
                break;
            case kWantFirstThread:
            case kThreadOrEnd:
                if (x == PARASON_TAG_THREAD) {
                    const int32_t k = static_cast<int32_t>(b.threads.size());
                    const int32_t type = k < static_cast<int32_t>(b.entries.size()) ? b.entries[k]
                                                                                     : kUntyped;
                    tokens[type] += 1;
                    ThreadRec t;
                    t.start = i;
                    t.block = f.block;
                    const int32_t ti = static_cast<int32_t>(out->threads.size());
                    out->threads.push_back(t);
                    b.threads.push_back(ti);
                    Frame nf{kThreadBody};
                    nf.type = type;
                    nf.block = f.block;
                    nf.thread = ti;
                    stack.push_back(nf);
                } else if (f.phase == kThreadOrEnd && x == PARASON_TAG_PARALLEL_END) {
                    b.end = i + 1;
                    // <Parallel>, the outlines block, the slowest thread, </Parallel>
                    const int64_t lat = (b.outlines_end - b.start) + f.latency + 1;
                    stack.pop_back();
                    --depth;
                    tokens[cur_type()] += 1;
                    stack.back().latency += lat;
                } else {
                    return fail(i);
                }
                break;
            default:
                return fail(i);
            }
            break;
        }
        case kEntry: {
            const int32_t close = f.type == kSubtask ? PARASON_TAG_SUBTASK_END : PARASON_TAG_TRIAL_END;
            if (is_text(x)) {
                tokens[cur_type()] += 1;
                f.phase += 1;
            } else if (x == close && f.phase > 0) {
                tokens[cur_type()] += 1;
                const int32_t type = f.type, bi = f.block;
                stack.pop_back();
                out->blocks[bi].entries.push_back(type);
                stack.back().phase = kEntryOrEnd;
            } else {
                return fail(i);
            }
            break;
        }
        }
    }
    if (!stack.empty()) return fail(n);       // the stream ended early
    if (i != n) return fail(i);               // symbols after </think>
    parason_trace_stats &st = out->st;
    st.total_tokens = n;
    st.subtask_tokens = tokens[kSubtask];
    st.trial_tokens = tokens[kTrial];
    st.parallel_blocks = static_cast<int32_t>(out->blocks.size());
    st.threads = static_cast<int32_t>(out->threads.size());
    st.max_depth = max_depth;
    st.top_level_blocks = static_cast<int32_t>(out->top_blocks.size());
    st.acceleration = static_cast<double>(n) / static_cast<double>(st.latency_tokens);
    st.eta = 1.0 - static_cast<double>(st.latency_tokens) / static_cast<double>(n);
    return true;
}

}  // namespace

extern "C" {

parason_status parason_trace_analyze(const int32_t *symbols, int64_t n, parason_trace_stats *out,
                                     int64_t *error_pos) {
    if (!out || n < 0 || (n > 0 && !symbols)) return PARASON_EINVAL;
    Parsed p;
    int64_t err = -1;
    const bool ok = parse(symbols, n, &p, &err);
    if (error_pos) *error_pos = ok ? -1 : err;
    if (!ok) return PARASON_EINVAL;
    *out = p.st;
    return PARASON_OK;
}

parason_status parason_trace_fork_tree(const int32_t *symbols, int64_t n, int32_t block,
                                       int32_t capacity, int32_t *parent, int32_t *node_len,
                                       int32_t *leaf_node, int32_t *num_nodes,
                                       int32_t *num_leaves) {
    if (!num_nodes || !num_leaves || n < 0 || (n > 0 && !symbols) || capacity < 0)
        return PARASON_EINVAL;
    Parsed p;
    int64_t err = -1;
    if (!parse(symbols, n, &p, &err)) return PARASON_EINVAL;
    if (block < 0 || block >= static_cast<int32_t>(p.top_blocks.size())) return PARASON_EINVAL;
    const BlockRec &root = p.blocks[p.top_blocks[block]];
    // node 0: every token before the block's first thread; then the threads
    // depth first (a thread with a nested block holds its tokens up to the
    // end of that block's outlines and has its threads as children)
    std::vector<int32_t> par{-1}, len{static_cast<int32_t>(p.threads[root.threads[0]].start)}, leaves;
    std::vector<std::pair<int32_t, int32_t>> todo;   // (thread record, parent node), in reverse
    for (size_t k = root.threads.size(); k-- > 0;) todo.emplace_back(root.threads[k], 0);
    while (!todo.empty()) {
        const auto [ti, pn] = todo.back();
        todo.pop_back();
        const ThreadRec &t = p.threads[ti];
        const int32_t me = static_cast<int32_t>(par.size());
        par.push_back(pn);
        if (t.first_nested < 0) {
            len.push_back(static_cast<int32_t>(t.end - t.start));
            leaves.push_back(me);
        } else {
            const BlockRec &nb = p.blocks[t.first_nested];
            len.push_back(static_cast<int32_t>(nb.outlines_end - t.start));
            for (size_t k = nb.threads.size(); k-- > 0;) todo.emplace_back(nb.threads[k], me);
        }
    }
    *num_nodes = static_cast<int32_t>(par.size());
    *num_leaves = static_cast<int32_t>(leaves.size());
    if (*num_nodes > capacity) return PARASON_EINVAL;   // counts tell the size needed
    if (!parent || !node_len || !leaf_node) return PARASON_EINVAL;
    for (size_t k = 0; k < par.size(); ++k) {
        parent[k] = par[k];
        node_len[k] = len[k];
    }
    for (size_t k = 0; k < leaves.size(); ++k) leaf_node[k] = leaves[k];
    return PARASON_OK;
}

}  // extern "C"
