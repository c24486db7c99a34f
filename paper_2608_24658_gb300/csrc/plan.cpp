// plan.cpp -- host planner and C ABI of libparason.
//
// The planner turns a fork tree (branches of Subtask/Trial parallel regions
// decoded as independent workers, paper Sec. 3.4; nested regions per Fig. 4)
// into work items for the attention kernel and merge lists for the merge
// kernel:
//
//  * every node n that some branch reads is processed once per kv head, with
//    all R_n = (#branches under n) * g query rows stacked into tiles of up to
//    64 rows, so the node's KV is read from HBM once for all of them;
//  * long nodes are cut into chunks of whole pages (split-K) so that the
//    grid fills the GPU; each (node, chunk, kv head) has R_n partial slots;
//  * branch b's result is the log-sum-exp merge of the partial slots of every
//    node on its root->leaf path and every chunk of those nodes.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <queue>
#include <vector>

#include <cudaTypedefs.h>

#include "internal.h"

using parason::WorkItem;

namespace {

constexpr int kNarrowRows = 16;         // nodes with at most this many rows: suffix pass
// autonomous warps per suffix-pass CTA (the kernel's count for the KV format)
// (the kernel's count for the KV format: 6 deeper warps for bf16 at head_dim
// 128 with g <= 4, where they are latency-bound)
int32_t narrow_warps(int32_t mode, int32_t head_dim, int32_t g) {
    if (mode == PARASON_FP8_E4M3_KV) return 12;
    return (mode == PARASON_BF16 && head_dim == 128 && g <= 4) ? 6 : 8;
}
// Suffix-pass pieces are at least kMinPiecePages long (4 against 8: tiny
// fork 13.8 -> 11.7 us, the Llama-3 shape, whose pieces are 8 pages long by
// the share below, level).
constexpr int kMinPiecePages = 4;
constexpr int kMaxPiecePages = 128;     // and at most this long
// The tcgen05 tile holds an item of up to 512 pages (its metadata slot).
constexpr int kMaxTileItemPages = 512;
constexpr int kWideBlockPages = 4;      // prefix pieces are whole 64-token blocks
// Prefix pieces: about one prefix CTA's share of the prefix work each, at
// most what the tile's metadata holds.  Every piece writes 64 KB of partial
// rows (128 rows) that the merge reads back and costs the tile an item
// change; the prefix CTAs join the suffix queue when theirs is empty, which
// evens out their uneven shares.  Same-box A/B against a third of a share
// and at most 128 pages: two-level step 81.8 -> 78.7 us, Llama-3 shape
// 39.8 -> 39.2 us, long prefix 854.5 -> 843 us (e4m3 KV 655.4 -> 600.2
// us), batched 2460 -> 2447 us.
constexpr int64_t kWidePiecesPerCta = 1;
// A prefill's queue is the whole launch, and nothing evens out the prefix
// CTAs' ends: its piece length is the one, of a few candidates, under which
// the queue, simulated, empties first.  An entry's start and its O cost
// about kPieceStartPages pages (join prefill, 8 -> 16 pieces per path: the
// kernel went from 606 to 672 us for 1024 more pairs on 152 CTAs, about 38
// pages of a pair each); a lone tile of a pair kLoneTileShare of a pair's
// time.
constexpr double kPieceStartPages = 32.0;
constexpr double kLoneTileShare = 0.6;
constexpr int kPieceCountCandidates = 16;
constexpr int64_t kPieceLengthSteps = 16;   // lengths tried per piece count, 4 pages apart
// suffix pieces: about this many per warp of the launch (at least
// kMinPiecePages and at most kMaxPiecePages pages).  Same-box A/B against
// 3: two-level step 79.7 -> 78.8 us, the Llama-3 shape level (its pieces
// were at an 8-page floor); 2 made the Llama-3-shape step 2 us slower.
constexpr double kNarrowPiecesPerWarp = 2.5;
constexpr double kWideProvision = 1.15;   // prefix CTAs relative to the cost model
// Decode: up to this many prefix queue entries per prefix CTA (num / den)
// become one CTA each; up to two, two entries each
constexpr int64_t kSpareEntriesNum = 3, kSpareEntriesDen = 2;
// pairs of tcgen05 row tiles when at least this share of the prefix
// tile-pages sits in pieces of two or more tiles.  Same-box A/B, pairs
// against single tiles: 32k prefix tile alone 207.4 -> 155.8 us, join
// prefill 856.6 -> 721.8 us, fork prefill 84.5 -> 75.2 us, long prefix
// 842.8 -> 839.4 us; the two-level tree (2/3 of its tile-pages in pieces of
// two or more tiles) 77.6 -> 87.8 us, so it stays on single tiles.
constexpr int64_t kPairShareNum = 3, kPairShareDen = 4;
constexpr int kFp32ChunkPages = 32;
// stream rows kept free after a branch's last item: half its pages, 4 to 64
// (an item that grows further makes the launch's tail: build a new plan)
constexpr int32_t kAppendSlackMin = 4, kAppendSlackMax = 64;
constexpr int kPatchesPerTail = 6;      // words one append may change per tail item
constexpr double kWideGroupPageCost = 1.0;   // one 16-row group of one page, in suffix pages
constexpr double kTcPageCost = 2.0;          // one page of a tcgen05 prefix tile (tuned)
constexpr double kTcPageCostE4m3 = 3.6;      // the same with e4m3 KV, whose suffix pages
                                             // take half the time (tuned)
constexpr int64_t kDefaultWaitNs = 2000000000LL;
constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Time of one page of a prefix-pass tile relative to one page of the suffix
// pass on the same SM.  The suffix pass runs 8 pages at once (one per warp);
// a prefix tile runs one 16-row MMA group of the page per warp, so a page of
// a tile with G groups costs G suffix pages of warp time.
//
// The prefix tile at head_dim 128 runs on tcgen05: one 128-row MMA per 64
// tokens, whatever the rows, at a cost measured against the suffix pass.
double wide_page_cost(int32_t rows, bool tensor_core_tile, bool e4m3) {
    if (tensor_core_tile) return e4m3 ? kTcPageCostE4m3 : kTcPageCost;
    const double groups = (rows + 15) / 16;
    return std::max(1.0, groups * kWideGroupPageCost);
}

// Pieces of a run of `pages` pages under the piece length `chunk`: equal
// pieces, multiples of `align` pages except the last.  Sets the pages of
// each piece but the last (`per`) and the piece count (`n`).
void piece_split(int64_t pages, int64_t chunk, int64_t align, int64_t &per, int64_t &n) {
    chunk = std::max<int64_t>(align, chunk / align * align);
    n = (pages + chunk - 1) / chunk;
    per = (pages + n - 1) / n;
    per = (per + align - 1) / align * align;
    n = (pages + per - 1) / per;
}

// Time, in pages, for `ctas` CTAs to empty a prefix queue whose (pages,
// tiles) groups are cut into pieces of at most `chunk` pages.  The queue
// hands its entries out longest first, the first `ctas` to the CTAs that own
// them, each later one to the CTA that frees first.  An entry is a tile, or
// with pairs two tiles (a lone tile at kLoneTileShare of a pair's time), and
// costs its pages plus kPieceStartPages for its start and its O.
double prefix_queue_time(const std::vector<std::pair<int64_t, int32_t>> &groups, int64_t chunk,
                         int32_t ctas, bool pairs) {
    std::vector<std::pair<int64_t, double>> entries;   // (pages, time)
    for (const auto &g : groups) {
        int64_t per = 0, n = 0;
        piece_split(g.first, chunk, kWideBlockPages, per, n);
        const int32_t full = pairs ? g.second / 2 : g.second;
        const int32_t lone = pairs ? g.second % 2 : 0;
        for (int64_t k = 0; k < n; ++k) {
            const int64_t np = std::min(per, g.first - k * per);
            for (int32_t t = 0; t < full; ++t)
                entries.emplace_back(np, static_cast<double>(np) + kPieceStartPages);
            for (int32_t t = 0; t < lone; ++t)
                entries.emplace_back(np, kLoneTileShare * static_cast<double>(np) + kPieceStartPages);
        }
    }
    std::stable_sort(entries.begin(), entries.end(),
                     [](const auto &a, const auto &b) { return a.first > b.first; });
    std::priority_queue<double, std::vector<double>, std::greater<double>> free_at;
    double end = 0.0;
    for (size_t e = 0; e < entries.size(); ++e) {
        double t0 = 0.0;
        if (e >= static_cast<size_t>(ctas)) {
            t0 = free_at.top();
            free_at.pop();
        }
        const double t1 = t0 + entries[e].second;
        free_at.push(t1);
        end = std::max(end, t1);
    }
    return end;
}

// Rows of one tile: a multiple of g (so a branch's rows never straddle two
// tiles) of at most 16 (fp32 mode and the suffix pass) or 128 (prefix pass).
int32_t tile_rows_for(int32_t rows, int32_t g, int32_t mode) {
    const int32_t cap = (mode == PARASON_FP32 || rows <= kNarrowRows) ? 16 : 128;
    if (g > cap) return 0;
    const int32_t t = (cap / g) * g;
    return std::min(t, ((rows + g - 1) / g) * g);
}

}  // namespace

struct parason_plan_s {
    parason_attn_config cfg{};
    int32_t group = 1;
    int32_t num_nodes = 0;
    int32_t num_leaves = 0;
    int64_t num_phys = 0;
    int32_t num_sms = 152;
    int32_t chunk_pages = kMinPiecePages;   // reported shortest piece
    std::vector<WorkItem> items;
    std::vector<int32_t> page_ids;
    std::vector<int32_t> dfs_leaf;
    std::vector<int2> merge_rng;       // per (branch, kv head): [begin, end) of its entries
    std::vector<int32_t> merge_ent;   // first partial slot of the branch's rows
    std::vector<int32_t> wide_queue;   // prefix-pass items, in pull order
    std::vector<int32_t> narrow_queue; // suffix-pass items, in pull order
    std::vector<int32_t> item_rows;    // per item: start of its page rows
    std::vector<int32_t> stream_rows;  // TMA row of every page, item by item
    std::vector<int32_t> item_rec;     // kRecWords per item (suffix-warp record)

    // the tree as it stands: appends grow branch nodes, forks add nodes and
    // branches (parason_plan_append / parason_plan_fork)
    std::vector<int32_t> tree_parent, tree_len, leaf_node;
    std::vector<std::vector<int32_t>> node_pages;   // physical pages of each node
    std::vector<int32_t> node_page_pos;             // each node's first position in page_ids
    std::vector<int32_t> dfs_pos;                   // branch -> its position in dfs_leaf
    std::vector<std::vector<int32_t>> tails;        // per branch: items ending at its node's last page
    std::vector<uint8_t> page_used;                 // physical pages some node owns
    int64_t narrow_chunk = kMinPiecePages;          // suffix piece length of the plan
    // room the device copy keeps for forks (a fork past it is PARASON_ENOSPACE)
    size_t cap_items = 0, cap_rows = 0, cap_leaves = 0, cap_ent = 0, cap_patch = 0;
    int32_t num_ctas = 0;
    int32_t num_wide_ctas = 0;
    int32_t suffix_warps = 8;          // suffix-pass warps per CTA (kernel instantiation)
    // the prefix queue holds pairs of row tiles (bf16 KV, head_dim 128):
    // position k is items 2k and 2k + 1, the second without rows when its
    // piece has an odd number of tiles
    bool tc_pairs = false;
    int64_t num_slots = 0;
    int64_t unique_tokens = 0;
    int64_t path_tokens = 0;
    bool prefill = false;              // a tree-masked prefill plan
    std::vector<int32_t> shard_branch; // sharded plans: global index of each branch
    std::vector<int32_t> item_key0;    // prefill: first key of a causal item, else -1

    // device side
    bool on_device = false;
    int device = -1;
    void *d_blob = nullptr;
    WorkItem *d_items = nullptr;
    int32_t *d_page_ids = nullptr;
    int32_t *d_dfs_leaf = nullptr;
    int2 *d_merge_rng = nullptr;
    int32_t *d_merge_ent = nullptr;
    int32_t *d_item_rec = nullptr;
    int2 *d_patch = nullptr;
    int32_t *d_item_key0 = nullptr;    // prefill plans only
    std::vector<int2> patches;         // host side of the last append's patch list
    size_t blob_words = 0;
    // word offsets of arrays in the blob (patch targets)
    size_t w_items = 0, w_rec = 0, w_strows = 0, w_mrng = 0, w_qnext = 0;
    int32_t *d_item_rows = nullptr;
    int32_t *d_stream_rows = nullptr;
    int32_t *d_queue_next = nullptr;   // 2 counters, set back to queue_start by the merge kernel
    int32_t queue_start[2] = {0, 0};   // positions past the ones CTAs own at launch
    int32_t *d_err = nullptr;
    uint32_t debug_flags = 0;
    int64_t wait_limit_ns = kDefaultWaitNs;

    // tensor maps of the last KV pools seen
    std::mutex tm_mutex;
    const void *tm_k_ptr = nullptr;
    const void *tm_v_ptr = nullptr;
    parason::KvMaps tm{};

    // timing
    int32_t timing_cap = 0;
    int32_t timing_n = 0;
    std::vector<cudaEvent_t> events;   // 3 per recorded call
};

namespace {

// ---------------------------------------------------------------------------
// validation and work decomposition (no CUDA calls)
// ---------------------------------------------------------------------------

parason_status validate_config(const parason_attn_config *cfg) {
    if (!cfg) return PARASON_EINVAL;
    if (cfg->num_q_heads <= 0 || cfg->num_kv_heads <= 0) return PARASON_EINVAL;
    if (cfg->num_q_heads % cfg->num_kv_heads != 0) return PARASON_EINVAL;
    if (cfg->head_dim != 64 && cfg->head_dim != 128) return PARASON_EINVAL;
    if (cfg->page_size != parason::kPageSize) return PARASON_EINVAL;
    if (cfg->mode != PARASON_BF16 && cfg->mode != PARASON_FP32 &&
        cfg->mode != PARASON_FP8_E4M3_KV)
        return PARASON_EINVAL;
    if (!(cfg->sm_scale >= 0.0f) || !std::isfinite(cfg->sm_scale)) return PARASON_EINVAL;
    if (cfg->mode == PARASON_FP8_E4M3_KV && cfg->head_dim != 128) return PARASON_EUNSUPPORTED;
    return PARASON_OK;
}

// The tree and its page table: parents before children, page counts that
// match the lengths, page ids in range and owned once, branches distinct,
// in range and childless.  (Pointer checks are the caller's.)
parason_status validate_tree(int32_t num_nodes, const int32_t *parent, const int32_t *node_len,
                             const int32_t *node_page_ptr, const int32_t *page_ids,
                             int32_t num_leaves, const int32_t *leaf_node, int64_t num_phys,
                             int32_t H_kv) {
    if (num_nodes < 0 || num_leaves < 0 || num_phys < 0) return PARASON_EINVAL;
    if (num_nodes > 0 && (!parent || !node_len || !node_page_ptr)) return PARASON_EINVAL;
    if (num_leaves > 0 && !leaf_node) return PARASON_EINVAL;
    if (num_leaves > 0 && num_nodes == 0) return PARASON_EINVAL;
    if (num_nodes > 0 && node_page_ptr[0] != 0) return PARASON_EINVAL;
    for (int32_t i = 0; i < num_nodes; ++i) {
        if (parent[i] < -1 || parent[i] >= i) return PARASON_EINVAL;
        if (node_len[i] < 0) return PARASON_EINVAL;
        const int64_t want = (static_cast<int64_t>(node_len[i]) + parason::kPageSize - 1) /
                             parason::kPageSize;
        if (static_cast<int64_t>(node_page_ptr[i + 1]) - node_page_ptr[i] != want)
            return PARASON_EINVAL;
    }
    const int64_t total_pages = num_nodes > 0 ? node_page_ptr[num_nodes] : 0;
    if (total_pages > 0 && !page_ids) return PARASON_EINVAL;
    // rows addressed by the kernels: (page * H_kv + kv_head) * 16 must fit int32
    if (num_phys > 0 &&
        (num_phys * static_cast<int64_t>(H_kv) * parason::kPageSize) > INT32_MAX)
        return PARASON_EUNSUPPORTED;
    {
        std::vector<int32_t> sorted(static_cast<size_t>(total_pages));
        if (total_pages > 0)
            std::memcpy(sorted.data(), page_ids, sizeof(int32_t) * static_cast<size_t>(total_pages));
        std::sort(sorted.begin(), sorted.end());
        for (int64_t i = 0; i < total_pages; ++i) {
            if (sorted[i] < 0 || sorted[i] >= num_phys) return PARASON_EINVAL;
            if (i > 0 && sorted[i] == sorted[i - 1]) return PARASON_EINVAL;
        }
    }
    std::vector<uint8_t> is_leaf(num_nodes, 0);
    std::vector<int32_t> nchild(num_nodes, 0);
    for (int32_t i = 0; i < num_nodes; ++i)
        if (parent[i] >= 0) nchild[parent[i]]++;
    for (int32_t b = 0; b < num_leaves; ++b) {
        const int32_t n = leaf_node[b];
        if (n < 0 || n >= num_nodes) return PARASON_EINVAL;
        if (is_leaf[n]) return PARASON_EINVAL;
        if (nchild[n] != 0) return PARASON_EINVAL;
        is_leaf[n] = 1;
    }
    return PARASON_OK;
}

// With `prefill`, leaf_node holds the chunk nodes of a tree-masked prefill:
// every token of a chunk is a query (numbered chunk by chunk), attending to
// every token of its node's ancestors and causally to its own node.
parason_status build_host(parason_plan_s *p, const parason_attn_config *cfg, int32_t num_nodes,
                          const int32_t *parent, const int32_t *node_len,
                          const int32_t *node_page_ptr, const int32_t *page_ids,
                          int32_t num_leaves, const int32_t *leaf_node,
                          int64_t num_phys, int32_t num_sms, bool prefill = false) {
    parason_status st = validate_config(cfg);
    if (st != PARASON_OK) return st;
    // the prefill's causal mask is in the tcgen05 tile: bf16 or e4m3 KV at head_dim 128
    if (prefill && (cfg->mode == PARASON_FP32 || cfg->head_dim != 128)) return PARASON_EUNSUPPORTED;
    p->prefill = prefill;
    if (num_nodes < 0 || num_leaves < 0 || num_phys < 0) return PARASON_EINVAL;

    const int32_t H_kv = cfg->num_kv_heads;
    const int32_t g = cfg->num_q_heads / H_kv;
    p->cfg = *cfg;
    p->group = g;
    p->num_nodes = num_nodes;
    p->num_leaves = num_leaves;
    p->num_phys = num_phys;
    p->num_sms = num_sms > 0 ? num_sms : 152;

    st = validate_tree(num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves, leaf_node,
                       num_phys, H_kv);
    if (st != PARASON_OK) return st;
    const int64_t total_pages = num_nodes > 0 ? node_page_ptr[num_nodes] : 0;
    p->page_ids.resize(static_cast<size_t>(total_pages));
    if (total_pages > 0)
        std::memcpy(p->page_ids.data(), page_ids, sizeof(int32_t) * static_cast<size_t>(total_pages));
    std::vector<int32_t> leaf_of_node(num_nodes, -1);
    for (int32_t b = 0; b < num_leaves; ++b) leaf_of_node[leaf_node[b]] = b;

    // branches under each node, and DFS order: parent[i] < i, so a reverse
    // sweep accumulates subtree counts and a forward sweep lays the subtrees
    // out contiguously (children in index order).
    std::vector<int64_t> cnt(num_nodes, 0), lo(num_nodes, 0), next_child(num_nodes, 0);
    for (int32_t i = 0; i < num_nodes; ++i) cnt[i] = leaf_of_node[i] >= 0 ? 1 : 0;
    for (int32_t i = num_nodes - 1; i >= 0; --i)
        if (parent[i] >= 0) cnt[parent[i]] += cnt[i];
    int64_t root_cursor = 0;
    for (int32_t i = 0; i < num_nodes; ++i) {
        if (parent[i] < 0) {
            lo[i] = root_cursor;
            root_cursor += cnt[i];
        } else {
            lo[i] = lo[parent[i]] + next_child[parent[i]];
            next_child[parent[i]] += cnt[i];
        }
    }
    // queries of a prefill: every token of every chunk, chunk by chunk
    std::vector<int64_t> qbase(static_cast<size_t>(num_leaves) + 1, 0);
    if (prefill) {
        for (int32_t c = 0; c < num_leaves; ++c) qbase[c + 1] = qbase[c] + node_len[leaf_node[c]];
        if (qbase[num_leaves] > INT32_MAX / 64) return PARASON_EUNSUPPORTED;
        p->num_leaves = static_cast<int32_t>(qbase[num_leaves]);
        p->dfs_leaf.resize(static_cast<size_t>(p->num_leaves));
        for (int32_t k = 0; k < p->num_leaves; ++k) p->dfs_leaf[k] = k;
    } else {
        p->dfs_leaf.assign(num_leaves, -1);
        for (int32_t b = 0; b < num_leaves; ++b) p->dfs_leaf[lo[leaf_node[b]]] = b;
    }

    // ------------------------------------------------------------------
    // work decomposition
    //
    // A run is (node, kv head, row tile) over all of the node's pages.  Runs
    // are cut into items along pages; every item owns `nrows` consecutive
    // partial slots.  Row tiles start at multiples of g, so each branch's g
    // rows of a node sit in one tile.
    const int32_t mode = cfg->mode;
    struct Run {
        int32_t node, head, row0, nrows;
        int64_t pages;              // pages the run covers (from the node's first)
        int64_t node_pages = 0;     // pages of the node
        int64_t leaf_lo = 0;        // position of its first row's branch (query)
        double cost_per_page;
        bool wide;
        bool causal = false;        // prefill: keys past the row's own token are masked
        int32_t span = -1;          // bf16 prefill: its page list in `spans`
    };
    // A bf16 prefill run reads its chunk's whole path in one list of pages:
    // every page of every non-empty ancestor, root first, then the chunk's
    // own pages up to the tile pair's last token.  Its pieces cross node
    // boundaries, so that each query row has a partial per piece of its path
    // rather than one per node.  An ancestor that ends inside a page is
    // followed by padding pages (zero-filled by TMA) up to the next 64-token
    // block, so that the keys no token stands for always end a block.
    struct Span {
        std::vector<int32_t> pos;     // position in page_ids of each page, -1: padding
        std::vector<int32_t> valid;   // valid tokens of each page
        int64_t own = 0;              // pages before the chunk's own ones
    };
    const int32_t pad_row = static_cast<int32_t>(num_phys * H_kv * parason::kPageSize);
    std::vector<Span> spans;
    std::vector<int32_t> item_span_rows;   // explicit page rows of span items, by item
    std::vector<int64_t> item_span_off;    // their start in item_span_rows, -1: none
    std::vector<Run> runs;
    int64_t narrow_pages = 0;
    double wide_cost = 0.0;
    if (prefill) {
        // chunk c: rows (token t, q head r) = t * g + r of every kv head, in
        // tiles; each tile reads every ancestor in full and its own node up
        // to the tile's last token
        for (int32_t c = 0; c < num_leaves; ++c) {
            const int32_t n = leaf_node[c];
            const int64_t C = node_len[n];
            if (C == 0) continue;
            const int64_t R = C * g;
            const int32_t rt = tile_rows_for(static_cast<int32_t>(std::min<int64_t>(R, 1 << 20)), g, mode);
            if (rt <= 0) return PARASON_EUNSUPPORTED;
            std::vector<int32_t> path;
            for (int32_t m = n; m >= 0; m = parent[m]) path.push_back(m);
            std::reverse(path.begin(), path.end());
            if (mode == PARASON_BF16 && cfg->head_dim == 128) {
                // one list per tile pair, up to the pair's last token; a pair's
                // first tile reads the few pages past its own last token masked
                const int64_t pair_rows = 2 * static_cast<int64_t>(rt);
                for (int64_t p0 = 0; p0 < R; p0 += pair_rows) {
                    const int64_t tb = std::min<int64_t>(R, p0 + pair_rows) / g;   // tokens [.., tb)
                    Span sp;
                    for (int32_t m : path) {
                        if (node_len[m] == 0) continue;
                        const int64_t P = node_page_ptr[m + 1] - node_page_ptr[m];
                        const int64_t use = m == n ? (tb + parason::kPageSize - 1) / parason::kPageSize : P;
                        if (m == n) sp.own = static_cast<int64_t>(sp.pos.size());
                        for (int64_t k = 0; k < use; ++k) {
                            sp.pos.push_back(node_page_ptr[m] + static_cast<int32_t>(k));
                            sp.valid.push_back(k == P - 1 ? node_len[m] - static_cast<int32_t>(P - 1) *
                                                                              parason::kPageSize
                                                          : parason::kPageSize);
                        }
                        while (m != n && sp.valid.back() < parason::kPageSize &&
                               sp.pos.size() % kWideBlockPages != 0) {
                            sp.pos.push_back(-1);
                            sp.valid.push_back(0);
                        }
                    }
                    spans.push_back(std::move(sp));
                    const int32_t si = static_cast<int32_t>(spans.size()) - 1;
                    for (int32_t j = 0; j < H_kv; ++j)
                        for (int64_t r0 = p0; r0 < std::min<int64_t>(R, p0 + pair_rows); r0 += rt) {
                            Run run;
                            run.node = n;
                            run.head = j;
                            run.row0 = static_cast<int32_t>(r0);
                            run.nrows = static_cast<int32_t>(std::min<int64_t>(rt, R - r0));
                            run.pages = static_cast<int64_t>(spans[si].pos.size());
                            run.node_pages = run.pages;
                            run.causal = true;
                            run.span = si;
                            run.leaf_lo = qbase[c];
                            run.wide = true;
                            run.cost_per_page = wide_page_cost(run.nrows, true, false);
                            wide_cost += run.cost_per_page * static_cast<double>(run.pages);
                            runs.push_back(run);
                        }
                }
                continue;
            }
            // (kv head, node, tile): the tiles of one ancestor read the same
            // pages and sit next to each other for the piece interleaving
            for (int32_t j = 0; j < H_kv; ++j)
                for (int32_t m : path) {
                    if (node_len[m] == 0) continue;
                    for (int64_t r0 = 0; r0 < R; r0 += rt) {
                        const int64_t nrows = std::min<int64_t>(rt, R - r0);
                        const int64_t tb = (r0 + nrows) / g;         // tokens [r0 / g, tb)
                        Run run;
                        run.node = m;
                        run.head = j;
                        run.row0 = static_cast<int32_t>(r0);
                        run.nrows = static_cast<int32_t>(nrows);
                        run.node_pages = node_page_ptr[m + 1] - node_page_ptr[m];
                        run.causal = m == n;
                        run.pages = run.causal ? (tb + parason::kPageSize - 1) / parason::kPageSize
                                               : run.node_pages;
                        run.leaf_lo = qbase[c];
                        run.wide = true;
                        run.cost_per_page = wide_page_cost(run.nrows, true, mode == PARASON_FP8_E4M3_KV);
                        wide_cost += run.cost_per_page * static_cast<double>(run.pages);
                        runs.push_back(run);
                    }
                }
        }
        for (int32_t n = 0; n < num_nodes; ++n)
            if (cnt[n] > 0) p->unique_tokens += node_len[n];
        // keys a query sees: its ancestors and its own node up to itself
        for (int32_t c = 0; c < num_leaves; ++c) {
            const int64_t C = node_len[leaf_node[c]];
            for (int32_t m = parent[leaf_node[c]]; m >= 0; m = parent[m]) p->path_tokens += C * node_len[m];
            p->path_tokens += C * (C + 1) / 2;
        }
    }
    for (int32_t n = 0; n < num_nodes && !prefill; ++n) {
        if (cnt[n] == 0 || node_len[n] == 0) continue;
        p->unique_tokens += node_len[n];
        const int64_t R = cnt[n] * g;
        if (R > INT32_MAX / 4) return PARASON_EUNSUPPORTED;
        const int64_t P = node_page_ptr[n + 1] - node_page_ptr[n];
        const int32_t rt = tile_rows_for(static_cast<int32_t>(std::min<int64_t>(R, 1 << 20)), g, mode);
        if (rt <= 0) return PARASON_EUNSUPPORTED;
        const bool wide = mode != PARASON_FP32 && R > kNarrowRows;
        for (int32_t j = 0; j < H_kv; ++j)
            for (int64_t r0 = 0; r0 < R; r0 += rt) {
                Run run;
                run.node = n;
                run.head = j;
                run.row0 = static_cast<int32_t>(r0);
                run.nrows = static_cast<int32_t>(std::min<int64_t>(rt, R - r0));
                run.pages = P;
                run.node_pages = P;
                run.leaf_lo = lo[n];
                run.wide = wide;
                run.cost_per_page =
                    // bf16 and e4m3 KV at head_dim 128 run the prefix on tcgen05
                    wide ? wide_page_cost(run.nrows, cfg->head_dim == 128, mode == PARASON_FP8_E4M3_KV)
                         : 1.0;
                if (wide)
                    wide_cost += run.cost_per_page * static_cast<double>(P);
                else
                    narrow_pages += P;
                runs.push_back(run);
            }
    }

    // The row tiles of one (node, kv head) over the same pages: runs [i, j)
    auto group_end = [&](size_t i) {
        size_t j = i + 1;
        while (j < runs.size() && runs[j].node == runs[i].node && runs[j].head == runs[i].head &&
               runs[j].pages == runs[i].pages)
            ++j;
        return j;
    };
    // Pairs of tiles: with bf16 KV at head_dim 128, when most prefix
    // tile-pages sit in pieces of two or more tiles, the tcgen05 tile runs
    // two tiles of a piece against each staged block.  The cost model and
    // the piece length still count tiles one by one (counting a pair as one
    // unit made fewer prefix CTAs and longer pieces, and was slower: long
    // prefix 841.8 -> 853.4 us, 32k prefix tile alone 156.1 -> 232.4 us).
    p->tc_pairs = false;
    if (mode == PARASON_BF16 && cfg->head_dim == 128) {
        int64_t multi = 0, all = 0;
        for (size_t i = 0; i < runs.size();) {
            const size_t j = group_end(i);
            if (runs[i].wide) {
                const int64_t tp = static_cast<int64_t>(j - i) * runs[i].pages;
                all += tp;
                if (j - i >= 2) multi += tp;
            }
            i = j;
        }
        p->tc_pairs = all > 0 && multi * kPairShareDen >= all * kPairShareNum;
    }
    int64_t wide_units = 0;                 // tile-pages of the prefix pass
    for (const Run &r : runs)
        if (r.wide) wide_units += r.pages;

    // CTAs of the persistent kernel: the first n_wide start on the prefix
    // queue and join the suffix queue when it runs dry, the others run the
    // suffix queue only.  Prefix CTAs are over-provisioned on purpose: spare
    // prefix capacity turns into suffix work, a prefix shortfall would be the
    // tail.  The fp32 kernel runs one item per CTA instead.
    int32_t n_wide = 0, n_narrow_ctas = 0;
    if (mode != PARASON_FP32) {
        const int32_t S = p->num_sms;
        const double narrow_cost = static_cast<double>(narrow_pages);
        if (prefill) {
            n_wide = S;
        } else if (wide_cost > 0 && narrow_cost > 0) {
            n_wide = static_cast<int32_t>(
                std::ceil(kWideProvision * S * wide_cost / (wide_cost + narrow_cost)));
            n_wide = std::min(std::max(n_wide, 1), std::max(S - 1, 1));
        } else if (wide_cost > 0) {
            n_wide = S;
        }
        n_narrow_ctas = narrow_cost > 0 ? std::max(S - n_wide, 1) : 0;
    }
    // Prefix pieces are about one prefix CTA's share each.  When the runs
    // cut that way give a few more queue entries than prefix CTAs, the CTAs
    // that take a second entry end a piece after the others, with little
    // left for them to even out on the suffix queue: then every entry gets
    // a CTA of its own, at the same piece length (up to 3/2 entries per
    // CTA, while that leaves half the SMs to the suffix queue), or every CTA
    // two entries (up to 2; the CTAs spared run the suffix queue).  Same-box
    // A/B: Llama-3 shape (24 entries, 18 -> 24 CTAs) step 42.9 -> 39.4 us;
    // two-level (128 entries, 68 -> 64 CTAs) 78.8 -> 77.2 us.  Slower, and
    // so left out: evening out 3 or more entries per CTA (long prefix bf16
    // 835.9 -> 843.0 us), and 128 prefix CTAs of 152 for the two-level tree
    // with e4m3 KV (71.8 -> 73.3 us).
    int64_t wide_chunk = std::min<int64_t>(
        kMaxTileItemPages,
        std::max<int64_t>(kWideBlockPages,
                          wide_units / std::max<int64_t>(1, static_cast<int64_t>(n_wide) * kWidePiecesPerCta)));
    if (!prefill && mode != PARASON_FP32 && n_wide > 0 && n_narrow_ctas > 0) {
        int64_t entries = 0;
        for (size_t i = 0; i < runs.size();) {
            const size_t j = group_end(i);
            if (runs[i].wide) {
                int64_t per = 0, n = 0;
                piece_split(runs[i].pages, wide_chunk, kWideBlockPages, per, n);
                const int64_t tiles = static_cast<int64_t>(j - i);
                entries += n * (p->tc_pairs ? (tiles + 1) / 2 : tiles);
            }
            i = j;
        }
        const int32_t S = p->num_sms;
        const bool one_each =
            entries * kSpareEntriesDen <= static_cast<int64_t>(n_wide) * kSpareEntriesNum;
        if (entries > n_wide && one_each && entries <= S / 2) {
            n_wide = static_cast<int32_t>(entries);
            n_narrow_ctas = S - n_wide;
        } else if (entries > n_wide && !one_each && entries <= 2 * static_cast<int64_t>(n_wide)) {
            n_wide = static_cast<int32_t>((entries + 1) / 2);
            n_narrow_ctas = S - n_wide;
        }
    }
    p->num_wide_ctas = n_wide;
    p->num_ctas = n_wide + n_narrow_ctas;
    // the kernel's CTAs own the first positions of each queue (one per
    // prefix CTA, one per warp of a suffix CTA); the counters start past them
    p->queue_start[0] = n_wide;
    p->suffix_warps = narrow_warps(mode, cfg->head_dim, g);
    p->queue_start[1] = n_narrow_ctas * p->suffix_warps;

    // Items: every run cut into pieces of at most `chunk` pages (the prefix
    // pass in whole 64-token blocks).  Each role's pieces form a queue,
    // longest first, that the kernel's workers pull from at run time; the
    // pieces are short enough that the last ones to be pulled end together.
    p->items.clear();
    int64_t slots = 0;
    std::vector<std::pair<int64_t, int32_t>> wide_q, narrow_q;   // (pages, item)
    std::vector<std::pair<int32_t, int32_t>> tails;              // (branch, item)
    std::vector<int32_t> key0;                                   // per item (prefill)
    // `queued`: the item starts a queue entry (the second tile of a pair
    // does not); `blank`: a pair's second tile without rows
    auto emit = [&](const Run &run, int64_t pg0, int64_t np, bool queued = true,
                    bool blank = false) -> bool {
        WorkItem it;
        const int64_t P = run.node_pages;
        // a span piece ends at its last page with keys, not in padding
        if (run.span >= 0)
            while (np > 1 && spans[run.span].pos[pg0 + np - 1] < 0) --np;
        it.num_pages = static_cast<int32_t>(np);
        int32_t k0 = run.causal && !blank ? static_cast<int32_t>(pg0 * parason::kPageSize) : -1;
        if (run.span >= 0) {
            // the item's page rows; a page that ends a node inside the item
            // carries 16 - its valid tokens in the row's low bits
            const Span &sp = spans[run.span];
            it.page_pos = sp.pos[pg0];
            it.last_valid = sp.valid[pg0 + np - 1];
            item_span_off.push_back(static_cast<int64_t>(item_span_rows.size()));
            for (int64_t k = pg0; k < pg0 + np; ++k) {
                int32_t row = pad_row;
                if (sp.pos[k] >= 0) {
                    row = (page_ids[sp.pos[k]] * H_kv + run.head) * parason::kPageSize;
                    if (k < pg0 + np - 1) row |= parason::kPageSize - sp.valid[k];
                }
                item_span_rows.push_back(row);
            }
            // the chunk's own keys start at stream position 16 (own - pg0)
            // when the item holds the first of them, at own token 16 (pg0 -
            // own) when it starts among them; none when it holds none
            k0 = blank || pg0 + np <= sp.own
                     ? -1
                     : (pg0 < sp.own ? -static_cast<int32_t>((sp.own - pg0) * parason::kPageSize)
                                     : static_cast<int32_t>((pg0 - sp.own) * parason::kPageSize));
        } else {
            it.page_pos = node_page_ptr[run.node] + static_cast<int32_t>(pg0);
            it.last_valid = (pg0 + np == P)
                                ? node_len[run.node] - static_cast<int32_t>(P - 1) * parason::kPageSize
                                : parason::kPageSize;
            item_span_off.push_back(-1);
        }
        it.leaf_lo = static_cast<int32_t>(run.leaf_lo);
        it.row0 = blank ? 0 : run.row0;
        it.nrows = blank ? 0 : run.nrows;
        it.kv_head = run.head;
        if (slots + it.nrows > INT32_MAX) return false;
        it.slot_base = static_cast<int32_t>(slots);
        slots += it.nrows;
        const int32_t id = static_cast<int32_t>(p->items.size());
        p->items.push_back(it);
        if (queued) (run.wide ? wide_q : narrow_q).emplace_back(np, id);
        key0.push_back(k0);
        if (!prefill && !blank && pg0 + np == P && leaf_of_node[run.node] >= 0)
            tails.emplace_back(leaf_of_node[run.node], id);
        return true;
    };
    auto cut = [&](const Run &r, int64_t chunk, int64_t align) -> bool {
        chunk = std::max<int64_t>(align, chunk / align * align);
        const int64_t n = (r.pages + chunk - 1) / chunk;
        // equal pieces (multiples of `align` except the last)
        int64_t per = (r.pages + n - 1) / n;
        per = (per + align - 1) / align * align;
        for (int64_t pg = 0; pg < r.pages; pg += per)
            if (!emit(r, pg, std::min(per, r.pages - pg))) return false;
        return true;
    };
    if (mode == PARASON_FP32) {
        for (const Run &r : runs)
            if (!cut(r, kFp32ChunkPages, 1)) return PARASON_EUNSUPPORTED;
    } else {
        const int64_t total_warps = static_cast<int64_t>(p->num_sms) * p->suffix_warps;
        const int64_t narrow_chunk = std::min<int64_t>(
            kMaxPiecePages,
            std::max<int64_t>(kMinPiecePages,
                              static_cast<int64_t>(static_cast<double>(narrow_pages) /
                                                   (kNarrowPiecesPerWarp * std::max<int64_t>(1, total_warps)))));
        p->narrow_chunk = narrow_chunk;
        if (prefill && n_wide > 0) {
            // candidates: the longest run cut into n pieces, n from the
            // fewest the tile allows up, and the lengths between that and
            // the shortest run cut into n pieces (which give the longer runs
            // n + 1 pieces and the shorter ones n)
            std::vector<std::pair<int64_t, int32_t>> groups;   // (pages, tiles)
            int64_t longest = 0, shortest = INT64_MAX;
            for (size_t i = 0; i < runs.size();) {
                const size_t j = group_end(i);
                groups.emplace_back(runs[i].pages, static_cast<int32_t>(j - i));
                longest = std::max(longest, runs[i].pages);
                shortest = std::min(shortest, runs[i].pages);
                i = j;
            }
            double best = prefix_queue_time(groups, wide_chunk, n_wide, p->tc_pairs);
            const int64_t n0 = (longest + kMaxTileItemPages - 1) / kMaxTileItemPages;
            for (int64_t n = n0; n < n0 + kPieceCountCandidates; ++n) {
                const int64_t hi = (longest + n - 1) / n;
                const int64_t lo = std::max<int64_t>((shortest + n - 1) / n, hi - kPieceLengthSteps * kWideBlockPages);
                for (int64_t c0 = hi; c0 >= lo; c0 -= kWideBlockPages) {
                    const int64_t c = std::min<int64_t>(kMaxTileItemPages, std::max<int64_t>(kWideBlockPages, c0));
                    const double tq = prefix_queue_time(groups, c, n_wide, p->tc_pairs);
                    if (tq < best) {
                        best = tq;
                        wide_chunk = c;
                    }
                }
            }
        }
        // The row tiles of one (node, kv head) read the same pages: their
        // pieces are emitted piece by piece across the tiles, so that the
        // queue hands out the copies of one page range together and all but
        // the first read of each page come from L2.
        for (size_t i = 0; i < runs.size();) {
            const size_t j = group_end(i);
            const Run &r = runs[i];
            const bool pairs = r.wide && p->tc_pairs;
            const int64_t align = r.wide ? kWideBlockPages : 1;
            int64_t per = 0, n = 0;
            piece_split(r.pages, r.wide ? wide_chunk : narrow_chunk, align, per, n);
            for (int64_t pg = 0; pg < r.pages; pg += per) {
                const int64_t np = std::min(per, r.pages - pg);
                for (size_t t = i; t < j; ++t) {
                    const bool second = pairs && (t - i) % 2 == 1;
                    if (!emit(runs[t], pg, np, !second)) return PARASON_EUNSUPPORTED;
                    if (pairs && !second && t + 1 == j && !emit(runs[t], pg, np, false, true))
                        return PARASON_EUNSUPPORTED;
                }
            }
            i = j;
        }
    }
    if (p->items.size() > static_cast<size_t>(INT32_MAX)) return PARASON_EUNSUPPORTED;
    p->num_slots = slots;

    // queues, longest piece first (ties in item order)
    auto order = [](std::vector<std::pair<int64_t, int32_t>> &q, std::vector<int32_t> &out) {
        std::stable_sort(q.begin(), q.end(),
                         [](const auto &a, const auto &b) { return a.first > b.first; });
        out.clear();
        for (auto &e : q) out.push_back(e.second);
    };
    order(wide_q, p->wide_queue);
    order(narrow_q, p->narrow_queue);
    if (p->tc_pairs) {       // each queued first tile brings its second along
        std::vector<int32_t> both;
        both.reserve(2 * p->wide_queue.size());
        for (int32_t id : p->wide_queue) {
            both.push_back(id);
            both.push_back(id + 1);
        }
        p->wide_queue.swap(both);
    }
    if (mode == PARASON_FP32) {        // one CTA per item, no queues
        p->wide_queue.clear();
        p->narrow_queue.clear();
    } else {
        // item ids in pull order: the prefix queue is items [0, W), the
        // suffix queue items [W, W + N), so a pull needs no queue lookup
        std::vector<WorkItem> sorted;
        std::vector<int32_t> new_id(p->items.size(), -1);
        sorted.reserve(p->items.size());
        for (int32_t id : p->wide_queue) {
            new_id[id] = static_cast<int32_t>(sorted.size());
            sorted.push_back(p->items[id]);
        }
        for (int32_t id : p->narrow_queue) {
            new_id[id] = static_cast<int32_t>(sorted.size());
            sorted.push_back(p->items[id]);
        }
        p->items.swap(sorted);
        for (auto &t : tails) t.second = new_id[t.second];
        std::vector<int32_t> key0_sorted(key0.size());
        for (size_t id = 0; id < key0.size(); ++id) key0_sorted[new_id[id]] = key0[id];
        key0.swap(key0_sorted);
        std::vector<int64_t> span_sorted(item_span_off.size());
        for (size_t id = 0; id < item_span_off.size(); ++id) span_sorted[new_id[id]] = item_span_off[id];
        item_span_off.swap(span_sorted);
        for (size_t k = 0; k < p->wide_queue.size(); ++k) p->wide_queue[k] = static_cast<int32_t>(k);
        for (size_t k = 0; k < p->narrow_queue.size(); ++k)
            p->narrow_queue[k] = static_cast<int32_t>(p->wide_queue.size() + k);
    }

    // the items that end at each branch node's last page (appends grow them)
    std::sort(tails.begin(), tails.end());
    p->tails.assign(static_cast<size_t>(num_leaves), {});
    std::vector<uint8_t> is_tail(p->items.size(), 0);
    for (const auto &t : tails) {
        p->tails[t.first].push_back(t.second);
        is_tail[t.second] = 1;
    }
    p->page_used.assign(static_cast<size_t>(num_phys), 0);
    for (int64_t i = 0; i < total_pages; ++i) p->page_used[page_ids[i]] = 1;
    // the tree, for appends and forks
    p->tree_parent.assign(parent, parent + num_nodes);
    p->tree_len.assign(node_len, node_len + num_nodes);
    p->leaf_node.assign(leaf_node, leaf_node + num_leaves);
    p->node_page_pos.assign(node_page_ptr, node_page_ptr + num_nodes);
    p->node_pages.assign(static_cast<size_t>(num_nodes), {});
    for (int32_t n = 0; n < num_nodes; ++n)
        p->node_pages[n].assign(page_ids + node_page_ptr[n], page_ids + node_page_ptr[n + 1]);
    p->dfs_pos.assign(static_cast<size_t>(p->num_leaves), 0);
    for (size_t k = 0; k < p->dfs_leaf.size(); ++k) p->dfs_pos[p->dfs_leaf[k]] = static_cast<int32_t>(k);

    // page streams: the TMA row (page * H_kv + kv head) * 16 of every page of
    // every item, item by item; a tail item is followed by kAppendSlack free
    // rows for the pages appends will add
    p->item_rows.assign(p->items.size() + 1, 0);
    p->stream_rows.clear();
    for (size_t i = 0; i < p->items.size(); ++i) {
        const WorkItem &it = p->items[i];
        if (item_span_off[i] >= 0)
            p->stream_rows.insert(p->stream_rows.end(), item_span_rows.begin() + item_span_off[i],
                                  item_span_rows.begin() + item_span_off[i] + it.num_pages);
        else
            for (int32_t pg = 0; pg < it.num_pages; ++pg)
                p->stream_rows.push_back((page_ids[it.page_pos + pg] * H_kv + it.kv_head) *
                                         parason::kPageSize);
        if (mode != PARASON_FP32 && is_tail[i])
            p->stream_rows.insert(p->stream_rows.end(),
                                  std::min(kAppendSlackMax, std::max(kAppendSlackMin, it.num_pages / 2)),
                                  0);
        if (p->stream_rows.size() > static_cast<size_t>(INT32_MAX)) return PARASON_EUNSUPPORTED;
        p->item_rows[i + 1] = static_cast<int32_t>(p->stream_rows.size());
    }
    // one 128-byte record per item for the suffix warps: the item, the start
    // of its page rows in the stream, and its first page rows
    p->item_rec.assign(p->items.size() * parason::kRecWords, 0);
    for (size_t i = 0; i < p->items.size(); ++i) {
        int32_t *rec = p->item_rec.data() + i * parason::kRecWords;
        std::memcpy(rec, &p->items[i], sizeof(WorkItem));
        rec[parason::kRecRowsOff] = p->item_rows[i];
        const int32_t np = p->items[i].num_pages;
        for (int32_t j = 0; j < std::min(np, parason::kRecRows); ++j)
            rec[parason::kRecRow0 + j] = p->stream_rows[p->item_rows[i] + j];
    }

    if (prefill) p->item_key0 = key0;
    else p->item_key0.clear();

    // merge lists per (branch, kv head): the first of the branch's g partial
    // slots in every item, on the branch's path, that covers its rows (in a
    // prefill, not the chunk's own items whose keys all follow the token)
    const int32_t L_rows = p->num_leaves;
    std::vector<std::vector<int32_t>> ent(static_cast<size_t>(L_rows) * H_kv);
    for (size_t ii = 0; ii < p->items.size(); ++ii) {
        const WorkItem &it = p->items[ii];
        if (it.nrows == 0) continue;                  // a pair's blank second tile
        const int32_t k0 = prefill ? key0[ii] : -1;
        const int32_t pos_lo = it.row0 / g, pos_hi = (it.row0 + it.nrows - 1) / g;
        for (int32_t pos = pos_lo; pos <= pos_hi; ++pos) {
            if (k0 > pos) continue;
            const int32_t b = p->dfs_leaf[it.leaf_lo + pos];
            ent[static_cast<size_t>(b) * H_kv + it.kv_head].push_back(it.slot_base + pos * g -
                                                                       it.row0);
        }
    }
    p->merge_rng.assign(static_cast<size_t>(L_rows) * H_kv, make_int2(0, 0));
    p->merge_ent.clear();
    for (size_t k = 0; k < ent.size(); ++k) {
        const int32_t e0 = static_cast<int32_t>(p->merge_ent.size());
        p->merge_ent.insert(p->merge_ent.end(), ent[k].begin(), ent[k].end());
        if (p->merge_ent.size() > static_cast<size_t>(INT32_MAX)) return PARASON_EUNSUPPORTED;
        p->merge_rng[k] = make_int2(e0, static_cast<int32_t>(p->merge_ent.size()));
    }
    for (int32_t b = 0; b < num_leaves && !prefill; ++b)
        for (int32_t n = leaf_node[b]; n >= 0; n = parent[n]) p->path_tokens += node_len[n];

    // room for forks: about as much again as the plan holds, with floors
    // that let a small plan take a few forks
    p->cap_items = p->items.size() + std::max<size_t>(4096, p->items.size());
    p->cap_rows = p->stream_rows.size() + std::max<size_t>(65536, p->stream_rows.size());
    p->cap_leaves = static_cast<size_t>(p->num_leaves) + std::max<size_t>(64, p->num_leaves);
    p->cap_ent = p->merge_ent.size() + std::max<size_t>(16384, p->merge_ent.size());
    // an append patches 6 words per tail item (at most H_kv per branch); a
    // fork one branch's merge ranges and the queue counters
    p->cap_patch = p->cap_leaves * H_kv * kPatchesPerTail + 2 * static_cast<size_t>(H_kv) + 2;
    return PARASON_OK;
}

// ---------------------------------------------------------------------------
// device side
// ---------------------------------------------------------------------------

parason_status upload(parason_plan_s *p, cudaStream_t stream) {
    if (cudaGetDevice(&p->device) != cudaSuccess) return PARASON_ECUDA;
    const int32_t H = p->cfg.num_kv_heads;
    // the arrays forks grow are allocated at their capacity
    const size_t n_items = p->cap_items * sizeof(WorkItem);
    const size_t n_pages = p->page_ids.size() * sizeof(int32_t);
    const size_t n_dfs = p->cap_leaves * sizeof(int32_t);
    const size_t n_mrng = p->cap_leaves * H * sizeof(int2);
    const size_t n_ment = p->cap_ent * sizeof(int32_t);
    const size_t n_rec = p->cap_items * parason::kRecWords * sizeof(int32_t);
    const size_t n_irows = (p->cap_items + 1) * sizeof(int32_t);
    // page rows are read 32 entries past their end by whole warps: pad
    const size_t n_strows = (p->cap_rows + 32) * sizeof(int32_t);
    const size_t n_qnext = 2 * sizeof(int32_t);
    const size_t n_err = parason::kErrWords * sizeof(int32_t);
    const size_t n_patch = p->cap_patch * sizeof(int2);
    const size_t n_key0 = p->item_key0.size() * sizeof(int32_t);
    constexpr int kArrays = 12;
    size_t off[kArrays], total = 0;
    // the queue counters and the error record are set separately; the patch
    // buffer is written by parason_plan_append and parason_plan_fork
    const size_t sizes[kArrays] = {n_items, n_pages,  n_dfs,   n_mrng, n_ment,  n_rec,
                                   n_irows, n_strows, n_qnext, n_err,  n_patch, n_key0};
    for (int i = 0; i < kArrays; ++i) {
        off[i] = total;
        total = align_up(total + std::max<size_t>(sizes[i], 4), kAlign);
    }
    if (cudaMalloc(&p->d_blob, total) != cudaSuccess) {
        cudaGetLastError();
        p->d_blob = nullptr;
        return PARASON_ENOMEM;
    }
    char *base = static_cast<char *>(p->d_blob);
    p->d_items = reinterpret_cast<WorkItem *>(base + off[0]);
    p->d_page_ids = reinterpret_cast<int32_t *>(base + off[1]);
    p->d_dfs_leaf = reinterpret_cast<int32_t *>(base + off[2]);
    p->d_merge_rng = reinterpret_cast<int2 *>(base + off[3]);
    p->d_merge_ent = reinterpret_cast<int32_t *>(base + off[4]);
    p->d_item_rec = reinterpret_cast<int32_t *>(base + off[5]);
    p->d_item_rows = reinterpret_cast<int32_t *>(base + off[6]);
    p->d_stream_rows = reinterpret_cast<int32_t *>(base + off[7]);
    p->d_queue_next = reinterpret_cast<int32_t *>(base + off[8]);
    p->d_err = reinterpret_cast<int32_t *>(base + off[9]);
    p->d_patch = reinterpret_cast<int2 *>(base + off[10]);
    p->d_item_key0 = p->prefill ? reinterpret_cast<int32_t *>(base + off[11]) : nullptr;
    p->w_items = off[0] / sizeof(int32_t);
    p->w_mrng = off[3] / sizeof(int32_t);
    p->w_rec = off[5] / sizeof(int32_t);
    p->w_strows = off[7] / sizeof(int32_t);
    p->w_qnext = off[8] / sizeof(int32_t);
    p->blob_words = total / sizeof(int32_t);
    const void *src[8] = {p->items.data(),     p->page_ids.data(),  p->dfs_leaf.data(),
                          p->merge_rng.data(), p->merge_ent.data(), p->item_rec.data(),
                          p->item_rows.data(), p->stream_rows.data()};
    const size_t copy[8] = {p->items.size() * sizeof(WorkItem), n_pages,
                            p->dfs_leaf.size() * sizeof(int32_t), p->merge_rng.size() * sizeof(int2),
                            p->merge_ent.size() * sizeof(int32_t), p->item_rec.size() * sizeof(int32_t),
                            p->item_rows.size() * sizeof(int32_t),
                            p->stream_rows.size() * sizeof(int32_t)};
    for (int i = 0; i < 8; ++i) {
        if (copy[i] == 0) continue;
        if (cudaMemcpyAsync(base + off[i], src[i], copy[i], cudaMemcpyHostToDevice, stream) !=
            cudaSuccess)
            return PARASON_ECUDA;
    }
    if (n_key0 > 0 && cudaMemcpyAsync(base + off[11], p->item_key0.data(), n_key0,
                                      cudaMemcpyHostToDevice, stream) != cudaSuccess)
        return PARASON_ECUDA;
    if (cudaMemsetAsync(p->d_err, 0, n_err, stream) != cudaSuccess) return PARASON_ECUDA;
    if (cudaMemcpyAsync(p->d_queue_next, p->queue_start, n_qnext, cudaMemcpyHostToDevice, stream) !=
        cudaSuccess)
        return PARASON_ECUDA;
    // the host vectors are pageable: make sure the copies have consumed them
    // before the caller can free its own arrays (ours stay alive anyway)
    if (cudaStreamSynchronize(stream) != cudaSuccess) return PARASON_ECUDA;
    p->on_device = true;
    return PARASON_OK;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    return fn;
}

// KV pool [P, H_kv, 16, d] seen as rows of 128-byte segments:
//   dim0 = 128 bytes of one segment (64 bf16 or 128 e4m3), dim1 = segment in
//   the token row, dim2 = token row (page * H_kv + kv_head) * 16 + slot.
// One box {seg, 1, 16} is one 128-byte column block of one page of one kv
// head (16 rows of 128 bytes, 128-byte swizzle).
parason_status encode_kv_map(CUtensorMap *map, const void *pages, int64_t num_phys,
                             int32_t H_kv, int32_t head_dim, int32_t mode) {
    auto fn = encode_fn();
    if (!fn) return PARASON_ECUDA;
    const int esize = (mode == PARASON_FP8_E4M3_KV) ? 1 : 2;
    const CUtensorMapDataType dt =
        (mode == PARASON_FP8_E4M3_KV) ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const int row_bytes = head_dim * esize;
    if (row_bytes % 128 != 0) return PARASON_EUNSUPPORTED;
    const int nseg = row_bytes / 128;
    const int seg_elems = 128 / esize;
    const cuuint64_t rows = static_cast<cuuint64_t>(num_phys) * H_kv * parason::kPageSize;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(seg_elems), static_cast<cuuint64_t>(nseg), rows};
    cuuint64_t strides[2] = {128, static_cast<cuuint64_t>(row_bytes)};
    cuuint32_t box[3] = {static_cast<cuuint32_t>(seg_elems), 1u,
                         static_cast<cuuint32_t>(parason::kPageSize)};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, dt, 3, const_cast<void *>(pages), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? PARASON_OK : PARASON_ECUDA;
}

// The same pool as a 5-D view: dim0 = 128 bytes of one segment, dim1 =
// segment, dim2 = slot in the page (16), dim3 = kv head, dim4 = page.  One
// box {seg, 1, 16, 1, kTcRunPages} is one 128-byte column block of
// kTcRunPages consecutive pages of one kv head: 16 kTcRunPages rows of 128
// bytes, laid out as the per-page boxes of those pages would be.
parason_status encode_kv_run_map(CUtensorMap *map, const void *pages, int64_t num_phys,
                                 int32_t H_kv, int32_t head_dim, int32_t mode) {
    auto fn = encode_fn();
    if (!fn) return PARASON_ECUDA;
    const int esize = (mode == PARASON_FP8_E4M3_KV) ? 1 : 2;
    const CUtensorMapDataType dt =
        (mode == PARASON_FP8_E4M3_KV) ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const int row_bytes = head_dim * esize;
    if (row_bytes % 128 != 0) return PARASON_EUNSUPPORTED;
    const int nseg = row_bytes / 128;
    const int seg_elems = 128 / esize;
    const cuuint64_t page_head_bytes = static_cast<cuuint64_t>(parason::kPageSize) * row_bytes;
    cuuint64_t dims[5] = {static_cast<cuuint64_t>(seg_elems), static_cast<cuuint64_t>(nseg),
                          static_cast<cuuint64_t>(parason::kPageSize), static_cast<cuuint64_t>(H_kv),
                          static_cast<cuuint64_t>(num_phys)};
    cuuint64_t strides[4] = {128, static_cast<cuuint64_t>(row_bytes), page_head_bytes,
                             page_head_bytes * static_cast<cuuint64_t>(H_kv)};
    cuuint32_t box[5] = {static_cast<cuuint32_t>(seg_elems), 1u,
                         static_cast<cuuint32_t>(parason::kPageSize), 1u,
                         static_cast<cuuint32_t>(parason::kTcRunPages)};
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    CUresult r = fn(map, dt, 5, const_cast<void *>(pages), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? PARASON_OK : PARASON_ECUDA;
}

// The same pool as a 4-D view whose dims are not in stride order: dim0 = 128
// bytes of one segment, dim1 = slot in the page (16, stride one token row),
// dim2 = segment (stride 128 bytes), dim3 = (page * H_kv + kv_head).  One box
// {seg, 16, nseg, 1} is a whole page of one kv head with its column blocks
// one after another, each 16 rows of 128 bytes (128-byte swizzle): what nseg
// boxes of the 3-D view give, in one copy.
parason_status encode_kv_page_map(CUtensorMap *map, const void *pages, int64_t num_phys,
                                  int32_t H_kv, int32_t head_dim, int32_t mode) {
    auto fn = encode_fn();
    if (!fn) return PARASON_ECUDA;
    const int esize = (mode == PARASON_FP8_E4M3_KV) ? 1 : 2;
    const CUtensorMapDataType dt =
        (mode == PARASON_FP8_E4M3_KV) ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const int row_bytes = head_dim * esize;
    if (row_bytes % 128 != 0) return PARASON_EUNSUPPORTED;
    const int nseg = row_bytes / 128;
    const int seg_elems = 128 / esize;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(seg_elems), static_cast<cuuint64_t>(parason::kPageSize),
                          static_cast<cuuint64_t>(nseg), static_cast<cuuint64_t>(num_phys) * H_kv};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(row_bytes), 128,
                             static_cast<cuuint64_t>(parason::kPageSize) * row_bytes};
    cuuint32_t box[4] = {static_cast<cuuint32_t>(seg_elems), static_cast<cuuint32_t>(parason::kPageSize),
                         static_cast<cuuint32_t>(nseg), 1u};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = fn(map, dt, 4, const_cast<void *>(pages), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? PARASON_OK : PARASON_ECUDA;
}

parason_status record_event(parason_plan_s *p, int which, cudaStream_t stream) {
    if (p->timing_cap <= 0 || p->timing_n >= p->timing_cap) return PARASON_OK;
    cudaEvent_t ev = p->events[3 * p->timing_n + which];
    return cudaEventRecord(ev, stream) == cudaSuccess ? PARASON_OK : PARASON_ECUDA;
}

void free_events(parason_plan_s *p) {
    for (auto e : p->events)
        if (e) cudaEventDestroy(e);
    p->events.clear();
    p->timing_cap = p->timing_n = 0;
}

parason_status plan_host(const parason_attn_config *cfg, int32_t num_nodes, const int32_t *parent,
                         const int32_t *node_len, const int32_t *node_page_ptr,
                         const int32_t *page_ids, int32_t num_leaves, const int32_t *leaf_node,
                         int64_t num_physical_pages, int32_t num_sms, bool prefill,
                         parason_plan *out) {
    if (!out) return PARASON_EINVAL;
    *out = nullptr;
    auto *p = new (std::nothrow) parason_plan_s();
    if (!p) return PARASON_ENOMEM;
    parason_status st;
    try {
        st = build_host(p, cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves,
                        leaf_node, num_physical_pages, num_sms, prefill);
    } catch (const std::bad_alloc &) {
        st = PARASON_ENOMEM;
    }
    if (st != PARASON_OK) {
        delete p;
        return st;
    }
    *out = p;
    return PARASON_OK;
}

parason_status plan_device(const parason_attn_config *cfg, int32_t num_nodes, const int32_t *parent,
                           const int32_t *node_len, const int32_t *node_page_ptr,
                           const int32_t *page_ids, int32_t num_leaves, const int32_t *leaf_node,
                           int64_t num_physical_pages, bool prefill, parason_stream_t stream,
                           parason_plan *out) {
    if (!out) return PARASON_EINVAL;
    *out = nullptr;
    // validate before touching CUDA, so malformed input is EINVAL everywhere
    parason_status st = validate_config(cfg);
    if (st != PARASON_OK) return st;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        // still report malformed trees as EINVAL on machines without a GPU
        parason_plan probe = nullptr;
        st = plan_host(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves,
                       leaf_node, num_physical_pages, 152, prefill, &probe);
        parason_plan_destroy(probe);
        cudaGetLastError();
        return st != PARASON_OK ? st : PARASON_ECUDA;
    }
    if (cfg->mode != PARASON_FP32) {
        int ctas_per_sm = 0;
        const cudaError_t e = parason::attn_mma_ctas_per_sm(cfg->head_dim, cfg->mode, &ctas_per_sm);
        if (e == cudaErrorNotSupported) return PARASON_EUNSUPPORTED;
        if (e != cudaSuccess) return PARASON_ECUDA;
        if (ctas_per_sm < 1) return PARASON_EUNSUPPORTED;
    }
    parason_plan p = nullptr;
    st = plan_host(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves, leaf_node,
                   num_physical_pages, sms, prefill, &p);
    if (st != PARASON_OK) return st;
    st = upload(p, reinterpret_cast<cudaStream_t>(stream));
    if (st != PARASON_OK) {
        parason_plan_destroy(p);
        return st;
    }
    *out = p;
    return PARASON_OK;
}

// ---------------------------------------------------------------------------
// sharding (one plan per rank, no exchange between ranks)
// ---------------------------------------------------------------------------

// The sub-forest of the requests (roots) of one rank, in the form build_host
// takes, with the global index of each of its branches.
struct SubForest {
    std::vector<int32_t> parent, len, ptr, pages, leaves, global_branch;
};

// Roots in index order are cut into `world` contiguous groups of about equal
// cost: a request's cost is the tokens of its nodes that some branch reads
// (the KV bytes its decode step moves, each shared node once) plus g per
// branch (its q and out rows, in the same units).  Rank `rank` gets group
// `rank`; a rank may get no request when there are fewer requests than ranks.
void shard_requests(int32_t num_nodes, const int32_t *parent, const int32_t *node_len,
                    const int32_t *node_page_ptr, const int32_t *page_ids, int32_t num_leaves,
                    const int32_t *leaf_node, int32_t g, int32_t rank, int32_t world,
                    SubForest *out) {
    std::vector<int32_t> root(num_nodes), root_idx(num_nodes, -1);
    std::vector<int64_t> cnt(num_nodes, 0);
    int32_t num_roots = 0;
    for (int32_t i = 0; i < num_nodes; ++i) {
        root[i] = parent[i] < 0 ? i : root[parent[i]];
        if (parent[i] < 0) root_idx[i] = num_roots++;
    }
    for (int32_t b = 0; b < num_leaves; ++b) cnt[leaf_node[b]] = 1;
    for (int32_t i = num_nodes - 1; i >= 0; --i)
        if (parent[i] >= 0) cnt[parent[i]] += cnt[i];
    std::vector<int64_t> cost(num_roots, 0);
    for (int32_t i = 0; i < num_nodes; ++i)
        if (cnt[i] > 0) cost[root_idx[root[i]]] += node_len[i];
    for (int32_t b = 0; b < num_leaves; ++b) cost[root_idx[root[leaf_node[b]]]] += g;
    std::vector<int64_t> prefix(num_roots + 1, 0);
    for (int32_t r = 0; r < num_roots; ++r) prefix[r + 1] = prefix[r] + cost[r];
    // boundary k: the prefix closest to k/world of the total, never moving back
    auto boundary = [&](int32_t k) -> int32_t {
        if (k <= 0) return 0;
        if (k >= world) return num_roots;
        const double target = static_cast<double>(prefix[num_roots]) * k / world;
        int32_t j = static_cast<int32_t>(std::lower_bound(prefix.begin(), prefix.end(),
                                                          static_cast<int64_t>(std::ceil(target))) -
                                         prefix.begin());
        j = std::min(j, num_roots);
        if (j > 0 && target - static_cast<double>(prefix[j - 1]) <
                         static_cast<double>(prefix[j]) - target)
            --j;
        return j;
    };
    int32_t lo = 0, hi = 0;
    for (int32_t k = 0; k <= rank; ++k) {
        lo = std::max(lo, boundary(k));
        hi = std::max(lo, boundary(k + 1));
    }
    std::vector<int32_t> remap(num_nodes, -1);
    out->ptr.assign(1, 0);
    for (int32_t i = 0; i < num_nodes; ++i) {
        const int32_t ri = root_idx[root[i]];
        if (ri < lo || ri >= hi) continue;
        remap[i] = static_cast<int32_t>(out->parent.size());
        out->parent.push_back(parent[i] < 0 ? -1 : remap[parent[i]]);
        out->len.push_back(node_len[i]);
        for (int32_t k = node_page_ptr[i]; k < node_page_ptr[i + 1]; ++k) out->pages.push_back(page_ids[k]);
        out->ptr.push_back(static_cast<int32_t>(out->pages.size()));
    }
    for (int32_t b = 0; b < num_leaves; ++b) {
        if (remap[leaf_node[b]] < 0) continue;
        out->leaves.push_back(remap[leaf_node[b]]);
        out->global_branch.push_back(b);
    }
}

parason_status plan_shard(const parason_attn_config *cfg, int32_t num_nodes, const int32_t *parent,
                          const int32_t *node_len, const int32_t *node_page_ptr,
                          const int32_t *page_ids, int32_t num_leaves, const int32_t *leaf_node,
                          int64_t num_phys, int32_t kind, int32_t rank, int32_t world,
                          bool host_only, int32_t num_sms, parason_stream_t stream,
                          parason_plan *out) {
    if (!out) return PARASON_EINVAL;
    *out = nullptr;
    parason_status st = validate_config(cfg);
    if (st != PARASON_OK) return st;
    if (world < 1 || rank < 0 || rank >= world) return PARASON_EINVAL;
    st = validate_tree(num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves, leaf_node,
                       num_phys, cfg->num_kv_heads);
    if (st != PARASON_OK) return st;
    parason_plan p = nullptr;
    if (kind == PARASON_SHARD_KV_HEADS) {
        // kv heads [rank H_kv / world, (rank + 1) H_kv / world) and their q heads
        if (cfg->num_kv_heads % world != 0) return PARASON_EINVAL;
        parason_attn_config c = *cfg;
        c.num_kv_heads = cfg->num_kv_heads / world;
        c.num_q_heads = cfg->num_q_heads / world;
        st = host_only ? plan_host(&c, num_nodes, parent, node_len, node_page_ptr, page_ids,
                                   num_leaves, leaf_node, num_phys, num_sms, false, &p)
                       : plan_device(&c, num_nodes, parent, node_len, node_page_ptr, page_ids,
                                     num_leaves, leaf_node, num_phys, false, stream, &p);
        if (st != PARASON_OK) return st;
        p->shard_branch.resize(static_cast<size_t>(num_leaves));
        for (int32_t b = 0; b < num_leaves; ++b) p->shard_branch[b] = b;
    } else if (kind == PARASON_SHARD_REQUESTS) {
        SubForest f;
        try {
            shard_requests(num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves,
                           leaf_node, cfg->num_q_heads / cfg->num_kv_heads, rank, world, &f);
        } catch (const std::bad_alloc &) {
            return PARASON_ENOMEM;
        }
        const int32_t n = static_cast<int32_t>(f.parent.size());
        const int32_t l = static_cast<int32_t>(f.leaves.size());
        st = host_only ? plan_host(cfg, n, f.parent.data(), f.len.data(), f.ptr.data(),
                                   f.pages.data(), l, f.leaves.data(), num_phys, num_sms, false, &p)
                       : plan_device(cfg, n, f.parent.data(), f.len.data(), f.ptr.data(),
                                     f.pages.data(), l, f.leaves.data(), num_phys, false, stream, &p);
        if (st != PARASON_OK) return st;
        p->shard_branch.swap(f.global_branch);
    } else {
        return PARASON_EINVAL;
    }
    *out = p;
    return PARASON_OK;
}

}  // namespace

int parason::plan_device(parason_plan p) { return (p && p->on_device) ? p->device : -1; }

extern "C" {

parason_status parason_attn_plan_host(const parason_attn_config *cfg, int32_t num_nodes,
                                      const int32_t *parent, const int32_t *node_len,
                                      const int32_t *node_page_ptr, const int32_t *page_ids,
                                      int32_t num_leaves, const int32_t *leaf_node,
                                      int64_t num_physical_pages, int32_t num_sms,
                                      parason_plan *out) {
    return plan_host(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves,
                     leaf_node, num_physical_pages, num_sms, false, out);
}

parason_status parason_attn_plan(const parason_attn_config *cfg, int32_t num_nodes,
                                 const int32_t *parent, const int32_t *node_len,
                                 const int32_t *node_page_ptr, const int32_t *page_ids,
                                 int32_t num_leaves, const int32_t *leaf_node,
                                 int64_t num_physical_pages, parason_stream_t stream,
                                 parason_plan *out) {
    return plan_device(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves,
                       leaf_node, num_physical_pages, false, stream, out);
}

parason_status parason_prefill_plan_host(const parason_attn_config *cfg, int32_t num_nodes,
                                         const int32_t *parent, const int32_t *node_len,
                                         const int32_t *node_page_ptr, const int32_t *page_ids,
                                         int32_t num_chunks, const int32_t *chunk_node,
                                         int64_t num_physical_pages, int32_t num_sms,
                                         parason_plan *out) {
    return plan_host(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_chunks,
                     chunk_node, num_physical_pages, num_sms, true, out);
}

parason_status parason_prefill_plan(const parason_attn_config *cfg, int32_t num_nodes,
                                    const int32_t *parent, const int32_t *node_len,
                                    const int32_t *node_page_ptr, const int32_t *page_ids,
                                    int32_t num_chunks, const int32_t *chunk_node,
                                    int64_t num_physical_pages, parason_stream_t stream,
                                    parason_plan *out) {
    return plan_device(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_chunks,
                       chunk_node, num_physical_pages, true, stream, out);
}

parason_status parason_attn_plan_shard(const parason_attn_config *cfg, int32_t num_nodes,
                                       const int32_t *parent, const int32_t *node_len,
                                       const int32_t *node_page_ptr, const int32_t *page_ids,
                                       int32_t num_leaves, const int32_t *leaf_node,
                                       int64_t num_physical_pages, int32_t kind, int32_t rank,
                                       int32_t world, parason_stream_t stream, parason_plan *out) {
    return plan_shard(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves,
                      leaf_node, num_physical_pages, kind, rank, world, false, 0, stream, out);
}

parason_status parason_attn_plan_shard_host(const parason_attn_config *cfg, int32_t num_nodes,
                                            const int32_t *parent, const int32_t *node_len,
                                            const int32_t *node_page_ptr, const int32_t *page_ids,
                                            int32_t num_leaves, const int32_t *leaf_node,
                                            int64_t num_physical_pages, int32_t kind, int32_t rank,
                                            int32_t world, int32_t num_sms, parason_plan *out) {
    return plan_shard(cfg, num_nodes, parent, node_len, node_page_ptr, page_ids, num_leaves,
                      leaf_node, num_physical_pages, kind, rank, world, true, num_sms, nullptr, out);
}

size_t parason_plan_workspace_bytes(parason_plan p) {
    if (!p) return 0;
    const size_t o = align_up(static_cast<size_t>(p->num_slots) * p->cfg.head_dim * sizeof(float), kAlign);
    const size_t ml = align_up(static_cast<size_t>(p->num_slots) * sizeof(float2), kAlign);
    return o + ml;
}

parason_status parason_attn_decode(parason_plan p, const void *q, const void *k_pages,
                                   const void *v_pages, const float *k_scale,
                                   const float *v_scale, void *out, float *lse,
                                   void *workspace, size_t workspace_bytes,
                                   parason_stream_t stream_) {
    if (!p || !p->on_device) return PARASON_EINVAL;
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    if (p->num_leaves == 0) return PARASON_OK;
    if (!q || !out) return PARASON_EINVAL;
    const bool has_items = !p->items.empty();
    if (has_items) {
        if (!k_pages || !v_pages || !workspace) return PARASON_EINVAL;
        if (workspace_bytes < parason_plan_workspace_bytes(p)) return PARASON_EINVAL;
        if (reinterpret_cast<uintptr_t>(workspace) % kAlign) return PARASON_EINVAL;
        if (reinterpret_cast<uintptr_t>(k_pages) % 16 || reinterpret_cast<uintptr_t>(v_pages) % 16)
            return PARASON_EINVAL;
        if (p->cfg.mode == PARASON_FP8_E4M3_KV && (!k_scale || !v_scale)) return PARASON_EINVAL;
    }
    if (reinterpret_cast<uintptr_t>(q) % 16 || reinterpret_cast<uintptr_t>(out) % 16)
        return PARASON_EINVAL;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return PARASON_ECUDA;
    if (dev != p->device) return PARASON_EINVAL;

    const int d = p->cfg.head_dim;
    float *part_o = static_cast<float *>(workspace);
    float2 *part_ml = reinterpret_cast<float2 *>(
        static_cast<char *>(workspace) +
        align_up(static_cast<size_t>(p->num_slots) * d * sizeof(float), kAlign));
    const float sm_scale = p->cfg.sm_scale > 0.0f ? p->cfg.sm_scale : 1.0f / std::sqrt(static_cast<float>(d));

    parason_status st = record_event(p, 0, stream);
    if (st != PARASON_OK) return st;
    if (has_items) {
        parason::AttnArgs a{};
        a.items = p->d_items;
        a.page_ids = p->d_page_ids;
        a.dfs_leaf = p->d_dfs_leaf;
        a.q = q;
        a.part_o = part_o;
        a.part_ml = part_ml;
        a.k_scale = k_scale;
        a.v_scale = v_scale;
        a.err = p->d_err;
        a.wait_limit_ns = p->wait_limit_ns;
        a.debug_flags = p->debug_flags;
        a.num_items = static_cast<int32_t>(p->items.size());
        a.num_q_heads = p->cfg.num_q_heads;
        a.num_kv_heads = p->cfg.num_kv_heads;
        a.group = p->group;
        a.scale_log2 = sm_scale * 1.4426950408889634f;
        a.item_rec = p->d_item_rec;
        a.num_wide_items = static_cast<int32_t>(p->wide_queue.size());
        a.num_narrow_items = static_cast<int32_t>(p->narrow_queue.size());
        a.item_rows = p->d_item_rows;
        a.stream_rows = p->d_stream_rows;
        a.queue_next = p->d_queue_next;
        a.num_ctas = p->num_ctas;
        a.num_wide_ctas = p->num_wide_ctas;
        a.kv_rows = static_cast<int32_t>(p->num_phys * p->cfg.num_kv_heads * parason::kPageSize);
        a.item_key0 = p->d_item_key0;
        a.suffix_warps = p->suffix_warps;
        a.tc_pairs = p->tc_pairs ? 1 : 0;
        cudaError_t e;
        if (p->cfg.mode == PARASON_FP32) {
            e = parason::launch_attn_fp32(a, static_cast<const float *>(k_pages),
                                          static_cast<const float *>(v_pages), d, stream);
        } else {
            parason::KvMaps maps;
            {
                std::lock_guard<std::mutex> lock(p->tm_mutex);
                const int32_t H = p->cfg.num_kv_heads, mode = p->cfg.mode;
                if (p->tm_k_ptr != k_pages) {
                    p->tm_k_ptr = nullptr;
                    st = encode_kv_map(&p->tm.k, k_pages, p->num_phys, H, d, mode);
                    if (st == PARASON_OK)
                        st = encode_kv_run_map(&p->tm.k_run, k_pages, p->num_phys, H, d, mode);
                    if (st == PARASON_OK)
                        st = encode_kv_page_map(&p->tm.k_page, k_pages, p->num_phys, H, d, mode);
                    if (st != PARASON_OK) return st;
                    p->tm_k_ptr = k_pages;
                }
                if (p->tm_v_ptr != v_pages) {
                    p->tm_v_ptr = nullptr;
                    st = encode_kv_map(&p->tm.v, v_pages, p->num_phys, H, d, mode);
                    if (st == PARASON_OK)
                        st = encode_kv_run_map(&p->tm.v_run, v_pages, p->num_phys, H, d, mode);
                    if (st == PARASON_OK)
                        st = encode_kv_page_map(&p->tm.v_page, v_pages, p->num_phys, H, d, mode);
                    if (st != PARASON_OK) return st;
                    p->tm_v_ptr = v_pages;
                }
                maps = p->tm;
            }
            e = (p->cfg.mode == PARASON_BF16) ? parason::launch_attn_bf16(a, maps, d, stream)
                                              : parason::launch_attn_fp8(a, maps, d, stream);
        }
        if (e == cudaErrorNotSupported) return PARASON_EUNSUPPORTED;
        if (e != cudaSuccess) return PARASON_ECUDA;
    }
    st = record_event(p, 1, stream);
    if (st != PARASON_OK) return st;
    parason::MergeArgs m{};
    m.merge_rng = p->d_merge_rng;
    m.merge_ent = p->d_merge_ent;
    m.part_o = part_o;
    m.part_ml = part_ml;
    m.out = out;
    m.lse = lse;
    m.num_leaves = p->num_leaves;
    m.num_q_heads = p->cfg.num_q_heads;
    m.group = p->group;
    m.num_kv_heads = p->cfg.num_kv_heads;
    m.queue_next = p->d_queue_next;
    m.queue_start[0] = p->queue_start[0];
    m.queue_start[1] = p->queue_start[1];
    // programmatic dependent launch after the persistent kernel: the merge
    // grid is launched while the attention grid drains, and waits for it
    const bool pdl = has_items && p->cfg.mode != PARASON_FP32;
    if (parason::launch_merge(m, d, p->cfg.mode, pdl, stream) != cudaSuccess) return PARASON_ECUDA;
    st = record_event(p, 2, stream);
    if (st != PARASON_OK) return st;
    if (p->timing_cap > 0 && p->timing_n < p->timing_cap) p->timing_n++;
    return PARASON_OK;
}

parason_status parason_lse_merge(const void *o_a, const float *lse_a, const void *o_b,
                                 const float *lse_b, void *o_out, float *lse_out, int64_t rows,
                                 int32_t head_dim, int32_t mode, parason_stream_t stream) {
    if (rows < 0 || (head_dim != 64 && head_dim != 128)) return PARASON_EINVAL;
    if (mode != PARASON_BF16 && mode != PARASON_FP32 && mode != PARASON_FP8_E4M3_KV)
        return PARASON_EINVAL;
    if (rows == 0) return PARASON_OK;
    if (!o_a || !lse_a || !o_b || !lse_b || !o_out || !lse_out) return PARASON_EINVAL;
    const uintptr_t mis = reinterpret_cast<uintptr_t>(o_a) | reinterpret_cast<uintptr_t>(o_b) |
                          reinterpret_cast<uintptr_t>(o_out);
    if (mis % 16) return PARASON_EINVAL;
    cudaError_t e = parason::launch_lse_merge(o_a, lse_a, o_b, lse_b, o_out, lse_out, rows, head_dim,
                                              mode, reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? PARASON_OK : PARASON_ECUDA;
}

parason_status parason_plan_check(parason_plan p, parason_stream_t stream) {
    if (!p || !p->on_device) return PARASON_EINVAL;
    if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return PARASON_ECUDA;
    int32_t rec[parason::kErrWords] = {0, 0, 0, 0};
    if (cudaMemcpy(rec, p->d_err, sizeof rec, cudaMemcpyDeviceToHost) != cudaSuccess)
        return PARASON_ECUDA;
    if (rec[0] != 0) {
        if (cudaMemset(p->d_err, 0, sizeof rec) != cudaSuccess) return PARASON_ECUDA;
        if (cudaMemcpy(p->d_queue_next, p->queue_start, 2 * sizeof(int32_t), cudaMemcpyHostToDevice) !=
            cudaSuccess)
            return PARASON_ECUDA;
        if (rec[0] == PARASON_ETIMEOUT || rec[0] == PARASON_ERANGE)
            return static_cast<parason_status>(rec[0]);
        return PARASON_ECUDA;
    }
    return PARASON_OK;
}

void parason_plan_destroy(parason_plan p) {
    if (!p) return;
    free_events(p);
    if (p->d_blob) cudaFree(p->d_blob);
    delete p;
}

const char *parason_status_string(parason_status s) {
    switch (s) {
    case PARASON_OK: return "ok";
    case PARASON_EINVAL: return "invalid argument";
    case PARASON_ENOMEM: return "out of memory";
    case PARASON_ECUDA: return "CUDA error";
    case PARASON_ETIMEOUT: return "device wait timed out";
    case PARASON_EUNSUPPORTED: return "unsupported";
    case PARASON_ENOSPACE: return "no room in the plan: build a new one";
    case PARASON_ERANGE: return "input value out of the kernel's range";
    }
    return "unknown status";
}

parason_status parason_plan_get_info(parason_plan p, parason_plan_info *info) {
    if (!p || !info) return PARASON_EINVAL;
    info->num_items = static_cast<int32_t>(p->items.size());
    info->num_leaves = p->num_leaves;
    info->num_merge_entries = static_cast<int32_t>(p->merge_ent.size());
    info->chunk_pages = p->chunk_pages;
    info->num_slots = p->num_slots;
    info->unique_tokens = p->unique_tokens;
    info->path_tokens = p->path_tokens;
    info->num_sms = p->num_sms;
    info->on_device = p->on_device ? 1 : 0;
    info->num_ctas = p->num_ctas;
    info->num_wide_ctas = p->num_wide_ctas;
    info->num_wide_items = static_cast<int32_t>(p->wide_queue.size());
    info->num_narrow_items = static_cast<int32_t>(p->narrow_queue.size());
    info->num_stream_rows = static_cast<int64_t>(p->stream_rows.size());
    info->tile_pairs = p->tc_pairs ? 1 : 0;
    return PARASON_OK;
}

parason_status parason_plan_append(parason_plan p, const int32_t *new_pages,
                                   parason_stream_t stream_) {
    if (!p) return PARASON_EINVAL;
    if (p->cfg.mode == PARASON_FP32 || p->prefill) return PARASON_EUNSUPPORTED;
    const int32_t L = p->num_leaves;
    if (L == 0) return PARASON_OK;
    if (p->on_device && p->blob_words > static_cast<size_t>(INT32_MAX)) return PARASON_EUNSUPPORTED;
    const int32_t H_kv = p->cfg.num_kv_heads;
    constexpr int32_t P16 = parason::kPageSize;

    // 1. check everything: on any error nothing changes
    std::vector<int32_t> claimed;
    auto refuse = [&](parason_status st) {
        for (int32_t pg : claimed) p->page_used[pg] = 0;
        return st;
    };
    if (p->on_device) {
        int dev = -1;
        if (cudaGetDevice(&dev) != cudaSuccess) {
            cudaGetLastError();
            return PARASON_ECUDA;
        }
        if (dev != p->device) return PARASON_EINVAL;
    }
    for (int32_t b = 0; b < L; ++b) {
        const int32_t len = p->tree_len[p->leaf_node[b]];
        if (p->tails[b].empty()) return refuse(PARASON_ENOSPACE);
        if (len == INT32_MAX) return refuse(PARASON_EUNSUPPORTED);
        if (len % P16 != 0) continue;
        if (!new_pages) return refuse(PARASON_EINVAL);
        const int32_t pg = new_pages[b];
        if (pg < 0 || pg >= p->num_phys || p->page_used[pg]) return refuse(PARASON_EINVAL);
        for (const int32_t t : p->tails[b]) {
            if (p->item_rows[t] + p->items[t].num_pages + 1 > p->item_rows[t + 1])
                return refuse(PARASON_ENOSPACE);
            if (p->items[t].num_pages == INT32_MAX) return refuse(PARASON_EUNSUPPORTED);
            // a prefix-pass item stays within what the tile's metadata holds
            if (t < static_cast<int32_t>(p->wide_queue.size()) &&
                p->items[t].num_pages + 1 > kMaxTileItemPages)
                return refuse(PARASON_ENOSPACE);
        }
        p->page_used[pg] = 1;
        claimed.push_back(pg);
    }

    // 2. the new values, without touching the plan yet: host words to write
    // and the device patch list (word offset in the device blob, value).
    // Each tail item belongs to one branch, so no word is written twice.
    std::vector<std::pair<int32_t *, int32_t>> host;
    std::vector<int2> &patches = p->patches;
    patches.clear();
    for (int32_t b = 0; b < L; ++b) {
        const bool opens_page = p->tree_len[p->leaf_node[b]] % P16 == 0;
        for (const int32_t t : p->tails[b]) {
            WorkItem &it = p->items[t];
            int32_t *rec = p->item_rec.data() + static_cast<size_t>(t) * parason::kRecWords;
            const size_t w_item = p->w_items + static_cast<size_t>(t) * (sizeof(WorkItem) / 4);
            const size_t w_rec = p->w_rec + static_cast<size_t>(t) * parason::kRecWords;
            int32_t last_valid = it.last_valid + 1;
            if (opens_page) {
                const int32_t j = it.num_pages;                   // the new page's index
                const int32_t row = (new_pages[b] * H_kv + it.kv_head) * P16;
                const int32_t np = it.num_pages + 1;
                last_valid = 1;
                host.emplace_back(&p->stream_rows[p->item_rows[t] + j], row);
                patches.push_back(make_int2(static_cast<int32_t>(p->w_strows + p->item_rows[t] + j), row));
                if (j < parason::kRecRows) {
                    host.emplace_back(&rec[parason::kRecRow0 + j], row);
                    patches.push_back(make_int2(static_cast<int32_t>(w_rec + parason::kRecRow0 + j), row));
                }
                host.emplace_back(&it.num_pages, np);
                host.emplace_back(&rec[1], np);
                patches.push_back(make_int2(static_cast<int32_t>(w_rec + 1), np));
                patches.push_back(make_int2(static_cast<int32_t>(w_item + 1), np));
            }
            host.emplace_back(&it.last_valid, last_valid);
            host.emplace_back(&rec[2], last_valid);
            patches.push_back(make_int2(static_cast<int32_t>(w_rec + 2), last_valid));
            patches.push_back(make_int2(static_cast<int32_t>(w_item + 2), last_valid));
        }
    }

    // 3. the device copy first: if it cannot be updated, neither is the host
    // copy, so the two never disagree
    if (p->debug_flags & PARASON_DEBUG_FAIL_UPDATE) return refuse(PARASON_ECUDA);
    if (p->on_device && !patches.empty()) {
        cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
        // a pageable source is staged before the call returns, so the host
        // list may be reused by the next append.  A failed copy or launch
        // leaves the plan's device blob as it was (only the patch buffer,
        // which nothing else reads, may have changed).
        if (cudaMemcpyAsync(p->d_patch, patches.data(), patches.size() * sizeof(int2),
                            cudaMemcpyHostToDevice, stream) != cudaSuccess ||
            parason::launch_scatter(static_cast<int32_t *>(p->d_blob), p->d_patch,
                                    static_cast<int32_t>(patches.size()), stream) != cudaSuccess) {
            cudaGetLastError();
            return refuse(PARASON_ECUDA);
        }
    }

    // 4. commit the host copy
    for (const auto &w : host) *w.first = w.second;
    for (int32_t b = 0; b < L; ++b) {
        const int32_t n = p->leaf_node[b];
        if (p->tree_len[n] % P16 == 0) p->node_pages[n].push_back(new_pages[b]);
        p->tree_len[n] += 1;
    }
    p->unique_tokens += L;
    p->path_tokens += L;
    return PARASON_OK;
}

parason_status parason_plan_fork(parason_plan p, int32_t branch, int32_t num_children,
                                 const int32_t *child_len, const int32_t *child_page_ptr,
                                 const int32_t *child_pages, parason_stream_t stream_) {
    if (!p) return PARASON_EINVAL;
    if (p->cfg.mode == PARASON_FP32 || p->prefill) return PARASON_EUNSUPPORTED;
    const int32_t L = p->num_leaves;
    const int32_t H = p->cfg.num_kv_heads, g = p->group;
    constexpr int32_t P16 = parason::kPageSize;
    if (branch < 0 || branch >= L || num_children < 1 || !child_len || !child_page_ptr)
        return PARASON_EINVAL;
    if (num_children > INT32_MAX - L || num_children > INT32_MAX - p->num_nodes) return PARASON_EINVAL;
    // a new branch's rows of every node on its path go to suffix-pass tiles
    if (g > kNarrowRows) return PARASON_EUNSUPPORTED;
    if (p->on_device && p->blob_words > static_cast<size_t>(INT32_MAX)) return PARASON_EUNSUPPORTED;

    // 1. check the children: lengths, page counts, fresh distinct pages
    if (child_page_ptr[0] != 0) return PARASON_EINVAL;
    for (int32_t c = 0; c < num_children; ++c) {
        if (child_len[c] < 0) return PARASON_EINVAL;
        const int64_t want = (static_cast<int64_t>(child_len[c]) + P16 - 1) / P16;
        if (static_cast<int64_t>(child_page_ptr[c + 1]) - child_page_ptr[c] != want)
            return PARASON_EINVAL;
    }
    const int32_t n_child_pages = child_page_ptr[num_children];
    if (n_child_pages > 0 && !child_pages) return PARASON_EINVAL;
    std::vector<int32_t> claimed;
    auto refuse = [&](parason_status st) {
        for (int32_t pg : claimed) p->page_used[pg] = 0;
        return st;
    };
    for (int32_t k = 0; k < n_child_pages; ++k) {
        const int32_t pg = child_pages[k];
        if (pg < 0 || pg >= p->num_phys || p->page_used[pg]) return refuse(PARASON_EINVAL);
        p->page_used[pg] = 1;
        claimed.push_back(pg);
    }
    if (p->on_device) {
        int dev = -1;
        if (cudaGetDevice(&dev) != cudaSuccess) {
            cudaGetLastError();
            return refuse(PARASON_ECUDA);
        }
        if (dev != p->device) return refuse(PARASON_EINVAL);
    }

    // 2. the new work, without touching the plan: branches L .. L + E - 1
    // are children 1 .. E (child 0 keeps index `branch`); node N0 + c is
    // child c, under the branch's node nb, which stops being a branch node
    const int32_t E = num_children - 1;
    const int32_t nb = p->leaf_node[branch];
    const int32_t N0 = p->num_nodes;
    const int32_t D0 = static_cast<int32_t>(p->dfs_leaf.size());   // new branches' DFS positions
    std::vector<int32_t> path;
    for (int32_t m = nb; m >= 0; m = p->tree_parent[m]) path.push_back(m);
    std::reverse(path.begin(), path.end());
    int64_t path_tok = 0;
    for (int32_t m : path) path_tok += p->tree_len[m];

    std::vector<WorkItem> items;
    std::vector<int32_t> rec, irows, rows;          // records, item row starts, page rows
    std::vector<std::vector<int32_t>> tails(num_children);
    // merge entries per (child, kv head); child 0 starts from the branch's list
    std::vector<std::vector<int32_t>> ent(static_cast<size_t>(num_children) * H);
    for (int32_t j = 0; j < H; ++j) {
        const int2 r = p->merge_rng[static_cast<size_t>(branch) * H + j];
        ent[j].assign(p->merge_ent.begin() + r.x, p->merge_ent.begin() + r.y);
    }
    int64_t slots = p->num_slots;
    const size_t item0 = p->items.size(), row0 = p->stream_rows.size();
    const int32_t page_pos0 = static_cast<int32_t>(p->page_ids.size());
    bool overflow = false;
    // one suffix-pass item: `np` pages of `pages` from `pg`, rows of DFS
    // positions [leaf_lo, leaf_lo + nrows / g) of kv head j
    auto add_item = [&](const std::vector<int32_t> &pages, int32_t node_len, int32_t page_pos,
                        int32_t pg, int32_t np, int32_t leaf_lo, int32_t nrows, int32_t j,
                        bool tail) -> int32_t {
        const int32_t P = static_cast<int32_t>(pages.size());
        WorkItem it;
        it.page_pos = page_pos + pg;
        it.num_pages = np;
        it.last_valid = pg + np == P ? node_len - (P - 1) * P16 : P16;
        it.leaf_lo = leaf_lo;
        it.row0 = 0;
        it.nrows = nrows;
        it.kv_head = j;
        if (slots + nrows > INT32_MAX) overflow = true;
        it.slot_base = static_cast<int32_t>(slots);
        slots += nrows;
        const int32_t start = static_cast<int32_t>(row0 + rows.size());
        irows.push_back(start);
        for (int32_t k = 0; k < np; ++k) rows.push_back((pages[pg + k] * H + j) * P16);
        if (tail) rows.insert(rows.end(), std::min(kAppendSlackMax, std::max(kAppendSlackMin, np / 2)), 0);
        const size_t r0 = rec.size();
        rec.resize(r0 + parason::kRecWords, 0);
        std::memcpy(&rec[r0], &it, sizeof(WorkItem));
        rec[r0 + parason::kRecRowsOff] = start;
        for (int32_t k = 0; k < std::min(np, parason::kRecRows); ++k)
            rec[r0 + parason::kRecRow0 + k] = (pages[pg + k] * H + j) * P16;
        items.push_back(it);
        return static_cast<int32_t>(item0 + items.size() - 1);
    };
    // equal pieces of at most the plan's suffix piece length
    auto pieces = [&](int32_t P, auto &&fn) {
        const int64_t chunk = std::max<int64_t>(1, p->narrow_chunk);
        const int64_t n = (P + chunk - 1) / chunk;
        const int32_t per = static_cast<int32_t>((P + n - 1) / std::max<int64_t>(1, n));
        for (int32_t pg = 0; pg < P; pg += per) fn(pg, std::min(per, P - pg));
    };
    // (a) the new branches on every node of the path, in tiles of whole
    // branches of at most 16 rows
    const int32_t bpt = kNarrowRows / g;
    for (int32_t m : path) {
        const int32_t P = static_cast<int32_t>(p->node_pages[m].size());
        if (p->tree_len[m] == 0 || P == 0) continue;
        for (int32_t j = 0; j < H; ++j)
            for (int32_t t0 = 0; t0 < E; t0 += bpt) {
                const int32_t nbr = std::min(bpt, E - t0);
                pieces(P, [&](int32_t pg, int32_t np) {
                    const int32_t id = add_item(p->node_pages[m], p->tree_len[m], p->node_page_pos[m],
                                                pg, np, D0 + t0, nbr * g, j, false);
                    for (int32_t i = 0; i < nbr; ++i)
                        ent[static_cast<size_t>(1 + t0 + i) * H + j].push_back(items[id - item0].slot_base +
                                                                              i * g);
                });
            }
    }
    // (b) every child's own node: one tile of its g rows per kv head; the
    // last piece is the branch's tail, followed by room for appends
    std::vector<std::vector<int32_t>> cpages(num_children);
    int32_t cpos = page_pos0;
    std::vector<int32_t> cpage_pos(num_children);
    for (int32_t c = 0; c < num_children; ++c) {
        cpages[c].assign(child_pages + child_page_ptr[c], child_pages + child_page_ptr[c + 1]);
        cpage_pos[c] = cpos;
        cpos += static_cast<int32_t>(cpages[c].size());
        const int32_t P = static_cast<int32_t>(cpages[c].size());
        if (P == 0) continue;
        const int32_t pos = c == 0 ? p->dfs_pos[branch] : D0 + c - 1;
        for (int32_t j = 0; j < H; ++j)
            pieces(P, [&](int32_t pg, int32_t np) {
                const bool tail = pg + np == P;
                const int32_t id = add_item(cpages[c], child_len[c], cpage_pos[c], pg, np, pos, g, j, tail);
                ent[static_cast<size_t>(c) * H + j].push_back(items[id - item0].slot_base);
                if (tail) tails[c].push_back(id);
            });
    }
    // merge lists, appended: the branch's moved list, then the new branches'
    std::vector<int32_t> ents;
    std::vector<int2> rng(static_cast<size_t>(num_children) * H);
    const size_t ent0 = p->merge_ent.size();
    for (size_t k = 0; k < ent.size(); ++k) {
        const int32_t e0 = static_cast<int32_t>(ent0 + ents.size());
        ents.insert(ents.end(), ent[k].begin(), ent[k].end());
        rng[k] = make_int2(e0, static_cast<int32_t>(ent0 + ents.size()));
    }
    // room in the device copy (the host copy keeps to it too)
    if (overflow || p->items.size() + items.size() > p->cap_items ||
        row0 + rows.size() > p->cap_rows || static_cast<size_t>(L) + E > p->cap_leaves ||
        ent0 + ents.size() > p->cap_ent || ent0 + ents.size() > static_cast<size_t>(INT32_MAX) ||
        row0 + rows.size() > static_cast<size_t>(INT32_MAX) ||
        (static_cast<size_t>(L) + E) * H * kPatchesPerTail + 2 * static_cast<size_t>(H) + 2 > p->cap_patch)
        return refuse(PARASON_ENOSPACE);
    std::vector<int32_t> dfs_new(static_cast<size_t>(E));
    for (int32_t i = 0; i < E; ++i) dfs_new[i] = L + i;
    // a plan that had no attention work has no grid yet: the new items get
    // one of suffix CTAs, whose warps own the first queue positions
    const bool new_grid = p->num_ctas == 0 && !items.empty();
    const int32_t queue_start1 = new_grid ? p->num_sms * p->suffix_warps : p->queue_start[1];

    // 3. the device copy: the appended regions lie past what the kernels
    // read until the host counts grow, and one scatter then moves the
    // branch's merge ranges -- so a failure leaves the device plan as it was
    if (p->debug_flags & PARASON_DEBUG_FAIL_UPDATE) return refuse(PARASON_ECUDA);
    if (p->on_device) {
        cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
        std::vector<int2> &patches = p->patches;
        patches.clear();
        for (int32_t j = 0; j < H; ++j) {
            const size_t w = p->w_mrng + 2 * (static_cast<size_t>(branch) * H + j);
            patches.push_back(make_int2(static_cast<int32_t>(w), rng[j].x));
            patches.push_back(make_int2(static_cast<int32_t>(w + 1), rng[j].y));
        }
        if (new_grid) patches.push_back(make_int2(static_cast<int32_t>(p->w_qnext + 1), queue_start1));
        struct Copy {
            void *dst;
            const void *src;
            size_t bytes;
        };
        const Copy copies[] = {
            {p->d_items + item0, items.data(), items.size() * sizeof(WorkItem)},
            {p->d_item_rec + item0 * parason::kRecWords, rec.data(), rec.size() * sizeof(int32_t)},
            // starts of the new items, and the end of the last one
            {p->d_item_rows + item0, irows.data(), irows.size() * sizeof(int32_t)},
            {p->d_stream_rows + row0, rows.data(), rows.size() * sizeof(int32_t)},
            {p->d_dfs_leaf + D0, dfs_new.data(), dfs_new.size() * sizeof(int32_t)},
            {p->d_merge_ent + ent0, ents.data(), ents.size() * sizeof(int32_t)},
            {p->d_merge_rng + static_cast<size_t>(L) * H, rng.data() + H,
             static_cast<size_t>(E) * H * sizeof(int2)},
        };
        const int32_t rows_end = static_cast<int32_t>(row0 + rows.size());
        bool ok = true;
        for (const Copy &c : copies)
            if (c.bytes && cudaMemcpyAsync(c.dst, c.src, c.bytes, cudaMemcpyHostToDevice, stream) !=
                               cudaSuccess)
                ok = false;
        if (ok && cudaMemcpyAsync(p->d_item_rows + item0 + irows.size(), &rows_end, sizeof(int32_t),
                                  cudaMemcpyHostToDevice, stream) != cudaSuccess)
            ok = false;
        if (ok && (cudaMemcpyAsync(p->d_patch, patches.data(), patches.size() * sizeof(int2),
                                   cudaMemcpyHostToDevice, stream) != cudaSuccess ||
                   parason::launch_scatter(static_cast<int32_t *>(p->d_blob), p->d_patch,
                                           static_cast<int32_t>(patches.size()), stream) != cudaSuccess))
            ok = false;
        if (!ok) {
            cudaGetLastError();
            return refuse(PARASON_ECUDA);
        }
    }

    // 4. commit the host copy
    p->items.insert(p->items.end(), items.begin(), items.end());
    p->item_rec.insert(p->item_rec.end(), rec.begin(), rec.end());
    p->item_rows.pop_back();                         // the old end is the first new start
    p->item_rows.insert(p->item_rows.end(), irows.begin(), irows.end());
    p->item_rows.push_back(static_cast<int32_t>(row0 + rows.size()));
    p->stream_rows.insert(p->stream_rows.end(), rows.begin(), rows.end());
    for (size_t i = item0; i < p->items.size(); ++i) p->narrow_queue.push_back(static_cast<int32_t>(i));
    p->merge_ent.insert(p->merge_ent.end(), ents.begin(), ents.end());
    for (int32_t j = 0; j < H; ++j) p->merge_rng[static_cast<size_t>(branch) * H + j] = rng[j];
    p->merge_rng.insert(p->merge_rng.end(), rng.begin() + H, rng.end());
    p->dfs_leaf.insert(p->dfs_leaf.end(), dfs_new.begin(), dfs_new.end());
    for (int32_t i = 0; i < E; ++i) p->dfs_pos.push_back(D0 + i);
    p->num_slots = slots;
    for (int32_t c = 0; c < num_children; ++c) {
        p->tree_parent.push_back(nb);
        p->tree_len.push_back(child_len[c]);
        p->node_pages.push_back(cpages[c]);
        p->node_page_pos.push_back(cpage_pos[c]);
        p->page_ids.insert(p->page_ids.end(), cpages[c].begin(), cpages[c].end());
        p->unique_tokens += child_len[c];
        p->path_tokens += child_len[c] + (c > 0 ? path_tok : 0);
    }
    p->tails[branch] = tails[0];
    for (int32_t c = 1; c < num_children; ++c) p->tails.push_back(tails[c]);
    p->leaf_node[branch] = N0;
    for (int32_t c = 1; c < num_children; ++c) p->leaf_node.push_back(N0 + c);
    p->num_nodes += num_children;
    p->num_leaves += E;
    if (new_grid) {
        p->num_ctas = p->num_sms;
        p->num_wide_ctas = 0;
        p->queue_start[1] = queue_start1;
    }
    return PARASON_OK;
}

parason_status parason_plan_export(parason_plan p, int32_t table, void *dst, size_t bytes) {
    if (!p) return PARASON_EINVAL;
    const void *src = nullptr;
    size_t n = 0;
    switch (table) {
    case PARASON_TABLE_ITEMS: src = p->items.data(); n = p->items.size() * sizeof(WorkItem); break;
    case PARASON_TABLE_DFS_LEAVES: src = p->dfs_leaf.data(); n = p->dfs_leaf.size() * 4; break;
    case PARASON_TABLE_MERGE_RANGES: src = p->merge_rng.data(); n = p->merge_rng.size() * 8; break;
    case PARASON_TABLE_MERGE: src = p->merge_ent.data(); n = p->merge_ent.size() * 4; break;
    case PARASON_TABLE_WIDE_QUEUE: src = p->wide_queue.data(); n = p->wide_queue.size() * 4; break;
    case PARASON_TABLE_NARROW_QUEUE: src = p->narrow_queue.data(); n = p->narrow_queue.size() * 4; break;
    case PARASON_TABLE_ITEM_ROWS: src = p->item_rows.data(); n = p->item_rows.size() * 4; break;
    case PARASON_TABLE_STREAM_ROWS: src = p->stream_rows.data(); n = p->stream_rows.size() * 4; break;
    case PARASON_TABLE_ITEM_KEY0: src = p->item_key0.data(); n = p->item_key0.size() * 4; break;
    case PARASON_TABLE_SHARD_BRANCHES:
        // an unsharded plan's branch b is branch b
        if (p->shard_branch.size() != static_cast<size_t>(p->num_leaves)) {
            p->shard_branch.resize(static_cast<size_t>(p->num_leaves));
            for (int32_t b = 0; b < p->num_leaves; ++b) p->shard_branch[b] = b;
        }
        src = p->shard_branch.data();
        n = p->shard_branch.size() * 4;
        break;
    default: return PARASON_EINVAL;
    }
    if (bytes < n || (n > 0 && !dst)) return PARASON_EINVAL;
    if (n) std::memcpy(dst, src, n);
    return PARASON_OK;
}

parason_status parason_plan_set_debug(parason_plan p, uint32_t flags, int64_t wait_limit_ns) {
    if (!p || wait_limit_ns < 0) return PARASON_EINVAL;
    p->debug_flags = flags;
    if (wait_limit_ns > 0) p->wait_limit_ns = wait_limit_ns;
    return PARASON_OK;
}

parason_status parason_plan_enable_timing(parason_plan p, int32_t max_calls) {
    if (!p || max_calls < 0 || !p->on_device) return PARASON_EINVAL;
    free_events(p);
    if (max_calls == 0) return PARASON_OK;
    p->events.assign(static_cast<size_t>(max_calls) * 3, nullptr);
    for (auto &e : p->events) {
        if (cudaEventCreate(&e) != cudaSuccess) {
            e = nullptr;
            free_events(p);
            return PARASON_ECUDA;
        }
    }
    p->timing_cap = max_calls;
    p->timing_n = 0;
    return PARASON_OK;
}

parason_status parason_plan_read_timing(parason_plan p, float *attn_ms, float *merge_ms,
                                        int32_t capacity, int32_t *count) {
    if (!p || !count || capacity < 0) return PARASON_EINVAL;
    const int32_t n = std::min(p->timing_n, capacity);
    if (p->timing_n > 0 && cudaEventSynchronize(p->events[3 * (p->timing_n - 1) + 2]) != cudaSuccess)
        return PARASON_ECUDA;
    for (int32_t i = 0; i < n; ++i) {
        float a = 0.f, m = 0.f;
        if (cudaEventElapsedTime(&a, p->events[3 * i], p->events[3 * i + 1]) != cudaSuccess ||
            cudaEventElapsedTime(&m, p->events[3 * i + 1], p->events[3 * i + 2]) != cudaSuccess)
            return PARASON_ECUDA;
        if (attn_ms) attn_ms[i] = a;
        if (merge_ms) merge_ms[i] = m;
    }
    *count = n;
    p->timing_n = 0;
    return PARASON_OK;
}

int32_t parason_plan_launches_per_decode(parason_plan p) {
    if (!p || p->num_leaves == 0) return 0;
    return (p->items.empty() ? 0 : 1) + 1;                // attention, then merge
}

const char *parason_version(void) { return "0.1.0"; }

}  // extern "C"
