// internal.h -- types shared by the planner and the kernels of libparason.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "parason.h"

namespace parason {

// One unit of attention work: a tile of query rows of one tree node and one
// kv head, against a run of that node's pages.
//
// The rows of node n are its branches in DFS order times the g = H_q/H_kv
// q heads of the kv head: node row r is branch dfs_leaf[leaf_lo + r / g],
// q head kv_head * g + r % g.  Tiles start at multiples of g.  The item
// writes the partial result (o, m, l) of its row row0 + i to partial slot
// slot_base + i.
struct WorkItem {
    int32_t page_pos;    // index in page_ids of the item's first page
    int32_t num_pages;   // pages in the item (>= 1)
    int32_t last_valid;  // valid tokens in the item's last page (1..16)
    int32_t leaf_lo;     // DFS position of the node's first branch
    int32_t row0;        // first node row of this tile
    int32_t nrows;       // rows in this tile (1..128)
    int32_t kv_head;
    int32_t slot_base;   // partial slot of the tile's first row
};
static_assert(sizeof(WorkItem) == 32, "WorkItem is a 32-byte device record");

constexpr int kPageSize = 16;

// Suffix-warp item record: 32 words (one 128-byte line, word i read by lane
// i): the WorkItem, the start of its page rows in the stream, its first rows.
constexpr int kRecWords = 32;
constexpr int kRecRowsOff = 8;
constexpr int kRecRow0 = 9;
constexpr int kRecRows = kRecWords - kRecRow0;   // 23
constexpr int kMaxTileRows = 128;
constexpr int kErrWords = 4;            // device error record: code, block, site, aux

// Where a bounded wait gave up (error record word 2).
enum WaitSite : int32_t {
    kSiteConsumerFull = 1,
    kSiteProducerEmpty = 2,
    kSiteBadItem = 3,        // an item the kernel cannot hold (planner contract broken)
    kSiteQRange = 4,         // e4m3 KV: a q element that f16 cannot hold (PARASON_ERANGE)
};

struct AttnArgs {
    const WorkItem *items;
    const int32_t *page_ids;
    const int32_t *dfs_leaf;
    const void *q;
    float *part_o;          // [num_slots, head_dim]   sum_t 2^(x_t - m) v_t
    float2 *part_ml;        // [num_slots]             (m, sum_t 2^(x_t - m))
    const float *k_scale;   // FP8 mode
    const float *v_scale;
    int32_t *err;           // kErrWords ints
    long long wait_limit_ns;
    uint32_t debug_flags;
    int32_t num_items;
    int32_t num_q_heads;
    int32_t num_kv_heads;
    int32_t group;
    float scale_log2;       // sm_scale * log2(e): x_t = scale_log2 * <q, k_t>

    // dynamic schedule: items are numbered in pull order, prefix-pass items
    // [0, num_wide_items) then suffix-pass items.  CTAs [0, num_wide_ctas)
    // pull prefix-pass items and then suffix-pass items; every warp of the
    // other CTAs pulls suffix-pass items.  queue_next[0] / [1] are the next
    // positions to claim.  The first claims need no atomic: position c of
    // the prefix queue belongs to prefix CTA c, position w Nc + (c - W) of
    // the suffix queue to warp w of suffix CTA c (Nc = num_ctas - W suffix
    // CTAs), so the counters start past them (queue_start; the merge kernel
    // sets them back).
    const int32_t *item_rec;        // kRecWords per item, items in pull order
    int32_t num_wide_items;
    int32_t num_narrow_items;
    int32_t *queue_next;
    // TMA rows (page * H_kv + kv head) * 16 of item i's pages:
    // stream_rows[item_rows[i] ...]
    const int32_t *item_rows;
    const int32_t *stream_rows;
    int32_t num_ctas;
    int32_t num_wide_ctas;
    int32_t kv_rows;        // rows of the KV tensor maps (pages * H_kv * 16); a
                            // TMA box starting there is out of range: zeros
    // tree-masked prefill: per item, the token index (in its node) of its
    // first key when the item is causal, else -1; null for decode plans
    const int32_t *item_key0;
    int32_t suffix_warps;   // suffix-pass warps per CTA the plan was made for
    // bf16 KV at head_dim 128: the prefix queue holds pairs of row tiles of
    // one piece (position k: items 2k and 2k + 1, the second without rows
    // when the piece has one tile), run by the tcgen05 tile in pair mode
    int32_t tc_pairs;
};

struct MergeArgs {
    const int2 *merge_rng;      // [num_leaves * H_kv]: [begin, end) in merge_ent
    const int32_t *merge_ent;   // first partial slot of the branch's rows
    const float *part_o;
    const float2 *part_ml;
    void *out;
    float *lse;
    int32_t num_leaves;
    int32_t num_q_heads;
    int32_t num_kv_heads;
    int32_t group;
    int32_t *queue_next;        // set back to queue_start for the next launch
    int32_t queue_start[2];
};

// Device a plan's metadata lives on (-1 for a host-only plan or NULL).
int plan_device(parason_plan plan);

// Resident CTAs per SM of the persistent attention kernel of a mode (sets its
// attributes); cudaErrorNotSupported for a shape it has no kernel for.
cudaError_t attn_mma_ctas_per_sm(int head_dim, int mode, int *ctas_per_sm);

// TMA views of the K and V pools.  k / v: one box is one 128-byte column
// block of one page of one kv head (16 rows).  k_run / v_run: one box is the
// same column block of kTcRunPages consecutive pages of one kv head, for
// blocks whose pages are consecutive in the pool.  k_page / v_page: one box
// is a whole page of one kv head, its column blocks one after another (the
// layout the per-block boxes of k / v give).
constexpr int kTcRunPages = 4;
struct KvMaps {
    CUtensorMap k, v, k_run, v_run, k_page, v_page;
};

// Kernel launchers; each returns the launch's cudaError_t.
cudaError_t launch_attn_bf16(const AttnArgs &a, const KvMaps &maps, int head_dim,
                             cudaStream_t stream);
cudaError_t launch_attn_fp8(const AttnArgs &a, const KvMaps &maps, int head_dim,
                            cudaStream_t stream);
cudaError_t launch_attn_fp32(const AttnArgs &a, const float *k_pages, const float *v_pages,
                             int head_dim, cudaStream_t stream);
cudaError_t launch_merge(const MergeArgs &a, int head_dim, int mode, bool programmatic,
                         cudaStream_t stream);
// base[patches[i].x] = patches[i].y for i < n (plan updates)
cudaError_t launch_scatter(int32_t *base, const int2 *patches, int32_t n, cudaStream_t stream);

cudaError_t launch_lse_merge(const void *o_a, const float *lse_a, const void *o_b,
                             const float *lse_b, void *o_out, float *lse_out, int64_t rows,
                             int head_dim, int mode, cudaStream_t stream);

}  // namespace parason
