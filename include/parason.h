/*
 * parason.h -- C ABI of the GB300 (sm_103a) fork-tree decode-attention library.
 *
 * Parallel reasoning forks one request into Subtask branches (all results
 * needed) and Trial branches (speculative attempts) (paper Sec. 3.1); threads
 * may nest further parallel regions (Fig. 4, rule W -> <Thread> B </Thread>),
 * so the live branches form a fork tree.  The runtime decodes every branch
 * as an independent worker (Sec. 3.4) and concatenates the branch outputs
 * into the context that follows (Fig. 1 caption), so each decode step needs,
 * for every branch b, softmax attention of b's query over b's whole context:
 * the KV of every tree node on the path root -> b, root first.
 *
 * This library computes exactly that, reading every shared node's KV from
 * HBM once for all the branches under it.  Sharing, tiling and splitting are
 * rearrangements of the same sums; the result is plain attention.
 *
 * Conventions for every entry point:
 *   - "host" pointers are read during the call only; "device" pointers are
 *     CUDA device memory owned by the caller and must stay valid until the
 *     work queued on `stream` has finished.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Every
 *     entry point that takes a stream only enqueues work on it, except
 *     parason_plan_check, which synchronises it.
 *   - No entry point throws; every failure is a parason_status.  Nothing is
 *     allocated by parason_attn_decode or parason_lse_merge.
 *
 * Layouts (row-major, innermost last):
 *   q         [num_leaves, H_q, head_dim]                 (branch b = row b)
 *   k_pages   [num_physical_pages, H_kv, page_size, head_dim]
 *   v_pages   same as k_pages
 *   out       [num_leaves, H_q, head_dim]   same dtype as q
 *   lse       [num_leaves, H_q] fp32, natural log of sum_t exp(s_t)
 *   q head h reads kv head h / (H_q / H_kv)  (grouped-query attention)
 *   s_t = sm_scale * <q, k_t>, sm_scale = 1/sqrt(head_dim) unless given.
 */
#ifndef PARASON_H
#define PARASON_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without including the CUDA headers (same type). */
struct CUstream_st;
typedef struct CUstream_st *parason_stream_t;

typedef enum {
    PARASON_OK = 0,
    PARASON_EINVAL = 1,       /* malformed argument, tree or page table   */
    PARASON_ENOMEM = 2,       /* host or device allocation failed (plan)  */
    PARASON_ECUDA = 3,        /* a CUDA runtime call failed               */
    PARASON_ETIMEOUT = 4,     /* a bounded device wait expired            */
    PARASON_EUNSUPPORTED = 5, /* valid but not implemented (shape / mode) */
    PARASON_ENOSPACE = 6,     /* the plan has no room for an update: build a new one */
    PARASON_ERANGE = 7        /* an input value outside what the mode's kernels hold
                                 (e4m3 KV: |q| >= 65520, see parason_attn_decode) */
} parason_status;

typedef enum {
    PARASON_BF16 = 0,         /* q, K, V, out bf16; fp32 accumulation     */
    PARASON_FP32 = 1,         /* q, K, V, out fp32; fp32 FMA throughout   */
    PARASON_FP8_E4M3_KV = 2   /* q, out bf16; K, V OCP e4m3 bytes with one
                                 fp32 scale per kv head for K and for V   */
} parason_mode;

typedef struct {
    int32_t num_q_heads;      /* H_q, multiple of H_kv                    */
    int32_t num_kv_heads;     /* H_kv                                     */
    int32_t head_dim;         /* 64 or 128                                */
    int32_t page_size;        /* tokens per KV page; must be 16           */
    int32_t mode;             /* a parason_mode                           */
    float sm_scale;           /* 0 => 1/sqrt(head_dim)                    */
} parason_attn_config;

typedef struct parason_plan_s *parason_plan;

/*
 * Build the decode plan of one fork tree (the branch set of Sec. 3.4 at one
 * decode step) and upload its metadata on `stream`.
 *
 * Tree, all host arrays:
 *   parent[num_nodes]        parent node, -1 for a root; parent[i] < i.
 *                            Several roots (several requests) are allowed.
 *   node_len[num_nodes]      tokens held by each node (>= 0); a branch's own
 *                            node includes the token decoded this step.
 *   node_page_ptr[num_nodes+1]  CSR offsets into page_ids; node i owns
 *                            exactly ceil(node_len[i] / page_size) pages.
 *   page_ids[node_page_ptr[num_nodes]]  physical page of node i's j-th page
 *                            at page_ids[node_page_ptr[i] + j], in
 *                            [0, num_physical_pages); no page is owned by two
 *                            nodes.  Token t of node i sits in slot
 *                            t % page_size of its page t / page_size.
 *   leaf_node[num_leaves]    node holding branch b's private suffix; distinct
 *                            nodes with no children.  Branch b's query is
 *                            row b of q.
 *
 * Returns PARASON_EINVAL for: bad config (H_q % H_kv != 0, head_dim not 64 or
 * 128, page_size != 16, unknown mode, negative or non-finite sm_scale), a
 * parent out of range or not smaller than its child, a negative length, a
 * page count that is not ceil(len/page_size), a page id out of range or owned
 * twice, a leaf out of range, repeated or with children, or a NULL pointer.
 * PARASON_EUNSUPPORTED for e4m3 KV with head_dim 64 (only 128 has a kernel).
 * PARASON_ENOMEM / PARASON_ECUDA if the metadata cannot be allocated or
 * copied.  On success *out owns host and device memory until
 * parason_plan_destroy.  The plan may be used by any number of decode calls,
 * one at a time: its device copy holds the work-queue positions that a
 * call's kernels advance and rewind, so two calls on one plan must not
 * overlap (issue them on one stream, or order their streams).
 */
parason_status parason_attn_plan(const parason_attn_config *cfg, int32_t num_nodes,
                                 const int32_t *parent, const int32_t *node_len,
                                 const int32_t *node_page_ptr, const int32_t *page_ids,
                                 int32_t num_leaves, const int32_t *leaf_node,
                                 int64_t num_physical_pages, parason_stream_t stream,
                                 parason_plan *out);

/*
 * Same validation and work decomposition as parason_attn_plan, but no device
 * memory and no CUDA call: the plan can be inspected (parason_plan_info,
 * parason_plan_export) on a machine without a GPU.  parason_attn_decode on
 * it returns PARASON_EINVAL.  `num_sms` is the SM count the work split
 * targets (152 on GB300).
 */
parason_status parason_attn_plan_host(const parason_attn_config *cfg, int32_t num_nodes,
                                      const int32_t *parent, const int32_t *node_len,
                                      const int32_t *node_page_ptr, const int32_t *page_ids,
                                      int32_t num_leaves, const int32_t *leaf_node,
                                      int64_t num_physical_pages, int32_t num_sms,
                                      parason_plan *out);

/*
 * Tree-masked prefill (the join, Sec. 3.1 and Fig. 1: after a parallel block
 * the threads' tokens become context of the main trajectory, and new text is
 * prefilled against the fork tree): plan one attention pass in which every
 * token of each chunk node is a query.
 *
 * Tree and pages as for parason_attn_plan; chunk_node[num_chunks] are
 * distinct childless nodes whose tokens (K and V already written) are
 * prefilled.  Queries are numbered chunk by chunk: query k = token t of
 * chunk c with k = (sum of the lengths of chunks 0 .. c-1) + t.  Query k
 * attends to every token of every ancestor of chunk_node[c] and to tokens
 * 0 .. t of chunk_node[c] itself (causal within the chunk).
 *
 * The plan is run with parason_attn_decode: q [num_queries, H_q, head_dim],
 * out the same shape, lse [num_queries, H_q]; parason_plan_info reports
 * num_queries as num_leaves.  The causal tile is the tcgen05 prefix tile:
 * PARASON_EUNSUPPORTED unless head_dim is 128 and the mode is PARASON_BF16
 * or PARASON_FP8_E4M3_KV (k_scale / v_scale as for decode), and
 * parason_plan_append on a prefill plan returns PARASON_EUNSUPPORTED.  Other
 * errors, ownership and concurrency as parason_attn_plan.
 */
parason_status parason_prefill_plan(const parason_attn_config *cfg, int32_t num_nodes,
                                    const int32_t *parent, const int32_t *node_len,
                                    const int32_t *node_page_ptr, const int32_t *page_ids,
                                    int32_t num_chunks, const int32_t *chunk_node,
                                    int64_t num_physical_pages, parason_stream_t stream,
                                    parason_plan *out);

/* parason_prefill_plan without device memory or CUDA calls (inspection), as
 * parason_attn_plan_host is to parason_attn_plan. */
parason_status parason_prefill_plan_host(const parason_attn_config *cfg, int32_t num_nodes,
                                         const int32_t *parent, const int32_t *node_len,
                                         const int32_t *node_page_ptr, const int32_t *page_ids,
                                         int32_t num_chunks, const int32_t *chunk_node,
                                         int64_t num_physical_pages, int32_t num_sms,
                                         parason_plan *out);

/*
 * One rank's part of a decode step that `world` ranks (one GPU each) share
 * with no exchange between them: the plan of the work rank `rank` computes.
 * The paper's runtime decodes each request's branches as independent
 * workers (Sec. 3.4), and requests do not read each other's KV; and the kv
 * heads of grouped-query attention are independent too.  So the step splits
 * either way with nothing to combine afterwards.
 *
 *   kind PARASON_SHARD_REQUESTS: the roots (requests), in index order, are
 *     cut into `world` contiguous groups of about equal cost (the tokens of
 *     a request's nodes that some branch reads, plus H_q/H_kv per branch);
 *     rank r plans the requests of group r.  Its branch b is global branch
 *     PARASON_TABLE_SHARD_BRANCHES[b] (increasing): q, out and lse of the
 *     rank hold those rows, in that order.  Page ids are the caller's, so
 *     the rank's pools are addressed as the whole pool would be
 *     (num_physical_pages pages); only the rank's pages are read.  A rank
 *     with no request gets a plan with no branch (decode does nothing).
 *   kind PARASON_SHARD_KV_HEADS: rank r takes kv heads [r H_kv / world,
 *     (r + 1) H_kv / world) and their q heads [r H_q / world, (r + 1) H_q /
 *     world); H_kv must be a multiple of world.  The plan is that of cfg
 *     with H_kv / world kv heads and H_q / world q heads over every branch:
 *     q, out and lse hold the rank's heads ([num_leaves, H_q / world, d]),
 *     the pools hold the rank's kv heads ([P, H_kv / world, 16, d]).
 *
 * The whole tree is validated as by parason_attn_plan (same errors), then
 * PARASON_EINVAL for world < 1, rank outside [0, world), an unknown kind, or
 * H_kv not a multiple of world (kv-head shards).  Ownership, concurrency and
 * every other call on the returned plan are as for parason_attn_plan.
 */
enum { PARASON_SHARD_REQUESTS = 0, PARASON_SHARD_KV_HEADS = 1 };
parason_status parason_attn_plan_shard(const parason_attn_config *cfg, int32_t num_nodes,
                                       const int32_t *parent, const int32_t *node_len,
                                       const int32_t *node_page_ptr, const int32_t *page_ids,
                                       int32_t num_leaves, const int32_t *leaf_node,
                                       int64_t num_physical_pages, int32_t kind, int32_t rank,
                                       int32_t world, parason_stream_t stream, parason_plan *out);

/* parason_attn_plan_shard without device memory or CUDA calls (inspection),
 * as parason_attn_plan_host is to parason_attn_plan. */
parason_status parason_attn_plan_shard_host(const parason_attn_config *cfg, int32_t num_nodes,
                                            const int32_t *parent, const int32_t *node_len,
                                            const int32_t *node_page_ptr, const int32_t *page_ids,
                                            int32_t num_leaves, const int32_t *leaf_node,
                                            int64_t num_physical_pages, int32_t kind, int32_t rank,
                                            int32_t world, int32_t num_sms, parason_plan *out);

/* Device workspace (bytes) that parason_attn_decode needs for this plan:
 * the split partial results (o, m, l) of every work item.  0 for NULL. */
size_t parason_plan_workspace_bytes(parason_plan plan);

/*
 * One decode step: out[b, h, :] = softmax(s) V over branch b's root->leaf KV.
 *
 * Defining passage: the runtime dispatches every <Subtask> / <Trial> entry of
 * a parallel region as an independent worker that decodes its own thread
 * (Sec. 3.4), and a branch's tokens are later concatenated into the context
 * rather than selected (Sec. 3.1, Trial Parallelism; Fig. 1 caption), so one
 * step needs every live branch's attention over its whole context: the KV
 * of each tree node on its root -> leaf path, root first (nested regions per
 * Fig. 4, rule W -> <Thread> B </Thread>).  The paper gives no attention
 * formula; this is plain softmax attention, s_t = sm_scale * <q, k_t>.
 *
 * Asynchronous on `stream`; allocates nothing; capturable in a CUDA graph.
 *
 *   q        device, [num_leaves, H_q, head_dim], bf16 (fp32 in FP32 mode),
 *            16-byte aligned; or page-locked host memory the device can
 *            address (cudaHostAlloc / cudaHostRegister), read in place
 *   k_pages  device, [num_physical_pages, H_kv, 16, head_dim], bf16 / fp32 /
 *            e4m3 bytes by mode, 16-byte aligned
 *   v_pages  device, same layout and dtype as k_pages
 *   k_scale, v_scale  device fp32 [H_kv] in FP8 mode (k = e4m3 * k_scale),
 *            ignored otherwise (may be NULL)
 *   out      device, [num_leaves, H_q, head_dim], dtype of q, 16-byte
 *            aligned; or page-locked host memory the device can address
 *            (cudaHostAlloc / cudaHostRegister): the merge kernel then
 *            writes the result straight to the host
 *   lse      device (or such host memory) fp32 [num_leaves, H_q], or NULL.
 *            A branch whose whole path holds no token gets out = 0 and
 *            lse = -inf.
 *   workspace  device, at least parason_plan_workspace_bytes(plan) bytes,
 *            256-byte aligned; no contents are kept between calls.
 *
 * Slots of a node's last page past node_len are never read into the result,
 * whatever they hold (NaN included).
 *
 * With e4m3 KV the kernels multiply q by the widened keys and values in f16
 * (f16 holds every e4m3 value exactly): q is narrowed from bf16 to f16,
 * which is exact for |q| < 65504 except in the low bits of values below
 * 2^-14.  A q element of magnitude 65520 or more (inf included) cannot be
 * narrowed: the kernel records PARASON_ERANGE, which the next
 * parason_plan_check returns, and that call's out and lse are undefined.  Returns PARASON_EINVAL on a host-only
 * plan, a NULL or misaligned buffer or a short workspace, PARASON_ECUDA if a
 * launch fails.  Device-side failures (a bounded wait that expired) are
 * reported by parason_plan_check.
 */
parason_status parason_attn_decode(parason_plan plan, const void *q, const void *k_pages,
                                   const void *v_pages, const float *k_scale,
                                   const float *v_scale, void *out, float *lse,
                                   void *workspace, size_t workspace_bytes,
                                   parason_stream_t stream);

/* Scratch, in bytes, that parason_attn_decode_no_alloc holds per device. */
#define PARASON_NO_ALLOC_SCRATCH_BYTES (64u << 20)

/*
 * parason_attn_decode without a caller workspace.  The paper has no
 * counterpart: this is a library convenience for callers that cannot hand
 * over device memory at decode time -- an engine whose HBM is fully
 * committed to its KV page pool and fixed buffers, or a C host with no device
 * allocator of its own.  The partial results go to a scratch array that is
 * part of the library's device image: PARASON_NO_ALLOC_SCRATCH_BYTES (64 MiB)
 * per device, reserved when the library's device code is loaded on that
 * device.  Neither this call nor anything it calls allocates device memory.
 *
 * Arguments, layouts, results and errors are those of parason_attn_decode,
 * plus:
 *   - PARASON_EUNSUPPORTED if parason_plan_workspace_bytes(plan) exceeds
 *     PARASON_NO_ALLOC_SCRATCH_BYTES (checked before anything else is
 *     touched; such a plan needs parason_attn_decode with a workspace).
 *     At head_dim 128 the scratch holds about 129,000 partial rows, e.g. a
 *     Llama-3-8B step of 16 branches over a 2048-token prefix needs 7.2 MB.
 *   - The first call on each device looks up the scratch's device address
 *     (with that device current) and keeps it for the life of the process;
 *     make that first call outside any stream capture.  The address is not
 *     looked up again, so the device's primary context must not be reset
 *     afterwards.
 *   - Nothing in the scratch has to start at zero and nothing in it is kept
 *     between calls: every partial row the merge reads is written earlier in
 *     the same call.
 *   - All calls on one device share the one scratch array, whatever their
 *     plan or stream: two calls that overlap in time race on it and both
 *     results are undefined.  Calls issued to a single stream never overlap.
 */
parason_status parason_attn_decode_no_alloc(parason_plan plan, const void *q,
                                            const void *k_pages, const void *v_pages,
                                            const float *k_scale, const float *v_scale,
                                            void *out, float *lse, parason_stream_t stream);

/*
 * Decode-loop update: one generated token appended to every branch's own
 * node (leaf_node[b] gains one token), without building a new plan.  The
 * paper's engine runs every branch for one token per step (Sec. 3.4); this
 * is the step between two parason_attn_decode calls, O(branches * H_kv).
 *
 *   new_pages  host int32 [num_leaves]: for a branch whose node length is a
 *              multiple of 16 (the new token opens a page), the physical
 *              page that takes it -- in range and owned by no node; entries
 *              of the other branches are ignored (pass -1).  May be NULL when
 *              no branch opens a page.
 *
 * The caller writes the new token's K and V into its slot (length % 16 of
 * the node's last page) before the next decode.  On a plan built with
 * parason_attn_plan the update is also made to the device copy, with one
 * host-to-device copy and one small kernel on `stream`.  A plan's appends
 * and decodes must be issued in order (one stream, or ordered streams).
 *
 * Returns PARASON_EINVAL for a missing, out-of-range or already used page;
 * PARASON_ENOSPACE if some branch's node has no pages yet, or its last work
 * item has no room left for another page: a plan leaves each branch room for
 * half as many pages as its last item had (4 to 64 pages), beyond which the
 * grown item would unbalance the decode; PARASON_EUNSUPPORTED in FP32 mode.  On any error
 * nothing is changed, on the host or on the device: the device copy is
 * updated first, and the host copy only once that succeeded.
 * PARASON_EINVAL if the current device is not the plan's.
 * PARASON_EUNSUPPORTED on a prefill plan.
 */
parason_status parason_plan_append(parason_plan plan, const int32_t *new_pages,
                                   parason_stream_t stream);

/*
 * Decode-loop update at a fork: branch `branch` reaches the end of an
 * <Outlines> block and its k = num_children threads start (Sec. 3.4: the
 * runtime dispatches each <Subtask> / <Trial> entry as an independent worker;
 * Fig. 4, rule W -> <Thread> B </Thread>: a thread may itself open a nested
 * region).  The branch's node stops being a branch node and gets k child
 * nodes; the plan is patched without being rebuilt.
 *
 *   child_len       host int32 [k]: tokens already held by each child (>= 0;
 *                   with 0 the child has no page, and appends to it need a
 *                   new plan)
 *   child_page_ptr  host int32 [k + 1]: CSR into child_pages; child c owns
 *                   ceil(child_len[c] / 16) pages
 *   child_pages     host int32: fresh physical pages (in range, owned by no
 *                   node); the caller has written their K and V
 *
 * Numbering: the children become nodes num_nodes .. num_nodes + k - 1 in
 * order, under the branch's node.  Child 0 is branch `branch` (row `branch`
 * of q, out, lse); child c >= 1 is the new branch num_leaves + c - 1.  So q,
 * out and lse of the next decode have num_leaves + k - 1 rows
 * (parason_plan_get_info reports the new count).
 *
 * The new branches' rows of every node on the branch's path, and every
 * child's own rows, become suffix-pass work items appended to the plan:
 * O(k * H_kv * (pages on the path) / piece) items, merge entries and page
 * rows, copied to the device with a few host-to-device copies and one small
 * kernel on `stream` (from pageable memory, so the call may wait for work
 * already queued on `stream`).  The ancestors' pages are then read once more
 * for the new branches than a new plan would read them: build a new plan
 * when convenient.  parason_plan_workspace_bytes grows by the new partial
 * rows: the next decode needs a workspace of the new size.
 *
 * Returns PARASON_EINVAL for a branch out of range, k < 1, a negative
 * length, a page count that is not ceil(len / 16), a page out of range, used
 * or repeated, a NULL array, or a current device that is not the plan's;
 * PARASON_EUNSUPPORTED in FP32 mode, on a prefill plan, or with more than 16
 * q heads per kv head; PARASON_ENOSPACE if the room the plan keeps for
 * forks (about as much again as it held when built) is used up -- build a
 * new plan then.  On any error nothing is changed, on the host or the
 * device.  Forks and appends of a plan are issued in order with its decodes.
 */
parason_status parason_plan_fork(parason_plan plan, int32_t branch, int32_t num_children,
                                 const int32_t *child_len, const int32_t *child_page_ptr,
                                 const int32_t *child_pages, parason_stream_t stream);

/*
 * Combine two attention results over disjoint key sets A and B (for example
 * two KV ranges of one branch, or a branch's context before and after a join)
 * into the result over A u B, row by row.
 *
 * Defining passage: a thread's result returns to the main trajectory and the
 * branches are concatenated into its context (Sec. 3.4; Sec. 3.1, Trial
 * Parallelism: the merge step concatenates rather than selects; Fig. 1), so
 * attention over the joined context is attention over the union of the key
 * sets; the paper gives no formula, and this is the exact log-sum-exp
 * identity for softmax over a union of disjoint sets:
 *   o = (e^{lse_a} o_a + e^{lse_b} o_b) / (e^{lse_a} + e^{lse_b})
 *   lse = ln(e^{lse_a} + e^{lse_b})
 * A side with lse = -inf is empty; both empty gives o = 0, lse = -inf.
 * o_a, o_b, o_out: device [rows, head_dim], bf16 (PARASON_BF16 and
 * PARASON_FP8_E4M3_KV) or fp32 (PARASON_FP32); lse_*: device fp32 [rows].
 * o_out / lse_out may alias the inputs row for row.  Asynchronous on stream.
 */
parason_status parason_lse_merge(const void *o_a, const float *lse_a, const void *o_b,
                                 const float *lse_b, void *o_out, float *lse_out,
                                 int64_t rows, int32_t head_dim, int32_t mode,
                                 parason_stream_t stream);

/* Synchronise `stream`, then read and clear the plan's device error word:
 * PARASON_ETIMEOUT if a kernel gave up a bounded wait since the last check,
 * PARASON_ERANGE if an e4m3-KV decode met a q element of magnitude 65520 or
 * more (the first error recorded wins), PARASON_ECUDA if the stream reports
 * an error, else PARASON_OK. */
parason_status parason_plan_check(parason_plan plan, parason_stream_t stream);

/* Release the plan's host and device memory.  NULL is a no-op.  Work queued
 * with the plan must have finished. */
void parason_plan_destroy(parason_plan plan);

/* Static English name of a status. */
const char *parason_status_string(parason_status status);

/* ---------------------------------------------------------------------------
 * Inspection, testing and measurement
 * ------------------------------------------------------------------------- */

typedef struct {
    int32_t num_items;          /* work items of the attention kernel       */
    int32_t num_leaves;
    int32_t num_merge_entries;  /* partial results folded by the merge      */
    int32_t chunk_pages;        /* shortest split-K piece, in pages         */
    int64_t num_slots;          /* partial (o, m, l) rows in the workspace  */
    int64_t unique_tokens;      /* tokens of nodes some branch reads, once  */
    int64_t path_tokens;        /* sum over branches of their path tokens   */
    int32_t num_sms;            /* SM count the split targeted              */
    int32_t on_device;          /* 1 if decode can run on this plan         */
    int32_t num_ctas;           /* CTAs of the persistent attention kernel  */
    int32_t num_wide_ctas;      /* of which start on the prefix pass        */
    int32_t num_wide_items;     /* prefix-pass items (tiles x pieces)       */
    int32_t num_narrow_items;   /* suffix-pass items                        */
    int64_t num_stream_rows;    /* entries of PARASON_TABLE_STREAM_ROWS     */
    int32_t tile_pairs;         /* 1: the prefix queue holds pairs of row
                                   tiles of one piece (bf16 KV, head_dim
                                   128): entries 2k and 2k + 1 are pulled
                                   together, and the second has no rows
                                   (row count 0) when the piece's tile
                                   count is odd                              */
} parason_plan_info;

parason_status parason_plan_get_info(parason_plan plan, parason_plan_info *info);

/*
 * Copy one of the plan's host-side tables into `dst` (host, `bytes` long):
 *   PARASON_TABLE_ITEMS      int32 [num_items][8]: first page position in
 *                            page_ids, page count, valid tokens in the last
 *                            page, first branch (index into the DFS branch
 *                            order), first node row, row count, kv head,
 *                            partial slot of the item's first row
 *   PARASON_TABLE_DFS_LEAVES int32 [num_leaves]: branches in DFS order
 *   PARASON_TABLE_MERGE_RANGES int32 [num_leaves * H_kv][2]: per (branch,
 *                            kv head), the begin and end of its entries in
 *                            PARASON_TABLE_MERGE (a fork moves a branch's
 *                            list to the end, so lists need not be in order)
 *   PARASON_TABLE_MERGE      int32 [num_merge_entries]: partial slot of the
 *                            branch's first q head of the kv head; q head
 *                            j*g + r reads slot entry + r
 *   PARASON_TABLE_WIDE_QUEUE int32 [num_wide_items]: prefix-pass items in the
 *                            order the kernel's prefix CTAs pull them (two
 *                            at a time when tile_pairs is set)
 *   PARASON_TABLE_NARROW_QUEUE int32 [num_narrow_items]: suffix-pass items in
 *                            the order the kernel's warps pull them
 *   PARASON_TABLE_ITEM_ROWS  int32 [num_items + 1]: start of each item's page
 *                            rows in the stream (an item's rows are the first
 *                            page-count entries from there)
 *   PARASON_TABLE_STREAM_ROWS int32 [num_stream_rows]: the TMA row
 *                            (page * H_kv + kv head) * 16 of every item page;
 *                            in a bf16 prefill piece over several nodes of a
 *                            path, a page that ends a node before the item's
 *                            last page adds 16 - its valid tokens (1..15),
 *                            and is followed up to the next 4-page block by
 *                            padding: the row num_physical_pages * H_kv * 16,
 *                            past the pool, which reads as zeros
 *   PARASON_TABLE_ITEM_KEY0  int32 [num_items] (prefill plans; empty for
 *                            decode plans): the causal mask's origin.  Query
 *                            token t of the chunk sees the key at position p
 *                            of the item's page stream (16 per page) iff
 *                            p <= t - key0: key0 is the own-node index of
 *                            the item's first key when the item starts in
 *                            the chunk's own node, minus the stream position
 *                            of the own node's first key when the item
 *                            reaches it from an ancestor, and -1 (no mask)
 *                            for an item with no key of the chunk's node
 *   PARASON_TABLE_SHARD_BRANCHES int32 [num_leaves]: the global index of
 *                            each of the plan's branches (parason_attn_plan_
 *                            shard); b for a plan that is not a shard
 * Returns PARASON_EINVAL if `bytes` is smaller than the table.
 */
enum {
    PARASON_TABLE_ITEMS = 0,
    PARASON_TABLE_DFS_LEAVES = 1,
    PARASON_TABLE_MERGE_RANGES = 2,
    PARASON_TABLE_MERGE = 3,
    PARASON_TABLE_WIDE_QUEUE = 4,
    PARASON_TABLE_NARROW_QUEUE = 5,
    PARASON_TABLE_ITEM_ROWS = 6,
    PARASON_TABLE_STREAM_ROWS = 7,
    PARASON_TABLE_ITEM_KEY0 = 8,
    PARASON_TABLE_SHARD_BRANCHES = 9
};
parason_status parason_plan_export(parason_plan plan, int32_t table, void *dst, size_t bytes);

/*
 * Debug controls.  `wait_limit_ns` bounds every device-side wait of the
 * plan's kernels (default 2e9 ns; 0 keeps the current value).  Flag
 * PARASON_DEBUG_SKIP_FIRST_LOAD makes each attention CTA skip issuing its
 * first KV load, so its consumers' wait can only expire: the kernel records
 * PARASON_ETIMEOUT, lets its other copies land, and exits; the output is
 * then undefined.  Used to test the timeout path without faulting the GPU.
 * Flag PARASON_DEBUG_FAIL_UPDATE makes parason_plan_append and
 * parason_plan_fork fail with PARASON_ECUDA at the point where they would
 * update the device copy (after every check, before anything is changed),
 * on host-only plans too: used to test that a failed update changes nothing.
 */
enum { PARASON_DEBUG_SKIP_FIRST_LOAD = 1u, PARASON_DEBUG_FAIL_UPDATE = 2u };
parason_status parason_plan_set_debug(parason_plan plan, uint32_t flags, int64_t wait_limit_ns);

/*
 * Per-kernel timing for benchmarks.  After parason_plan_enable_timing(plan,
 * n) every decode records CUDA events on its stream around its attention
 * kernel and its merge kernel, for up to n calls.  parason_plan_read_timing
 * synchronises on the last event and writes the durations (ms) of the
 * recorded calls to attn_ms[] and merge_ms[] (either may be NULL), sets
 * *count, and starts a new recording.  n = 0 disables timing.
 */
parason_status parason_plan_enable_timing(parason_plan plan, int32_t max_calls);
parason_status parason_plan_read_timing(parason_plan plan, float *attn_ms, float *merge_ms,
                                        int32_t capacity, int32_t *count);

/* Number of kernel launches one parason_attn_decode call of this plan makes. */
int32_t parason_plan_launches_per_decode(parason_plan plan);

/* ------------------------------------------------------------------------
 * Reasoning traces: the tag stream of the parallel-reasoning grammar (Fig. 4)
 *
 *   S -> <think> B </think>        B -> T B | P B | (empty)
 *   P -> <Parallel> O H </Parallel> O -> <Outlines> G </Outlines>
 *   G -> E G | E                   E -> <Subtask> T </Subtask> | <Trial> T </Trial>
 *   H -> W H | W                   W -> <Thread> B </Thread>
 *   T -> one or more text tokens
 *
 * A trace is an array of int32 symbols: a text token is any id >= 0, a tag
 * is one of the codes below (one generated token each).
 * ------------------------------------------------------------------------ */
enum {
    PARASON_TAG_THINK = -1, PARASON_TAG_THINK_END = -2,
    PARASON_TAG_PARALLEL = -3, PARASON_TAG_PARALLEL_END = -4,
    PARASON_TAG_OUTLINES = -5, PARASON_TAG_OUTLINES_END = -6,
    PARASON_TAG_SUBTASK = -7, PARASON_TAG_SUBTASK_END = -8,
    PARASON_TAG_TRIAL = -9, PARASON_TAG_TRIAL_END = -10,
    PARASON_TAG_THREAD = -11, PARASON_TAG_THREAD_END = -12
};

typedef struct {
    int64_t total_tokens;     /* every symbol of the trace                          */
    int64_t latency_tokens;   /* token length of the longest generation path
                                 (Sec. 4): sequential tokens count one each, a
                                 <Parallel> block counts its tags and outlines
                                 plus its slowest thread                          */
    int64_t subtask_tokens;   /* tokens whose innermost thread is a Subtask: thread
                                 k of a block has the type of outline entry k     */
    int64_t trial_tokens;     /* same for Trial (threads past the last entry are
                                 untyped)                                         */
    int32_t parallel_blocks;  /* <Parallel> blocks at any depth                     */
    int32_t threads;          /* threads at any depth                              */
    int32_t max_depth;        /* deepest nesting of blocks (0: none)               */
    int32_t top_level_blocks; /* blocks directly in the <think> body               */
    double acceleration;      /* total / latency (Tab. 4)                          */
    double eta;               /* 1 - latency / total (Sec. 3.5)                    */
} parason_trace_stats;

/*
 * Check a trace against the grammar and compute its token metrics (host
 * only, no CUDA call).  `symbols` is host memory of n int32.  Returns
 * PARASON_EINVAL for NULL pointers or a trace outside the grammar; then
 * *error_pos (if not NULL) is the first symbol no derivation can accept (n if
 * the trace ends early).  The grammar is LL(1), so that position is unique.
 */
parason_status parason_trace_analyze(const int32_t *symbols, int64_t n, parason_trace_stats *out,
                                     int64_t *error_pos);

/*
 * Fork tree of top-level block `block` (0-based, in trace order), in the form
 * parason_attn_plan takes: the decode state in which every innermost thread
 * of the block runs, each at its full length in the trace.
 *   node 0       every token before the block's first <Thread> (earlier
 *                blocks are joined, so all of it is context);
 *   thread node  its tokens up to the end of its first nested outlines block,
 *                whose threads become its children -- or all its tokens, as
 *                a branch, if it has no nested block.
 * Nodes are in depth-first order (parent[i] < i); leaf_node lists the
 * branches in that order.  parent and node_len hold `capacity` entries,
 * leaf_node as many.  *num_nodes and *num_leaves are set whenever the trace
 * parses; PARASON_EINVAL if it does not, if `block` is out of range or if
 * capacity < *num_nodes (call again with a larger capacity).  Host only.
 */
parason_status parason_trace_fork_tree(const int32_t *symbols, int64_t n, int32_t block,
                                       int32_t capacity, int32_t *parent, int32_t *node_len,
                                       int32_t *leaf_node, int32_t *num_nodes,
                                       int32_t *num_leaves);

/* Library version, "major.minor.patch". */
const char *parason_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PARASON_H */
