// attn_bf16.cu -- fork-tree decode attention for bf16 KV on sm_103a.
//
// Persistent kernel, two CTAs per SM.  Each CTA runs a planner-made list of
// work items back to back; an item is up to 64 stacked query rows (the
// branches under one fork-tree node times the q heads of one kv head)
// against one chunk of that node's pages.  A node's KV is read from HBM once
// for all the rows stacked on it: this is what turns the shared prefix of many
// Subtask/Trial branches (paper Sec. 3.1, 3.4) into one read.
//
//   warp 4 (producer)   TMA: one 3-D box per (page, kv head) for K and for V,
//                       128-byte swizzle, into a ring of single-page stages
//                       that runs continuously across item boundaries, so the
//                       next item's pages load during this item's epilogue.
//   warps 0-3           tensor-core QK^T and PV with mma.sync m16n8k16 (bf16
//                       in, fp32 accumulate) from ldmatrix fragments, online
//                       softmax in registers with quad shuffles.  The warps
//                       split the tile's rows (16 per warp) and, for small
//                       tiles, the item's pages (page p to warp p % tgc).
//
// Epilogue of an item: the warps of a row group combine through shared memory
// and write the item's partial (o, m, l) rows; then the item is counted into
// every (branch, kv head) it feeds, and the item that completes a pair runs
// that pair's log-sum-exp merge (merge_epilogue.cuh) -- no second kernel.
//
// Scores are kept in the log2 domain: x = sm_scale*log2(e)*<q,k>, so the
// partial is m = max x, l = sum 2^(x-m), o = sum 2^(x-m) v (unnormalised).
#include "device_common.cuh"
#include "merge_epilogue.cuh"

namespace parason {
namespace {

constexpr int kConsumerWarps = 4;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kThreads = kConsumerThreads + 32;
constexpr int kCtasPerSm = 2;
constexpr long long kDrainLimitNs = 1000000000LL;
// shared memory one CTA may use when two share an SM (228 KB per SM, 1 KB
// reserved per CTA, a little static shared memory)
constexpr int kCtaSmemBudget = (228 * 1024) / kCtasPerSm - 1024 - 512;

template <int D>
struct Bf16Shape {
    static constexpr int kPageBytes = kPageSize * D * 2;        // one page of one kv head
    static constexpr int kSeg = D * 2 / 128;                     // 128-byte rows per token
    static constexpr int kStageBytes = 2 * kPageBytes;           // K and V of one page
    // combine scratch: [warp][16 rows][D/2 + 8] floats (two column halves)
    static constexpr int kHalf = D / 2;
    static constexpr int kScratchStride = kHalf + 8;
    static constexpr int kCombineBytes = kConsumerWarps * 16 * (kScratchStride * 4 + 8);
    static constexpr int kScratchBytes =
        kCombineBytes > dev::kMergeStageBytes ? kCombineBytes : dev::kMergeStageBytes;
    static constexpr int kBarBytesMax = 2 * 64 * 8;
    static constexpr int kStages =
        (kCtaSmemBudget - kScratchBytes - kBarBytesMax - 1024) / kStageBytes;
    static constexpr int kRingBytes = kStages * kStageBytes;
    static constexpr int kBarBytes = 2 * kStages * 8;
    static constexpr int kSmemBytes = kRingBytes + kScratchBytes + kBarBytes + 1024;
    static_assert(kStages >= 4 && kStages <= 64, "ring depth");
    static_assert(kSmemBytes <= kCtaSmemBudget, "two CTAs per SM must fit");
};

// Online-softmax state of one warp: 16 rows, thread holds rows gid, gid+8.
template <int D>
struct WarpState {
    float o[D / 8][4];
    float m[2];
    float l[2];
};

// One 16-token page: S = Q K^T, online softmax, O += P V.
template <int D>
__device__ __forceinline__ void page_step(uint32_t kbase, uint32_t vbase, int valid,
                                          const uint32_t (&qa)[D / 16][4], WarpState<D> &st,
                                          float scale_log2, int lane) {
    using S = Bf16Shape<D>;
    const int tig = lane & 3;
    const int mi = lane >> 3, r8 = lane & 7;

    // two accumulator pairs (first and second half of d) halve the MMA chain
    float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    float sd[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    {
        const int tok = r8 + ((mi >> 1) << 3);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            const int dch = 2 * ks + (mi & 1);
            const uint32_t row = tok * S::kSeg + (dch >> 3);
            uint32_t b00, b01, b10, b11;
            dev::ldsm_x4(kbase + dev::swz128(row, dch & 7), b00, b01, b10, b11);
            if (ks < D / 32) {
                dev::mma_bf16_16816(sc[0], qa[ks], b00, b01);
                dev::mma_bf16_16816(sc[1], qa[ks], b10, b11);
            } else {
                dev::mma_bf16_16816(sd[0], qa[ks], b00, b01);
                dev::mma_bf16_16816(sd[1], qa[ks], b10, b11);
            }
        }
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) sc[nt][e] += sd[nt][e];
    }

    // online softmax (log2 domain), rows gid (e = 0,1) and gid + 8 (e = 2,3)
    float x[2][4];
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int tok = nt * 8 + 2 * tig + (e & 1);
            x[nt][e] = tok < valid ? sc[nt][e] * scale_log2 : -INFINITY;
        }
    float mx0 = fmaxf(fmaxf(x[0][0], x[0][1]), fmaxf(x[1][0], x[1][1]));
    float mx1 = fmaxf(fmaxf(x[0][2], x[0][3]), fmaxf(x[1][2], x[1][3]));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    // token 0 of every page in a chunk is valid, so mx0/mx1 are finite
    const float mn0 = fmaxf(st.m[0], mx0), mn1 = fmaxf(st.m[1], mx1);
    const float al0 = dev::fast_exp2(st.m[0] - mn0), al1 = dev::fast_exp2(st.m[1] - mn1);
    st.m[0] = mn0;
    st.m[1] = mn1;
    float p[2][4];
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
        p[nt][0] = dev::fast_exp2(x[nt][0] - mn0);
        p[nt][1] = dev::fast_exp2(x[nt][1] - mn0);
        p[nt][2] = dev::fast_exp2(x[nt][2] - mn1);
        p[nt][3] = dev::fast_exp2(x[nt][3] - mn1);
    }
    st.l[0] = st.l[0] * al0 + (p[0][0] + p[0][1] + p[1][0] + p[1][1]);
    st.l[1] = st.l[1] * al1 + (p[0][2] + p[0][3] + p[1][2] + p[1][3]);
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) {
        st.o[dt][0] *= al0;
        st.o[dt][1] *= al0;
        st.o[dt][2] *= al1;
        st.o[dt][3] *= al1;
    }

    // O += P V: P (16 rows x 16 tokens) straight from the S accumulators
    const uint32_t pa[4] = {dev::pack_bf16(p[0][0], p[0][1]), dev::pack_bf16(p[0][2], p[0][3]),
                            dev::pack_bf16(p[1][0], p[1][1]), dev::pack_bf16(p[1][2], p[1][3])};
    // slots past the node's length may hold anything (NaN included): their
    // P is 0, but 0 * NaN is NaN, so their V values are zeroed
    uint32_t keep_lo = 0xffffffffu, keep_hi = 0xffffffffu;
    if (valid < kPageSize) {
        const int t0 = 2 * tig;
        keep_lo = (t0 < valid ? 0x0000ffffu : 0u) | (t0 + 1 < valid ? 0xffff0000u : 0u);
        keep_hi = (t0 + 8 < valid ? 0x0000ffffu : 0u) | (t0 + 9 < valid ? 0xffff0000u : 0u);
    }
    const int vtok = r8 + ((mi & 1) << 3);
#pragma unroll
    for (int dt = 0; dt < D / 8; dt += 2) {
        const int dch = dt + (mi >> 1);
        const uint32_t row = vtok * S::kSeg + (dch >> 3);
        uint32_t v0, v1, v2, v3;
        dev::ldsm_x4_trans(vbase + dev::swz128(row, dch & 7), v0, v1, v2, v3);
        v0 &= keep_lo;
        v1 &= keep_hi;
        v2 &= keep_lo;
        v3 &= keep_hi;
        dev::mma_bf16_16816(st.o[dt], pa, v0, v1);
        dev::mma_bf16_16816(st.o[dt + 1], pa, v2, v3);
    }
}

// Q fragments (A operand, row-major 16 x D) for rows rg*16 + {gid, gid+8}.
template <int D>
__device__ __forceinline__ void load_q_fragments(const AttnArgs &a, const WorkItem &it, int rg,
                                                 int lane, uint32_t (&qa)[D / 16][4]) {
    const int gid = lane >> 2, tig = lane & 3;
    const __nv_bfloat16 *qb = static_cast<const __nv_bfloat16 *>(a.q);
    const __nv_bfloat16 *qrow[2] = {nullptr, nullptr};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int r = rg * 16 + gid + 8 * h;
        if (r < it.nrows) {
            const int nr = it.row0 + r;
            const int leaf = a.dfs_leaf[it.leaf_lo + nr / a.group];
            const int head = it.kv_head * a.group + nr % a.group;
            qrow[h] = qb + (static_cast<int64_t>(leaf) * a.num_q_heads + head) * D;
        }
    }
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int c0 = ks * 16 + 2 * tig;
            qa[ks][h] = qrow[h] ? *reinterpret_cast<const uint32_t *>(qrow[h] + c0) : 0u;
            qa[ks][2 + h] = qrow[h] ? *reinterpret_cast<const uint32_t *>(qrow[h] + c0 + 8) : 0u;
        }
}

// Write the partial (o, m, l) of an item: straight from registers when each
// warp owns its rows, else combining the warps of a row group through shared
// memory, one column half at a time.
template <int D>
__device__ __forceinline__ void write_partials(const AttnArgs &a, const WorkItem &it,
                                               WarpState<D> &st, int tgc, int rg, int warp,
                                               int lane, float *sc_o, float2 *sc_ml) {
    using S = Bf16Shape<D>;
    const int gid = lane >> 2, tig = lane & 3;
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 1);
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 2);
    st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 1);
    st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 2);
    if (tgc == 1) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int r = rg * 16 + gid + 8 * h;
            if (r >= it.nrows) continue;
            const int64_t slot = static_cast<int64_t>(it.slot_base) + it.row0 + r;
            float *dst = a.part_o + slot * D;
#pragma unroll
            for (int dt = 0; dt < D / 8; ++dt)
                *reinterpret_cast<float2 *>(dst + dt * 8 + 2 * tig) =
                    make_float2(st.o[dt][2 * h], st.o[dt][2 * h + 1]);
            if (tig == 0) a.part_ml[slot] = make_float2(st.m[h], st.l[h]);
        }
        return;
    }
    const int tid = threadIdx.x;
    if (tig == 0) {
        sc_ml[warp * 16 + gid] = make_float2(st.m[0], st.l[0]);
        sc_ml[warp * 16 + gid + 8] = make_float2(st.m[1], st.l[1]);
    }
    constexpr int kVec = S::kHalf / 4;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        float *wo = sc_o + warp * 16 * S::kScratchStride;
#pragma unroll
        for (int dt = 0; dt < D / 16; ++dt) {
            const int c = dt * 8 + 2 * tig;
            const int src = half * (D / 16) + dt;
            *reinterpret_cast<float2 *>(wo + gid * S::kScratchStride + c) =
                make_float2(st.o[src][0], st.o[src][1]);
            *reinterpret_cast<float2 *>(wo + (gid + 8) * S::kScratchStride + c) =
                make_float2(st.o[src][2], st.o[src][3]);
        }
        dev::bar_sync<kConsumerThreads>(1);
        for (int idx = tid; idx < it.nrows * kVec; idx += kConsumerThreads) {
            const int r = idx / kVec, c4 = idx % kVec;
            const int grp = r >> 4, rr = r & 15;
            float M = -INFINITY;
            for (int w = 0; w < tgc; ++w) M = fmaxf(M, sc_ml[(grp * tgc + w) * 16 + rr].x);
            float L = 0.f;
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int w = 0; w < tgc; ++w) {
                const int ww = grp * tgc + w;
                const float2 ml = sc_ml[ww * 16 + rr];
                const float sc = dev::fast_exp2(ml.x - M);
                L += sc * ml.y;
                const float4 v = *reinterpret_cast<const float4 *>(
                    sc_o + (ww * 16 + rr) * S::kScratchStride + 4 * c4);
                acc.x += sc * v.x;
                acc.y += sc * v.y;
                acc.z += sc * v.z;
                acc.w += sc * v.w;
            }
            const int64_t slot = static_cast<int64_t>(it.slot_base) + it.row0 + r;
            *reinterpret_cast<float4 *>(a.part_o + slot * D + half * S::kHalf + 4 * c4) = acc;
            if (half == 0 && c4 == 0) a.part_ml[slot] = make_float2(M, L);
        }
        dev::bar_sync<kConsumerThreads>(1);
    }
}

// Persistent kernel: CTA c runs its planner-assigned items back to back.
// Two CTAs of 5 warps per SM: 10 warps over 4 sub-partitions of 16K
// registers allow at most 168 registers per thread.
template <int D>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    attn_bf16_kernel(const __grid_constant__ CUtensorMap tmap_k,
                     const __grid_constant__ CUtensorMap tmap_v, const AttnArgs a) {
    using S = Bf16Shape<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t ring = dev::smem_addr(smem);
    uint8_t *scratch = smem + S::kRingBytes;
    float *sc_o = reinterpret_cast<float *>(scratch);
    float2 *sc_ml = reinterpret_cast<float2 *>(scratch + kConsumerWarps * 16 * S::kScratchStride * 4);
    const uint32_t bar_full = dev::smem_addr(smem + S::kRingBytes + S::kScratchBytes);
    const uint32_t bar_empty = bar_full + S::kStages * 8;
    __shared__ int abort_flag;
    __shared__ int merge_count;
    __shared__ int merge_list[kMaxTileRows + 1];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int i_begin = a.cta_ptr[blockIdx.x], i_end = a.cta_ptr[blockIdx.x + 1];
    auto k_page = [&](int s) { return ring + s * S::kStageBytes; };
    auto v_page = [&](int s) { return ring + s * S::kStageBytes + S::kPageBytes; };

    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int s = 0; s < S::kStages; ++s) {
            dev::mbar_init(bar_full + 8 * s, 1);
            dev::mbar_init(bar_empty + 8 * s, kConsumerWarps);
        }
        dev::fence_mbar_init();
    }
    __syncthreads();

    if (warp == kConsumerWarps) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            dev::prefetch_tensormap(&tmap_k);
            dev::prefetch_tensormap(&tmap_v);
            int last_issue[S::kStages];
            for (int s = 0; s < S::kStages; ++s) last_issue[s] = -1;
            int stage = 0;
            bool ok = true;
            for (int ii = i_begin; ii < i_end && ok; ++ii) {
                const WorkItem it = a.items[a.cta_items[ii]];
                for (int pg = 0; pg < it.num_pages; ++pg, ++stage) {
                    const int s = stage % S::kStages;
                    if (stage >= S::kStages &&
                        !dev::mbar_wait_bounded(bar_empty + 8 * s, ((stage / S::kStages) - 1) & 1,
                                                a.wait_limit_ns, &abort_flag)) {
                        if (!abort_flag) {
                            abort_flag = 1;
                            dev::record_error(a.err, PARASON_ETIMEOUT, kSiteProducerEmpty);
                        }
                        ok = false;
                        break;
                    }
                    if (abort_flag) {
                        ok = false;
                        break;
                    }
                    if ((a.debug_flags & PARASON_DEBUG_SKIP_FIRST_LOAD) && stage == 0) continue;
                    const int page = a.page_ids[it.page_pos + pg];
                    const int row = (page * a.num_kv_heads + it.kv_head) * kPageSize;
                    dev::mbar_arrive_expect_tx(bar_full + 8 * s, S::kStageBytes);
                    dev::tma_load_3d(k_page(s), &tmap_k, 0, 0, row, bar_full + 8 * s);
                    dev::tma_load_3d(v_page(s), &tmap_v, 0, 0, row, bar_full + 8 * s);
                    last_issue[s] = stage;
                }
            }
            // every copy this CTA issued must land before its shared memory goes
            for (int s = 0; s < S::kStages; ++s)
                if (last_issue[s] >= 0)
                    dev::mbar_wait_bounded(bar_full + 8 * s, (last_issue[s] / S::kStages) & 1,
                                           kDrainLimitNs, nullptr);
        }
        return;
    }

    // ---------------------------------------------------------------- consumers
    const int tid = threadIdx.x;                     // 0 .. 127
    if (blockIdx.x == 0 && a.num_empty_leaves > 0)
        dev::write_empty_branches<D>(a, tid, kConsumerThreads);

    int stage = 0;
    for (int ii = i_begin; ii < i_end; ++ii) {
        const WorkItem it = a.items[a.cta_items[ii]];
        const int rgc = it.nrows <= 16 ? 1 : (it.nrows <= 32 ? 2 : 4);
        const int tgc = kConsumerWarps / rgc;
        const int rg = warp / tgc, tg = warp % tgc;

        uint32_t qa[D / 16][4];
        load_q_fragments<D>(a, it, rg, lane, qa);
        WarpState<D> st;
#pragma unroll
        for (int dt = 0; dt < D / 8; ++dt)
            st.o[dt][0] = st.o[dt][1] = st.o[dt][2] = st.o[dt][3] = 0.f;
        st.m[0] = st.m[1] = -INFINITY;
        st.l[0] = st.l[1] = 0.f;

        // page pg is processed by token-group warp pg % tgc of each row group;
        // every warp waits for every page (which keeps the empty barrier's
        // phases exact) and releases it
        bool ok = true;
        for (int pg = 0; pg < it.num_pages; ++pg, ++stage) {
            const int s = stage % S::kStages;
            if (!dev::mbar_wait_bounded(bar_full + 8 * s, (stage / S::kStages) & 1,
                                        a.wait_limit_ns, &abort_flag)) {
                ok = false;
                break;
            }
            if (pg % tgc == tg) {
                const int valid = (pg == it.num_pages - 1) ? it.last_valid : kPageSize;
                page_step<D>(k_page(s), v_page(s), valid, qa, st, a.scale_log2, lane);
            }
            __syncwarp();
            if (lane == 0) dev::mbar_arrive(bar_empty + 8 * s);
        }
        if (!ok && lane == 0 && !abort_flag) {
            abort_flag = 1;
            dev::record_error(a.err, PARASON_ETIMEOUT, kSiteConsumerFull);
        }
        // one decision for all consumer warps, whatever the producer does meanwhile
        if (dev::bar_sync_or<kConsumerThreads>(1, !ok || abort_flag)) break;

        write_partials<D>(a, it, st, tgc, rg, warp, lane, sc_o, sc_ml);

        // ------------------------------- count this item into its branches
        __threadfence();
        dev::bar_sync<kConsumerThreads>(1);
        if (tid == 0) {
            int n = 0;
            const int pos_lo = it.row0 / a.group;
            const int pos_hi = (it.row0 + it.nrows - 1) / a.group;
            for (int pos = pos_lo; pos <= pos_hi; ++pos) {
                const int b = a.dfs_leaf[it.leaf_lo + pos];
                const int idx = b * a.num_kv_heads + it.kv_head;
                if (atomicAdd(a.counters + idx, 1) == a.targets[idx] - 1) {
                    a.counters[idx] = 0;           // ready for the next decode call
                    merge_list[n++] = b;
                }
            }
            __threadfence();
            merge_count = n;
        }
        dev::bar_sync<kConsumerThreads>(1);
        for (int m = 0; m < merge_count; ++m)
            dev::merge_branch_head<D, kConsumerThreads>(a, merge_list[m], it.kv_head, tid, scratch);
    }
}

// Shared memory and carveout are set once per device; returns the number of
// CTAs the hardware keeps resident per SM (the persistent grid's width).
template <int D>
cudaError_t configure(int *ctas_per_sm) {
    using S = Bf16Shape<D>;
    static int configured_device = -1;
    static int resident = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (configured_device != dev) {
        e = cudaFuncSetAttribute(attn_bf16_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 S::kSmemBytes);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(attn_bf16_kernel<D>,
                                 cudaFuncAttributePreferredSharedMemoryCarveout,
                                 cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&resident, attn_bf16_kernel<D>, kThreads,
                                                          S::kSmemBytes);
        if (e != cudaSuccess) return e;
        configured_device = dev;
    }
    if (ctas_per_sm) *ctas_per_sm = resident;
    return cudaSuccess;
}

template <int D>
cudaError_t launch(const AttnArgs &a, const CUtensorMap &tk, const CUtensorMap &tv,
                   cudaStream_t stream) {
    using S = Bf16Shape<D>;
    cudaError_t e = configure<D>(nullptr);
    if (e != cudaSuccess) return e;
    attn_bf16_kernel<D><<<a.num_ctas, kThreads, S::kSmemBytes, stream>>>(tk, tv, a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t attn_bf16_ctas_per_sm(int head_dim, int *ctas_per_sm) {
    if (head_dim == 128) return configure<128>(ctas_per_sm);
    if (head_dim == 64) return configure<64>(ctas_per_sm);
    return cudaErrorNotSupported;
}

cudaError_t launch_attn_bf16(const AttnArgs &a, const CUtensorMap &tk, const CUtensorMap &tv,
                             int head_dim, cudaStream_t stream) {
    if (a.num_items <= 0) return cudaSuccess;
    if (head_dim == 128) return launch<128>(a, tk, tv, stream);
    if (head_dim == 64) return launch<64>(a, tk, tv, stream);
    return cudaErrorNotSupported;
}

}  // namespace parason
