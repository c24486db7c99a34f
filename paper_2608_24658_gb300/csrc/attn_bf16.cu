// attn_bf16.cu -- node-chunk attention for bf16 KV on sm_103a.
//
// One CTA runs one work item: up to 64 stacked query rows (the branches under
// one fork-tree node times the q heads of one kv head) against one chunk of
// that node's pages.  The KV of the chunk is read from HBM exactly once per
// item, whatever the number of rows: this is what turns the shared prefix of
// many Subtask/Trial branches (paper Sec. 3.1, 3.4) into one read.
//
//   warp 4 (producer)   TMA: one 3-D box per (page, kv head) for K and for V,
//                       128-byte swizzle, into a ring of kStages stages of
//                       kStagePages pages, completion on mbarriers.
//   warps 0-3           tensor-core QK^T and PV with mma.sync m16n8k16 (bf16
//                       in, fp32 accumulate) from ldmatrix fragments, online
//                       softmax in registers with quad shuffles.  The warps
//                       split the tile's rows (16 per warp) and, for small
//                       tiles, the chunk's pages; they combine through shared
//                       memory at the end and write the partial (o, m, l).
//
// Scores are kept in the log2 domain: x = sm_scale*log2(e)*<q,k>, so the
// partial is m = max x, l = sum 2^(x-m), o = sum 2^(x-m) v (unnormalised).
#include "device_common.cuh"

namespace parason {
namespace {

constexpr int kConsumerWarps = 4;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kStagePages = 4;
constexpr int kStages = 3;
constexpr long long kDrainLimitNs = 1000000000LL;

template <int D>
struct Bf16Shape {
    static constexpr int kPageBytes = kPageSize * D * 2;        // one page of one kv head
    static constexpr int kSeg = D * 2 / 128;                     // 128-byte rows per token
    static constexpr int kStageBytes = 2 * kStagePages * kPageBytes;
    static constexpr int kRingBytes = kStages * kStageBytes;
    static constexpr int kScratchStride = D + 8;                 // floats per scratch row
    static constexpr int kScratchBytes =
        kConsumerWarps * 16 * (kScratchStride * 4 + 8);
    static_assert(kScratchBytes <= kRingBytes, "combine scratch must fit in the ring");
    static constexpr int kBarBytes = 2 * kStages * 8;
    static constexpr int kSmemBytes = kRingBytes + kBarBytes + 1024;   // + alignment slack
};

// Online-softmax state of one warp: 16 rows, thread holds rows gid, gid+8.
template <int D>
struct WarpState {
    float o[D / 8][4];
    float m[2];
    float l[2];
};

template <int D>
__device__ __forceinline__ void page_step(uint32_t kbase, uint32_t vbase, int valid,
                                          const uint32_t (&qa)[D / 16][4], WarpState<D> &st,
                                          float scale_log2, int lane) {
    using S = Bf16Shape<D>;
    const int tig = lane & 3;
    const int mi = lane >> 3, r8 = lane & 7;

    // S = Q K^T: 16 rows x 16 tokens (two n-tiles of 8 tokens)
    float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    {
        const int tok = r8 + ((mi >> 1) << 3);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            const int dch = 2 * ks + (mi & 1);
            const uint32_t row = tok * S::kSeg + (dch >> 3);
            uint32_t b00, b01, b10, b11;
            dev::ldsm_x4(kbase + dev::swz128(row, dch & 7), b00, b01, b10, b11);
            dev::mma_bf16_16816(sc[0], qa[ks], b00, b01);
            dev::mma_bf16_16816(sc[1], qa[ks], b10, b11);
        }
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

template <int D>
__global__ void __launch_bounds__(kThreads, 2)
    attn_bf16_kernel(const __grid_constant__ CUtensorMap tmap_k,
                     const __grid_constant__ CUtensorMap tmap_v, const AttnArgs a) {
    using S = Bf16Shape<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t ring = dev::smem_addr(smem);
    const uint32_t bar_full = dev::smem_addr(smem + S::kRingBytes);
    const uint32_t bar_empty = bar_full + kStages * 8;
    __shared__ int abort_flag;

    const WorkItem it = a.items[blockIdx.x];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_iters = (it.num_pages + kStagePages - 1) / kStagePages;
    auto k_page = [&](int s, int j) { return ring + s * S::kStageBytes + j * S::kPageBytes; };
    auto v_page = [&](int s, int j) {
        return ring + s * S::kStageBytes + (kStagePages + j) * S::kPageBytes;
    };

    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int s = 0; s < kStages; ++s) {
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
            int last_issue[kStages];
            for (int s = 0; s < kStages; ++s) last_issue[s] = -1;
            for (int i = 0; i < n_iters; ++i) {
                const int s = i % kStages;
                if (i >= kStages &&
                    !dev::mbar_wait_bounded(bar_empty + 8 * s, ((i / kStages) - 1) & 1,
                                            a.wait_limit_ns, &abort_flag)) {
                    if (!abort_flag) {
                        abort_flag = 1;
                        dev::record_error(a.err, PARASON_ETIMEOUT, kSiteProducerEmpty);
                    }
                    break;
                }
                if (abort_flag) break;
                if ((a.debug_flags & PARASON_DEBUG_SKIP_FIRST_LOAD) && i == 0) continue;
                const int p0 = i * kStagePages;
                const int np = min(kStagePages, it.num_pages - p0);
                dev::mbar_arrive_expect_tx(bar_full + 8 * s, np * 2 * S::kPageBytes);
                for (int j = 0; j < np; ++j) {
                    const int page = a.page_ids[it.page_pos + p0 + j];
                    const int row = (page * a.num_kv_heads + it.kv_head) * kPageSize;
                    dev::tma_load_3d(k_page(s, j), &tmap_k, 0, 0, row, bar_full + 8 * s);
                    dev::tma_load_3d(v_page(s, j), &tmap_v, 0, 0, row, bar_full + 8 * s);
                }
                last_issue[s] = i;
            }
            // every copy this CTA issued must land before its shared memory goes
            for (int s = 0; s < kStages; ++s)
                if (last_issue[s] >= 0)
                    dev::mbar_wait_bounded(bar_full + 8 * s, (last_issue[s] / kStages) & 1,
                                           kDrainLimitNs, nullptr);
        }
        return;
    }

    // ---------------------------------------------------------------- consumers
    const int rgc = it.nrows <= 16 ? 1 : (it.nrows <= 32 ? 2 : 4);
    const int tgc = kConsumerWarps / rgc;
    const int rg = warp / tgc, tg = warp % tgc;
    const int gid = lane >> 2, tig = lane & 3;

    // Q fragments (A operand, row-major 16 x D) for rows rg*16 + {gid, gid+8}
    uint32_t qa[D / 16][4];
    {
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

    WarpState<D> st;
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) st.o[dt][0] = st.o[dt][1] = st.o[dt][2] = st.o[dt][3] = 0.f;
    st.m[0] = st.m[1] = -INFINITY;
    st.l[0] = st.l[1] = 0.f;

    bool ok = true;
    for (int i = 0; i < n_iters; ++i) {
        const int s = i % kStages;
        if (!dev::mbar_wait_bounded(bar_full + 8 * s, (i / kStages) & 1, a.wait_limit_ns,
                                    &abort_flag)) {
            ok = false;
            break;
        }
        const int p0 = i * kStagePages;
        const int np = min(kStagePages, it.num_pages - p0);
        for (int j = tg; j < np; j += tgc) {
            const int valid = (p0 + j == it.num_pages - 1) ? it.last_valid : kPageSize;
            page_step<D>(k_page(s, j), v_page(s, j), valid, qa, st, a.scale_log2, lane);
        }
        __syncwarp();
        if (lane == 0) dev::mbar_arrive(bar_empty + 8 * s);
    }
    if (!ok && lane == 0) {
        if (!abort_flag) {
            abort_flag = 1;
            dev::record_error(a.err, PARASON_ETIMEOUT, kSiteConsumerFull);
        }
    }
    // consumers only: the producer warp does not take part
    asm volatile("bar.sync 1, %0;" ::"n"(kConsumerWarps * 32) : "memory");
    if (abort_flag) return;

    // ------------------------------------------- combine the warps of each row group
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 1);
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 2);
    st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 1);
    st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 2);
    float *sc_o = reinterpret_cast<float *>(smem);                       // [warp][16][stride]
    float2 *sc_ml = reinterpret_cast<float2 *>(smem + kConsumerWarps * 16 * S::kScratchStride * 4);
    {
        float *wo = sc_o + warp * 16 * S::kScratchStride;
#pragma unroll
        for (int dt = 0; dt < D / 8; ++dt) {
            const int c = dt * 8 + 2 * tig;
            *reinterpret_cast<float2 *>(wo + gid * S::kScratchStride + c) =
                make_float2(st.o[dt][0], st.o[dt][1]);
            *reinterpret_cast<float2 *>(wo + (gid + 8) * S::kScratchStride + c) =
                make_float2(st.o[dt][2], st.o[dt][3]);
        }
        if (tig == 0) {
            sc_ml[warp * 16 + gid] = make_float2(st.m[0], st.l[0]);
            sc_ml[warp * 16 + gid + 8] = make_float2(st.m[1], st.l[1]);
        }
    }
    asm volatile("bar.sync 1, %0;" ::"n"(kConsumerWarps * 32) : "memory");

    constexpr int kVec = D / 4;    // float4 columns per row
    for (int idx = threadIdx.x; idx < it.nrows * kVec; idx += kConsumerWarps * 32) {
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
            const float4 v = *reinterpret_cast<const float4 *>(sc_o + (ww * 16 + rr) * S::kScratchStride + 4 * c4);
            acc.x += sc * v.x;
            acc.y += sc * v.y;
            acc.z += sc * v.z;
            acc.w += sc * v.w;
        }
        const int64_t slot = static_cast<int64_t>(it.slot_base) + it.row0 + r;
        *reinterpret_cast<float4 *>(a.part_o + slot * D + 4 * c4) = acc;
        if (c4 == 0) a.part_ml[slot] = make_float2(M, L);
    }
}

template <int D>
cudaError_t launch(const AttnArgs &a, const CUtensorMap &tk, const CUtensorMap &tv,
                   cudaStream_t stream) {
    using S = Bf16Shape<D>;
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(attn_bf16_kernel<D>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             S::kSmemBytes);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    attn_bf16_kernel<D><<<a.num_items, kThreads, S::kSmemBytes, stream>>>(tk, tv, a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_attn_bf16(const AttnArgs &a, const CUtensorMap &tk, const CUtensorMap &tv,
                             int head_dim, cudaStream_t stream) {
    if (a.num_items <= 0) return cudaSuccess;
    if (head_dim == 128) return launch<128>(a, tk, tv, stream);
    if (head_dim == 64) return launch<64>(a, tk, tv, stream);
    return cudaErrorNotSupported;
}

}  // namespace parason
