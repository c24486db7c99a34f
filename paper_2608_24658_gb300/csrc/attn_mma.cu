// attn_mma.cu -- fork-tree decode attention for bf16 or e4m3 KV on sm_103a.
//
// One persistent launch, one CTA per SM, two roles (the planner decides how
// many SMs each gets so that both finish together):
//
//  * prefix pass (CTAs [0, num_wide_ctas)): nodes that many branches share
//    (the request prefix, a subtask thread).  Up to 128 query rows -- the
//    branches under the node times the q heads of one kv head -- are stacked
//    into one tile against the node's pages, so the node's KV is read from
//    HBM once for all of them, which is what the shared prefix of
//    Subtask/Trial branches buys (paper Sec. 3.1, 3.4).
//      - head_dim 128 (bf16 or e4m3 KV): a tcgen05 tile (prefix_cta_tc).
//        Warp roles: a scheduler warp stages each item's metadata; a
//        producer warp moves 64-token blocks of K and V by TMA (one 5-D box
//        per column block when the block's 4 pages are consecutive in the
//        pool, else 3-D boxes per page) into a 6-stage ring (with e4m3 KV,
//        4 raw stages and 4 converted ones); one thread issues S = Q K^T and
//        another O += P V as tcgen05.mma with Q, S/P and O in TMEM and K, V
//        from shared memory; 4 softmax warps own one row per thread (TMEM
//        lane) and write P over S; 4 epilogue warps store an item's O and
//        load Q two items ahead (with e4m3 KV they also convert each staged
//        block to f16).
//      - bf16 at head_dim 128, when the planner pairs row tiles: two
//        128-row tiles of a piece against each staged block
//        (prefix_cta_tc_pair), Q in shared memory, each tile's S/P and O in
//        TMEM, so that a block is staged once for 256 rows.
//      - head_dim 64: mma.sync (prefix_cta): a producer warp streams pages
//        into a ring, 8 consumer warps of 16 rows share the pages and combine
//        through shared memory.
//  * suffix pass (the other CTAs, and prefix CTAs once the prefix queue is
//    empty): nodes of at most 16 rows (a branch's own suffix).  Each warp is
//    an independent worker with its own TMA ring that pulls split-K pieces
//    from a queue: no CTA barrier, no cross-warp combine.  QK^T and PV are
//    mma.sync m16n8k16 with fp32 accumulation and a quad-shuffle online
//    softmax; tiles of 5 to 8 rows run the transposed step (S^T = K Q^T),
//    with e4m3 KV two pages per softmax update.  A bf16 page at head_dim 128
//    comes in one TMA box per tensor (the 4-D page maps).
//
// Every item writes a partial (o, m, l) per row.  The merge kernel (merge.cu)
// folds the partials of every branch's path; it is launched as a
// programmatic dependent of this grid.
//
// KV formats:
//  * bf16: fragments by ldmatrix (V transposed by ldmatrix.trans), bf16 MMA.
//  * e4m3 (one fp32 scale per kv head for K and for V): 4- and 16-byte
//    shared loads, every e4m3 pair widened to f16 exactly (cvt.rn.f16x2.
//    e4m3x2), f16 MMA; q is narrowed from bf16 to f16 (exact for |q| in the
//    f16 normal range; a q element that would overflow f16 is reported as
//    PARASON_ERANGE through the plan's error record).  The K scale joins the
//    softmax scale, the V scale multiplies the partial o.  The suffix
//    fragment layouts permute d so that each thread's bytes are contiguous:
//    the 16-row step's QK^T takes d = 16ks + 4t + {0..3} for thread t of a
//    quad, the transposed step's two 16-byte runs per token row, and PV
//    gives each thread one 16-byte chunk of V's columns.
//
// Scores are kept in the log2 domain: x = scale*log2(e)*<q,k>, so a partial
// is m = max x, l = sum 2^(x-m), o = sum 2^(x-m) v (unnormalised).
#include <mutex>

#include "device_common.cuh"
#include "tcgen05.cuh"

namespace parason {
namespace {

constexpr int kConsumerWarps = 8;                          // prefix pass on mma.sync
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kMaxSuffixWarps = 12;                        // suffix pass: warps per CTA, at most
// 12 warps: the suffix pass runs 6, 8 or 12 autonomous warps (by KV type);
// the prefix pass on tcgen05 uses all 12 (softmax 4, epilogue 4, producer,
// S issuer, scheduler, PV issuer), the one on mma.sync 9 (8 consumers and a
// producer)
constexpr int kThreads = 12 * 32;
constexpr long long kDrainLimitNs = 1000000000LL;
constexpr int kSmemBudget = 220 * 1024;                    // dynamic, one CTA per SM
constexpr int kIdSlots = 8;      // prefix-pass item ids in flight from producer to consumers
constexpr int kGrabSlots = 8;    // suffix-pass item ids a warp has pulled but not finished
constexpr float kLazyRescaleLog2 = 8.f;   // mma.sync softmax: move the reference max past 2^8

// KV formats, with the number of suffix-pass warps per CTA (each with a
// private ring; the 192 KB of rings is split between them).  An e4m3 page
// costs more issue per byte (widening to f16), so that pass runs more,
// shallower warps; bf16 with few rows per tile (g <= 4) runs fewer, deeper
// ones, whose extra pages in flight shorten the tail of the launch.
// kStepPages: pages of a suffix item under one softmax update of the
// transposed step (e4m3 pages are cheap to stream and costly to widen: two
// pages per update give each warp two independent MMA chains)
struct KvBf16 {
    static constexpr int kElemBytes = 2;
    static constexpr int kSuffixWarps = 8;
    static constexpr int kStepPages = 1;
};
struct KvBf16Deep {
    static constexpr int kElemBytes = 2;
    static constexpr int kSuffixWarps = 6;
    static constexpr int kStepPages = 1;
};
struct KvE4m3 {
    static constexpr int kElemBytes = 1;
    static constexpr int kSuffixWarps = 12;
    static constexpr int kStepPages = 2;
};

template <int D, class KV>
struct Shape {
    static constexpr int kRowBytes = D * KV::kElemBytes;    // one token of one kv head
    static constexpr int kPageBytes = kPageSize * kRowBytes; // one page of one kv head
    // a page lands as kSeg column blocks of 16 tokens x 128 bytes, so that 8
    // consecutive tokens hit 8 different 128-byte swizzle rows
    static constexpr int kSeg = kRowBytes / 128;
    static constexpr int kSegBytes = kPageSize * 128;
    static constexpr int kStageBytes = 2 * kPageBytes;      // K and V of one page

    // suffix pass: a private ring per warp
    static constexpr int kSuffixWarps = KV::kSuffixWarps;
    static constexpr int kWarpStages = (192 * 1024) / (kSuffixWarps * kStageBytes);
    static constexpr int kWarpRingBytes = kWarpStages * kStageBytes;
    static constexpr int kNarrowBytes = kSuffixWarps * kWarpRingBytes;
    static constexpr int kNarrowBars = kSuffixWarps * kWarpStages;

    // prefix pass: one ring + combine scratch [warp][16 rows][D/2 + 8] floats
    static constexpr int kHalf = D / 2;
    static constexpr int kScratchStride = kHalf + 8;
    static constexpr int kScratchBytes = kConsumerWarps * 16 * (kScratchStride * 4 + 8);
    static constexpr int kWideStages = (kNarrowBytes - kScratchBytes) / kStageBytes;
    static constexpr int kWideRingBytes = kWideStages * kStageBytes;
    static constexpr int kWideBars = 2 * kWideStages;

    // + kIdSlots item-id barriers of the prefix pass, + the tcgen05 tile's 16
    static constexpr int kWideAll = kWideBars + kIdSlots;
    static constexpr int kBars0 = kNarrowBars > kWideAll ? kNarrowBars : kWideAll;
    static constexpr int kBars = kBars0 > 16 + kIdSlots ? kBars0 : 16 + kIdSlots;
    static constexpr int kBodyBytes =
        kNarrowBytes > kWideRingBytes + kScratchBytes ? kNarrowBytes : kWideRingBytes + kScratchBytes;
    static constexpr int kSmemBytes = kBodyBytes + kBars * 8 + 1024;   // + alignment slack
    static_assert(kRowBytes % 128 == 0, "token rows are whole 128-byte blocks");
    static_assert(kWarpStages >= 2, "suffix ring depth");
    static_assert(kSuffixWarps <= kMaxSuffixWarps, "suffix-pass warps fit the item rings");
    static_assert(kWideStages >= 4, "prefix ring depth");
    static_assert(kSmemBytes <= kSmemBudget, "shared memory budget");

};

// K then V of one (page, kv head) into a stage: one TMA box {128 bytes, 1
// block, 16 tokens} per column block and tensor (the prefix pass of the
// mma.sync path; a prefix page may be read again by another row tile of its
// node and keeps the normal L2 policy).
template <int D, class KV>
__device__ __forceinline__ void load_page(uint32_t dst, const CUtensorMap *tmap_k,
                                          const CUtensorMap *tmap_v, int row, uint32_t bar) {
    using S = Shape<D, KV>;
#pragma unroll
    for (int sg = 0; sg < S::kSeg; ++sg) {
        dev::tma_load_3d(dst + sg * S::kSegBytes, tmap_k, 0, sg, row, bar);
        dev::tma_load_3d(dst + S::kPageBytes + sg * S::kSegBytes, tmap_v, 0, sg, row, bar);
    }
}

// The same for a suffix page, in one box per tensor (the page maps) where a
// page has several column blocks: half the copies at head_dim 128 bf16, in
// the same shared-memory layout (same-box A/B: two-level step 81.8 -> 79.6
// us, long prefix 839.6 -> 834.2 us).  A suffix page is read by one item
// only, so its lines go first when L2 needs room (the partials written
// meanwhile stay for the merge).
template <int D, class KV>
__device__ __forceinline__ void load_suffix_page(uint32_t dst, const KvMaps &maps, int row,
                                                 uint32_t bar) {
    using S = Shape<D, KV>;
    const uint64_t pol = dev::l2_evict_first_policy();
    if constexpr (S::kSeg > 1) {
        const int ph = row / kPageSize;
        dev::tma_load_4d_hint(dst, &maps.k_page, 0, 0, 0, ph, bar, pol);
        dev::tma_load_4d_hint(dst + S::kPageBytes, &maps.v_page, 0, 0, 0, ph, bar, pol);
    } else {
        dev::tma_load_3d_hint(dst, &maps.k, 0, 0, row, bar, pol);
        dev::tma_load_3d_hint(dst + S::kPageBytes, &maps.v, 0, 0, row, bar, pol);
    }
}

template <int D>
struct WarpState {
    float o[D / 8][4];
    float m[2];
    float l[2];
};

template <int D>
__device__ __forceinline__ void reset(WarpState<D> &st) {
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) st.o[dt][0] = st.o[dt][1] = st.o[dt][2] = st.o[dt][3] = 0.f;
    st.m[0] = st.m[1] = -INFINITY;
    st.l[0] = st.l[1] = 0.f;
}

// Output column of accumulator o[nt][e] of thread (gid, tig): its row is gid
// (e < 2) or gid + 8, its column below.
template <class KV>
__device__ __forceinline__ int out_col(int nt, int e, int tig) {
    if constexpr (KV::kElemBytes == 2)
        return nt * 8 + 2 * tig + (e & 1);
    else
        return 16 * (2 * tig + (e & 1)) + nt;
}

__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t two_bytes) {
    uint32_t out;
    asm("{\n\t.reg .b16 lo, hi;\n\t"
        "mov.b32 {lo, hi}, %1;\n\t"
        "cvt.rn.f16x2.e4m3x2 %0, lo;\n\t}"
        : "=r"(out)
        : "r"(two_bytes));
    return out;
}

// Four e4m3 values (one word) widened exactly to two f16 pairs: bytes 0-1
// to `lo`, bytes 2-3 to `hi`.
__device__ __forceinline__ void e4m3x4_to_f16x2x2(uint32_t four_bytes, uint32_t &lo, uint32_t &hi) {
    asm("{\n\t.reg .b16 l, h;\n\t"
        "mov.b32 {l, h}, %2;\n\t"
        "cvt.rn.f16x2.e4m3x2 %0, l;\n\t"
        "cvt.rn.f16x2.e4m3x2 %1, h;\n\t}"
        : "=r"(lo), "=r"(hi)
        : "r"(four_bytes));
}

// A bf16 pair of q narrowed to an f16 pair for the e4m3 MMAs.  The f16
// values are exact for |q| < 65504 (tiny values lose low bits); an element
// of magnitude 65520 or more (including inf) would round to inf, so `big` is
// set and the caller reports PARASON_ERANGE rather than returning a silently
// wrong result.  NaN is passed through and not flagged.
__device__ __forceinline__ uint32_t q_pair_to_f16(uint32_t two, bool &big) {
    const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&two);
    const float lo = __low2float(b), hi = __high2float(b);
    big |= fmaxf(fabsf(lo), fabsf(hi)) >= 65520.f;
    return dev::pack_f16(lo, hi);
}

// Record PARASON_ERANGE once per warp if any lane saw an out-of-range q.
__device__ __forceinline__ void report_q_range(const AttnArgs &a, bool big, int lane) {
    if (__any_sync(0xffffffffu, big) && lane == 0) dev::record_error(a.err, PARASON_ERANGE, kSiteQRange);
}

__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(addr));
    return v;
}

// Online softmax over one page's scores s (two n-tiles of 8 tokens), then
// rescale o; returns P packed as the A operand of the PV MMA.
template <int D, class KV>
__device__ __forceinline__ void softmax_page(const float (&sc)[2][4], int valid, float scale_log2,
                                             WarpState<D> &st, int tig, uint32_t (&pa)[4]) {
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
    // token 0 of every page of an item is valid, so mx0/mx1 are finite.
    // Lazy rescale: the reference max m (and with it o and l) moves only when
    // some row's max grows by more than 2^8 (always at an item's first page,
    // where m = -inf); otherwise P = 2^(x - m) stays below 2^8 and o, l keep
    // accumulating against the old m, which the merge takes as it is.
    const bool grow = mx0 > st.m[0] + kLazyRescaleLog2 || mx1 > st.m[1] + kLazyRescaleLog2;
    if (__any_sync(0xffffffffu, grow)) {
        const float mn0 = fmaxf(st.m[0], mx0), mn1 = fmaxf(st.m[1], mx1);
        const float al0 = dev::fast_exp2(st.m[0] - mn0), al1 = dev::fast_exp2(st.m[1] - mn1);
        st.m[0] = mn0;
        st.m[1] = mn1;
        st.l[0] *= al0;
        st.l[1] *= al1;
#pragma unroll
        for (int dt = 0; dt < D / 8; ++dt) {
            st.o[dt][0] *= al0;
            st.o[dt][1] *= al0;
            st.o[dt][2] *= al1;
            st.o[dt][3] *= al1;
        }
    }
    const float mn0 = st.m[0], mn1 = st.m[1];
    float p[2][4];
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
        p[nt][0] = dev::fast_exp2(x[nt][0] - mn0);
        p[nt][1] = dev::fast_exp2(x[nt][1] - mn0);
        p[nt][2] = dev::fast_exp2(x[nt][2] - mn1);
        p[nt][3] = dev::fast_exp2(x[nt][3] - mn1);
    }
    st.l[0] += p[0][0] + p[0][1] + p[1][0] + p[1][1];
    st.l[1] += p[0][2] + p[0][3] + p[1][2] + p[1][3];
    if constexpr (KV::kElemBytes == 2) {
        pa[0] = dev::pack_bf16(p[0][0], p[0][1]);
        pa[1] = dev::pack_bf16(p[0][2], p[0][3]);
        pa[2] = dev::pack_bf16(p[1][0], p[1][1]);
        pa[3] = dev::pack_bf16(p[1][2], p[1][3]);
    } else {
        pa[0] = dev::pack_f16(p[0][0], p[0][1]);
        pa[1] = dev::pack_f16(p[0][2], p[0][3]);
        pa[2] = dev::pack_f16(p[1][0], p[1][1]);
        pa[3] = dev::pack_f16(p[1][2], p[1][3]);
    }
}

// One 16-token page: S = Q K^T, online softmax, O += P V.
template <int D, class KV>
__device__ __forceinline__ void page_step(uint32_t kbase, uint32_t vbase, int valid,
                                          const uint32_t (&qa)[D / 16][4], WarpState<D> &st,
                                          float scale_log2, int lane) {
    using S = Shape<D, KV>;
    const int gid = lane >> 2, tig = lane & 3;
    const int mi = lane >> 3, r8 = lane & 7;

    // two accumulator pairs (first and second half of d) halve the MMA chain
    float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    float sd[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    if constexpr (KV::kElemBytes == 2) {
        const int tok = r8 + ((mi >> 1) << 3);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            const int dch = 2 * ks + (mi & 1);
            uint32_t b00, b01, b10, b11;
            dev::ldsm_x4(kbase + (dch >> 3) * S::kSegBytes + dev::swz128(tok, dch & 7), b00, b01,
                         b10, b11);
            float(&acc)[2][4] = ks < D / 32 ? sc : sd;
            dev::mma_bf16_16816(acc[0], qa[ks], b00, b01);
            dev::mma_bf16_16816(acc[1], qa[ks], b10, b11);
        }
    } else {
        // thread (gid, tig) reads bytes 4tig..4tig+3 of 16-byte chunk ks of token gid
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            float(&acc)[2][4] = ks < D / 32 ? sc : sd;
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                const uint32_t w = lds32(kbase + dev::swz128(nt * 8 + gid, ks) + 4 * tig);
                uint32_t b0, b1;
                e4m3x4_to_f16x2x2(w, b0, b1);
                dev::mma_f16_16816(acc[nt], qa[ks], b0, b1);
            }
        }
    }
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) sc[nt][e] += sd[nt][e];

    uint32_t pa[4];
    softmax_page<D, KV>(sc, valid, scale_log2, st, tig, pa);

    if constexpr (KV::kElemBytes == 2) {
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
            uint32_t v0, v1, v2, v3;
            dev::ldsm_x4_trans(vbase + (dch >> 3) * S::kSegBytes + dev::swz128(vtok, dch & 7), v0,
                               v1, v2, v3);
            v0 &= keep_lo;
            v1 &= keep_hi;
            v2 &= keep_lo;
            v3 &= keep_hi;
            dev::mma_bf16_16816(st.o[dt], pa, v0, v1);
            dev::mma_bf16_16816(st.o[dt + 1], pa, v2, v3);
        }
    } else {
        // thread gid owns output columns 16gid .. 16gid+15: one 16-byte chunk
        // of each of its four tokens 2tig, 2tig+1, 2tig+8, 2tig+9
        static_assert(D == 128, "e4m3 KV path is written for head_dim 128");
        const int t0 = 2 * tig;
        uint4 va = lds128(vbase + dev::swz128(t0, gid));
        uint4 vb = lds128(vbase + dev::swz128(t0 + 1, gid));
        uint4 vc = lds128(vbase + dev::swz128(t0 + 8, gid));
        uint4 vd = lds128(vbase + dev::swz128(t0 + 9, gid));
        if (valid < kPageSize) {
            const uint4 z = make_uint4(0u, 0u, 0u, 0u);
            if (t0 >= valid) va = z;
            if (t0 + 1 >= valid) vb = z;
            if (t0 + 8 >= valid) vc = z;
            if (t0 + 9 >= valid) vd = z;
        }
        const uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
        const uint32_t wc[4] = {vc.x, vc.y, vc.z, vc.w}, wd[4] = {vd.x, vd.y, vd.z, vd.w};
#pragma unroll
        for (int nt = 0; nt < 16; ++nt) {
            const uint32_t sel = (nt & 3) | ((4 + (nt & 3)) << 4);   // byte nt of x, byte nt of y
            const uint32_t lo = __byte_perm(wa[nt >> 2], wb[nt >> 2], sel);
            const uint32_t hi = __byte_perm(wc[nt >> 2], wd[nt >> 2], sel);
            dev::mma_f16_16816(st.o[nt], pa, e4m3x2_to_f16x2(lo), e4m3x2_to_f16x2(hi));
        }
    }
}

// ---------------------------------------------------------------------------
// Transposed page step for tiles of at most 8 rows (a suffix tile holds one
// branch, g <= 8 q heads): S^T = K Q^T and O^T += V^T P^T, so that every
// m16n8k16 MMA runs 16 tokens (or 16 output columns) against the 8 rows,
// instead of 16 rows -- half of them padding -- against 8 tokens: half the
// MMAs of page_step, and half its accumulators.
//   S^T fragment: c0, c1 = token gid, rows 2tig and 2tig + 1; c2, c3 = token
//   gid + 8.  O^T fragment of column tile dt: c0, c1 = column tcol(dt, gid),
//   rows 2tig and 2tig + 1; c2, c3 = column tcol(dt, gid + 8).
// The reduction index d of S^T may be permuted (the same way in K and Q); the
// e4m3 path does so to read 16 bytes of K at a time, and picks its output
// columns so that each lane's columns are one 16-byte chunk of V.
// ---------------------------------------------------------------------------
template <int D>
struct WarpStateT {
    float o[D / 16][4];
    float m[2];        // rows 2tig, 2tig + 1 (equal in the 8 lanes of a tig)
    float l[2];        // this lane's tokens; summed over the lanes at the end
};

template <int D>
__device__ __forceinline__ void reset(WarpStateT<D> &st) {
#pragma unroll
    for (int dt = 0; dt < D / 16; ++dt) st.o[dt][0] = st.o[dt][1] = st.o[dt][2] = st.o[dt][3] = 0.f;
    st.m[0] = st.m[1] = -INFINITY;
    st.l[0] = st.l[1] = 0.f;
}

// output column of O^T row `r` (gid or gid + 8) of column tile dt
template <class KV>
__device__ __forceinline__ int tcol(int dt, int r) {
    if constexpr (KV::kElemBytes == 2)
        return dt * 16 + r;
    else
        return 16 * (r & 7) + 2 * dt + (r >> 3);
}

// Q^T fragments (B operand, d x 8 rows): row gid of the tile, d pairs of
// k-step ks -- (16 ks + 2 tig, 16 ks + 8 + 2 tig) for bf16; for e4m3, widened
// to f16, (e, e + 2) with e = 32 tig + 16 (ks / 4) + 4 (ks % 4), the slice
// that word ks % 4 of the lane's 16-byte K chunk 2 tig + ks / 4 holds
template <int D, class KV>
__device__ __forceinline__ void load_q_fragments_t(const AttnArgs &a, const WorkItem &it, int lane,
                                                   uint32_t (&qb)[D / 16][2]) {
    const int gid = lane >> 2, tig = lane & 3;
    const __nv_bfloat16 *qrow = nullptr;
    if (gid < it.nrows) {
        const int nr = it.row0 + gid;
        const int leaf = a.dfs_leaf[it.leaf_lo + nr / a.group];
        const int head = it.kv_head * a.group + nr % a.group;
        qrow = static_cast<const __nv_bfloat16 *>(a.q) + (static_cast<int64_t>(leaf) * a.num_q_heads + head) * D;
    }
    bool big = false;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
        if constexpr (KV::kElemBytes == 2) {
            qb[ks][0] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + ks * 16 + 2 * tig) : 0u;
            qb[ks][1] = qrow ? *reinterpret_cast<const uint32_t *>(qrow + ks * 16 + 8 + 2 * tig) : 0u;
        } else {
            uint2 u = make_uint2(0u, 0u);
            if (qrow) u = *reinterpret_cast<const uint2 *>(qrow + 32 * tig + 16 * (ks >> 2) + 4 * (ks & 3));
            qb[ks][0] = q_pair_to_f16(u.x, big);
            qb[ks][1] = q_pair_to_f16(u.y, big);
        }
    }
    if constexpr (KV::kElemBytes == 1) report_q_range(a, big, lane);
}

// S^T of one page, unscaled: s[e] for token gid + 8 (e / 2), row 2 tig + e % 2
template <int D, class KV>
__device__ __forceinline__ void scores_t(uint32_t kbase, const uint32_t (&qb)[D / 16][2], int lane,
                                         float (&s)[4]) {
    using S = Shape<D, KV>;
    const int gid = lane >> 2, tig = lane & 3;
    const int mi = lane >> 3, r8 = lane & 7;
    // S^T = K Q^T, two accumulators (first and second half of d)
    float sc[4] = {0.f, 0.f, 0.f, 0.f}, sd[4] = {0.f, 0.f, 0.f, 0.f};
    if constexpr (KV::kElemBytes == 2) {
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            float(&acc)[4] = ks < D / 32 ? sc : sd;
            uint32_t ka[4];
            const int tok = r8 + ((mi & 1) << 3), dch = 2 * ks + (mi >> 1);
            dev::ldsm_x4(kbase + (dch >> 3) * S::kSegBytes + dev::swz128(tok, dch & 7), ka[0], ka[1],
                         ka[2], ka[3]);
            dev::mma_bf16_16816(acc, ka, qb[ks][0], qb[ks][1]);
        }
    } else {
        static_assert(D == 128, "e4m3 KV path is written for head_dim 128");
        // 16-byte chunks 2 tig and 2 tig + 1 of tokens gid and gid + 8 (the
        // eight lanes of a phase read eight distinct swizzled chunks)
        uint4 kg[2], kh[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            kg[j] = lds128(kbase + dev::swz128(gid, 2 * tig + j));
            kh[j] = lds128(kbase + dev::swz128(gid + 8, 2 * tig + j));
        }
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            float(&acc)[4] = ks < D / 32 ? sc : sd;
            const uint4 &g = kg[ks >> 2], &h = kh[ks >> 2];
            const int i = ks & 3;
            const uint32_t w0 = i == 0 ? g.x : i == 1 ? g.y : i == 2 ? g.z : g.w;
            const uint32_t w1 = i == 0 ? h.x : i == 1 ? h.y : i == 2 ? h.z : h.w;
            uint32_t ka[4];
            e4m3x4_to_f16x2x2(w0, ka[0], ka[2]);
            e4m3x4_to_f16x2x2(w1, ka[1], ka[3]);
            dev::mma_f16_16816(acc, ka, qb[ks][0], qb[ks][1]);
        }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) s[e] = sc[e] + sd[e];
}

// O^T += V^T P^T of one page
template <int D, class KV>
__device__ __forceinline__ void pv_t(uint32_t vbase, int valid, uint32_t pb0, uint32_t pb1,
                                     WarpStateT<D> &st, int lane) {
    using S = Shape<D, KV>;
    const int gid = lane >> 2, tig = lane & 3;
    const int mi = lane >> 3, r8 = lane & 7;
    if constexpr (KV::kElemBytes == 2) {
        // slots past the node's length may hold anything (NaN included): V
        // of those tokens is zeroed (this lane's A columns are tokens 2tig,
        // 2tig + 1 and 2tig + 8, 2tig + 9)
        uint32_t keep_lo = 0xffffffffu, keep_hi = 0xffffffffu;
        if (valid < kPageSize) {
            const int t0 = 2 * tig;
            keep_lo = (t0 < valid ? 0x0000ffffu : 0u) | (t0 + 1 < valid ? 0xffff0000u : 0u);
            keep_hi = (t0 + 8 < valid ? 0x0000ffffu : 0u) | (t0 + 9 < valid ? 0xffff0000u : 0u);
        }
        const int vtok = r8 + ((mi >> 1) << 3);
#pragma unroll
        for (int dt = 0; dt < D / 16; ++dt) {
            const int dch = 2 * dt + (mi & 1);
            uint32_t va[4];
            dev::ldsm_x4_trans(vbase + (dch >> 3) * S::kSegBytes + dev::swz128(vtok, dch & 7), va[0],
                               va[1], va[2], va[3]);
            va[0] &= keep_lo;
            va[1] &= keep_lo;
            va[2] &= keep_hi;
            va[3] &= keep_hi;
            dev::mma_bf16_16816(st.o[dt], va, pb0, pb1);
        }
    } else {
        // this lane's output columns are 16 gid .. 16 gid + 15: chunk gid of
        // its four tokens 2tig, 2tig + 1, 2tig + 8, 2tig + 9
        const int t0 = 2 * tig;
        uint4 va = lds128(vbase + dev::swz128(t0, gid));
        uint4 vb = lds128(vbase + dev::swz128(t0 + 1, gid));
        uint4 vc = lds128(vbase + dev::swz128(t0 + 8, gid));
        uint4 vd = lds128(vbase + dev::swz128(t0 + 9, gid));
        if (valid < kPageSize) {
            const uint4 z = make_uint4(0u, 0u, 0u, 0u);
            if (t0 >= valid) va = z;
            if (t0 + 1 >= valid) vb = z;
            if (t0 + 8 >= valid) vc = z;
            if (t0 + 9 >= valid) vd = z;
        }
        const uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
        const uint32_t wc[4] = {vc.x, vc.y, vc.z, vc.w}, wd[4] = {vd.x, vd.y, vd.z, vd.w};
#pragma unroll
        for (int dt = 0; dt < D / 16; ++dt) {
            // columns 16 gid + 2 dt (+1): bytes b, b + 1 of word dt / 2
            const uint32_t b = 2 * (dt & 1);
            const uint32_t sel = b | ((4 + b) << 4) | ((b + 1) << 8) | ((5 + b) << 12);
            const uint32_t lo = __byte_perm(wa[dt >> 1], wb[dt >> 1], sel);   // tokens 2tig, 2tig+1
            const uint32_t hi = __byte_perm(wc[dt >> 1], wd[dt >> 1], sel);   // tokens 2tig+8, 2tig+9
            uint32_t a4[4];
            e4m3x4_to_f16x2x2(lo, a4[0], a4[1]);   // columns 16 gid + 2 dt, + 1
            e4m3x4_to_f16x2x2(hi, a4[2], a4[3]);
            dev::mma_f16_16816(st.o[dt], a4, pb0, pb1);
        }
    }
}

// NP consecutive pages of one item under one online-softmax update (their
// scores share the row maxima, the rescale and the shuffles); all pages but
// the last are full.
template <int D, class KV, int NP>
__device__ __forceinline__ void pages_step_t(const uint32_t *kbase, const uint32_t *vbase,
                                             int valid_last, const uint32_t (&qb)[D / 16][2],
                                             WarpStateT<D> &st, float scale_log2, int lane) {
    const int gid = lane >> 2;
    float x[NP][4];
#pragma unroll
    for (int p = 0; p < NP; ++p) {
        float sp[4];
        scores_t<D, KV>(kbase[p], qb, lane, sp);
        const int valid = p == NP - 1 ? valid_last : kPageSize;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int tok = gid + ((e >> 1) << 3);
            x[p][e] = tok < valid ? sp[e] * scale_log2 : -INFINITY;
        }
    }
    // row maxima over the pages' tokens: the 8 lanes of a tig
    float mx0 = fmaxf(x[0][0], x[0][2]), mx1 = fmaxf(x[0][1], x[0][3]);
#pragma unroll
    for (int p = 1; p < NP; ++p) {
        mx0 = fmaxf(mx0, fmaxf(x[p][0], x[p][2]));
        mx1 = fmaxf(mx1, fmaxf(x[p][1], x[p][3]));
    }
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
    }
    // (token 0 of every page of an item is valid: the maxima are finite)
    const bool grow = mx0 > st.m[0] + kLazyRescaleLog2 || mx1 > st.m[1] + kLazyRescaleLog2;
    if (__any_sync(0xffffffffu, grow)) {
        const float mn0 = fmaxf(st.m[0], mx0), mn1 = fmaxf(st.m[1], mx1);
        const float al0 = dev::fast_exp2(st.m[0] - mn0), al1 = dev::fast_exp2(st.m[1] - mn1);
        st.m[0] = mn0;
        st.m[1] = mn1;
        st.l[0] *= al0;
        st.l[1] *= al1;
#pragma unroll
        for (int dt = 0; dt < D / 16; ++dt) {
            st.o[dt][0] *= al0;
            st.o[dt][1] *= al1;
            st.o[dt][2] *= al0;
            st.o[dt][3] *= al1;
        }
    }
#pragma unroll
    for (int p = 0; p < NP; ++p) {
        const float p0 = dev::fast_exp2(x[p][0] - st.m[0]), p1 = dev::fast_exp2(x[p][1] - st.m[1]);
        const float p2 = dev::fast_exp2(x[p][2] - st.m[0]), p3 = dev::fast_exp2(x[p][3] - st.m[1]);
        st.l[0] += p0 + p2;
        st.l[1] += p1 + p3;
        // P^T as the B operand (tokens x rows): transpose the two 8 x 8 halves
        uint32_t pb0, pb1;
        if constexpr (KV::kElemBytes == 2) {
            pb0 = dev::movmatrix_trans(dev::pack_bf16(p0, p1));
            pb1 = dev::movmatrix_trans(dev::pack_bf16(p2, p3));
        } else {
            pb0 = dev::movmatrix_trans(dev::pack_f16(p0, p1));
            pb1 = dev::movmatrix_trans(dev::pack_f16(p2, p3));
        }
        pv_t<D, KV>(vbase[p], p == NP - 1 ? valid_last : kPageSize, pb0, pb1, st, lane);
    }
}

// Q fragments (A operand, row-major 16 x D) for tile rows rg*16 + {gid, gid+8}:
// bf16 as stored, or widened to f16 with d permuted as the e4m3 QK^T wants.
template <int D, class KV>
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
    bool big = false;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            if constexpr (KV::kElemBytes == 2) {
                const int c0 = ks * 16 + 2 * tig;
                qa[ks][h] = qrow[h] ? *reinterpret_cast<const uint32_t *>(qrow[h] + c0) : 0u;
                qa[ks][2 + h] = qrow[h] ? *reinterpret_cast<const uint32_t *>(qrow[h] + c0 + 8) : 0u;
            } else {
                uint2 u = make_uint2(0u, 0u);
                if (qrow[h]) u = *reinterpret_cast<const uint2 *>(qrow[h] + ks * 16 + 4 * tig);
                qa[ks][h] = q_pair_to_f16(u.x, big);
                qa[ks][2 + h] = q_pair_to_f16(u.y, big);
            }
        }
    if constexpr (KV::kElemBytes == 1) report_q_range(a, big, lane);
}

// Softmax scale of an item and the factor of its partial o (the kv head's
// e4m3 scales for K and V; 1 for bf16).
template <class KV>
__device__ __forceinline__ float2 item_scales(const AttnArgs &a, const WorkItem &it) {
    if constexpr (KV::kElemBytes == 2)
        return make_float2(a.scale_log2, 1.f);
    else
        return make_float2(a.scale_log2 * a.k_scale[it.kv_head], a.v_scale[it.kv_head]);
}

// A warp that owns rows rg*16 .. rg*16+15 of an item writes their partials
// straight from registers.
template <int D, class KV>
__device__ __forceinline__ void store_warp_partials(const AttnArgs &a, const WorkItem &it,
                                                    WarpState<D> &st, int rg, int lane,
                                                    float o_scale) {
    const int gid = lane >> 2, tig = lane & 3;
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 1);
    st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 2);
    st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 1);
    st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 2);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int r = rg * 16 + gid + 8 * h;
        if (r >= it.nrows) continue;
        const int64_t slot = static_cast<int64_t>(it.slot_base) + r;
        float *dst = a.part_o + slot * D;
#pragma unroll
        for (int dt = 0; dt < D / 8; ++dt) {
            if constexpr (KV::kElemBytes == 2) {
                *reinterpret_cast<float2 *>(dst + dt * 8 + 2 * tig) =
                    make_float2(st.o[dt][2 * h], st.o[dt][2 * h + 1]);
            } else {
                dst[out_col<KV>(dt, 0, tig)] = st.o[dt][2 * h] * o_scale;
                dst[out_col<KV>(dt, 1, tig)] = st.o[dt][2 * h + 1] * o_scale;
            }
        }
        if (tig == 0) a.part_ml[slot] = make_float2(st.m[h], st.l[h]);
    }
}

// The same for the transposed state: the lanes of a tig hold its two rows.
template <int D, class KV>
__device__ __forceinline__ void store_warp_partials_t(const AttnArgs &a, const WorkItem &it,
                                                      WarpStateT<D> &st, int lane, float o_scale) {
    const int gid = lane >> 2, tig = lane & 3;
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
        st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], o);
        st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], o);
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int r = 2 * tig + h;
        if (r >= it.nrows) continue;
        const int64_t slot = static_cast<int64_t>(it.slot_base) + r;
        float *dst = a.part_o + slot * D;
#pragma unroll
        for (int dt = 0; dt < D / 16; ++dt) {
            if constexpr (KV::kElemBytes == 2) {
                dst[tcol<KV>(dt, gid)] = st.o[dt][h];
                dst[tcol<KV>(dt, gid + 8)] = st.o[dt][2 + h];
            } else {
                // columns 16 gid + 2 dt and the next: one pair
                *reinterpret_cast<float2 *>(dst + tcol<KV>(dt, gid)) =
                    make_float2(st.o[dt][h] * o_scale, st.o[dt][2 + h] * o_scale);
            }
        }
        if (gid == 0) a.part_ml[slot] = make_float2(st.m[h], st.l[h]);
    }
}

// Work queues.  A queue position is taken with one atomicAdd; items are
// numbered in pull order, so position k of the prefix queue is item k and
// position k of the suffix queue item num_wide_items + k.  The merge kernel
// rewinds both counters after every launch.
__device__ __forceinline__ int queue_item(const AttnArgs &a, int which, int k) {
    if (which == 0) return k < a.num_wide_items ? k : -1;
    return k < a.num_narrow_items ? a.num_wide_items + k : -1;
}

__device__ __forceinline__ int pull(const AttnArgs &a, int which, int lane) {
    int id = -1;
    if (lane == 0) id = queue_item(a, which, atomicAdd(a.queue_next + which, 1));
    return __shfl_sync(0xffffffffu, id, 0);
}

// The TMA rows of one item's pages, read by one whole warp 32 at a time: lane
// i holds row base + i; row(pg) returns the row of page pg (pg uniform over
// the warp, nondecreasing within an item).
struct ItemRows {
    const int32_t *rows = nullptr;
    int base = -1;
    int win = 0;
    __device__ void start(const AttnArgs &a, int item) {
        rows = a.stream_rows + a.item_rows[item];
        base = -1;
    }
    __device__ __forceinline__ int row(int pg, int lane) {
        if (base < 0 || pg >= base + 32) {
            base = pg & ~31;
            win = rows[base + lane];        // the row array is padded by 32 entries
        }
        return __shfl_sync(0xffffffffu, win, pg - base);
    }
};

// ---------------------------------------------------------------------------
// suffix pass: every warp pulls items from the suffix queue and streams their
// pages through its own ring
// ---------------------------------------------------------------------------
template <int D, class KV>
__device__ void suffix_warp(const KvMaps &maps, const AttnArgs &a, uint32_t ring, uint32_t bars,
                            int warp, int lane, WorkItem *grab) {
    using S = Shape<D, KV>;
    constexpr int NS = S::kWarpStages;
    const uint32_t my_ring = ring + warp * S::kWarpRingBytes;
    const uint32_t my_bar = bars + warp * NS * 8;
    const bool skip_first = (a.debug_flags & PARASON_DEBUG_SKIP_FIRST_LOAD) && warp == 0 &&
                            static_cast<int>(blockIdx.x) >= a.num_wide_ctas;

    // Issue side (whole warp, uniform).  The next item is fetched in steps
    // spread over the current item's last pages -- claim a queue position,
    // then read the item's record, then switch to it -- so that no step waits
    // on the one before: the warp keeps streaming while they complete, and
    // holds no more than one item beyond the one it is issuing.
    constexpr int kFetchPages = 2;
    int pulled = 0, iss_pg = 0, iss_np = 0, issued = 0;
    bool iss_done = false;
    int fetch = 0;                   // 0: idle, 1: position claimed, 2: record requested
    // lane 0: the claimed queue position.  Warp w of suffix CTA c owns
    // position w * Nc + c (Nc suffix CTAs): consecutive positions, often
    // neighbouring pieces of one run, start on different SMs instead of all
    // on one (same-box A/B: the Llama-3-shape step 40.1 -> 39.7 us, the
    // other workloads level)
    const int own_first = static_cast<int>(blockIdx.x) - a.num_wide_ctas;
    int claimed = own_first >= 0 ? warp * (a.num_ctas - a.num_wide_ctas) + own_first : -1;
    int nxt_id = -1;
    int32_t nxt_w = 0;               // lane i: word i of the next item's record
    int32_t cur_w = 0;               // lane i: word i of the current item's record
    int rows_off = 0, win_base = -1;
    int32_t win = 0;
    auto fetch_step = [&]() {
        if (fetch == 0) {
            if (lane == 0 && (pulled > 0 || claimed < 0)) claimed = atomicAdd(a.queue_next + 1, 1);
            fetch = 1;
        } else if (fetch == 1) {
            int id = -1;
            if (lane == 0) id = queue_item(a, 1, claimed);
            nxt_id = __shfl_sync(0xffffffffu, id, 0);
            if (nxt_id >= 0) nxt_w = a.item_rec[static_cast<int64_t>(nxt_id) * kRecWords + lane];
            fetch = 2;
        }
    };
    // TMA row of page pg of the current item: from the record, then from the
    // page stream 32 rows at a time (the stream is padded by 32 entries)
    auto row_of = [&](int pg) {
        if (pg < kRecRows) return __shfl_sync(0xffffffffu, cur_w, kRecRow0 + pg);
        const int base = kRecRows + ((pg - kRecRows) & ~31);
        if (base != win_base) {
            win = a.stream_rows[rows_off + base + lane];
            win_base = base;
        }
        return __shfl_sync(0xffffffffu, win, pg - base);
    };
    auto issue_next = [&]() {
        if (iss_done) return;
        if (iss_pg + kFetchPages >= iss_np) fetch_step();
        while (iss_pg >= iss_np) {
            while (fetch < 2) fetch_step();
            if (nxt_id < 0) {
                iss_done = true;
                return;
            }
            cur_w = nxt_w;
            fetch = 0;
            iss_np = __shfl_sync(0xffffffffu, cur_w, 1);          // WorkItem::num_pages
            rows_off = __shfl_sync(0xffffffffu, cur_w, kRecRowsOff);
            win_base = -1;
            iss_pg = 0;
            // hand the item to the consume side
            if (lane < 8) reinterpret_cast<int32_t *>(grab + pulled % kGrabSlots)[lane] = cur_w;
            ++pulled;
        }
        const int row = row_of(iss_pg);
        if (lane == 0 && !(skip_first && issued == 0)) {
            const int s = issued % NS;
            const uint32_t bar = my_bar + s * 8;
            dev::mbar_arrive_expect_tx(bar, S::kStageBytes);
            load_suffix_page<D, KV>(my_ring + s * S::kStageBytes, maps, row, bar);
        }
        ++iss_pg;
        ++issued;
    };
    for (int i = 0; i < NS; ++i) issue_next();

    // consume side: the pulled items in order
    int consumed = 0;
    bool ok = true;
    for (int k = 0; consumed < issued && ok; ++k) {
        __syncwarp();
        const WorkItem it = grab[k % kGrabSlots];
        const float2 scl = item_scales<KV>(a, it);
        if (it.nrows > 4 && it.nrows <= 8) {
            // one branch of 5 to 8 q heads: the transposed step (tiles of up
            // to 4 rows measured faster, at the tail, with the 16-row step)
            uint32_t qb[D / 16][2];
            load_q_fragments_t<D, KV>(a, it, lane, qb);
            WarpStateT<D> st;
            reset<D>(st);
            for (int pg = 0; pg < it.num_pages;) {
                // kStepPages pages per softmax update while the item has them
                const int np = it.num_pages - pg >= KV::kStepPages ? KV::kStepPages : 1;
                uint32_t kb[KV::kStepPages], vb[KV::kStepPages];
#pragma unroll
                for (int p = 0; p < KV::kStepPages; ++p) {
                    const int c = consumed + (p < np ? p : 0);
                    const int s = c % NS;
                    kb[p] = my_ring + s * S::kStageBytes;
                    vb[p] = kb[p] + S::kPageBytes;
                    if (p < np && !dev::mbar_wait_bounded(my_bar + s * 8, (c / NS) & 1,
                                                          a.wait_limit_ns, nullptr))
                        ok = false;
                }
                if (!ok) break;
                const int valid = pg + np == it.num_pages ? it.last_valid : kPageSize;
                if (KV::kStepPages > 1 && np == KV::kStepPages)
                    pages_step_t<D, KV, KV::kStepPages>(kb, vb, valid, qb, st, scl.x, lane);
                else
                    pages_step_t<D, KV, 1>(kb, vb, valid, qb, st, scl.x, lane);
                __syncwarp();
                for (int p = 0; p < np; ++p) issue_next();
                pg += np;
                consumed += np;
            }
            if (!ok) break;
            store_warp_partials_t<D, KV>(a, it, st, lane, scl.y);
            continue;
        }
        uint32_t qa[D / 16][4];
        load_q_fragments<D, KV>(a, it, 0, lane, qa);
        WarpState<D> st;
        reset<D>(st);
        for (int pg = 0; pg < it.num_pages; ++pg, ++consumed) {
            const int s = consumed % NS;
            if (!dev::mbar_wait_bounded(my_bar + s * 8, (consumed / NS) & 1, a.wait_limit_ns,
                                        nullptr)) {
                ok = false;
                break;
            }
            const int valid = (pg == it.num_pages - 1) ? it.last_valid : kPageSize;
            page_step<D, KV>(my_ring + s * S::kStageBytes,
                             my_ring + s * S::kStageBytes + S::kPageBytes, valid, qa, st, scl.x,
                             lane);
            // refill this slot: its shared-memory reads are complete, since
            // every MMA that consumed them has issued (in order) before this point
            __syncwarp();
            issue_next();
        }
        if (!ok) break;
        store_warp_partials<D, KV>(a, it, st, 0, lane, scl.y);
    }
    if (!ok && lane == 0) dev::record_error(a.err, PARASON_ETIMEOUT, kSiteConsumerFull);
    // copies still in flight must land before the CTA's shared memory goes
    if (lane == 0) {
        for (int q = consumed; q < issued; ++q) {
            if (skip_first && q == 0) continue;
            dev::mbar_wait_bounded(my_bar + (q % NS) * 8, (q / NS) & 1, kDrainLimitNs, nullptr);
        }
    }
    __syncwarp();
}

// Prefix pass: the producer warp pulls items and hands their ids to the
// consumer warps through kIdSlots shared slots, each with an mbarrier (id -1
// ends the queue).  The producer is never more than a few items ahead of the
// slowest consumer (it waits for ring stages they release), so the slots
// are never overwritten before they are read.
__device__ __forceinline__ void publish_id(volatile int *slots, uint32_t id_bars, int k, int id) {
    slots[k % kIdSlots] = id;
    dev::mbar_arrive(id_bars + 8 * (k % kIdSlots));
}

__device__ __forceinline__ int take_id(const volatile int *slots, uint32_t id_bars, int k,
                                       long long limit, volatile int *abort, bool *ok) {
    if (!dev::mbar_wait_bounded(id_bars + 8 * (k % kIdSlots), (k / kIdSlots) & 1, limit, abort)) {
        *ok = false;
        return -1;
    }
    return slots[k % kIdSlots];
}

// ---------------------------------------------------------------------------
// prefix pass: up to 128 stacked rows share one page stream
// ---------------------------------------------------------------------------
template <int D, class KV>
__device__ void prefix_cta(const CUtensorMap *tmap_k, const CUtensorMap *tmap_v,
                           const AttnArgs &a, uint8_t *smem, uint32_t ring, uint32_t bars,
                           int warp, int lane, volatile int *abort_flag, volatile int *id_slots) {
    using S = Shape<D, KV>;
    constexpr int NS = S::kWideStages;
    const uint32_t bar_full = bars, bar_empty = bars + NS * 8;
    const uint32_t id_bars = bars + 2 * NS * 8;
    auto k_page = [&](int s) { return ring + s * S::kStageBytes; };

    if (warp == kConsumerWarps) {
        // ------------------------------------------------------------ producer
        // the whole warp pulls items and walks their pages; lane 0 waits and issues
        int last_issue[NS];
        for (int s = 0; s < NS; ++s) last_issue[s] = -1;
        const bool skip_first = a.debug_flags & PARASON_DEBUG_SKIP_FIRST_LOAD;
        int stage = 0;
        bool go = true;
        for (int k = 0; go; ++k) {
            // a prefix CTA owns position blockIdx.x of the prefix queue
            const int id = *abort_flag ? -1
                                       : (k == 0 ? queue_item(a, 0, static_cast<int>(blockIdx.x))
                                                 : pull(a, 0, lane));
            if (lane == 0) publish_id(id_slots, id_bars, k, id);
            if (id < 0) break;
            ItemRows rows;
            rows.start(a, id);
            const int np = a.items[id].num_pages;
            for (int pg = 0; pg < np; ++pg, ++stage) {
                const int s = stage % NS;
                int stop = 0;
                if (lane == 0) {
                    if (stage >= NS && !dev::mbar_wait_bounded(bar_empty + 8 * s,
                                                               ((stage / NS) - 1) & 1,
                                                               a.wait_limit_ns, abort_flag)) {
                        if (!*abort_flag) {
                            *abort_flag = 1;
                            dev::record_error(a.err, PARASON_ETIMEOUT, kSiteProducerEmpty);
                        }
                        stop = 1;
                    } else if (*abort_flag) {
                        stop = 1;
                    }
                }
                if (__shfl_sync(0xffffffffu, stop, 0)) {
                    go = false;
                    break;
                }
                const int row = rows.row(pg, lane);
                if (lane == 0 && !(skip_first && stage == 0)) {
                    dev::mbar_arrive_expect_tx(bar_full + 8 * s, S::kStageBytes);
                    load_page<D, KV>(k_page(s), tmap_k, tmap_v, row, bar_full + 8 * s);
                    last_issue[s] = stage;
                }
            }
        }
        // every copy this CTA issued must land before its shared memory goes
        if (lane == 0)
            for (int s = 0; s < NS; ++s)
                if (last_issue[s] >= 0)
                    dev::mbar_wait_bounded(bar_full + 8 * s, (last_issue[s] / NS) & 1, kDrainLimitNs,
                                           nullptr);
        return;
    }
    if (warp > kConsumerWarps) return;

    // ---------------------------------------------------------------- consumers
    uint8_t *scratch = smem + S::kWideRingBytes;
    float *sc_o = reinterpret_cast<float *>(scratch);
    float2 *sc_ml = reinterpret_cast<float2 *>(scratch + kConsumerWarps * 16 * S::kScratchStride * 4);
    const int tid = threadIdx.x;
    const int gid = lane >> 2, tig = lane & 3;
    int stage = 0;
    for (int k = 0;; ++k) {
        bool got = true;
        const int id = take_id(id_slots, id_bars, k, a.wait_limit_ns, abort_flag, &got);
        if (dev::bar_sync_or<kConsumerThreads>(1, !got || id < 0)) break;
        const WorkItem it = a.items[id];
        const float2 scl = item_scales<KV>(a, it);
        const int groups = (it.nrows + 15) >> 4;
        const int rgc = groups <= 2 ? 2 : (groups <= 4 ? 4 : 8);
        const int tgc = kConsumerWarps / rgc;
        const int rg = warp / tgc, tg = warp % tgc;
        const bool has_rows = rg * 16 < it.nrows;

        uint32_t qa[D / 16][4];
        load_q_fragments<D, KV>(a, it, rg, lane, qa);
        WarpState<D> st;
        reset<D>(st);

        // page pg goes to token-group warp pg % tgc of each row group; every
        // warp waits for every page (keeping the empty barrier's phases exact)
        // and releases it
        bool ok = true;
        for (int pg = 0; pg < it.num_pages; ++pg, ++stage) {
            const int s = stage % NS;
            if (!dev::mbar_wait_bounded(bar_full + 8 * s, (stage / NS) & 1, a.wait_limit_ns,
                                        abort_flag)) {
                ok = false;
                break;
            }
            if (has_rows && pg % tgc == tg) {
                const int valid = (pg == it.num_pages - 1) ? it.last_valid : kPageSize;
                page_step<D, KV>(k_page(s), k_page(s) + S::kPageBytes, valid, qa, st, scl.x, lane);
            }
            __syncwarp();
            if (lane == 0) dev::mbar_arrive(bar_empty + 8 * s);
        }
        if (!ok && lane == 0 && !*abort_flag) {
            *abort_flag = 1;
            dev::record_error(a.err, PARASON_ETIMEOUT, kSiteConsumerFull);
        }
        // one decision for all consumer warps, whatever the producer does meanwhile
        if (dev::bar_sync_or<kConsumerThreads>(1, !ok || *abort_flag)) break;

        if (tgc == 1) {
            if (has_rows) store_warp_partials<D, KV>(a, it, st, rg, lane, scl.y);
            continue;
        }
        // combine the token-group warps of each row group, one column half at a time
        st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 1);
        st.l[0] += __shfl_xor_sync(0xffffffffu, st.l[0], 2);
        st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 1);
        st.l[1] += __shfl_xor_sync(0xffffffffu, st.l[1], 2);
        if (tig == 0) {
            sc_ml[warp * 16 + gid] = make_float2(st.m[0], st.l[0]);
            sc_ml[warp * 16 + gid + 8] = make_float2(st.m[1], st.l[1]);
        }
        constexpr int kVec = S::kHalf / 4;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            float *wo = sc_o + warp * 16 * S::kScratchStride;
#pragma unroll
            for (int dt = 0; dt < D / 8; ++dt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int col = out_col<KV>(dt, e, tig);
                    if (col / S::kHalf == half)
                        wo[(gid + 8 * (e >> 1)) * S::kScratchStride + col % S::kHalf] =
                            st.o[dt][e] * scl.y;
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
                const int64_t slot = static_cast<int64_t>(it.slot_base) + r;
                *reinterpret_cast<float4 *>(a.part_o + slot * D + half * S::kHalf + 4 * c4) = acc;
                if (half == 0 && c4 == 0) a.part_ml[slot] = make_float2(M, L);
            }
            dev::bar_sync<kConsumerThreads>(1);
        }
    }
}


// ---------------------------------------------------------------------------
// prefix pass on tcgen05 (bf16 or e4m3 KV, head_dim 128): a tile of up to 128
// stacked rows against 64-token blocks (4 pages) of the node's pages
//
//   warp 10     scheduler: pulls items from the prefix queue and stages each
//               one's metadata (the item, the TMA row of each page, the
//               branch of each group of g rows) in one of kTcMeta shared
//               slots, so that no other role waits on a dependent chain of
//               global loads when it moves to the next item
//   warp 8      producer: TMA of K and V, one block per ring stage: one box
//               per column block of K and of V when the block's 4 pages are
//               consecutive in the pool (the 5-D run maps), else one per
//               page and column block; pages past the item's end are loaded
//               from an out-of-range row, which TMA fills with zeros
//   warp 9      S issuer (one thread): S = Q K^T (M 128, N 64, K 128) into
//               one of two TMEM buffers, once PV of the block two back has
//               freed it; runs ahead across item boundaries
//   warp 11     PV issuer (one thread): O += P V (M 128, N 128, K 64) into
//               the item's TMEM accumulator (two, alternating by item).
//               A (Q or P) comes from TMEM, B (K or V) from shared memory.
//               tcgen05.commit releases ring stages and signals completion.
//   warps 0-3   softmax: thread r owns row r (TMEM lane r); online softmax in
//               the log2 domain with a lazy rescale of O (only when a row's
//               max grows by more than 2^8); P (bf16, f16 with e4m3 KV)
//               overwrites the first 32 columns of its S buffer, the A
//               operand of PV; writes the row's (m, l) at the end of an item
//   warps 4-7   epilogue: once an item's O is complete, stores its rows to the
//               partials and loads the Q rows of the item two ahead into the
//               TMEM Q buffer that item frees (Q of items 0 and 1 at start);
//               with e4m3 KV they also convert every staged block to f16
//
// TMEM, 512 columns: O[2] at 0 and 128, S/P[2] at 256 and 320, Q[2] at 384
// and 448.  Shared memory: the ring [6][K: 2 col blocks x 64 tokens x 128 B |
// V: same], 128-byte swizzled (K-major descriptors for K, MN-major for V),
// and the metadata slots; with e4m3 KV the first 64 KB stage the raw blocks
// (4 x 16 KB) and the next 128 KB hold 4 converted f16 blocks.
// ---------------------------------------------------------------------------
constexpr int kTcRows = 128;
constexpr int kTcBlockPages = 4;
constexpr int kTcBlockTokens = kTcBlockPages * kPageSize;    // 64
static_assert(kTcRunPages == kTcBlockPages, "a run box holds one block's pages");
constexpr int kTcStages = 6;
constexpr int kTcColBlockBytes = kTcBlockTokens * 128;        // 8 KB: 64 tokens x 128 B
constexpr int kTcKBytes = 2 * kTcColBlockBytes;               // d = 128: two column blocks
constexpr int kTcStageBytes = 2 * kTcKBytes;                  // K + V
constexpr int kTcRingBytes = kTcStages * kTcStageBytes;       // 192 KB
// e4m3 KV: TMA stages the raw bytes (K and V of a block, 64 rows of 128 B
// each: 16 KB) in kTcF8Stages stages; the epilogue warps convert each block
// to f16 (exactly) into kTcCvStages stages laid out like a bf16 stage.
constexpr int kTcF8Bytes = kTcBlockTokens * 128;              // 8 KB: K (or V) of a block
constexpr int kTcF8StageBytes = 2 * kTcF8Bytes;
constexpr int kTcF8Stages = 4;                                 // raw e4m3 stages
constexpr int kTcCvStages = 4;
constexpr int kTcCvOffset = kTcF8Stages * kTcF8StageBytes;    // 64 KB
static_assert(kTcF8Stages <= kTcStages, "raw e4m3 stages use the ring's barriers");
static_assert(kTcCvOffset + kTcCvStages * kTcStageBytes <= kTcRingBytes, "e4m3 rings fit");
constexpr int kTcTmemCols = 512;
constexpr uint32_t kTmemO = 0, kTmemS = 256, kTmemQ = 384;    // TMEM column bases
constexpr float kTcRescaleLog2 = 8.f;                         // lazy rescale threshold
constexpr int kTcMeta = 4;                                    // item metadata slots
constexpr int kTcMetaPages = 512;                             // pages of one item at most
constexpr int kTcSoftmaxWarps = 4;                            // warps 0-3
constexpr int kTcEpilogueWarp = 4;                            // warps 4-7
constexpr int kTcProducerWarp = 8;
constexpr int kTcMmaWarp = 9;
constexpr int kTcSchedulerWarp = 10;
constexpr int kTcPvWarp = 11;
static_assert(kTcRingBytes <= Shape<128, KvBf16>::kBodyBytes, "tcgen05 ring fits the CTA's memory");
static_assert(kTcRingBytes <= Shape<128, KvBf16Deep>::kBodyBytes, "tcgen05 ring fits the CTA's memory");
static_assert(kTcRingBytes <= Shape<128, KvE4m3>::kBodyBytes, "tcgen05 ring fits the CTA's memory");
static_assert(kTcSchedulerWarp < kThreads / 32 && kTcPvWarp < kThreads / 32,
              "every tcgen05 role has a warp");
static_assert(kMaxSuffixWarps <= kThreads / 32, "every suffix-pass warp exists");

// Metadata of one prefix item, staged by the scheduler warp.
struct TcMeta {
    WorkItem it;
    int32_t id;                      // -1: the queue is empty
    int32_t key0;                    // causal item: its first key's token index, else -1
    int32_t key0B;                   // pair mode: the same for the second tile
    int32_t pad;
    WorkItem itB;                    // pair mode: the second tile (no rows: none)
    int32_t rows[kTcMetaPages];      // TMA row of each page
    int32_t leaves[kTcRows];         // branch of rows [g i, g i + g)
    int32_t leavesB[kTcRows];        // pair mode: the same for the second tile
    // leading valid tokens of each 64-token block (64 but where a node ends
    // inside the item: a prefill piece over a path pads each node that ends
    // inside a page with zero-filled pages up to the next block); the item's
    // last block also goes by last_valid
    uint8_t block_valid[kTcMetaPages / 4];
};

// causal mask: -1 when the item's rows see all of its keys
constexpr int32_t kNoKey0 = -1;

// 32 consecutive fp32 values of one partial row (128 bytes, 32-byte
// aligned), scaled, as four 32-byte stores: every store fills whole sectors
// (16-byte stores from the 32 rows of a warp left each sector to be filled
// by two instructions).
__device__ __forceinline__ void store_row32(float *dst, const uint32_t (&v)[32], float scale) {
#pragma unroll
    for (int q = 0; q < 32; q += 8)
        asm volatile("st.global.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(dst + q),
                     "f"(__uint_as_float(v[q]) * scale), "f"(__uint_as_float(v[q + 1]) * scale),
                     "f"(__uint_as_float(v[q + 2]) * scale), "f"(__uint_as_float(v[q + 3]) * scale),
                     "f"(__uint_as_float(v[q + 4]) * scale), "f"(__uint_as_float(v[q + 5]) * scale),
                     "f"(__uint_as_float(v[q + 6]) * scale), "f"(__uint_as_float(v[q + 7]) * scale)
                     : "memory");
}

// An item's page rows into its metadata slot: the TMA row of every page
// (padding pages carry the first row past the pool, which TMA fills with
// zeros), and the leading valid tokens of every block, from the low 4 bits
// of the stream rows (16 - the valid tokens of a page that ends a node;
// a TMA row (page * H_kv + kv head) * 16 leaves them zero).
__device__ __forceinline__ void stage_item_rows(TcMeta &m, const int32_t *src, int np, int kv_rows,
                                                int lane) {
    // lane b takes block b: its 4 rows are loaded before any is looked at
    for (int b = lane; b * 4 < np; b += 32) {
        int32_t row[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) row[j] = b * 4 + j < np ? src[b * 4 + j] : kv_rows;
        int v = 0;
        bool open = true;                                  // no node has ended in the block yet
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int low = row[j] & (kPageSize - 1);
            if (open && row[j] < kv_rows) v += kPageSize - low;
            open = open && row[j] < kv_rows && low == 0;   // padding, or a node's last page
            if (b * 4 + j < np) m.rows[b * 4 + j] = row[j] & ~(kPageSize - 1);
        }
        m.block_valid[b] = static_cast<uint8_t>(v);
    }
}

// barrier slots (8 bytes each) in the CTA's barrier area
enum TcBar : int {
    kBarKvFull = 0,                          // [stages] producer -> MMA (TMA bytes)
    kBarKvEmpty = kBarKvFull + kTcStages,    // [stages] MMA commit -> producer
    kBarSFull = kBarKvEmpty + kTcStages,     // [2] MMA commit -> softmax
    kBarPFull = kBarSFull + 2,               // [2] softmax (128 arrivals) -> MMA
    kBarPvDone = kBarPFull + 2,              // [2] MMA commit -> softmax (before a rescale)
    kBarQReady = kBarPvDone + 2,             // [2] epilogue (128 arrivals) -> MMA
    kBarOFull = kBarQReady + 2,              // [2] MMA commit -> epilogue
    kBarOEmpty = kBarOFull + 2,              // [2] epilogue (4 arrivals) -> MMA
    kBarMetaFull = kBarOEmpty + 2,           // [kTcMeta] scheduler -> every role
    kBarMetaEmpty = kBarMetaFull + kTcMeta,  // [kTcMeta] epilogue (4 arrivals) -> scheduler
    kBarDrain = kBarMetaEmpty + kTcMeta,     // both issuers' commits -> issuers, before TMEM is freed
    kBarCvFull,                              // [kTcCvStages] converters (4 arrivals) -> MMA
    kBarCvEmpty = kBarCvFull + kTcCvStages,  // [kTcCvStages] MMA commit -> converters
    kTcBars = kBarCvEmpty + kTcCvStages
};

// arrivals each barrier waits for; with e4m3 KV the 4 converter warps free
// the staging stages
__host__ __device__ constexpr int tc_bar_count(int i, bool f8) {
    return (i == kBarPFull || i == kBarPFull + 1 || i == kBarQReady || i == kBarQReady + 1)
               ? kTcRows
               : ((i == kBarOEmpty || i == kBarOEmpty + 1 ||
                   (i >= kBarMetaEmpty && i < kBarMetaEmpty + kTcMeta) ||
                   (f8 && i >= kBarKvEmpty && i < kBarKvEmpty + kTcStages))
                      ? 4
                      : ((i >= kBarCvFull && i < kBarCvFull + kTcCvStages)
                             ? kTcRows
                             : (i == kBarDrain ? 2 : 1)));
}

// e4m3 -> f16 of one 64-token block by 128 threads (8 of its 1024 16-byte
// chunks each): staged K and V rows of 128 bytes (128-byte swizzled) into two
// 8 KB column blocks per operand (128-byte swizzled), the layout TMA gives a
// bf16 block; rows from `valid` on become zeros.  The thread's 8 chunks are
// loaded before any is stored, so that their latencies overlap (a load may
// not pass an earlier shared store).
__device__ __forceinline__ void convert_block_e4m3(uint32_t src, uint32_t dst, int valid, int t) {
    uint4 w[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const int idx = t + kTcRows * q;
        const int op = idx >> 9;                 // 0: K, 1: V
        const int r = (idx >> 3) & 63;           // token
        const int c = idx & 7;                   // elements 16c .. 16c + 15
        w[q] = lds128(src + op * kTcF8Bytes + r * 128 + ((c ^ (r & 7)) << 4));
    }
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const int idx = t + kTcRows * q;
        const int op = idx >> 9;
        const int r = (idx >> 3) & 63;
        const int c = idx & 7;
        if (r >= valid) w[q] = make_uint4(0u, 0u, 0u, 0u);
        // chunks c and c + 4 of a row widen into the same 16-byte slots of
        // the two column blocks; the 8 threads of a quarter warp (one row)
        // would store two to a bank group, so the c >= 4 threads store their
        // second half first
        const bool second_first = (c & 4) != 0;
        const uint4 v = second_first ? make_uint4(w[q].z, w[q].w, w[q].x, w[q].y) : w[q];
        uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
        e4m3x4_to_f16x2x2(v.x, a0, a1);
        e4m3x4_to_f16x2x2(v.y, a2, a3);
        e4m3x4_to_f16x2x2(v.z, b0, b1);
        e4m3x4_to_f16x2x2(v.w, b2, b3);
        const int c2 = 2 * (c & 3);              // f16 chunk in column block c / 4
        const int first = second_first ? c2 + 1 : c2;
        const uint32_t row = dst + op * kTcKBytes + (c >> 2) * kTcColBlockBytes + r * 128;
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(row + ((first ^ (r & 7)) << 4)),
                     "r"(a0), "r"(a1), "r"(a2), "r"(a3)
                     : "memory");
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(row + (((first ^ 1) ^ (r & 7)) << 4)),
                     "r"(b0), "r"(b1), "r"(b2), "r"(b3)
                     : "memory");
    }
}

__device__ __forceinline__ bool tc_wait(uint32_t bar, uint32_t parity, long long limit,
                                        volatile int *abort) {
    return dev::mbar_wait_bounded(bar, parity, limit, abort);
}

// one warp: lane 0 waits, the warp agrees on the outcome
__device__ __forceinline__ bool tc_warp_wait(uint32_t bar, uint32_t parity, long long limit,
                                             volatile int *abort, int lane) {
    int ok = 1;
    if (lane == 0) ok = tc_wait(bar, parity, limit, abort) ? 1 : 0;
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

__device__ __forceinline__ void tc_fail(const AttnArgs &a, volatile int *abort, int site) {
    if (!*abort) {
        *abort = 1;
        dev::record_error(a.err, PARASON_ETIMEOUT, site);
    }
}

__device__ __forceinline__ int tc_blocks(int num_pages) {
    return (num_pages + kTcBlockPages - 1) / kTcBlockPages;
}

template <int D, class KV>
__device__ void prefix_cta_tc(const KvMaps *maps, const AttnArgs &a, uint8_t *smem, uint32_t bars,
                              uint32_t tmem, int warp, int lane, volatile int *abort_flag,
                              TcMeta *meta) {
    static_assert(D == 128, "the tcgen05 prefix tile is written for head_dim 128");
    constexpr bool kF8 = KV::kElemBytes == 1;
    const uint32_t ring = dev::smem_addr(smem);
    auto bar = [&](int i) { return bars + 8u * static_cast<uint32_t>(i); };
    const long long limit = a.wait_limit_ns;

    if (warp == kTcSchedulerWarp) {
        // ------------------------------------------------------------ scheduler
        for (int k = 0;; ++k) {
            const int s = k % kTcMeta;
            if (k >= kTcMeta &&
                !tc_warp_wait(bar(kBarMetaEmpty + s), ((k / kTcMeta) - 1) & 1, limit, abort_flag, lane)) {
                if (lane == 0) tc_fail(a, abort_flag, kSiteProducerEmpty);
                break;
            }
            // a prefix CTA owns position blockIdx.x of the prefix queue
            int id = *abort_flag ? -1
                                 : (k == 0 ? queue_item(a, 0, static_cast<int>(blockIdx.x))
                                           : pull(a, 0, lane));
            TcMeta &m = meta[s];
            if (id >= 0) {
                const WorkItem it = a.items[id];
                if (it.num_pages <= 0 || it.num_pages > kTcMetaPages || it.nrows <= 0 ||
                    it.nrows > kTcRows || it.row0 % a.group != 0) {
                    if (lane == 0 && !*abort_flag) {
                        *abort_flag = 1;
                        dev::record_error(a.err, PARASON_EINVAL, kSiteBadItem);
                    }
                    id = -1;
                } else {
                    if (lane == 0) {
                        m.it = it;
                        m.key0 = a.item_key0 ? a.item_key0[id] : kNoKey0;
                    }
                    stage_item_rows(m, a.stream_rows + a.item_rows[id], it.num_pages, a.kv_rows, lane);
                    const int nbr = (it.nrows + a.group - 1) / a.group;
                    const int32_t *lv = a.dfs_leaf + it.leaf_lo + it.row0 / a.group;
                    for (int i = lane; i < nbr; i += 32) m.leaves[i] = lv[i];
                }
            }
            if (lane == 0) m.id = id;
            __syncwarp();
            if (lane == 0) dev::mbar_arrive(bar(kBarMetaFull + s));
            if (id < 0) break;
        }
    } else if (warp == kTcProducerWarp) {
        // ------------------------------------------------------------ producer
        const bool skip_first = a.debug_flags & PARASON_DEBUG_SKIP_FIRST_LOAD;
        // bf16 KV: the tile's K and V go to L2 as evict-last (measured: the
        // Llama-3-shape step 42.9 -> 41.4 us, the long-prefix one -1 us, the
        // join prefill +1%; no gain with e4m3 KV, which keeps the default)
        const uint64_t last_pol = dev::l2_evict_last_policy();
        // e4m3 blocks keep the default L2 policy (the per-page boxes use no hint)
        const uint64_t f8_pol = dev::l2_evict_normal_policy();
        const int kv_page_rows = a.num_kv_heads * kPageSize;   // TMA rows between consecutive pages
        constexpr int NS = kF8 ? kTcF8Stages : kTcStages;
        int last_issue[NS];
        for (int s = 0; s < NS; ++s) last_issue[s] = -1;
        int blk = 0;
        bool ok = true;
        for (int k = 0; ok; ++k) {
            const int ms = k % kTcMeta;
            if (!tc_warp_wait(bar(kBarMetaFull + ms), (k / kTcMeta) & 1, limit, abort_flag, lane)) {
                if (lane == 0) tc_fail(a, abort_flag, kSiteProducerEmpty);
                break;
            }
            const TcMeta &m = meta[ms];
            if (m.id < 0) break;
            const int np = m.it.num_pages;
            const int nb = tc_blocks(np);
            for (int bi = 0; bi < nb; ++bi, ++blk) {
                const int s = blk % NS;
                if (blk >= NS &&
                    !tc_warp_wait(bar(kBarKvEmpty + s), ((blk / NS) - 1) & 1, limit, abort_flag,
                                  lane)) {
                    if (lane == 0) tc_fail(a, abort_flag, kSiteProducerEmpty);
                    ok = false;
                    break;
                }
                if (!(skip_first && blk == 0)) {
                    // the block's boxes are issued by one lane each (one
                    // thread issuing them all was the tile's bottleneck); the
                    // expected bytes are registered first
                    const uint32_t fb = bar(kBarKvFull + s);
                    if (lane == 0)
                        dev::mbar_arrive_expect_tx(fb, kF8 ? kTcF8StageBytes : kTcStageBytes);
                    __syncwarp();
                    // the TMA unit takes about 90 cycles a box, so a block of
                    // pages that are consecutive in the pool (the common case)
                    // goes in one box per column block of K and of V
                    const int pg0 = bi * kTcBlockPages;
                    bool run = pg0 + kTcBlockPages <= np;
                    const int row0 = m.rows[pg0 < np ? pg0 : 0];
#pragma unroll
                    for (int j = 1; j < kTcBlockPages; ++j)
                        run = run && m.rows[pg0 + j] == row0 + j * kv_page_rows;
                    if (run) {
                        const int page = row0 / kv_page_rows;
                        if constexpr (kF8) {
                            if (lane < 2)
                                dev::tma_load_5d_hint(ring + s * kTcF8StageBytes + lane * kTcF8Bytes,
                                                      lane ? &maps->v_run : &maps->k_run, 0, 0, 0,
                                                      m.it.kv_head, page, fb, f8_pol);
                        } else {
                            // lane: K (even) or V, column block lane / 2
                            if (lane < 4)
                                dev::tma_load_5d_hint(ring + s * kTcStageBytes + (lane & 1) * kTcKBytes +
                                                          (lane >> 1) * kTcColBlockBytes,
                                                      (lane & 1) ? &maps->v_run : &maps->k_run, 0,
                                                      lane >> 1, 0, m.it.kv_head, page, fb, last_pol);
                        }
                    } else if constexpr (kF8) {
                        // raw e4m3 rows: one 2 KB box per page of K (even lanes) and of V
                        if (lane < 2 * kTcBlockPages) {
                            const int j = lane >> 1;
                            const int pg = bi * kTcBlockPages + j;
                            const int row = pg < np ? m.rows[pg] : a.kv_rows;   // kv_rows: zero fill
                            const uint32_t st = ring + s * kTcF8StageBytes + (lane & 1) * kTcF8Bytes;
                            dev::tma_load_3d(st + j * kPageSize * 128, (lane & 1) ? &maps->v : &maps->k,
                                             0, 0, row, fb);
                        }
                    } else {
                        // page j = lane / 4, column block (lane / 2) % 2, K (even lanes) or V
                        if (lane < 4 * kTcBlockPages) {
                            const int j = lane >> 2, cb = (lane >> 1) & 1;
                            const int pg = bi * kTcBlockPages + j;
                            const int row = pg < np ? m.rows[pg] : a.kv_rows;   // kv_rows: zero fill
                            const uint32_t off = cb * kTcColBlockBytes + j * kPageSize * 128;
                            const uint32_t st = ring + s * kTcStageBytes + (lane & 1) * kTcKBytes;
                            dev::tma_load_3d_hint(st + off, (lane & 1) ? &maps->v : &maps->k, 0, cb,
                                                  row, fb, last_pol);
                        }
                    }
                    last_issue[s] = blk;
                }
            }
        }
        // every copy this CTA issued must land before its shared memory is reused
        if (lane == 0)
            for (int s = 0; s < NS; ++s)
                if (last_issue[s] >= 0)
                    dev::mbar_wait_bounded(bar(kBarKvFull + s), (last_issue[s] / NS) & 1,
                                           kDrainLimitNs, nullptr);
    } else if (warp == kTcMmaWarp || warp == kTcPvWarp) {
        // ------------------------------------------------------------ MMA issuers
        if (lane == 0) {
            // Two threads issue, so that neither product waits behind the other's
            // issue (an MMA takes about 45 cycles to issue; twelve per block on
            // one thread held the tile back).  Warp 9 issues S = Q K^T of every
            // block, warp 11 O += P V.  S(b) overwrites the buffer of P(b - 2),
            // so it waits for PV(b - 2) to complete.
            constexpr uint32_t kIdS = kF8 ? tc::idesc_f16_f32(kTcRows, kTcBlockTokens, false)
                                          : tc::idesc_bf16_f32(kTcRows, kTcBlockTokens, false);
            constexpr uint32_t kIdPV = kF8 ? tc::idesc_f16_f32(kTcRows, D, true)
                                           : tc::idesc_bf16_f32(kTcRows, D, true);
            constexpr int kMmaStages = kF8 ? kTcCvStages : kTcStages;
            auto wait = [&](int i, int parity) {
                return tc_wait(bar(i), static_cast<uint32_t>(parity & 1), limit, abort_flag);
            };
            // descriptors of stage 0; a stage, a column block or a K step moves
            // the start address field (address / 16) by a constant
            const uint32_t mma_ring = kF8 ? ring + kTcCvOffset : ring;
            const uint64_t desc_k = tc::smem_desc_sw128(mma_ring, 16, 1024);
            const uint64_t desc_v = tc::smem_desc_sw128(mma_ring + kTcKBytes, kTcColBlockBytes, 1024);
            constexpr uint32_t kStageStep = kTcStageBytes >> 4;
            bool ok = true;
            int b = 0;                       // block of the CTA's stream
            int st = 0, ph = 0;              // its stage and the stage's phase parity
            for (int k = 0; ok; ++k) {
                const int ms = k % kTcMeta;
                if (!wait(kBarMetaFull + ms, k / kTcMeta)) {
                    ok = false;
                    break;
                }
                if (meta[ms].id < 0) break;
                const int nb = tc_blocks(meta[ms].it.num_pages);
                if (warp == kTcMmaWarp) {
                    // S of the item's blocks, with its Q (buffer k & 1)
                    if (!wait(kBarQReady + (k & 1), k >> 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t tQ = tmem + kTmemQ + 64u * (k & 1);
                    for (int i = 0; i < nb; ++i, ++b) {
                        if (!wait((kF8 ? kBarCvFull : kBarKvFull) + st, ph) ||
                            (b >= 2 && !wait(kBarPvDone + (b & 1), (b - 2) >> 1))) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
                        const uint32_t tS = tmem + kTmemS + 64u * (b & 1);
                        const uint64_t kd = desc_k + static_cast<uint64_t>(st * kStageStep);
#pragma unroll
                        for (int ks = 0; ks < D / 16; ++ks) {
                            constexpr uint32_t kCb = kTcColBlockBytes;
                            const uint32_t off = ((ks >> 2) * kCb + (ks & 3) * 32) >> 4;
                            tc::mma_bf16_tmem_a(tS, tQ + 8u * ks, kd + off, kIdS, ks > 0);
                        }
                        tc::commit(bar(kBarSFull + (b & 1)));
                        if (++st == kMmaStages) {
                            st = 0;
                            ph ^= 1;
                        }
                    }
                } else {
                    // PV of the item's blocks into O (buffer k & 1)
                    const uint32_t tO = tmem + kTmemO + 128u * (k & 1);
                    for (int i = 0; i < nb; ++i, ++b) {
                        if (!wait(kBarPFull + (b & 1), b >> 1) ||
                            // the O buffer was last used by item k - 2: its epilogue must be done
                            (i == 0 && k >= 2 && !wait(kBarOEmpty + (k & 1), (k >> 1) - 1))) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
                        const uint32_t tP = tmem + kTmemS + 64u * (b & 1);
                        const uint64_t vd = desc_v + static_cast<uint64_t>(st * kStageStep);
#pragma unroll
                        for (int kk = 0; kk < kTcBlockTokens / 16; ++kk)
                            tc::mma_bf16_tmem_a(tO, tP + 8u * kk,
                                                vd + static_cast<uint32_t>((kk * 2048) >> 4), kIdPV,
                                                i > 0 || kk > 0);
                        // S(b) completed before P(b) was written: both products
                        // of the stage are done when these arrive
                        tc::commit(bar((kF8 ? kBarCvEmpty : kBarKvEmpty) + st));
                        tc::commit(bar(kBarPvDone + (b & 1)));
                        if (i == nb - 1) tc::commit(bar(kBarOFull + (k & 1)));
                        if (++st == kMmaStages) st = 0;
                    }
                }
            }
            if (!ok) tc_fail(a, abort_flag, kSiteConsumerFull);
            // every MMA of both issuers must finish before TMEM is freed
            tc::commit(bar(kBarDrain));
            dev::mbar_wait_bounded(bar(kBarDrain), 0, kDrainLimitNs, nullptr);
        }
        __syncwarp();
    } else if (warp < kTcSoftmaxWarps) {
        // ------------------------------------------------------------ softmax
        const int r = threadIdx.x;                       // tile row == TMEM lane
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(warp * 32) << 16);
        int blk = 0;
        for (int k = 0;; ++k) {
            const int ms = k % kTcMeta;
            if (!tc_warp_wait(bar(kBarMetaFull + ms), (k / kTcMeta) & 1, limit, abort_flag, lane)) {
                if (lane == 0) tc_fail(a, abort_flag, kSiteConsumerFull);
                break;
            }
            if (meta[ms].id < 0) break;
            const WorkItem it = meta[ms].it;
            const int nb = tc_blocks(it.num_pages);
            const int tokens = (it.num_pages - 1) * kPageSize + it.last_valid;
            const uint32_t tO = lane_base + kTmemO + 128u * (k & 1);
            // causal item (tree-masked prefill): the row's token, relative to
            // the item's first key, is the last key it sees
            const int key0 = meta[ms].key0;
            const int t_rel = key0 == kNoKey0 ? (1 << 30) : (it.row0 + r) / a.group - key0;
            // e4m3 K: the kv head's scale goes into the logits
            const float sl = kF8 ? a.scale_log2 * a.k_scale[it.kv_head] : a.scale_log2;
            float m_use = -INFINITY, l = 0.f;
            bool ok = true;
            for (int i = 0; i < nb; ++i) {
                const int b = blk + i;
                const int valid = min(static_cast<int>(meta[ms].block_valid[i]), tokens - i * kTcBlockTokens);
                const int seen = min(valid, t_rel - i * kTcBlockTokens + 1);   // keys the row sees
                const uint32_t tS = lane_base + kTmemS + 64u * (b & 1);
                if (!tc_warp_wait(bar(kBarSFull + (b & 1)), (b >> 1) & 1, limit, abort_flag, lane)) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
                uint32_t sr[2][32];
                tc::ld32(tS, sr[0]);
                tc::ld32(tS + 32, sr[1]);
                tc::wait_ld();
                // raw scores; keys the row does not see (past the item's last
                // token, or past the row's own token in a causal item) -inf
                float x[64];
#pragma unroll
                for (int j = 0; j < 64; ++j) x[j] = __uint_as_float(sr[j >> 5][j & 31]);
                if (seen < kTcBlockTokens) {
#pragma unroll
                    for (int j = 0; j < 64; ++j) x[j] = j < seen ? x[j] : -INFINITY;
                }
                // the block's max in the log2 domain (sl > 0)
                float mr = x[0];
#pragma unroll
                for (int j = 1; j + 1 < 64; j += 2) mr = dev::max3(mr, x[j], x[j + 1]);
                mr = fmaxf(mr, x[63]);
                const float mb = mr * sl;
                if (i == 0) {
                    m_use = mb;
                } else if (__any_sync(0xffffffffu, mb > m_use + kTcRescaleLog2)) {
                    // O must hold PV(b - 1) before it is rescaled
                    if (!tc_warp_wait(bar(kBarPvDone + ((b - 1) & 1)), ((b - 1) >> 1) & 1, limit,
                                      abort_flag, lane)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    const float m_new = fmaxf(m_use, mb);
                    // (a row with no visible key yet keeps m = -inf and alpha 1)
                    const float alpha = m_new == m_use ? 1.f : dev::fast_exp2(m_use - m_new);
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t ov[32];
                        tc::ld32(tO + 32 * c, ov);
                        tc::wait_ld();
#pragma unroll
                        for (int j = 0; j < 32; ++j) ov[j] = __float_as_uint(__uint_as_float(ov[j]) * alpha);
                        tc::st32(tO + 32 * c, ov);
                    }
                    tc::wait_st();
                    l *= alpha;
                    m_use = m_new;
                }
                // P = 2^(x - m) as bf16 pairs over the first 32 columns of S
                // (0 for a row that has seen no key: every x is -inf)
                const float m_ref = m_use == -INFINITY ? 0.f : m_use;
                // 2^(x sl - m) with pairs of fp32 lanes: one packed FMA per
                // two exponents, and two running sums
                const unsigned long long slp = dev::f32x2(sl, sl), nmp = dev::f32x2(-m_ref, -m_ref);
                unsigned long long lsum = dev::f32x2(0.f, 0.f);
                uint32_t pw[32];
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    float e0, e1;
                    dev::f32x2_split(dev::fma_f32x2(dev::f32x2(x[2 * c], x[2 * c + 1]), slp, nmp), e0, e1);
                    const float p0 = dev::fast_exp2(e0), p1 = dev::fast_exp2(e1);
                    lsum = dev::add_f32x2(lsum, dev::f32x2(p0, p1));
                    pw[c] = kF8 ? dev::pack_f16(p0, p1) : dev::pack_bf16(p0, p1);
                }
                {
                    float l0, l1;
                    dev::f32x2_split(lsum, l0, l1);
                    l += l0 + l1;
                }
                tc::st32(tS, pw);
                tc::wait_st();
                // V rows past the block's valid tokens may hold anything (NaN
                // included); P is 0 there but 0 * NaN is NaN, so zero them (the
                // e4m3 converters write those rows as zeros)
                if (!kF8 && valid < kTcBlockTokens) {
                    const uint32_t vst = ring + (b % kTcStages) * kTcStageBytes + kTcKBytes;
                    const int n16 = (kTcBlockTokens - valid) * 2 * 8;     // 16-byte chunks
                    for (int q = r; q < n16; q += kTcRows) {
                        const int t = valid + q / 16, cb = (q / 8) & 1, c = q & 7;
                        asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};" ::"r"(
                                         vst + cb * kTcColBlockBytes + t * 128 + (c << 4)),
                                     "r"(0u)
                                     : "memory");
                    }
                    tc::fence_proxy_async_smem();
                }
                tc::fence_before_sync();
                dev::mbar_arrive(bar(kBarPFull + (b & 1)));
            }
            if (!ok) {
                if (lane == 0) tc_fail(a, abort_flag, kSiteConsumerFull);
                break;
            }
            if (r < it.nrows) a.part_ml[static_cast<int64_t>(it.slot_base) + r] = make_float2(m_use, l);
            blk += nb;
        }
    } else if (warp >= kTcEpilogueWarp && warp < kTcEpilogueWarp + 4) {
        // ------------------------------------------------------------ epilogue
        const int quarter = warp - kTcEpilogueWarp;      // == warp % 4: its TMEM lanes
        const int r = quarter * 32 + lane;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        bool ok = true;
        // wait for slot k; true if it holds an item
        auto has_item = [&](int k) {
            if (!tc_warp_wait(bar(kBarMetaFull + k % kTcMeta), (k / kTcMeta) & 1, limit, abort_flag,
                              lane)) {
                ok = false;
                return false;
            }
            return meta[k % kTcMeta].id >= 0;
        };
        // Q row r of item k: global loads into registers ...
        auto fetch_q = [&](int k, uint4 (&qv)[16]) {
            const TcMeta &m = meta[k % kTcMeta];
            if (r < m.it.nrows) {
                const int leaf = m.leaves[r / a.group];
                const int head = m.it.kv_head * a.group + r % a.group;
                const uint4 *src = reinterpret_cast<const uint4 *>(
                    static_cast<const __nv_bfloat16 *>(a.q) +
                    (static_cast<int64_t>(leaf) * a.num_q_heads + head) * D);
#pragma unroll
                for (int c = 0; c < 16; ++c) qv[c] = src[c];
            } else {
#pragma unroll
                for (int c = 0; c < 16; ++c) qv[c] = make_uint4(0u, 0u, 0u, 0u);
            }
        };
        // ... then into TMEM Q buffer k & 1 (bf16 pairs, or f16 pairs for
        // the e4m3 tile, lane r)
        auto put_q = [&](int k, const uint4 (&qv)[16]) {
            bool big = false;
            auto cv = [&big](uint32_t two) {
                if constexpr (!kF8) return two;
                return q_pair_to_f16(two, big);
            };
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                uint32_t w[32];
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    w[4 * c] = cv(qv[8 * h + c].x);
                    w[4 * c + 1] = cv(qv[8 * h + c].y);
                    w[4 * c + 2] = cv(qv[8 * h + c].z);
                    w[4 * c + 3] = cv(qv[8 * h + c].w);
                }
                tc::st32(lane_base + kTmemQ + 64u * (k & 1) + 32u * h, w);
            }
            if constexpr (kF8) report_q_range(a, big, lane);
            tc::wait_st();
            tc::fence_before_sync();
            dev::mbar_arrive(bar(kBarQReady + (k & 1)));
        };
        if constexpr (kF8) {
        // item j's O rows to its partials, times the kv head's V scale
        auto store_o = [&](int j, const WorkItem &it) {
            const float vs = a.v_scale[it.kv_head];
            const uint32_t tO = lane_base + kTmemO + 128u * (j & 1);
            float *dst = a.part_o + (static_cast<int64_t>(it.slot_base) + r) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t ov[32];
                tc::ld32(tO + 32 * c, ov);
                tc::wait_ld();
                if (r < it.nrows) store_row32(dst + 32 * c, ov, vs);
            }
        };
            // The converters take every block of every item in order.  An
            // item's O is stored once the next item's first block is
            // converted (the S issuer needs that block before the item's
            // last PV can follow, so waiting for the O first could never
            // end), and its second block too where there is one, so that the
            // wait for the O is short (long-prefix step with e4m3 KV: 668 ->
            // 655 us).
            auto convert = [&](int gb, int valid) -> bool {
                const int s = gb % kTcF8Stages, c = gb % kTcCvStages;
                if (!tc_warp_wait(bar(kBarKvFull + s), (gb / kTcF8Stages) & 1, limit, abort_flag, lane))
                    return false;
                if (gb >= kTcCvStages &&
                    !tc_warp_wait(bar(kBarCvEmpty + c), ((gb / kTcCvStages) - 1) & 1, limit, abort_flag,
                                  lane))
                    return false;
                convert_block_e4m3(ring + s * kTcF8StageBytes, ring + kTcCvOffset + c * kTcStageBytes,
                                   valid, r);
                tc::fence_proxy_async_smem();
                dev::mbar_arrive(bar(kBarCvFull + c));
                __syncwarp();
                if (lane == 0) dev::mbar_arrive(bar(kBarKvEmpty + s));
                return true;
            };
            // store item j's O; load item j + 2's Q into the buffer j frees
            auto finish = [&](int j, bool next_exists) -> bool {
                const WorkItem it = meta[j % kTcMeta].it;
                if (!tc_warp_wait(bar(kBarOFull + (j & 1)), (j >> 1) & 1, limit, abort_flag, lane))
                    return false;
                tc::fence_after_sync();
                const bool has_j2 = next_exists && has_item(j + 2);
                if (!ok) return false;
                uint4 qv[16];
                if (has_j2) fetch_q(j + 2, qv);
                store_o(j, it);
                if (has_j2) put_q(j + 2, qv);
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) {
                    dev::mbar_arrive(bar(kBarOEmpty + (j & 1)));
                    dev::mbar_arrive(bar(kBarMetaEmpty + j % kTcMeta));
                }
                return true;
            };
            if (has_item(0)) {
                uint4 qv[16];
                fetch_q(0, qv);
                put_q(0, qv);
                if (has_item(1)) {
                    fetch_q(1, qv);
                    put_q(1, qv);
                }
                for (int k = 0, gb = 0; ok; ++k) {
                    const WorkItem it = meta[k % kTcMeta].it;
                    const int nb = tc_blocks(it.num_pages);
                    const int tokens = (it.num_pages - 1) * kPageSize + it.last_valid;
                    for (int i = 0; i < nb && ok; ++i, ++gb) {
                        ok = convert(gb, min(kTcBlockTokens, tokens - i * kTcBlockTokens));
                        if (ok && k > 0 && i == min(1, nb - 1)) ok = finish(k - 1, true);
                    }
                    if (!ok) break;
                    const bool more = has_item(k + 1);
                    if (!ok) break;
                    if (!more) {
                        ok = finish(k, false);
                        break;
                    }
                }
            }
            if (!ok && lane == 0) tc_fail(a, abort_flag, kSiteConsumerFull);
            return;
        }
        bool has_k = has_item(0), has_k1 = false;
        if (has_k) {
            uint4 qv[16];
            fetch_q(0, qv);
            put_q(0, qv);
            has_k1 = has_item(1);
            if (has_k1) {
                fetch_q(1, qv);
                put_q(1, qv);
            }
        }
        for (int k = 0; ok && has_k; ++k) {
            const WorkItem it = meta[k % kTcMeta].it;
            if (!tc_warp_wait(bar(kBarOFull + (k & 1)), (k >> 1) & 1, limit, abort_flag, lane)) {
                ok = false;
                break;
            }
            tc::fence_after_sync();
            // item k's S MMAs are complete, so its Q buffer takes item k + 2's rows;
            // their loads are in flight while O is stored
            const bool has_k2 = has_k1 && has_item(k + 2);
            uint4 qv[16];
            if (has_k2) fetch_q(k + 2, qv);
            const uint32_t tO = lane_base + kTmemO + 128u * (k & 1);
            float *dst = a.part_o + (static_cast<int64_t>(it.slot_base) + r) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t ov[32];
                tc::ld32(tO + 32 * c, ov);
                tc::wait_ld();
                if (r < it.nrows) {
#pragma unroll
                    for (int j = 0; j < 32; j += 4)
                        *reinterpret_cast<float4 *>(dst + 32 * c + j) =
                            make_float4(__uint_as_float(ov[j]), __uint_as_float(ov[j + 1]),
                                        __uint_as_float(ov[j + 2]), __uint_as_float(ov[j + 3]));
                }
            }
            if (has_k2) put_q(k + 2, qv);
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) {
                dev::mbar_arrive(bar(kBarOEmpty + (k & 1)));
                dev::mbar_arrive(bar(kBarMetaEmpty + k % kTcMeta));
            }
            has_k = has_k1;
            has_k1 = has_k2;
        }
        if (!ok && lane == 0) tc_fail(a, abort_flag, kSiteConsumerFull);
    }
}

// ---------------------------------------------------------------------------
// prefix pass on tcgen05, pair mode (bf16 KV, head_dim 128): two 128-row
// tiles of one piece -- consecutive row tiles of one node and kv head, over
// the same pages -- against every staged 64-token block, so that each block
// is staged once for 256 rows.  The prefix queue holds pairs: position k is
// items 2k (tile A) and 2k + 1 (tile B, no rows when the piece has one
// tile).
//
//   warp 10     scheduler: pulls pairs and stages their metadata
//   warp 8      producer: TMA of each block of the pair's pages, once, into
//               a 4-stage ring
//   warp 9      S issuer (one thread): S_t = Q_t K^T for t = A, B of a block,
//               A and B from shared memory
//   warp 11     PV issuer (one thread): O_t += P_t V; the stage goes back to
//               the producer after the block's last PV
//   warps 0-3   tile A: softmax (thread r owns row r, TMEM lane r), the next
//               pair's Q rows into shared memory, then the row's (m, l) and O
//   warps 4-7   tile B: the same for the second tile
//
// TMEM, 512 columns: O_A, O_B at 0 and 128; S/P of tile A at 256 and 320, of
// tile B at 384 and 448 (each tile alternates its two buffers by block, as
// the single-tile pass does).  Shared memory: the ring [4][K | V] as in the
// single-tile pass, then Q_A and Q_B, 32 KB each, in the layout TMA gives a
// K block (two 16 KB column blocks of 128 rows x 128 bytes, 128-byte
// swizzle).  Every wait is bounded, as in the single-tile pass.
// ---------------------------------------------------------------------------
constexpr int kTpStages = 4;
constexpr int kTpQOffset = kTpStages * kTcStageBytes;         // 128 KB
constexpr int kTpQColBlockBytes = kTcRows * 128;              // 16 KB
constexpr int kTpQBytes = 2 * kTpQColBlockBytes;              // 32 KB: d = 128
static_assert(kTpQOffset + 2 * kTpQBytes <= kTcRingBytes, "pair-mode ring and Q fit");

enum TcPairBar : int {
    kPbKvFull = 0,                            // [stages] producer -> S issuer (TMA bytes)
    kPbKvEmpty = kPbKvFull + kTpStages,       // [stages] PV issuer commit -> producer
    kPbSFull = kPbKvEmpty + kTpStages,        // [2 tiles x 2] S issuer commit -> tile warps
    kPbPFull = kPbSFull + 4,                  // [2 x 2] tile warps (128 arrivals) -> PV issuer
    kPbPvDone = kPbPFull + 4,                 // [2 x 2] PV commit -> S issuer, tile warps (rescale)
    kPbQReady = kPbPvDone + 4,                // [2] tile warps (128 arrivals) -> S issuer
    kPbOFull = kPbQReady + 2,                 // [2] PV commit -> tile warps
    kPbOEmpty = kPbOFull + 2,                 // [2] tile warps (4 arrivals) -> PV issuer
    kPbMetaFull = kPbOEmpty + 2,              // [kTcMeta] scheduler -> every role
    kPbMetaEmpty = kPbMetaFull + kTcMeta,     // [kTcMeta] the 8 tile warps -> scheduler
    kPbDrain = kPbMetaEmpty + kTcMeta,        // both issuers' commits -> issuers
    kTcPairBars
};

__host__ __device__ constexpr int tc_pair_bar_count(int i) {
    return ((i >= kPbPFull && i < kPbPFull + 4) || (i >= kPbQReady && i < kPbQReady + 2))
               ? kTcRows
               : ((i >= kPbOEmpty && i < kPbOEmpty + 2)
                      ? 4
                      : ((i >= kPbMetaEmpty && i < kPbMetaEmpty + kTcMeta) ? 8
                                                                          : (i == kPbDrain ? 2 : 1)));
}

// Queue position k of the prefix queue in pair mode: item 2k (-1: empty).
__device__ __forceinline__ int pair_item(const AttnArgs &a, int k) {
    return 2 * k + 1 < a.num_wide_items ? 2 * k : -1;
}

template <int D>
__device__ void prefix_cta_tc_pair(const KvMaps *maps, const AttnArgs &a, uint8_t *smem, uint32_t bars,
                                   uint32_t tmem, int warp, int lane, volatile int *abort_flag,
                                   TcMeta *meta) {
    static_assert(D == 128, "the tcgen05 prefix tile is written for head_dim 128");
    const uint32_t ring = dev::smem_addr(smem);
    auto bar = [&](int i) { return bars + 8u * static_cast<uint32_t>(i); };
    const long long limit = a.wait_limit_ns;

    if (warp == kTcSchedulerWarp) {
        // ------------------------------------------------------------ scheduler
        for (int k = 0;; ++k) {
            const int s = k % kTcMeta;
            if (k >= kTcMeta &&
                !tc_warp_wait(bar(kPbMetaEmpty + s), ((k / kTcMeta) - 1) & 1, limit, abort_flag, lane)) {
                if (lane == 0) tc_fail(a, abort_flag, kSiteProducerEmpty);
                break;
            }
            // a prefix CTA owns pair blockIdx.x of the prefix queue
            int id = -1;
            if (!*abort_flag) {
                if (k == 0) {
                    id = pair_item(a, static_cast<int>(blockIdx.x));
                } else {
                    int pos = 0;
                    if (lane == 0) pos = atomicAdd(a.queue_next, 1);
                    id = pair_item(a, __shfl_sync(0xffffffffu, pos, 0));
                }
            }
            TcMeta &m = meta[s];
            if (id >= 0) {
                const WorkItem it = a.items[id], itB = a.items[id + 1];
                bool bad = it.num_pages <= 0 || it.num_pages > kTcMetaPages || it.nrows <= 0 ||
                           it.nrows > kTcRows || it.row0 % a.group != 0;
                if (itB.nrows != 0)
                    bad = bad || itB.nrows < 0 || itB.nrows > kTcRows || itB.row0 % a.group != 0 ||
                          itB.num_pages != it.num_pages || itB.page_pos != it.page_pos ||
                          itB.last_valid != it.last_valid || itB.kv_head != it.kv_head;
                if (bad) {
                    if (lane == 0 && !*abort_flag) {
                        *abort_flag = 1;
                        dev::record_error(a.err, PARASON_EINVAL, kSiteBadItem);
                    }
                    id = -1;
                } else {
                    if (lane == 0) {
                        m.it = it;
                        m.itB = itB;
                        m.key0 = a.item_key0 ? a.item_key0[id] : kNoKey0;
                        m.key0B = a.item_key0 ? a.item_key0[id + 1] : kNoKey0;
                    }
                    stage_item_rows(m, a.stream_rows + a.item_rows[id], it.num_pages, a.kv_rows, lane);
                    const int nbr = (it.nrows + a.group - 1) / a.group;
                    const int32_t *lv = a.dfs_leaf + it.leaf_lo + it.row0 / a.group;
                    for (int i = lane; i < nbr; i += 32) m.leaves[i] = lv[i];
                    if (itB.nrows > 0) {
                        const int nbrB = (itB.nrows + a.group - 1) / a.group;
                        const int32_t *lvB = a.dfs_leaf + itB.leaf_lo + itB.row0 / a.group;
                        for (int i = lane; i < nbrB; i += 32) m.leavesB[i] = lvB[i];
                    }
                }
            }
            if (lane == 0) m.id = id;
            __syncwarp();
            if (lane == 0) dev::mbar_arrive(bar(kPbMetaFull + s));
            if (id < 0) break;
        }
    } else if (warp == kTcProducerWarp) {
        // ------------------------------------------------------------ producer
        const bool skip_first = a.debug_flags & PARASON_DEBUG_SKIP_FIRST_LOAD;
        const uint64_t last_pol = dev::l2_evict_last_policy();
        const int kv_page_rows = a.num_kv_heads * kPageSize;
        int last_issue[kTpStages];
        for (int s = 0; s < kTpStages; ++s) last_issue[s] = -1;
        int blk = 0;
        bool ok = true;
        for (int k = 0; ok; ++k) {
            const int ms = k % kTcMeta;
            if (!tc_warp_wait(bar(kPbMetaFull + ms), (k / kTcMeta) & 1, limit, abort_flag, lane)) {
                if (lane == 0) tc_fail(a, abort_flag, kSiteProducerEmpty);
                break;
            }
            const TcMeta &m = meta[ms];
            if (m.id < 0) break;
            const int np = m.it.num_pages;
            const int nb = tc_blocks(np);
            for (int bi = 0; bi < nb; ++bi, ++blk) {
                const int s = blk % kTpStages;
                if (blk >= kTpStages &&
                    !tc_warp_wait(bar(kPbKvEmpty + s), ((blk / kTpStages) - 1) & 1, limit, abort_flag,
                                  lane)) {
                    if (lane == 0) tc_fail(a, abort_flag, kSiteProducerEmpty);
                    ok = false;
                    break;
                }
                if (!(skip_first && blk == 0)) {
                    const uint32_t fb = bar(kPbKvFull + s);
                    if (lane == 0) dev::mbar_arrive_expect_tx(fb, kTcStageBytes);
                    __syncwarp();
                    const int pg0 = bi * kTcBlockPages;
                    bool run = pg0 + kTcBlockPages <= np;
                    const int row0 = m.rows[pg0 < np ? pg0 : 0];
#pragma unroll
                    for (int j = 1; j < kTcBlockPages; ++j)
                        run = run && m.rows[pg0 + j] == row0 + j * kv_page_rows;
                    if (run) {
                        const int page = row0 / kv_page_rows;
                        // lane: K (even) or V, column block lane / 2
                        if (lane < 4)
                            dev::tma_load_5d_hint(ring + s * kTcStageBytes + (lane & 1) * kTcKBytes +
                                                      (lane >> 1) * kTcColBlockBytes,
                                                  (lane & 1) ? &maps->v_run : &maps->k_run, 0, lane >> 1,
                                                  0, m.it.kv_head, page, fb, last_pol);
                    } else if (lane < 4 * kTcBlockPages) {
                        // page j = lane / 4, column block (lane / 2) % 2, K (even lanes) or V
                        const int j = lane >> 2, cb = (lane >> 1) & 1;
                        const int pg = bi * kTcBlockPages + j;
                        const int row = pg < np ? m.rows[pg] : a.kv_rows;   // kv_rows: zero fill
                        const uint32_t off = cb * kTcColBlockBytes + j * kPageSize * 128;
                        const uint32_t st = ring + s * kTcStageBytes + (lane & 1) * kTcKBytes;
                        dev::tma_load_3d_hint(st + off, (lane & 1) ? &maps->v : &maps->k, 0, cb, row, fb,
                                              last_pol);
                    }
                    last_issue[s] = blk;
                }
            }
        }
        // every copy this CTA issued must land before its shared memory is reused
        if (lane == 0)
            for (int s = 0; s < kTpStages; ++s)
                if (last_issue[s] >= 0)
                    dev::mbar_wait_bounded(bar(kPbKvFull + s), (last_issue[s] / kTpStages) & 1,
                                           kDrainLimitNs, nullptr);
    } else if (warp == kTcMmaWarp || warp == kTcPvWarp) {
        // ------------------------------------------------------------ MMA issuers
        if (lane == 0) {
            constexpr uint32_t kIdS = tc::idesc_bf16_f32(kTcRows, kTcBlockTokens, false);
            constexpr uint32_t kIdPV = tc::idesc_bf16_f32(kTcRows, D, true);
            auto wait = [&](int i, int parity) {
                return tc_wait(bar(i), static_cast<uint32_t>(parity & 1), limit, abort_flag);
            };
            const uint64_t desc_k = tc::smem_desc_sw128(ring, 16, 1024);
            const uint64_t desc_v = tc::smem_desc_sw128(ring + kTcKBytes, kTcColBlockBytes, 1024);
            const uint64_t desc_q[2] = {tc::smem_desc_sw128(ring + kTpQOffset, 16, 1024),
                                        tc::smem_desc_sw128(ring + kTpQOffset + kTpQBytes, 16, 1024)};
            constexpr uint32_t kStageStep = kTcStageBytes >> 4;
            bool ok = true;
            int st = 0, ph = 0;              // stage of the block and the stage's phase parity
            int u[2] = {0, 0};               // blocks of each tile so far
            int j[2] = {0, 0};               // pairs in which each tile had rows
            for (int k = 0; ok; ++k) {
                const int ms = k % kTcMeta;
                if (!wait(kPbMetaFull + ms, k / kTcMeta)) {
                    ok = false;
                    break;
                }
                if (meta[ms].id < 0) break;
                const bool on[2] = {true, meta[ms].itB.nrows > 0};
                const int nb = tc_blocks(meta[ms].it.num_pages);
                if (warp == kTcMmaWarp) {
                    for (int t = 0; t < 2 && ok; ++t)
                        if (on[t] && !wait(kPbQReady + t, j[t])) ok = false;
                    if (ok) tc::fence_after_sync();
                    for (int i = 0; i < nb && ok; ++i) {
                        if (!wait(kPbKvFull + st, ph)) {
                            ok = false;
                            break;
                        }
                        const uint64_t kd = desc_k + static_cast<uint64_t>(st * kStageStep);
                        for (int t = 0; t < 2; ++t) {
                            if (!on[t]) continue;
                            const int buf = u[t] & 1;
                            // the buffer holds the tile's P of two blocks back until its PV is done
                            if (u[t] >= 2 && !wait(kPbPvDone + 2 * t + buf, (u[t] - 2) >> 1)) {
                                ok = false;
                                break;
                            }
                            tc::fence_after_sync();
                            const uint32_t tS = tmem + kTmemS + 128u * t + 64u * buf;
#pragma unroll
                            for (int ks = 0; ks < D / 16; ++ks) {
                                const uint32_t koff = ((ks >> 2) * kTcColBlockBytes + (ks & 3) * 32) >> 4;
                                const uint32_t qoff = ((ks >> 2) * kTpQColBlockBytes + (ks & 3) * 32) >> 4;
                                tc::mma_bf16(tS, desc_q[t] + qoff, kd + koff, kIdS, ks > 0);
                            }
                            tc::commit(bar(kPbSFull + 2 * t + buf));
                            ++u[t];
                        }
                        if (++st == kTpStages) {
                            st = 0;
                            ph ^= 1;
                        }
                    }
                } else {
                    for (int i = 0; i < nb && ok; ++i) {
                        const uint64_t vd = desc_v + static_cast<uint64_t>(st * kStageStep);
                        for (int t = 0; t < 2; ++t) {
                            if (!on[t]) continue;
                            const int buf = u[t] & 1;
                            if (!wait(kPbPFull + 2 * t + buf, u[t] >> 1) ||
                                // the tile's O was last used by its previous pair: stored?
                                (i == 0 && j[t] > 0 && !wait(kPbOEmpty + t, j[t] - 1))) {
                                ok = false;
                                break;
                            }
                            tc::fence_after_sync();
                            const uint32_t tO = tmem + kTmemO + 128u * t;
                            const uint32_t tP = tmem + kTmemS + 128u * t + 64u * buf;
#pragma unroll
                            for (int kk = 0; kk < kTcBlockTokens / 16; ++kk)
                                tc::mma_bf16_tmem_a(tO, tP + 8u * kk,
                                                    vd + static_cast<uint32_t>((kk * 2048) >> 4), kIdPV,
                                                    i > 0 || kk > 0);
                            tc::commit(bar(kPbPvDone + 2 * t + buf));
                            if (i == nb - 1) tc::commit(bar(kPbOFull + t));
                            ++u[t];
                        }
                        if (!ok) break;
                        // both tiles' products of the stage are done when this arrives
                        // (each S completed before its P was written)
                        tc::commit(bar(kPbKvEmpty + st));
                        if (++st == kTpStages) st = 0;
                    }
                }
                for (int t = 0; t < 2; ++t)
                    if (on[t]) ++j[t];
            }
            if (!ok) tc_fail(a, abort_flag, kSiteConsumerFull);
            // every MMA of both issuers must finish before TMEM is freed
            tc::commit(bar(kPbDrain));
            dev::mbar_wait_bounded(bar(kPbDrain), 0, kDrainLimitNs, nullptr);
        }
        __syncwarp();
    } else if (warp < 8) {
        // ------------------------------------------------------------ tile warps
        const int t = warp >> 2;                         // tile A (warps 0-3) or B (4-7)
        const int quarter = warp & 3;                    // its TMEM lanes
        const int r = quarter * 32 + lane;               // tile row == TMEM lane
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        const uint32_t tO = lane_base + kTmemO + 128u * t;
        const uint32_t q_smem = ring + kTpQOffset + t * kTpQBytes;
        bool ok = true;
        int u = 0, jp = 0;                               // this tile's blocks and pairs so far
        auto tile_of = [&](const TcMeta &m) -> const WorkItem & { return t == 0 ? m.it : m.itB; };
        // Q rows of the tile in pair k into the tile's Q buffer in shared
        // memory (row r: 16 chunks of 16 bytes, 128-byte swizzle) by
        // asynchronous copies (zeros past the tile's rows) ...
        auto issue_q = [&](int k) {
            const TcMeta &m = meta[k % kTcMeta];
            const WorkItem &it = tile_of(m);
            const bool live = r < it.nrows;
            const int leaf = live ? (t == 0 ? m.leaves : m.leavesB)[r / a.group] : 0;
            const int head = live ? it.kv_head * a.group + r % a.group : 0;
            const char *src = reinterpret_cast<const char *>(
                static_cast<const __nv_bfloat16 *>(a.q) +
                (static_cast<int64_t>(leaf) * a.num_q_heads + head) * D);
            const uint32_t bytes = live ? 16u : 0u;
#pragma unroll
            for (int c = 0; c < 16; ++c) {
                const uint32_t dst = q_smem + (c >> 3) * kTpQColBlockBytes + r * 128 +
                                     (((c & 7) ^ (r & 7)) << 4);
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst),
                             "l"(src + 16 * c), "r"(bytes)
                             : "memory");
            }
        };
        // ... that are waited for, made visible to the tensor cores and
        // announced to the S issuer later
        auto publish_q = [&]() {
            asm volatile("cp.async.wait_all;" ::: "memory");
            tc::fence_proxy_async_smem();
            dev::mbar_arrive(bar(kPbQReady + t));
        };
        // wait for slot k; true if it holds a pair
        auto has_pair = [&](int k) {
            if (!tc_warp_wait(bar(kPbMetaFull + k % kTcMeta), (k / kTcMeta) & 1, limit, abort_flag, lane)) {
                ok = false;
                return false;
            }
            return meta[k % kTcMeta].id >= 0;
        };
        auto on_in = [&](int k) { return t == 0 || meta[k % kTcMeta].itB.nrows > 0; };
        bool have = has_pair(0);
        if (have && on_in(0)) {
            issue_q(0);
            publish_q();
        }
        for (int k = 0; ok && have; ++k) {
            const TcMeta &m = meta[k % kTcMeta];
            const bool on = on_in(k);
            bool more = false, loaded_next = false;
            if (on) {
                const WorkItem it = tile_of(m);
                const int nb = tc_blocks(it.num_pages);
                const int tokens = (it.num_pages - 1) * kPageSize + it.last_valid;
                const int key0 = t == 0 ? m.key0 : m.key0B;
                const int t_rel = key0 == kNoKey0 ? (1 << 30) : (it.row0 + r) / a.group - key0;
                float m_use = -INFINITY, l = 0.f;
                for (int i = 0; i < nb; ++i) {
                    const int buf = u & 1;
                    const uint32_t tS = lane_base + kTmemS + 128u * t + 64u * buf;
                    const int valid = min(static_cast<int>(m.block_valid[i]), tokens - i * kTcBlockTokens);
                    const int seen = min(valid, t_rel - i * kTcBlockTokens + 1);
                    if (!tc_warp_wait(bar(kPbSFull + 2 * t + buf), (u >> 1) & 1, limit, abort_flag, lane)) {
                        ok = false;
                        break;
                    }
                    tc::fence_after_sync();
                    uint32_t sr[2][32];
                    tc::ld32(tS, sr[0]);
                    tc::ld32(tS + 32, sr[1]);
                    tc::wait_ld();
                    // the tile's last S of the pair is done: its Q buffer takes the
                    // next pair's rows while this block's softmax runs
                    if (i == nb - 1) {
                        more = has_pair(k + 1);
                        if (!ok) break;
                        if (more && on_in(k + 1)) {
                            issue_q(k + 1);
                            loaded_next = true;
                        }
                    }
                    float x[64];
#pragma unroll
                    for (int q = 0; q < 64; ++q) x[q] = __uint_as_float(sr[q >> 5][q & 31]);
                    if (seen < kTcBlockTokens) {
#pragma unroll
                        for (int q = 0; q < 64; ++q) x[q] = q < seen ? x[q] : -INFINITY;
                    }
                    float mr = x[0];
#pragma unroll
                    for (int q = 1; q + 1 < 64; q += 2) mr = dev::max3(mr, x[q], x[q + 1]);
                    mr = fmaxf(mr, x[63]);
                    const float sl = a.scale_log2;
                    const float mb = mr * sl;
                    if (i == 0) {
                        m_use = mb;
                    } else if (__any_sync(0xffffffffu, mb > m_use + kTcRescaleLog2)) {
                        // O must hold the tile's previous PV before it is rescaled
                        if (!tc_warp_wait(bar(kPbPvDone + 2 * t + ((u - 1) & 1)), ((u - 1) >> 1) & 1, limit,
                                          abort_flag, lane)) {
                            ok = false;
                            break;
                        }
                        tc::fence_after_sync();
                        const float m_new = fmaxf(m_use, mb);
                        const float alpha = m_new == m_use ? 1.f : dev::fast_exp2(m_use - m_new);
#pragma unroll
                        for (int c = 0; c < D / 32; ++c) {
                            uint32_t ov[32];
                            tc::ld32(tO + 32 * c, ov);
                            tc::wait_ld();
#pragma unroll
                            for (int q = 0; q < 32; ++q)
                                ov[q] = __float_as_uint(__uint_as_float(ov[q]) * alpha);
                            tc::st32(tO + 32 * c, ov);
                        }
                        tc::wait_st();
                        l *= alpha;
                        m_use = m_new;
                    }
                    const float m_ref = m_use == -INFINITY ? 0.f : m_use;
                    const unsigned long long slp = dev::f32x2(sl, sl), nmp = dev::f32x2(-m_ref, -m_ref);
                    unsigned long long lsum = dev::f32x2(0.f, 0.f);
                    uint32_t pw[32];
#pragma unroll
                    for (int c = 0; c < 32; ++c) {
                        float e0, e1;
                        dev::f32x2_split(dev::fma_f32x2(dev::f32x2(x[2 * c], x[2 * c + 1]), slp, nmp), e0, e1);
                        const float p0 = dev::fast_exp2(e0), p1 = dev::fast_exp2(e1);
                        lsum = dev::add_f32x2(lsum, dev::f32x2(p0, p1));
                        pw[c] = dev::pack_bf16(p0, p1);
                    }
                    {
                        float l0, l1;
                        dev::f32x2_split(lsum, l0, l1);
                        l += l0 + l1;
                    }
                    tc::st32(tS, pw);
                    tc::wait_st();
                    // V rows past the block's valid tokens may hold anything (NaN
                    // included); P is 0 there but 0 * NaN is NaN, so tile A zeroes
                    // them before its PV -- tile B's PV of the block is issued after
                    if (t == 0 && valid < kTcBlockTokens) {
                        const int stage = u % kTpStages;   // tile A has a block of every stage
                        const uint32_t vst = ring + stage * kTcStageBytes + kTcKBytes;
                        const int n16 = (kTcBlockTokens - valid) * 2 * 8;
                        for (int q = r; q < n16; q += kTcRows) {
                            const int tt = valid + q / 16, cb = (q / 8) & 1, c = q & 7;
                            asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};" ::"r"(
                                             vst + cb * kTcColBlockBytes + tt * 128 + (c << 4)),
                                         "r"(0u)
                                         : "memory");
                        }
                        tc::fence_proxy_async_smem();
                    }
                    tc::fence_before_sync();
                    dev::mbar_arrive(bar(kPbPFull + 2 * t + buf));
                    ++u;
                }
                if (!ok) break;
                if (loaded_next) publish_q();
                if (r < it.nrows) a.part_ml[static_cast<int64_t>(it.slot_base) + r] = make_float2(m_use, l);
                // the tile's O, once its last PV is done
                if (!tc_warp_wait(bar(kPbOFull + t), jp & 1, limit, abort_flag, lane)) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
                float *dst = a.part_o + (static_cast<int64_t>(it.slot_base) + r) * D;
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t ov[32];
                    tc::ld32(tO + 32 * c, ov);
                    tc::wait_ld();
                    if (r < it.nrows) store_row32(dst + 32 * c, ov, 1.f);
                }
                tc::fence_before_sync();
                __syncwarp();
                if (lane == 0) dev::mbar_arrive(bar(kPbOEmpty + t));
                ++jp;
            } else {
                // the tile has no rows in this pair; its Q buffer is free
                more = has_pair(k + 1);
                if (!ok) break;
                if (more && on_in(k + 1)) {
                    issue_q(k + 1);
                    publish_q();
                }
            }
            __syncwarp();
            if (lane == 0) dev::mbar_arrive(bar(kPbMetaEmpty + k % kTcMeta));
            have = more;
        }
        if (!ok && lane == 0) tc_fail(a, abort_flag, kSiteConsumerFull);
    }
}

// One CTA per SM: 12 warps leave at most 168 registers per thread (three warps
// on one sub-partition of 16K registers).
template <int D, class KV>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ KvMaps maps, const AttnArgs a) {
    using S = Shape<D, KV>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t ring = dev::smem_addr(smem);
    const uint32_t bars = dev::smem_addr(smem + S::kBodyBytes);
    __shared__ int abort_flag;
    __shared__ int id_slots[kIdSlots];                        // prefix-pass item ids
    __shared__ WorkItem grab_items[kMaxSuffixWarps][kGrabSlots];  // suffix-pass items per warp
    const bool wide = static_cast<int>(blockIdx.x) < a.num_wide_ctas;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // the prefix pass at head_dim 128 (bf16 or e4m3 KV) runs on tcgen05; with
    // bf16 KV the plan may hand it pairs of row tiles (pair mode)
    constexpr bool kTcPrefix = D == 128;
    const bool tc_pairs = kTcPrefix && KV::kElemBytes == 2 && a.tc_pairs != 0;
    const int prefix_bars =
        kTcPrefix ? (tc_pairs ? static_cast<int>(kTcPairBars) : static_cast<int>(kTcBars))
                  : 2 * S::kWideStages + kIdSlots;
    static_assert(!kTcPrefix || (kTcBars <= S::kBars && kTcPairBars <= S::kBars),
                  "barrier area holds the tcgen05 barriers");
    __shared__ TcMeta tc_meta[kTcPrefix ? kTcMeta : 1];
    __shared__ uint32_t tmem_base;
    if (threadIdx.x == 0) {
        abort_flag = 0;
        if (wide && kTcPrefix && tc_pairs) {
            for (int i = 0; i < kTcPairBars; ++i) dev::mbar_init(bars + 8 * i, tc_pair_bar_count(i));
        } else if (wide && kTcPrefix) {
            for (int i = 0; i < kTcBars; ++i)
                dev::mbar_init(bars + 8 * i, tc_bar_count(i, KV::kElemBytes == 1));
        } else if (wide) {
            for (int s = 0; s < S::kWideStages; ++s) {
                dev::mbar_init(bars + 8 * s, 1);
                dev::mbar_init(bars + 8 * (S::kWideStages + s), kConsumerWarps);
            }
            for (int i = 0; i < kIdSlots; ++i) dev::mbar_init(bars + 8 * (2 * S::kWideStages + i), 1);
        } else {
            for (int s = 0; s < S::kNarrowBars; ++s) dev::mbar_init(bars + 8 * s, 1);
        }
        dev::fence_mbar_init();
        dev::prefetch_tensormap(&maps.k);
        dev::prefetch_tensormap(&maps.v);
        if constexpr (S::kSeg > 1) {
            dev::prefetch_tensormap(&maps.k_page);
            dev::prefetch_tensormap(&maps.v_page);
        }
    }
    if constexpr (kTcPrefix) {
        if (wide && warp == kTcMmaWarp) tc::alloc<kTcTmemCols>(dev::smem_addr(&tmem_base));
        tc::fence_before_sync();
    }
    __syncthreads();
    // let the merge grid launch now; it waits for this grid to complete
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (wide) {
        if constexpr (kTcPrefix) {
            tc::fence_after_sync();
            if constexpr (KV::kElemBytes == 2) {
                if (tc_pairs)
                    prefix_cta_tc_pair<D>(&maps, a, smem, bars, tmem_base, warp, lane, &abort_flag,
                                          tc_meta);
                else
                    prefix_cta_tc<D, KV>(&maps, a, smem, bars, tmem_base, warp, lane, &abort_flag,
                                         tc_meta);
            } else {
                prefix_cta_tc<D, KV>(&maps, a, smem, bars, tmem_base, warp, lane, &abort_flag,
                                     tc_meta);
            }
            tc::fence_before_sync();
            __syncthreads();
            tc::fence_after_sync();
            if (warp == kTcMmaWarp) tc::dealloc<kTcTmemCols>(tmem_base);
        } else {
            prefix_cta<D, KV>(&maps.k, &maps.v, a, smem, ring, bars, warp, lane, &abort_flag,
                              id_slots);
        }
        // the prefix queue is empty: this CTA joins the suffix queue with the
        // same shared memory (every copy it issued has landed), unless every
        // suffix position is already claimed (the counter only grows, so a
        // stale read can only send the CTA to find the queue empty)
        __shared__ int suffix_open;
        if (threadIdx.x == 0)
            suffix_open = *static_cast<volatile int *>(a.queue_next + 1) < a.num_narrow_items;
        __syncthreads();
        if (abort_flag || !suffix_open) return;
        // barrier i is invalidated and re-initialised by thread i
        for (int i = threadIdx.x; i < prefix_bars || i < S::kNarrowBars; i += blockDim.x) {
            if (i < prefix_bars)
                asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(bars + 8 * i) : "memory");
            if (i < S::kNarrowBars) dev::mbar_init(bars + 8 * i, 1);
        }
        dev::fence_mbar_init();
        __syncthreads();
    }
    if (warp < S::kSuffixWarps)
        suffix_warp<D, KV>(maps, a, ring, bars, warp, lane, grab_items[warp]);
}

// Shared memory and carveout are set once per device (with that device
// current); reports the number of CTAs that fit per SM (the persistent grid
// needs one).  The per-device results sit in an array guarded by a mutex, so
// threads that plan or decode on different devices neither race nor read
// another device's count.
constexpr int kMaxConfigDevices = 64;

template <int D, class KV>
cudaError_t configure(int *ctas_per_sm) {
    using S = Shape<D, KV>;
    static std::mutex mu;
    static int resident[kMaxConfigDevices] = {};   // 0: not configured yet
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxConfigDevices) return cudaErrorNotSupported;
    std::lock_guard<std::mutex> lock(mu);
    if (resident[dev] == 0) {
        e = cudaFuncSetAttribute(attn_kernel<D, KV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 S::kSmemBytes);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(attn_kernel<D, KV>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        int n = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attn_kernel<D, KV>, kThreads,
                                                          S::kSmemBytes);
        if (e != cudaSuccess) return e;
        // a kernel that does not fit is remembered as -1 (never configured again)
        resident[dev] = n > 0 ? n : -1;
    }
    if (ctas_per_sm) *ctas_per_sm = resident[dev] > 0 ? resident[dev] : 0;
    return cudaSuccess;
}

template <int D, class KV>
cudaError_t launch(const AttnArgs &a, const KvMaps &maps, cudaStream_t stream) {
    using S = Shape<D, KV>;
    cudaError_t e = configure<D, KV>(nullptr);
    if (e != cudaSuccess) return e;
    attn_kernel<D, KV><<<a.num_ctas, kThreads, S::kSmemBytes, stream>>>(maps, a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t attn_mma_ctas_per_sm(int head_dim, int mode, int *ctas_per_sm) {
    if (mode == PARASON_FP8_E4M3_KV)
        return head_dim == 128 ? configure<128, KvE4m3>(ctas_per_sm) : cudaErrorNotSupported;
    if (head_dim == 128) {
        const cudaError_t e = configure<128, KvBf16Deep>(nullptr);
        if (e != cudaSuccess) return e;
        return configure<128, KvBf16>(ctas_per_sm);
    }
    if (head_dim == 64) return configure<64, KvBf16>(ctas_per_sm);
    return cudaErrorNotSupported;
}

cudaError_t launch_attn_bf16(const AttnArgs &a, const KvMaps &maps, int head_dim,
                             cudaStream_t stream) {
    if (a.num_items <= 0 || a.num_ctas <= 0) return cudaSuccess;
    if (head_dim == 128)
        return a.suffix_warps == KvBf16Deep::kSuffixWarps ? launch<128, KvBf16Deep>(a, maps, stream)
                                                          : launch<128, KvBf16>(a, maps, stream);
    if (head_dim == 64) return launch<64, KvBf16>(a, maps, stream);
    return cudaErrorNotSupported;
}

cudaError_t launch_attn_fp8(const AttnArgs &a, const KvMaps &maps, int head_dim,
                            cudaStream_t stream) {
    if (a.num_items <= 0 || a.num_ctas <= 0) return cudaSuccess;
    if (head_dim == 128) return launch<128, KvE4m3>(a, maps, stream);
    return cudaErrorNotSupported;
}

}  // namespace parason
