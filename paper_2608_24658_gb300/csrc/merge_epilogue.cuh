// merge_epilogue.cuh -- the log-sum-exp merge of one (branch, kv head), run
// inside the attention kernel by the CTA that completes its last partial.
//
// Branch b's attention over its root->leaf context is the softmax over the
// union of the key sets of all (node, chunk) partials on its path; with the
// partials in the log2 domain (m, l = sum 2^(x-m), o = sum 2^(x-m) v):
//   M = max_i m_i, L = sum_i l_i 2^(m_i - M), out = sum_i o_i 2^(m_i - M) / L,
//   lse = (M + log2 L) ln 2.
// Every branch's output is needed because all branch outputs are
// concatenated into the context that follows (paper Fig. 1, Sec. 3.1).
#pragma once

#include <cuda_bf16.h>

#include "device_common.cuh"
#include "internal.h"

namespace parason {
namespace dev {

constexpr float kLn2 = 0.69314718055994530942f;

// Partials are read with ld.global.cg: other SMs wrote them during this
// launch, so they must come from L2, never from a stale L1 line.
__device__ __forceinline__ float4 ldcg_f4(const float *p) {
    return __ldcg(reinterpret_cast<const float4 *>(p));
}

// Shared memory a merge may stage: slot, weight and m of up to kMergeBatch
// partials for up to kMergeMaxGroup q heads, plus per-row (M, L).
constexpr int kMergeBatch = 64;
constexpr int kMergeMaxGroup = 16;
constexpr int kMergeStageBytes = kMergeBatch * kMergeMaxGroup * 12 + kMergeMaxGroup * 8;

// Fallback for very long merge lists: one thread per output float4, the
// partials folded one after another (online max).
template <int D, int NT>
__device__ void merge_branch_head_serial(const AttnArgs &a, int b, int j, int tid) {
    constexpr int kVec = D / 4;
    const int g = a.group;
    const int e0 = a.merge_ptr[b], e1 = a.merge_ptr[b + 1];
    for (int w = tid; w < g * kVec; w += NT) {
        const int r = w / kVec, c4 = w % kVec;
        float M = -INFINITY, L = 0.f;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int e = e0; e < e1; ++e) {
            const int2 ent = a.merge_ent[e];
            const int64_t slot = static_cast<int64_t>(ent.x) + static_cast<int64_t>(j) * ent.y + r;
            const float2 ml = __ldcg(a.part_ml + slot);
            const float4 o = ldcg_f4(a.part_o + slot * D + 4 * c4);
            const float Mn = fmaxf(M, ml.x);
            const float s_old = exp2f(M - Mn), s_new = exp2f(ml.x - Mn);
            L = L * s_old + ml.y * s_new;
            acc.x = acc.x * s_old + o.x * s_new;
            acc.y = acc.y * s_old + o.y * s_new;
            acc.z = acc.z * s_old + o.z * s_new;
            acc.w = acc.w * s_old + o.w * s_new;
            M = Mn;
        }
        const float inv = L > 0.f ? 1.f / L : 0.f;
        const int64_t row = static_cast<int64_t>(b) * a.num_q_heads + j * g + r;
        __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x * inv, acc.y * inv);
        __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z * inv, acc.w * inv);
        uint2 u;
        u.x = *reinterpret_cast<uint32_t *>(&lo);
        u.y = *reinterpret_cast<uint32_t *>(&hi);
        *reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(a.out) + row * D + 4 * c4) = u;
        if (a.lse && c4 == 0) a.lse[row] = L > 0.f ? (M + log2f(L)) * kLn2 : -INFINITY;
    }
}

// Merge of (branch b, kv head j) by the NT consumer threads of a CTA (named
// barrier 1).  Three phases so that loads overlap instead of chaining:
//   1. every (partial, row) pair: its slot and (m, l), one load round trip;
//   2. per row: M, L and the weights 2^(m_i - M) / L;
//   3. every (row, float4 column): sum_i w_i o_i with independent loads.
template <int D, int NT>
__device__ void merge_branch_head(const AttnArgs &a, int b, int j, int tid, uint8_t *stage) {
    constexpr int kVec = D / 4;
    const int g = a.group;
    const int e0 = a.merge_ptr[b], e1 = a.merge_ptr[b + 1];
    const int n = e1 - e0;
    if (n > kMergeBatch || g > kMergeMaxGroup) {
        merge_branch_head_serial<D, NT>(a, b, j, tid);
        return;
    }
    const int ng = n * g;
    int *s_slot = reinterpret_cast<int *>(stage);
    float *s_w = reinterpret_cast<float *>(s_slot + kMergeBatch * kMergeMaxGroup);
    float *s_m = s_w + kMergeBatch * kMergeMaxGroup;
    float2 *s_row = reinterpret_cast<float2 *>(s_m + kMergeBatch * kMergeMaxGroup);
    for (int idx = tid; idx < ng; idx += NT) {
        const int e = idx / g, r = idx % g;
        const int2 ent = a.merge_ent[e0 + e];
        const int slot = ent.x + j * ent.y + r;      // < num_slots, which fits int32
        const float2 ml = __ldcg(a.part_ml + slot);
        s_slot[idx] = slot;
        s_m[idx] = ml.x;
        s_w[idx] = ml.y;
    }
    bar_sync<NT>(1);
    for (int r = tid; r < g; r += NT) {
        float M = -INFINITY;
        for (int e = 0; e < n; ++e) M = fmaxf(M, s_m[e * g + r]);
        float L = 0.f;
        for (int e = 0; e < n; ++e) L += s_w[e * g + r] * exp2f(s_m[e * g + r] - M);
        const float inv = L > 0.f ? 1.f / L : 0.f;
        for (int e = 0; e < n; ++e) s_w[e * g + r] = exp2f(s_m[e * g + r] - M) * inv;
        s_row[r] = make_float2(M, L);
    }
    bar_sync<NT>(1);
    for (int w = tid; w < g * kVec; w += NT) {
        const int r = w / kVec, c4 = w % kVec;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
        for (int e = 0; e < n; ++e) {
            const float wt = s_w[e * g + r];
            const float4 o = ldcg_f4(a.part_o + static_cast<int64_t>(s_slot[e * g + r]) * D + 4 * c4);
            acc.x += wt * o.x;
            acc.y += wt * o.y;
            acc.z += wt * o.z;
            acc.w += wt * o.w;
        }
        const int64_t row = static_cast<int64_t>(b) * a.num_q_heads + j * g + r;
        __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
        __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
        uint2 u;
        u.x = *reinterpret_cast<uint32_t *>(&lo);
        u.y = *reinterpret_cast<uint32_t *>(&hi);
        *reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(a.out) + row * D + 4 * c4) = u;
        if (a.lse && c4 == 0) {
            const float2 ML = s_row[r];
            a.lse[row] = ML.y > 0.f ? (ML.x + log2f(ML.y)) * kLn2 : -INFINITY;
        }
    }
    bar_sync<NT>(1);
}

// Branches whose whole path holds no token: out = 0, lse = -inf.
template <int D>
__device__ void write_empty_branches(const AttnArgs &a, int tid, int nthreads) {
    const int64_t per = static_cast<int64_t>(a.num_q_heads) * D;
    for (int i = 0; i < a.num_empty_leaves; ++i) {
        const int b = a.empty_leaves[i];
        __nv_bfloat16 *o = static_cast<__nv_bfloat16 *>(a.out) + b * per;
        for (int64_t k = tid; k < per; k += nthreads) o[k] = __float2bfloat16(0.f);
        if (a.lse)
            for (int h = tid; h < a.num_q_heads; h += nthreads)
                a.lse[static_cast<int64_t>(b) * a.num_q_heads + h] = -INFINITY;
    }
}

}  // namespace dev
}  // namespace parason
