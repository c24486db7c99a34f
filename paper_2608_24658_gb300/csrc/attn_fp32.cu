// attn_fp32.cu -- node-chunk attention for fp32 q/K/V (the fp32 parity mode).
//
// Same work items as the bf16 kernel (tiles of at most 16 rows in this mode),
// computed with plain fp32 FMAs so that results stay within 1e-5 of fp64:
// each of the 4 warps takes every 4th page of the chunk, each lane holds
// D/32 consecutive elements of a K/V row (coalesced 8- or 16-byte loads), a
// warp-wide shuffle reduction forms each score, and the online softmax is
// updated token by token.  The warps combine through shared memory.
#include "internal.h"

namespace parason {
namespace {

constexpr int kWarps = 4;
constexpr int kRows = 16;

template <int N>
__device__ __forceinline__ void load_vec(const float *p, float (&v)[N]) {
    if constexpr (N == 4) {
        const float4 t = *reinterpret_cast<const float4 *>(p);
        v[0] = t.x, v[1] = t.y, v[2] = t.z, v[3] = t.w;
    } else {
        const float2 t = *reinterpret_cast<const float2 *>(p);
        v[0] = t.x, v[1] = t.y;
    }
}

template <int D>
__global__ void __launch_bounds__(kWarps * 32)
    attn_fp32_kernel(const AttnArgs a, const float *__restrict__ kp, const float *__restrict__ vp) {
    constexpr int N = D / 32;
    __shared__ float sc_o[kWarps][kRows][D];
    __shared__ float2 sc_ml[kWarps][kRows];
    const WorkItem it = a.items[blockIdx.x];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float *qf = static_cast<const float *>(a.q);

    float q[kRows][N], o[kRows][N], m[kRows], l[kRows];
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
        m[r] = -INFINITY;
        l[r] = 0.f;
#pragma unroll
        for (int i = 0; i < N; ++i) o[r][i] = q[r][i] = 0.f;
        if (r < it.nrows) {
            const int nr = it.row0 + r;
            const int leaf = a.dfs_leaf[it.leaf_lo + nr / a.group];
            const int head = it.kv_head * a.group + nr % a.group;
            load_vec<N>(qf + (static_cast<int64_t>(leaf) * a.num_q_heads + head) * D + lane * N, q[r]);
        }
    }

    for (int pg = warp; pg < it.num_pages; pg += kWarps) {
        const int page = a.page_ids[it.page_pos + pg];
        const int valid = (pg == it.num_pages - 1) ? it.last_valid : kPageSize;
        const int64_t base = static_cast<int64_t>(page * a.num_kv_heads + it.kv_head) * kPageSize * D;
        for (int t = 0; t < valid; ++t) {
            float k[N], v[N];
            load_vec<N>(kp + base + t * D + lane * N, k);
            load_vec<N>(vp + base + t * D + lane * N, v);
#pragma unroll
            for (int r = 0; r < kRows; ++r) {
                if (r >= it.nrows) break;
                float dot = 0.f;
#pragma unroll
                for (int i = 0; i < N; ++i) dot = fmaf(q[r][i], k[i], dot);
#pragma unroll
                for (int s = 16; s > 0; s >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, s);
                const float x = dot * a.scale_log2;
                const float mn = fmaxf(m[r], x);
                const float al = exp2f(m[r] - mn);
                const float p = exp2f(x - mn);
                l[r] = l[r] * al + p;
#pragma unroll
                for (int i = 0; i < N; ++i) o[r][i] = fmaf(p, v[i], o[r][i] * al);
                m[r] = mn;
            }
        }
    }

#pragma unroll
    for (int r = 0; r < kRows; ++r) {
#pragma unroll
        for (int i = 0; i < N; ++i) sc_o[warp][r][lane * N + i] = o[r][i];
        if (lane == 0) sc_ml[warp][r] = make_float2(m[r], l[r]);
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < it.nrows * D; idx += kWarps * 32) {
        const int r = idx / D, c = idx % D;
        float M = -INFINITY;
        for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sc_ml[w][r].x);
        float L = 0.f, acc = 0.f;
        for (int w = 0; w < kWarps; ++w) {
            const float s = exp2f(sc_ml[w][r].x - M);
            L += s * sc_ml[w][r].y;
            acc += s * sc_o[w][r][c];
        }
        const int64_t slot = static_cast<int64_t>(it.slot_base) + r;
        a.part_o[slot * D + c] = acc;
        if (c == 0) a.part_ml[slot] = make_float2(M, L);
    }
}

}  // namespace

cudaError_t launch_attn_fp32(const AttnArgs &a, const float *k_pages, const float *v_pages,
                             int head_dim, cudaStream_t stream) {
    if (a.num_items <= 0) return cudaSuccess;
    if (head_dim == 128)
        attn_fp32_kernel<128><<<a.num_items, kWarps * 32, 0, stream>>>(a, k_pages, v_pages);
    else if (head_dim == 64)
        attn_fp32_kernel<64><<<a.num_items, kWarps * 32, 0, stream>>>(a, k_pages, v_pages);
    else
        return cudaErrorNotSupported;
    return cudaGetLastError();
}

}  // namespace parason
