// merge.cu -- log-sum-exp merge kernels.
//
// tree merge: branch b's attention over its root->leaf KV is the softmax over
// the union of the key sets of every (node, chunk) partial on its path, so
//   M = max_i m_i,  L = sum_i l_i 2^(m_i - M),  o = sum_i o_i 2^(m_i - M) / L,
//   lse = (M + log2 L) ln 2
// with the partials in the log2 domain of the attention kernels.  Every
// branch's result is needed because branch outputs are concatenated into the
// context that follows (paper Fig. 1, Sec. 3.1).
//
// lse merge: two normalised results over disjoint key sets with natural-log
// lse combine with weights e^{lse_a}, e^{lse_b}.
#include <cuda_bf16.h>

#include "internal.h"

namespace parason {
namespace {

constexpr int kMergeThreads = 128;
constexpr float kLn2 = 0.69314718055994530942f;

template <int D>
struct Vec;
template <>
struct Vec<128> {
    static constexpr int N = 4;
};
template <>
struct Vec<64> {
    static constexpr int N = 2;
};

template <int N>
__device__ __forceinline__ void load_f32(const float *p, float (&v)[N]) {
    if constexpr (N == 4) {
        const float4 t = *reinterpret_cast<const float4 *>(p);
        v[0] = t.x, v[1] = t.y, v[2] = t.z, v[3] = t.w;
    } else {
        const float2 t = *reinterpret_cast<const float2 *>(p);
        v[0] = t.x, v[1] = t.y;
    }
}

template <int N>
__device__ __forceinline__ void store_out(void *out, int64_t off, const float (&v)[N], bool bf16) {
    if (bf16) {
        __nv_bfloat16 *o = static_cast<__nv_bfloat16 *>(out) + off;
        if constexpr (N == 4) {
            __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]);
            __nv_bfloat162 b = __floats2bfloat162_rn(v[2], v[3]);
            uint2 u;
            u.x = *reinterpret_cast<uint32_t *>(&a);
            u.y = *reinterpret_cast<uint32_t *>(&b);
            *reinterpret_cast<uint2 *>(o) = u;
        } else {
            *reinterpret_cast<__nv_bfloat162 *>(o) = __floats2bfloat162_rn(v[0], v[1]);
        }
    } else {
        float *o = static_cast<float *>(out) + off;
        if constexpr (N == 4)
            *reinterpret_cast<float4 *>(o) = make_float4(v[0], v[1], v[2], v[3]);
        else
            *reinterpret_cast<float2 *>(o) = make_float2(v[0], v[1]);
    }
}

template <int N>
__device__ __forceinline__ void load_in(const void *in, int64_t off, float (&v)[N], bool bf16) {
    if (bf16) {
        const __nv_bfloat16 *p = static_cast<const __nv_bfloat16 *>(in) + off;
        if constexpr (N == 4) {
            const uint2 u = *reinterpret_cast<const uint2 *>(p);
            const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(&u.x);
            const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&u.y);
            v[0] = __low2float(a), v[1] = __high2float(a);
            v[2] = __low2float(b), v[3] = __high2float(b);
        } else {
            const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(p);
            v[0] = __low2float(a), v[1] = __high2float(a);
        }
    } else {
        load_f32<N>(static_cast<const float *>(in) + off, v);
    }
}

// W warps per (branch, q head), 4 / W rows per CTA of 4 warps (W = 4 when
// there are few rows, so that enough loads are in flight; 1 when there are
// many).  Warp w of a row folds entries w, w + W, w + 2W, ... of the row's
// list into its own (M_w, L_w, acc_w): lane e loads entry e's (m, l) (one
// round trip for up to 32 entries), the pass's max and weights come from warp
// reductions, then every lane accumulates its D/32 columns with the partial
// rows requested 8 at a time.  The W results combine through shared memory
// by the same rule.  Runs as a dependent grid of the attention kernel:
// griddepcontrol.wait returns once that grid has completed and its writes
// are visible.
template <int D, int W>
__global__ void __launch_bounds__(kMergeThreads)
    tree_merge_kernel(const MergeArgs a, bool out_bf16) {
    constexpr int N = Vec<D>::N;
    constexpr int kWarps = kMergeThreads / 32;
    constexpr int kRowsPerCta = kWarps / W;
    __shared__ float s_acc[W > 1 ? kWarps : 1][D];
    __shared__ float s_m[kWarps], s_l[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int w = warp % W;
    const int64_t row = static_cast<int64_t>(blockIdx.x) * kRowsPerCta + warp / W;   // b * H_q + h
    const bool active = row < static_cast<int64_t>(a.num_leaves) * a.num_q_heads;
    const int b = active ? static_cast<int>(row / a.num_q_heads) : 0;
    const int h = active ? static_cast<int>(row % a.num_q_heads) : 0;
    const int j = h / a.group, r = h % a.group;
    const int64_t pair = static_cast<int64_t>(b) * a.num_kv_heads + j;
    // the merge lists are plan data: read them while the attention grid drains
    const int2 rg = active ? a.merge_rng[pair] : make_int2(0, 0);
    const int e0 = rg.x, e1 = rg.y;
    const int first_e = e0 + w + W * lane;
    const int first_slot = first_e < e1 ? a.merge_ent[first_e] + r : 0;
    asm volatile("griddepcontrol.wait;" ::: "memory");
    // the attention grid is complete: rewind its work queues for the next call
    if (blockIdx.x == 0 && threadIdx.x == 0 && a.queue_next) {
        a.queue_next[0] = a.queue_start[0];
        a.queue_next[1] = a.queue_start[1];
    }

    float M = -INFINITY, L = 0.f;
    float acc[N];
#pragma unroll
    for (int i = 0; i < N; ++i) acc[i] = 0.f;
    // this warp's entries e0 + w + W * i, 32 per pass
    for (int i0 = 0; e0 + w + W * i0 < e1; i0 += 32) {
        const int e = e0 + w + W * (i0 + lane);
        const bool valid = e < e1;
        const int slot = valid ? (i0 == 0 ? first_slot : a.merge_ent[e] + r) : 0;
        const int cnt = min(32, (e1 - (e0 + w) + W - 1) / W - i0);
        // With few rows (W = 4: up to 8 entries a warp) the pass's first 8
        // partial rows are requested together with the (m, l) of its entries,
        // since they do not depend on the weights.  With many rows the extra
        // registers cost more occupancy than the round trip they save.
        constexpr int kEarly = W == 4 ? 8 : 0;
        float v0[kEarly > 0 ? kEarly : 1][N];
#pragma unroll
        for (int k = 0; k < kEarly; ++k) {
            const int si = __shfl_sync(0xffffffffu, slot, k);
            if (k < cnt) load_f32<N>(a.part_o + static_cast<int64_t>(si) * D + lane * N, v0[k]);
        }
        float m = -INFINITY, l = 0.f;
        if (valid) {
            const float2 ml = a.part_ml[slot];
            m = ml.x;
            l = ml.y;
        }
        float mb = m;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, o));
        const float Mn = fmaxf(M, mb);             // finite: the pass has a valid entry
        const float s_old = exp2f(M - Mn);
        const float wgt = valid ? exp2f(m - Mn) : 0.f;
        float lw = l * wgt;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) lw += __shfl_xor_sync(0xffffffffu, lw, o);
        L = L * s_old + lw;
#pragma unroll
        for (int i = 0; i < N; ++i) acc[i] *= s_old;
#pragma unroll
        for (int k = 0; k < kEarly; ++k) {
            const float wk = __shfl_sync(0xffffffffu, wgt, k);
            if (k < cnt)
#pragma unroll
                for (int c = 0; c < N; ++c) acc[c] += wk * v0[k][c];
        }
        for (int k0 = kEarly; k0 < cnt; k0 += 8) {
            float v[8][N];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int si = __shfl_sync(0xffffffffu, slot, (k0 + k) & 31);
                if (k0 + k < cnt) load_f32<N>(a.part_o + static_cast<int64_t>(si) * D + lane * N, v[k]);
            }
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float wk = __shfl_sync(0xffffffffu, wgt, (k0 + k) & 31);
                if (k0 + k < cnt)
#pragma unroll
                    for (int c = 0; c < N; ++c) acc[c] += wk * v[k][c];
            }
        }
        M = Mn;
    }
    if constexpr (W > 1) {
#pragma unroll
        for (int c = 0; c < N; ++c) s_acc[warp][lane * N + c] = acc[c];
        if (lane == 0) {
            s_m[warp] = M;
            s_l[warp] = L;
        }
        __syncthreads();
        if (w != 0) return;
        const int base = warp;                     // the row's first warp
        float Mg = -INFINITY;
#pragma unroll
        for (int u = 0; u < W; ++u) Mg = fmaxf(Mg, s_m[base + u]);
        L = 0.f;
#pragma unroll
        for (int c = 0; c < N; ++c) acc[c] = 0.f;
        if (Mg != -INFINITY) {
#pragma unroll
            for (int u = 0; u < W; ++u) {
                const float su = s_m[base + u] == -INFINITY ? 0.f : exp2f(s_m[base + u] - Mg);
                L += s_l[base + u] * su;
#pragma unroll
                for (int c = 0; c < N; ++c) acc[c] += su * s_acc[base + u][lane * N + c];
            }
        }
        M = Mg;
    }
    if (!active) return;
    const bool empty = !(L > 0.f);
    const float inv = empty ? 0.f : 1.f / L;
#pragma unroll
    for (int c = 0; c < N; ++c) acc[c] *= inv;
    store_out<N>(a.out, row * D + lane * N, acc, out_bf16);
    if (a.lse && lane == 0) a.lse[row] = empty ? -INFINITY : (M + log2f(L)) * kLn2;
}

// Many rows: one warp per (branch, kv head).  The kv head's G q heads share
// its merge list (q head j G + r reads slot entry + r), so the warp reads the
// list once and keeps the G rows' loads in flight together; per pass of up to
// 32 entries, every row's weights come from warp reductions as above, then
// the partial rows are requested 8 at a time over entries and heads.
template <int D, int G>
__global__ void __launch_bounds__(kMergeThreads)
    tree_merge_group_kernel(const MergeArgs a, bool out_bf16) {
    constexpr int N = Vec<D>::N;
    constexpr int KB = G >= 8 ? 1 : 8 / G;          // entries per batch of loads
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t pair = static_cast<int64_t>(blockIdx.x) * (kMergeThreads / 32) + warp;
    const bool active = pair < static_cast<int64_t>(a.num_leaves) * a.num_kv_heads;
    // the merge lists are plan data: read them while the attention grid drains
    const int2 rg = active ? a.merge_rng[pair] : make_int2(0, 0);
    const int e0 = rg.x, e1 = rg.y;
    const int first_slot = e0 + lane < e1 ? a.merge_ent[e0 + lane] : 0;
    asm volatile("griddepcontrol.wait;" ::: "memory");
    // the attention grid is complete: rewind its work queues for the next call
    if (blockIdx.x == 0 && threadIdx.x == 0 && a.queue_next) {
        a.queue_next[0] = a.queue_start[0];
        a.queue_next[1] = a.queue_start[1];
    }
    if (!active) return;

    float M[G], L[G], acc[G][N];
#pragma unroll
    for (int r = 0; r < G; ++r) {
        M[r] = -INFINITY;
        L[r] = 0.f;
#pragma unroll
        for (int c = 0; c < N; ++c) acc[r][c] = 0.f;
    }
    for (int i0 = 0; e0 + i0 < e1; i0 += 32) {
        const int e = e0 + i0 + lane;
        const bool valid = e < e1;
        const int slot = valid ? (i0 == 0 ? first_slot : a.merge_ent[e]) : 0;
        const int cnt = min(32, e1 - e0 - i0);
        float wgt[G];
#pragma unroll
        for (int r = 0; r < G; ++r) {
            float m = -INFINITY, l = 0.f;
            if (valid) {
                const float2 ml = a.part_ml[slot + r];
                m = ml.x;
                l = ml.y;
            }
            float mb = m;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, o));
            const float Mn = fmaxf(M[r], mb);       // finite: the pass has a valid entry
            const float s_old = exp2f(M[r] - Mn);
            wgt[r] = valid ? exp2f(m - Mn) : 0.f;
            float lw = l * wgt[r];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) lw += __shfl_xor_sync(0xffffffffu, lw, o);
            L[r] = L[r] * s_old + lw;
#pragma unroll
            for (int c = 0; c < N; ++c) acc[r][c] *= s_old;
            M[r] = Mn;
        }
        for (int k0 = 0; k0 < cnt; k0 += KB) {
            float v[KB][G][N];
#pragma unroll
            for (int k = 0; k < KB; ++k) {
                const int si = __shfl_sync(0xffffffffu, slot, (k0 + k) & 31);
#pragma unroll
                for (int r = 0; r < G; ++r)
                    if (k0 + k < cnt)
                        load_f32<N>(a.part_o + static_cast<int64_t>(si + r) * D + lane * N, v[k][r]);
            }
#pragma unroll
            for (int k = 0; k < KB; ++k)
#pragma unroll
                for (int r = 0; r < G; ++r) {
                    const float wk = __shfl_sync(0xffffffffu, wgt[r], (k0 + k) & 31);
                    if (k0 + k < cnt)
#pragma unroll
                        for (int c = 0; c < N; ++c) acc[r][c] += wk * v[k][r][c];
                }
        }
    }
#pragma unroll
    for (int r = 0; r < G; ++r) {
        const int64_t row = pair * G + r;            // b * H_q + j * G + r
        const bool empty = !(L[r] > 0.f);
        const float inv = empty ? 0.f : 1.f / L[r];
#pragma unroll
        for (int c = 0; c < N; ++c) acc[r][c] *= inv;
        store_out<N>(a.out, row * D + lane * N, acc[r], out_bf16);
        if (a.lse && lane == 0) a.lse[row] = empty ? -INFINITY : (M[r] + log2f(L[r])) * kLn2;
    }
}

template <int D>
__global__ void __launch_bounds__(kMergeThreads)
    lse_merge_kernel(const void *o_a, const float *lse_a, const void *o_b, const float *lse_b,
                     void *o_out, float *lse_out, int64_t rows, bool bf16) {
    constexpr int N = Vec<D>::N;
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * kMergeThreads + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (row >= rows) return;
    const float la = lse_a[row], lb = lse_b[row];
    float va[N], vb[N], o[N];
    load_in<N>(o_a, row * D + lane * N, va, bf16);
    load_in<N>(o_b, row * D + lane * N, vb, bf16);
    float lse;
    if (la == -INFINITY && lb == -INFINITY) {
#pragma unroll
        for (int i = 0; i < N; ++i) o[i] = 0.f;
        lse = -INFINITY;
    } else {
        const float mx = fmaxf(la, lb);
        const float wa = expf(la - mx), wb = expf(lb - mx);
        const float inv = 1.f / (wa + wb);
#pragma unroll
        for (int i = 0; i < N; ++i) o[i] = (wa * va[i] + wb * vb[i]) * inv;
        lse = mx + logf(wa + wb);
    }
    __syncwarp();   // every lane has read its inputs before any lane writes (aliasing)
    store_out<N>(o_out, row * D + lane * N, o, bf16);
    if (lane == 0) lse_out[row] = lse;
}

}  // namespace

cudaError_t launch_merge(const MergeArgs &a, int head_dim, int mode, bool programmatic,
                         cudaStream_t stream) {
    const int64_t rows = static_cast<int64_t>(a.num_leaves) * a.num_q_heads;
    if (rows == 0) return cudaSuccess;
    // warps per row: as many as keep the grid near 4096 warps, at most 4.
    // With at least 4096 (branch, kv head) pairs and groups of 2 or 4, one
    // warp per pair (measured: faster there; with groups of 8, or fewer
    // pairs, too few warps are left to hide the loads' latency)
    const int W = rows * 4 <= 4096 ? 4 : (rows * 2 <= 4096 ? 2 : 1);
    const int g = a.group;
    const bool grouped = W < 4 && (g == 2 || g == 4) && rows / g >= 4096;
    const int64_t warps = grouped ? rows / g : rows * W;
    const int64_t blocks = (warps + kMergeThreads / 32 - 1) / (kMergeThreads / 32);
    if (blocks > 0x7fffffff) return cudaErrorInvalidValue;
    const bool bf16 = mode != PARASON_FP32;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(blocks));
    cfg.blockDim = dim3(kMergeThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = programmatic ? 1 : 0;
    if (grouped) {
        if (head_dim == 128)
            return g == 2 ? cudaLaunchKernelEx(&cfg, tree_merge_group_kernel<128, 2>, a, bf16)
                          : cudaLaunchKernelEx(&cfg, tree_merge_group_kernel<128, 4>, a, bf16);
        if (head_dim == 64)
            return g == 2 ? cudaLaunchKernelEx(&cfg, tree_merge_group_kernel<64, 2>, a, bf16)
                          : cudaLaunchKernelEx(&cfg, tree_merge_group_kernel<64, 4>, a, bf16);
        return cudaErrorNotSupported;
    }
    if (head_dim == 128) {
        if (W == 4) return cudaLaunchKernelEx(&cfg, tree_merge_kernel<128, 4>, a, bf16);
        if (W == 2) return cudaLaunchKernelEx(&cfg, tree_merge_kernel<128, 2>, a, bf16);
        return cudaLaunchKernelEx(&cfg, tree_merge_kernel<128, 1>, a, bf16);
    }
    if (head_dim == 64) {
        if (W == 4) return cudaLaunchKernelEx(&cfg, tree_merge_kernel<64, 4>, a, bf16);
        if (W == 2) return cudaLaunchKernelEx(&cfg, tree_merge_kernel<64, 2>, a, bf16);
        return cudaLaunchKernelEx(&cfg, tree_merge_kernel<64, 1>, a, bf16);
    }
    return cudaErrorNotSupported;
}

cudaError_t launch_lse_merge(const void *o_a, const float *lse_a, const void *o_b,
                             const float *lse_b, void *o_out, float *lse_out, int64_t rows,
                             int head_dim, int mode, cudaStream_t stream) {
    if (rows <= 0) return cudaSuccess;
    const int64_t blocks = (rows * 32 + kMergeThreads - 1) / kMergeThreads;
    const bool bf16 = mode != PARASON_FP32;
    if (head_dim == 128)
        lse_merge_kernel<128><<<static_cast<unsigned>(blocks), kMergeThreads, 0, stream>>>(
            o_a, lse_a, o_b, lse_b, o_out, lse_out, rows, bf16);
    else if (head_dim == 64)
        lse_merge_kernel<64><<<static_cast<unsigned>(blocks), kMergeThreads, 0, stream>>>(
            o_a, lse_a, o_b, lse_b, o_out, lse_out, rows, bf16);
    else
        return cudaErrorNotSupported;
    return cudaGetLastError();
}

namespace {
__global__ void scatter_kernel(int32_t *base, const int2 *patches, int32_t n) {
    const int32_t i = static_cast<int32_t>(blockIdx.x * blockDim.x + threadIdx.x);
    if (i < n) base[patches[i].x] = patches[i].y;
}
}  // namespace

cudaError_t launch_scatter(int32_t *base, const int2 *patches, int32_t n, cudaStream_t stream) {
    if (n <= 0) return cudaSuccess;
    scatter_kernel<<<(n + 255) / 256, 256, 0, stream>>>(base, patches, n);
    return cudaGetLastError();
}

}  // namespace parason
