// Grouped-query attention with one query per row over that row's KV history:
//     out[r, h] = softmax(q[r, h] . K[0..ctx_r)^T / sqrt(hd)) V[0..ctx_r),  ctx_r = pos_r + 1
// Used for decode (row = live rollout, KV = its slot) and for prefill (row = one prompt
// token, KV = the prompt's slot, causal by construction).
//
// q and the KV cache are fp16; the output is a bf16 hi/lo pair (the next GEMM's operand).
//
// Work item = (row, split of `chunk` positions) for one KV head (blockIdx.y): the CTA loads
// the G = n_heads / n_kv query heads that share the KV head once and streams the split's K
// and V rows (256 contiguous bytes each at hd = 128) exactly once with 16-byte loads, the
// next iteration's rows in flight while the current ones are used.  Each half-warp owns
// one position at a time, each lane hd/16 dimensions; scores are reduced with xor-shuffles
// inside the half-warp (the warp's two halves always iterate together) and folded into an
// online softmax (base-2, exp2f) four positions at a time.  The 8 half-warp states are
// merged in shared memory; rows with several splits write fp32 partials and the last split
// to arrive (per-row counter, no spinning) merges them in split order.
#pragma once
#include "device_common.cuh"

namespace sara {

constexpr int kAttnThreads = 128;
constexpr int kAttnMaxG = 8;
constexpr int kAttnPPI = 4;         // positions per half-warp per iteration
constexpr int kAttnMaxSplits = 96;  // largest split count the merge handles in shared memory

struct AttnParams {
    const uint16_t *q;        // [rows][n_heads][hd] fp16
    uint16_t *out;            // [rows][n_heads][hd] bf16 hi
    uint16_t *out_lo;         // [rows][n_heads][hd] bf16 lo (may be null)
    const uint16_t *kv;       // slot s at kv + s * slot_stride: [2][n_kv][cap][hd] fp16
    int64_t slot_stride;
    int cap;
    const int *row_slot;      // [rows]
    const int *row_pos;       // [rows] position of the query token (ctx = pos + 1)
    const int2 *items;        // [n_items] (row, split)
    const int *n_items_dev;   // device item count (nullptr -> n_items_fixed)
    int n_items_fixed;
    const int *row_item0;     // [rows] index of the row's first item
    int n_heads, n_kv, chunk;
    float scale_log2;         // log2(e) / sqrt(hd)
    float *part;              // [items][n_kv][G][hd + 2] fp32 partials (m, l, o[hd])
    int *cnt;                 // [rows][n_kv] arrival counters, zero between launches
    int *err;
    uint64_t *stamps;         // optional [blocks][16] phase timestamps (profiling builds)
};

#ifdef SARA_STAMPS
#define ATTN_STAMP(i) do { if (p.stamps && threadIdx.x == 0 && blockIdx.y == 0 && blockIdx.x < 152) p.stamps[(size_t)blockIdx.x * 16 + (i)] = globaltimer_ns(); } while (0)
#else
#define ATTN_STAMP(i) do { } while (0)
#endif

__device__ __forceinline__ float2 half2_bits_to_float2(uint32_t w) {
    __half2 h;
    *reinterpret_cast<uint32_t *>(&h) = w;
    return __half22float2(h);
}

// bf16 hi/lo store of one output element
__device__ __forceinline__ void attn_store(const AttnParams &p, int64_t idx, float v) {
    uint16_t hi, lo;
    split_bf16(v, hi, lo);
    p.out[idx] = hi;
    if (p.out_lo) p.out_lo[idx] = lo;
}

template <int DPL>
__device__ __forceinline__ void attn_load_words(const uint16_t *p, uint32_t (&w)[DPL / 2]) {
    if constexpr (DPL == 8) {
        const uint4 x = *reinterpret_cast<const uint4 *>(p);
        w[0] = x.x; w[1] = x.y; w[2] = x.z; w[3] = x.w;
    } else if constexpr (DPL == 4) {
        const uint2 x = *reinterpret_cast<const uint2 *>(p);
        w[0] = x.x; w[1] = x.y;
    } else {
        w[0] = *reinterpret_cast<const uint32_t *>(p);
    }
}

template <int HD, int G>
__global__ void __launch_bounds__(kAttnThreads)
attn_rows_kernel(AttnParams p) {
    constexpr int DPL = HD / 16;  // dims per lane
    constexpr int NW = DPL / 2;   // packed bf16 words per lane and position
    static_assert(DPL == 2 || DPL == 4 || DPL == 8, "head_dim must be 32, 64 or 128");
    static_assert(G >= 1 && G <= kAttnMaxG, "query group must be 1..8");
    __shared__ float s_m[8][G], s_l[8][G];
    __shared__ float s_o[8][G][HD];
    __shared__ float s_fin_m[G], s_fin_l[G];
    __shared__ float s_w[G][kAttnMaxSplits];
    __shared__ int s_last;

    ATTN_STAMP(0);
    pdl_wait_prior_grids();
    pdl_allow_dependents();
    const int n_items = p.n_items_dev ? *p.n_items_dev : p.n_items_fixed;
    const int kvh = blockIdx.y;
    ATTN_STAMP(1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int half = lane >> 4, dl = lane & 15;
    const int hw = warp * 2 + half;  // half-warp id 0..7
    const unsigned fmask = 0xffffffffu;
    constexpr int kStride = 8 * kAttnPPI;  // positions per CTA iteration

    for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
        const int2 it = p.items[item];
        const int row = it.x, split = it.y;
        const int ctx = p.row_pos[row] + 1;
        const int p0 = split * p.chunk, p1 = min(ctx, p0 + p.chunk);
        const int nsplit = (ctx + p.chunk - 1) / p.chunk;
        const uint16_t *Kb = p.kv + (int64_t)p.row_slot[row] * p.slot_stride + (int64_t)kvh * p.cap * HD + dl * DPL;
        const uint16_t *Vb = Kb + (int64_t)p.n_kv * p.cap * HD;

        // q slice of every head in the group, pre-scaled by log2(e)/sqrt(hd)
        float q[G][DPL];
#pragma unroll
        for (int g = 0; g < G; ++g) {
            uint32_t w[NW];
            attn_load_words<DPL>(p.q + ((int64_t)row * p.n_heads + kvh * G + g) * HD + dl * DPL, w);
#pragma unroll
            for (int i = 0; i < NW; ++i) {
                const float2 f = half2_bits_to_float2(w[i]);
                q[g][2 * i] = f.x * p.scale_log2;
                q[g][2 * i + 1] = f.y * p.scale_log2;
            }
        }
        float m[G], l[G], o[G][DPL];
#pragma unroll
        for (int g = 0; g < G; ++g) {
            m[g] = -INFINITY;
            l[g] = 0.f;
#pragma unroll
            for (int d = 0; d < DPL; ++d) o[g][d] = 0.f;
        }

        // the trip count is uniform across the warp (full-warp shuffles below)
        const int wstart = p0 + warp * 2 * kAttnPPI;
        uint32_t kw[kAttnPPI][NW], vw[kAttnPPI][NW];
        auto load_rows = [&](int wb, uint32_t (&K)[kAttnPPI][NW], uint32_t (&V)[kAttnPPI][NW]) {
#pragma unroll
            for (int j = 0; j < kAttnPPI; ++j) {
                const int pp = wb + half * kAttnPPI + j;
                const int pc = pp < p1 ? pp : p0;
                attn_load_words<DPL>(Kb + (int64_t)pc * HD, K[j]);
                attn_load_words<DPL>(Vb + (int64_t)pc * HD, V[j]);
            }
        };
        ATTN_STAMP(2);
        if (wstart < p1) load_rows(wstart, kw, vw);
        for (int wbase = wstart; wbase < p1; wbase += kStride) {
            uint32_t nk[kAttnPPI][NW], nv[kAttnPPI][NW];
            const bool more = wbase + kStride < p1;
            if (more) load_rows(wbase + kStride, nk, nv);
            const int base = wbase + half * kAttnPPI;
            float kf[kAttnPPI][DPL], vf[kAttnPPI][DPL];
#pragma unroll
            for (int j = 0; j < kAttnPPI; ++j)
#pragma unroll
                for (int i = 0; i < NW; ++i) {
                    const float2 k2 = half2_bits_to_float2(kw[j][i]);
                    const float2 v2 = half2_bits_to_float2(vw[j][i]);
                    kf[j][2 * i] = k2.x;
                    kf[j][2 * i + 1] = k2.y;
                    vf[j][2 * i] = v2.x;
                    vf[j][2 * i + 1] = v2.y;
                }
#pragma unroll
            for (int g = 0; g < G; ++g) {
                float sc[kAttnPPI];
#pragma unroll
                for (int j = 0; j < kAttnPPI; ++j) {
                    float s = 0.f;
#pragma unroll
                    for (int d = 0; d < DPL; ++d) s = fmaf(q[g][d], kf[j][d], s);
                    s += __shfl_xor_sync(fmask, s, 8);
                    s += __shfl_xor_sync(fmask, s, 4);
                    s += __shfl_xor_sync(fmask, s, 2);
                    s += __shfl_xor_sync(fmask, s, 1);
                    sc[j] = (base + j < p1) ? s : -INFINITY;
                }
                float mn = m[g];
#pragma unroll
                for (int j = 0; j < kAttnPPI; ++j) mn = fmaxf(mn, sc[j]);
                if (mn == -INFINITY) continue;  // nothing valid yet for this half-warp
                const float corr = exp2f(m[g] - mn);
                float pj[kAttnPPI], ps = 0.f;
#pragma unroll
                for (int j = 0; j < kAttnPPI; ++j) { pj[j] = exp2f(sc[j] - mn); ps += pj[j]; }
                l[g] = l[g] * corr + ps;
                m[g] = mn;
#pragma unroll
                for (int d = 0; d < DPL; ++d) {
                    float acc = o[g][d] * corr;
#pragma unroll
                    for (int j = 0; j < kAttnPPI; ++j) acc = fmaf(pj[j], vf[j][d], acc);
                    o[g][d] = acc;
                }
            }
            if (more) {
#pragma unroll
                for (int j = 0; j < kAttnPPI; ++j)
#pragma unroll
                    for (int i = 0; i < NW; ++i) { kw[j][i] = nk[j][i]; vw[j][i] = nv[j][i]; }
            }
        }
        ATTN_STAMP(3);
        // merge the 8 half-warp states
#pragma unroll
        for (int g = 0; g < G; ++g) {
            if (dl == 0) { s_m[hw][g] = m[g]; s_l[hw][g] = l[g]; }
#pragma unroll
            for (int d = 0; d < DPL; ++d) s_o[hw][g][dl * DPL + d] = o[g][d];
        }
        __syncthreads();
        if (threadIdx.x < G) {
            const int g = threadIdx.x;
            float M = -INFINITY;
            for (int h = 0; h < 8; ++h) M = fmaxf(M, s_m[h][g]);
            float L = 0.f;
            for (int h = 0; h < 8; ++h) L += (s_m[h][g] == -INFINITY) ? 0.f : s_l[h][g] * exp2f(s_m[h][g] - M);
            s_fin_m[g] = M;
            s_fin_l[g] = L;
        }
        __syncthreads();
        constexpr int per = G * HD;
        if (nsplit == 1) {
            for (int e = threadIdx.x; e < per; e += kAttnThreads) {
                const int g = e / HD, d = e - g * HD;
                const float M = s_fin_m[g];
                float acc = 0.f;
#pragma unroll
                for (int h = 0; h < 8; ++h)
                    if (s_m[h][g] != -INFINITY) acc += s_o[h][g][d] * exp2f(s_m[h][g] - M);
                attn_store(p, ((int64_t)row * p.n_heads + kvh * G + g) * HD + d, acc / s_fin_l[g]);
            }
        } else {
            float *mine = p.part + ((int64_t)item * p.n_kv + kvh) * G * (HD + 2);
            for (int e = threadIdx.x; e < per; e += kAttnThreads) {
                const int g = e / HD, d = e - g * HD;
                const float M = s_fin_m[g];
                float acc = 0.f;
#pragma unroll
                for (int h = 0; h < 8; ++h)
                    if (s_m[h][g] != -INFINITY) acc += s_o[h][g][d] * exp2f(s_m[h][g] - M);
                mine[g * (HD + 2) + 2 + d] = acc;
            }
            if (threadIdx.x < G) {
                mine[threadIdx.x * (HD + 2)] = s_fin_m[threadIdx.x];
                mine[threadIdx.x * (HD + 2) + 1] = s_fin_l[threadIdx.x];
            }
            __threadfence();
            __syncthreads();
            ATTN_STAMP(4);
            if (threadIdx.x == 0) {
                const int old = atomicAdd(&p.cnt[row * p.n_kv + kvh], 1);
                s_last = (old == nsplit - 1);
                if (s_last) p.cnt[row * p.n_kv + kvh] = 0;
            }
            __syncthreads();
            ATTN_STAMP(5);
            if (s_last) {
                __threadfence();
                const int i0 = p.row_item0[row];
                const float *base = p.part + ((int64_t)i0 * p.n_kv + kvh) * G * (HD + 2);
                const int64_t sp_stride = (int64_t)p.n_kv * G * (HD + 2);
                // per head: M = max_s m_s, weights w_s = 2^(m_s - M), L = sum_s w_s l_s (warp g)
                for (int g = warp; g < G; g += kAttnThreads / 32) {
                    float M = -INFINITY;
                    for (int sp = lane; sp < nsplit; sp += 32) M = fmaxf(M, __ldcg(base + sp * sp_stride + g * (HD + 2)));
#pragma unroll
                    for (int o2 = 16; o2 > 0; o2 >>= 1) M = fmaxf(M, __shfl_xor_sync(fmask, M, o2));
                    float L = 0.f;
                    for (int sp = lane; sp < nsplit; sp += 32) {
                        const float ms = __ldcg(base + sp * sp_stride + g * (HD + 2));
                        const float w = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
                        if (sp < kAttnMaxSplits) s_w[g][sp] = w;
                        L += w * __ldcg(base + sp * sp_stride + g * (HD + 2) + 1);
                    }
#pragma unroll
                    for (int o2 = 16; o2 > 0; o2 >>= 1) L += __shfl_xor_sync(fmask, L, o2);
                    if (lane == 0) s_fin_l[g] = L;
                }
                __syncthreads();
                for (int e = threadIdx.x; e < per; e += kAttnThreads) {
                    const int g = e / HD, d = e - g * HD;
                    float acc = 0.f;
                    const float *src = base + g * (HD + 2) + 2 + d;
#pragma unroll 4
                    for (int sp = 0; sp < nsplit; ++sp) acc += s_w[g][sp] * __ldcg(src + sp * sp_stride);
                    attn_store(p, ((int64_t)row * p.n_heads + kvh * G + g) * HD + d, acc / s_fin_l[g]);
                }
                ATTN_STAMP(6);
            }
        }
        __syncthreads();  // shared state reused by the next item
    }
    ATTN_STAMP(7);
}

}  // namespace sara
