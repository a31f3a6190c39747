// Grouped-query attention with one query per row over that row's KV history:
//     out[r, h] = softmax(q[r, h] . K[0..ctx_r)^T / sqrt(hd)) V[0..ctx_r),  ctx_r = pos_r + 1
// Used for decode (row = live rollout, KV = its slot) and for prefill (row = one prompt
// token, KV = the prompt's slot, causal by construction).
//
// Work item = (row, split of `chunk` positions) for one KV head (blockIdx.y): the CTA loads
// the G = n_heads / n_kv query heads that share the KV head once and streams the split's K
// and V rows (256 contiguous bytes each at hd = 128) exactly once with 16-byte loads.  Each
// half-warp owns one position at a time, each lane hd/16 dimensions; scores are reduced
// with xor-shuffles inside the half-warp (the warp's two halves always iterate together)
// and folded into an online softmax (base-2,
// exp2f) four positions at a time.  The 8 half-warp states are merged in shared memory;
// rows with several splits write fp32 partials and the last split to arrive (per-row
// counter, no spinning) merges them in split order.
#pragma once
#include "device_common.cuh"

namespace sara {

constexpr int kAttnThreads = 128;
constexpr int kAttnMaxG = 8;
constexpr int kAttnPPI = 4;  // positions per half-warp per iteration

struct AttnParams {
    const uint16_t *q;        // [rows][n_heads][hd]
    uint16_t *out;            // [rows][n_heads][hd]
    const uint16_t *kv;       // slot s at kv + s * slot_stride: [2][n_kv][cap][hd]
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
};

template <int HD>
__global__ void __launch_bounds__(kAttnThreads)
attn_rows_kernel(AttnParams p) {
    constexpr int DPL = HD / 16;  // dims per lane
    static_assert(DPL == 2 || DPL == 4 || DPL == 8, "head_dim must be 32, 64 or 128");
    __shared__ float s_m[8][kAttnMaxG], s_l[8][kAttnMaxG];
    __shared__ float s_o[8][kAttnMaxG][HD];
    __shared__ float s_fin_m[kAttnMaxG], s_fin_l[kAttnMaxG];
    __shared__ int s_last;

    pdl_wait_prior_grids();
    pdl_allow_dependents();
    const int n_items = p.n_items_dev ? *p.n_items_dev : p.n_items_fixed;
    const int kvh = blockIdx.y;
    const int G = p.n_heads / p.n_kv;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int half = lane >> 4, dl = lane & 15;
    const int hw = warp * 2 + half;  // half-warp id 0..7
    const unsigned fmask = 0xffffffffu;

    for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
        const int2 it = p.items[item];
        const int row = it.x, split = it.y;
        const int ctx = p.row_pos[row] + 1;
        const int p0 = split * p.chunk, p1 = min(ctx, p0 + p.chunk);
        const int nsplit = (ctx + p.chunk - 1) / p.chunk;
        const uint16_t *Kb = p.kv + (int64_t)p.row_slot[row] * p.slot_stride + (int64_t)kvh * p.cap * HD;
        const uint16_t *Vb = Kb + (int64_t)p.n_kv * p.cap * HD;

        // q slice of every head in the group, pre-scaled by log2(e)/sqrt(hd)
        float q[kAttnMaxG][DPL];
#pragma unroll
        for (int g = 0; g < kAttnMaxG; ++g) {
#pragma unroll
            for (int d = 0; d < DPL; ++d)
                q[g][d] = (g < G) ? bf16_to_f32(p.q[((int64_t)row * p.n_heads + kvh * G + g) * HD + dl * DPL + d]) *
                                        p.scale_log2
                                  : 0.f;
        }
        float m[kAttnMaxG], l[kAttnMaxG], o[kAttnMaxG][DPL];
#pragma unroll
        for (int g = 0; g < kAttnMaxG; ++g) {
            m[g] = -INFINITY;
            l[g] = 0.f;
#pragma unroll
            for (int d = 0; d < DPL; ++d) o[g][d] = 0.f;
        }

        // The trip count is uniform across the warp (both half-warps iterate together) because
        // the score reduction below uses full-warp shuffles; positions past p1 are masked.
        for (int wbase = p0 + warp * 2 * kAttnPPI; wbase < p1; wbase += 8 * kAttnPPI) {
            const int base = wbase + half * kAttnPPI;
            float kf[kAttnPPI][DPL], vf[kAttnPPI][DPL];
            bool valid[kAttnPPI];
#pragma unroll
            for (int j = 0; j < kAttnPPI; ++j) {
                const int pp = base + j;
                valid[j] = pp < p1;
                const int pc = valid[j] ? pp : p0;
                const uint16_t *kr = Kb + (int64_t)pc * HD + dl * DPL;
                const uint16_t *vr = Vb + (int64_t)pc * HD + dl * DPL;
                uint32_t kw[DPL / 2], vw[DPL / 2];
                if constexpr (DPL == 8) {
                    const uint4 kk = *reinterpret_cast<const uint4 *>(kr);
                    const uint4 vv = *reinterpret_cast<const uint4 *>(vr);
                    kw[0] = kk.x; kw[1] = kk.y; kw[2] = kk.z; kw[3] = kk.w;
                    vw[0] = vv.x; vw[1] = vv.y; vw[2] = vv.z; vw[3] = vv.w;
                } else if constexpr (DPL == 4) {
                    const uint2 kk = *reinterpret_cast<const uint2 *>(kr);
                    const uint2 vv = *reinterpret_cast<const uint2 *>(vr);
                    kw[0] = kk.x; kw[1] = kk.y;
                    vw[0] = vv.x; vw[1] = vv.y;
                } else {
                    kw[0] = *reinterpret_cast<const uint32_t *>(kr);
                    vw[0] = *reinterpret_cast<const uint32_t *>(vr);
                }
#pragma unroll
                for (int w = 0; w < DPL / 2; ++w) {
                    kf[j][2 * w] = __uint_as_float(kw[w] << 16);
                    kf[j][2 * w + 1] = __uint_as_float(kw[w] & 0xffff0000u);
                    vf[j][2 * w] = __uint_as_float(vw[w] << 16);
                    vf[j][2 * w + 1] = __uint_as_float(vw[w] & 0xffff0000u);
                }
            }
#pragma unroll
            for (int g = 0; g < kAttnMaxG; ++g) {
                if (g >= G) break;
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
                    sc[j] = valid[j] ? s : -INFINITY;
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
        }
        // merge the 8 half-warp states
#pragma unroll
        for (int g = 0; g < kAttnMaxG; ++g) {
            if (g < G) {
                if (dl == 0) { s_m[hw][g] = m[g]; s_l[hw][g] = l[g]; }
#pragma unroll
                for (int d = 0; d < DPL; ++d) s_o[hw][g][dl * DPL + d] = o[g][d];
            }
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
        const int per = G * HD;
        if (nsplit == 1) {
            for (int e = threadIdx.x; e < per; e += kAttnThreads) {
                const int g = e / HD, d = e - g * HD;
                const float M = s_fin_m[g];
                float acc = 0.f;
                for (int h = 0; h < 8; ++h)
                    if (s_m[h][g] != -INFINITY) acc += s_o[h][g][d] * exp2f(s_m[h][g] - M);
                p.out[((int64_t)row * p.n_heads + kvh * G + g) * HD + d] = f32_to_bf16(acc / s_fin_l[g]);
            }
        } else {
            float *mine = p.part + ((int64_t)item * p.n_kv + kvh) * G * (HD + 2);
            for (int e = threadIdx.x; e < per; e += kAttnThreads) {
                const int g = e / HD, d = e - g * HD;
                const float M = s_fin_m[g];
                float acc = 0.f;
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
            if (threadIdx.x == 0) {
                const int old = atomicAdd(&p.cnt[row * p.n_kv + kvh], 1);
                s_last = (old == nsplit - 1);
                if (s_last) p.cnt[row * p.n_kv + kvh] = 0;
            }
            __syncthreads();
            if (s_last) {
                __threadfence();
                const int i0 = p.row_item0[row];
                for (int e = threadIdx.x; e < per; e += kAttnThreads) {
                    const int g = e / HD, d = e - g * HD;
                    float M = -INFINITY;
                    for (int sp = 0; sp < nsplit; ++sp)
                        M = fmaxf(M, __ldcg(p.part + ((int64_t)(i0 + sp) * p.n_kv + kvh) * G * (HD + 2) + g * (HD + 2)));
                    float L = 0.f, acc = 0.f;
                    for (int sp = 0; sp < nsplit; ++sp) {
                        const float *src = p.part + ((int64_t)(i0 + sp) * p.n_kv + kvh) * G * (HD + 2) + g * (HD + 2);
                        const float ms = __ldcg(src);
                        if (ms == -INFINITY) continue;
                        const float w = exp2f(ms - M);
                        L += __ldcg(src + 1) * w;
                        acc += __ldcg(src + 2 + d) * w;
                    }
                    p.out[((int64_t)row * p.n_heads + kvh * G + g) * HD + d] = f32_to_bf16(acc / L);
                }
            }
        }
        __syncthreads();  // shared state reused by the next item
    }
}

}  // namespace sara
