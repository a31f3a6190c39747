// Small kernels of the step graph: embedding gather for the prefill rows (with the first
// RMSNorm's inputs), sampling reduction + per-step bookkeeping, and the teacher-forcing
// round setup.
#pragma once
#include "controller.cuh"
#include "device_common.cuh"
#include "step_state.cuh"

namespace sara {

// x_f32[r] = E[tok[r]]; xg[r] = x * g as a bf16 hi/lo pair; ssq[t][r] = sum over features
// [128t, 128t+128) of x^2.  One CTA (128 threads) per row; rows >= *rows_dev exit.
static __global__ void __launch_bounds__(128) embed_kernel(const uint16_t *E, const uint16_t *g, const int *rows_dev,
                                                           const int *row_tok, int d, int rows_cap, int vocab,
                                                           float *x_f32, uint16_t *xg, uint16_t *xg_lo, float *ssq,
                                                           int *err) {
    pdl_wait_prior_grids();
    pdl_allow_dependents();
    const int rows = min(*rows_dev, rows_cap);
    __shared__ float red[4];
    for (int r = blockIdx.x; r < rows; r += gridDim.x) {
        int tok = row_tok[r];
        if (tok < 0 || tok >= vocab) {  // token ids come from the caller: never read outside E
            if (threadIdx.x == 0) report_error(err, ERR_BOUNDS);
            tok = 0;
        }
        const uint16_t *er = E + (int64_t)tok * d;
        for (int t = 0; t < d / 128; ++t) {
            const int f = t * 128 + threadIdx.x;
            const float x = bf16_to_f32(er[f]);
            x_f32[(int64_t)r * d + f] = x;
            uint16_t hi, lo;
            split_bf16(x * bf16_to_f32(g[f]), hi, lo);
            xg[(int64_t)r * d + f] = hi;
            xg_lo[(int64_t)r * d + f] = lo;
            const float s = warp_sum(x * x);
            if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
            __syncthreads();
            if (threadIdx.x == 0) ssq[(int64_t)t * rows_cap + r] = red[0] + red[1] + red[2] + red[3];
            __syncthreads();
        }
    }
}

// 256-thread exclusive scan helper (blockDim.x == 256): returns the prefix, sets total.
__device__ __forceinline__ int scan256(int v, int &total, int *warp_tot) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    int before = 0, tot = 0;
    for (int w = 0; w < 8; ++w) {
        if (w < warp) before += warp_tot[w];
        tot += warp_tot[w];
    }
    __syncthreads();
    total = tot;
    return before + x - v;
}

// Sampling finish + step bookkeeping, after the decode-step kernel.  That kernel's lm_head
// epilogue left, per live row, the first maximum of logit + Gumbel noise of every (256-token
// tile, 128-token half) (arg_val / arg_idx [rows][2 * tiles]); CTA r reduces row r's maxima
// to its token (ties: lowest token id).  The last CTA to finish appends each row's token to
// its rollout, retires rollouts that reached their length, compacts the live rows (order
// kept) and writes the next step's rows and attention items.
static __global__ void __launch_bounds__(256) sample_finish_kernel(StepPtrs c, int vocab) {
    __shared__ float sv[8];
    __shared__ int si[8];
    __shared__ int s_last;
    __shared__ int warp_tot[8];
    pdl_wait_prior_grids();
    pdl_allow_dependents();
    StepVars &V = *c.v;
    const int live = V.live;
    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (r < live) {
        const int tiles = (vocab + 255) / 256, nparts = 2 * tiles;
        float best = -INFINITY;
        int bi = 0x7fffffff;
        for (int j = tid; j < nparts; j += blockDim.x) {
            if ((j & 1) * 128 >= min(256, vocab - 256 * (j >> 1))) continue;  // a half tile past the vocabulary
            const float v = __ldcg(&c.arg_val[(int64_t)r * nparts + j]);
            const int id = __ldcg(&c.arg_idx[(int64_t)r * nparts + j]);
            if (v > best || (v == best && id < bi)) { best = v; bi = id; }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ob = __shfl_xor_sync(0xffffffffu, best, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (ob > best || (ob == best && oi < bi)) { best = ob; bi = oi; }
        }
        if (lane == 0) { sv[warp] = best; si[warp] = bi; }
        __syncthreads();
        if (tid == 0) {
            for (int w = 1; w < 8; ++w)
                if (sv[w] > best || (sv[w] == best && si[w] < bi)) { best = sv[w]; bi = si[w]; }
            c.sampled[r] = bi;
        }
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
        const int old = atomicAdd(&V.fin_count, 1);
        s_last = (old == (int)gridDim.x - 1);
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (tid == 0) {
        V.fin_count = 0;
        // the preceding decode-step launch's duration into the step's kernel-time total
        if (V.kt1 > V.kt0) V.kernel_ns += (int64_t)(V.kt1 - V.kt0);
        V.kt0 = ~0ull;
        V.kt1 = 0ull;
    }
    if (live == 0) return;
    const StepConst &K = *c.kc;
    const int Lp = K.Lp, B = K.attn_chunk;
    const int nsh = shared_blocks(Lp, B);
    // bookkeeping over the live rows (several passes of 256)
    int out = 0;
    int top = V.blk_top, low = V.blk_low;  // the KV block free stack (same value in every thread)
    int stop = V.slot_top;                 // the free rollout slots (asynchronous schedule)
    for (int base = 0; base < live; base += 256) {
        const int i = base + tid;
        int keep = 0, slot = 0, gen = 0, next_tok = 0;
        if (i < live) {
            slot = c.row_slot[i];
            gen = c.seq_gen[slot];
            const int tok = __ldcg(&c.sampled[i]);
            if (K.teacher) {
                c.sampled_out[(int64_t)slot * K.T_forced + gen] = tok;
                next_tok = (gen + 1 < K.T_forced) ? c.forced[(int64_t)slot * K.T_forced + gen] : 0;
            } else {
                c.gen_tok[((int64_t)c.seq_q[slot] * K.k + c.seq_j[slot]) * K.max_gen + gen] = tok;
                next_tok = tok;
            }
            gen += 1;
            c.seq_gen[slot] = gen;
            keep = gen < c.seq_len[slot];
        }
        // KV blocks, in row order: a finished rollout returns its private blocks (positions
        // up to Lp - 2 + gen), then a kept one whose next position opens a block takes one
        int32_t *bt = c.blk_tab + (int64_t)slot * c.nblk_max;
        int nfree = 0, need = 0;
        if (i < live) {
            if (!keep) nfree = (Lp + gen - 2) / B - nsh + 1;
            else need = ((Lp - 1 + gen) % B) == 0;
        }
        int ftot;
        const int foff = scan256(nfree, ftot, warp_tot);
        for (int j = 0; j < nfree; ++j) c.blk_free[top + foff + j] = bt[nsh + j];
        top += ftot;
        __syncthreads();
        int atot;
        const int aoff = scan256(need, atot, warp_tot);
        if (need) {
            const int at = top - 1 - aoff;
            if (at >= 0) bt[(Lp - 1 + gen) / B] = c.blk_free[at];
            else report_error(&V.err, ERR_CAPACITY);
        }
        top = max(0, top - atot);
        low = min(low, top);
        if (K.schedule != 0) {
            // asynchronous schedule: a finished rollout returns its slot, and the prompt whose
            // batch it completes is listed for the decisions at this step boundary
            const int fin = (i < live && !keep) ? 1 : 0;
            int stot;
            const int soff = scan256(fin, stot, warp_tot);
            if (fin) {
                c.slot_free[stop + soff] = slot;
                const int q = c.seq_q[slot];
                if (atomicSub(&c.q_inflight[q], 1) == 1) c.dec_list[atomicAdd(&V.n_dec, 1)] = q;
            }
            stop += stot;
        }
        // stable in-place compaction: a kept row lands at or before its own index
        int tot;
        const int before = scan256(keep, tot, warp_tot);
        if (keep) {
            const int dst = out + before;
            c.row_slot[dst] = slot;
            c.row_pos[dst] = Lp - 1 + gen;
            c.row_tok[dst] = next_tok;
            c.row_seed[dst] = sampler_row_seed(K.sample_seed, c.seq_uid[slot], gen);
        }
        __syncthreads();
        out += tot;
    }
    // attention items of the next step: splits of `span` KV blocks
    int blocks = 0;
    for (int base = 0; base < out; base += 256) {
        const int i = base + tid;
        int tot;
        scan256(i < out ? (c.row_pos[i] + K.attn_chunk) / K.attn_chunk : 0, tot, warp_tot);
        blocks += tot;
    }
    const int span = att_span_for(blocks, K.att_slots, out);
    int items = 0;
    for (int base = 0; base < out; base += 256) {
        const int i = base + tid;
        const int ns = (i < out) ? ((c.row_pos[i] + K.attn_chunk) / K.attn_chunk + span - 1) / span : 0;
        int tot;
        const int before = scan256(ns, tot, warp_tot);
        if (i < out) {
            const int i0 = items + before;
            c.row_item0[i] = i0;
            for (int sp = 0; sp < ns; ++sp) {
                if (i0 + sp < c.att_cap) c.att_items[i0 + sp] = make_int2(i, sp);
                else report_error(&V.err, ERR_CAPACITY);
            }
        }
        items += tot;
    }
    if (tid == 0) {
        V.live = out;
        V.att_items = min(items, c.att_cap);
        V.att_span = span;
        V.exec_steps += 1;
        V.round_steps += 1;
        V.blk_top = top;
        V.blk_low = low;
        V.slot_top = stop;
    }
}

// Teacher forcing: n rollouts, rollout i uses prompt slot i and rollout slot i, lengths T.
static __global__ void __launch_bounds__(kCtlThreads, 1) teacher_setup_kernel(StepPtrs c, int n, const int64_t *uid) {
    pdl_wait_prior_grids();
    const StepConst &K = *c.kc;
    StepVars &V = *c.v;
    const int Lp = K.Lp, Lpre = Lp - 1;
    const int nblk = (Lp + K.attn_chunk - 1) / K.attn_chunk;
    const int span = att_span_for((int64_t)n * nblk, K.att_slots, n);
    const int nsplit = (nblk + span - 1) / span;
    const int nsh = shared_blocks(Lp, K.attn_chunk);
    for (int i = threadIdx.x; i < c.n_priv; i += kCtlThreads) c.blk_free[i] = c.n_shared + c.n_priv - 1 - i;
    __syncthreads();
    for (int r = threadIdx.x; r < n; r += kCtlThreads) {
        int32_t *bt = c.blk_tab + (int64_t)r * c.nblk_max;  // prompt r's full blocks, then a private one
        for (int j = 0; j < nsh; ++j) bt[j] = r * c.nsh_max + j;
        bt[nsh] = r < c.n_priv ? c.blk_free[c.n_priv - 1 - r] : c.n_shared;  // (n > n_priv: an error)
        c.fresh_pslot[r] = r;
        c.new_slots[r] = r;
        c.seq_q[r] = r;
        c.seq_j[r] = 0;
        c.seq_len[r] = K.T_forced;
        c.seq_gen[r] = 0;
        c.seq_pslot[r] = r;
        c.seq_uid[r] = uid[r];
        c.row_slot[r] = r;
        c.row_pos[r] = Lp - 1;
        c.row_tok[r] = c.p_tok[(int64_t)r * Lp + Lp - 1];
        c.row_seed[r] = sampler_row_seed(K.sample_seed, uid[r], 0);
        c.row_item0[r] = r * nsplit;
        for (int sp = 0; sp < nsplit; ++sp) c.att_items[r * nsplit + sp] = make_int2(r, sp);
    }
    for (int r = threadIdx.x; r < n * Lpre; r += kCtlThreads) {
        const int f = r / Lpre, t = r - f * Lpre;
        c.pre_slot[r] = f;
        c.pre_pos[r] = t;
        c.pre_tok[r] = c.p_tok[(int64_t)f * Lp + t];
        c.pre_items[r] = make_int2(r, 0);
        c.pre_item0[r] = r;
    }
    if (threadIdx.x == 0) {
        StepVars z;
        memset(&z, 0, sizeof(z));
        z.round = 0;
        z.live = n;
        z.att_items = n * nsplit;
        z.att_span = span;
        z.pre_rows = n * Lpre;
        z.n_fresh = n;
        z.round_maxL = K.T_forced;
        z.kt0 = ~0ull;
        z.blk_top = z.blk_low = c.n_priv - n;
        z.n_new = n;
        if (n > c.n_priv) z.err |= ERR_CAPACITY;
        V = z;
    }
}

// Gumbel-max over given fp32 logits (kernel-level entry point): one CTA per row.
static __global__ void __launch_bounds__(256) sample_rows_kernel(const float *logits, int V, uint64_t sample_seed,
                                                                 const int64_t *uid, const int *t, int *token) {
    __shared__ float sv[8];
    __shared__ int si[8];
    const int r = blockIdx.x;
    const uint64_t rs = sampler_row_seed(sample_seed, uid[r], t[r]);
    float best = -INFINITY;
    int bi = 0x7fffffff;
    for (int v = threadIdx.x; v < V; v += blockDim.x) {
        const float z = logits[(int64_t)r * V + v] + gumbel_from_hash(splitmix_at(rs, (uint64_t)v + 1));
        if (z > best) { best = z; bi = v; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ob = __shfl_xor_sync(0xffffffffu, best, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (ob > best || (ob == best && oi < bi)) { best = ob; bi = oi; }
    }
    if ((threadIdx.x & 31) == 0) { sv[threadIdx.x >> 5] = best; si[threadIdx.x >> 5] = bi; }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < 8; ++w)
            if (sv[w] > best || (sv[w] == best && si[w] < bi)) { best = sv[w]; bi = si[w]; }
        token[r] = bi;
    }
}

}  // namespace sara
