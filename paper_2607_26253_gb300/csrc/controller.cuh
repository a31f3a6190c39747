// SARA controller on the GPU (Algorithm 1 of arxiv 2607.26253), one CTA of 1024 threads.
//
// Runs at the top of every loop iteration of the step graph.  Mid-round (live rows > 0) it
// only checks the round's step bound.  When a round has finished (or before the probe) it
//   1. applies the round's verdicts to each issued prompt's posterior counts (n, s);
//   2. DECIDEs every active prompt with the exact table of Eq. (decide) built from the
//      closed-form predictor p_eff of Prop. 1 (integer prior, exact 128-bit rationals);
//   3. funds one more rollout for each continuing prompt while the budget N allows, the
//      highest p_eff first (ties: lower stream index), the rest become INCOMPLETE;
//   4. refills the working set toward B - |C| with fresh prompts (n0-rollout probes);
//   5. (decode) assigns prompt-KV slots and rollout slots, writes the prefill rows of the
//      fresh prompts and the first decode step's rows, and opens the round-start branch of
//      the graph; sets the loop condition to 0 once nothing more can be issued.
#pragma once
#include <cuda_runtime.h>

#include "device_common.cuh"
#include "step_state.cuh"

namespace sara {

constexpr int kCtlThreads = 1024;

// ---------------------------------------------------------------------------------------
// block-wide helpers (blockDim.x == kCtlThreads)
struct CtlShared {
    int warp_tot[32];
    long long warp_tot64[32];
    int bcast[8];
    int hist[2 * kMaxK + 2];
    unsigned pslot_used[256];  // bitmap of prompt slots (<= 8192)
};

__device__ __forceinline__ int blk_excl_scan(int v, int &total, CtlShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh.warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = sh.warp_tot[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        sh.warp_tot[lane] = w;  // inclusive
    }
    __syncthreads();
    const int before = (warp > 0 ? sh.warp_tot[warp - 1] : 0) + x - v;
    total = sh.warp_tot[31];
    __syncthreads();
    return before;
}

__device__ __forceinline__ long long blk_sum64(long long v, CtlShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) sh.warp_tot64[warp] = v;
    __syncthreads();
    long long t = 0;
    for (int w = 0; w < 32; ++w) t += sh.warp_tot64[w];
    __syncthreads();
    return t;
}

__device__ __forceinline__ int blk_max(int v, CtlShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    if (lane == 0) sh.warp_tot[warp] = v;
    __syncthreads();
    int t = sh.warp_tot[0];
    for (int w = 1; w < 32; ++w) t = max(t, sh.warp_tot[w]);
    __syncthreads();
    return t;
}

// Stable compaction of list[0..n) by flag(i) into dst; returns the kept count.
template <typename Flag>
__device__ __forceinline__ int blk_compact(const int32_t *list, int n, int32_t *dst, Flag flag, CtlShared &sh) {
    int out = 0;
    for (int base = 0; base < n; base += kCtlThreads) {
        const int i = base + threadIdx.x;
        const int keep = (i < n) ? (flag(i) ? 1 : 0) : 0;
        int tot;
        const int off = blk_excl_scan(keep, tot, sh);
        if (keep) dst[out + off] = list[i];
        out += tot;
    }
    __syncthreads();
    return out;
}

// ---------------------------------------------------------------------------------------
// exact predictor: prod_{i<a} (b+i) / (b+r+i) and p_eff = 1 - that for a saturated prefix
typedef unsigned __int128 u128;

__device__ __forceinline__ void saturated_ratio(int a, int b, int r, u128 &num, u128 &den) {
    num = 1;
    den = 1;
    for (int i = 0; i < a; ++i) {
        num *= (u128)(b + i);
        den *= (u128)(b + r + i);
    }
}
// p_eff(n, s) for n >= 1 as (num, den)
__device__ __forceinline__ void peff_frac(int n, int s, int k, int a0, int b0, u128 &pn, u128 &pd) {
    if (s >= 1 && n - s >= 1) { pn = 1; pd = 1; return; }
    u128 rn, rd;
    if (s == 0) saturated_ratio(a0, b0 + n, k - n, rn, rd);  // all-fail prefix
    else saturated_ratio(b0, a0 + n, k - n, rn, rd);         // all-pass prefix
    pn = rd - rn;
    pd = rd;
}

// dec_tab[n][s] (Eq. decide) and rank_tab[n][s] = number of keys (mixed, (m,0), (m,m)) with a
// strictly larger p_eff, so a smaller rank means a higher priority; 0 = mixed.  1 <= n <= k.
static __device__ void ctl_build_tables(const StepConst &K, const StepPtrs &c) {
    const int k = K.k;
    for (int e = threadIdx.x; e < kTabDim * kTabDim; e += kCtlThreads) {
        const int n = e / kTabDim, s = e % kTabDim;
        uint8_t d = D_CONTINUE, rk = 0;
        if (n >= 1 && n <= k && s <= n) {
            const bool mixed = s >= 1 && n - s >= 1;
            u128 pn, pd;
            peff_frac(n, s, k, K.a0, K.b0, pn, pd);
            if (mixed) d = (n >= K.commit_min) ? D_COMMIT : D_CONTINUE;
            else if (n >= k) d = D_ABANDON;
            else d = (pn * (u128)K.tau_den < (u128)K.tau_num * pd) ? D_ABANDON : D_CONTINUE;
            int cntg = 0;
            if (!mixed) {
                cntg = (pn == pd) ? 0 : 1;  // the mixed class (p_eff = 1)
                for (int mm = 1; mm <= k; ++mm) {
                    for (int side = 0; side < 2; ++side) {
                        u128 qn, qd;
                        peff_frac(mm, side ? mm : 0, k, K.a0, K.b0, qn, qd);
                        if (qn * pd > pn * qd) ++cntg;
                    }
                }
            }
            rk = (uint8_t)min(cntg, 2 * kMaxK + 1);
        }
        c.dec_tab[e] = d;
        c.rank_tab[e] = rk;
    }
}

// ------------------------------------------------------------------------------------------
// Warm-start (App. D): a prompt's prior Beta(a, b) is real, carried from earlier steps, so the
// predictor of Prop. 1 / Eq. (peff) is evaluated in fp64 through log-Gamma and Eq. (decide)
// compares it with tau_low in fp64 (decisions agree with exact arithmetic away from ties).
__device__ __forceinline__ double log_beta(double x, double y) { return lgamma(x) + lgamma(y) - lgamma(x + y); }
__device__ __forceinline__ double peff_real(int n, int s, int k, double a, double b) {
    if (s > 0 && s < n) return 1.0;
    const double ap = a + s, bp = b + (n - s);
    const int r = k - n;
    double out = 1.0;
    if (s == 0) out -= exp(log_beta(ap, bp + r) - log_beta(ap, bp));  // the rest all fail
    if (s == n) out -= exp(log_beta(ap + r, bp) - log_beta(ap, bp));  // the rest all succeed
    return out;
}
__device__ __forceinline__ int decide_real(int n, int s, const StepConst &K, double a, double b) {
    if (s > 0 && s < n && n >= K.commit_min) return D_COMMIT;
    if (n == K.k) return D_ABANDON;
    return peff_real(n, s, K.k, a, b) < K.tau_f ? D_ABANDON : D_CONTINUE;
}

__device__ __forceinline__ int verdict_of(uint64_t seed, int64_t q, int j, uint64_t thr) {
    return (splitmix_at(seed, (uint64_t)q * 64u + (uint64_t)j + 1u) >> 32) < thr ? 1 : 0;
}

__device__ __forceinline__ uint64_t sampler_row_seed(uint64_t sample_seed, int64_t uid, int t) {
    return splitmix_at(sample_seed, (uint64_t)uid * (1ull << 20) + (uint64_t)t + 1u);
}

// The step graph's conditions: h[0] loop, h[1] rollouts join (their KV set-up runs), h[2] fresh
// prompts are prefilled first (-1: whenever rollouts join).  use_handles: bit 0 = h[0] exists,
// bit 1 = h[1] and h[2] exist.
struct CondHandles {
    cudaGraphConditionalHandle h[3];
};
__device__ __forceinline__ void set_conds(const CondHandles &hs, int loop, int round_start, int use_handles,
                                          int prefill = -1) {
    if (threadIdx.x == 0) {
        if (use_handles & 1) cudaGraphSetConditional(hs.h[0], loop ? 1u : 0u);
        if (use_handles & 2) {
            cudaGraphSetConditional(hs.h[1], round_start ? 1u : 0u);
            cudaGraphSetConditional(hs.h[2], (prefill < 0 ? round_start : prefill) ? 1u : 0u);
        }
    }
}

// Decode rows of a round's first step and the prefill rows of its fresh prompts.
static __device__ void ctl_round_setup(const StepConst &K, StepVars &V, const StepPtrs &c, CtlShared &sh,
                                       int n_funded, int n_fresh, int first_fresh_q) {
    const int k = K.k, Lp = K.Lp;
    // prompt slots: continuing prompts keep theirs, fresh prompts take free ones in order
    for (int w = threadIdx.x; w < 256; w += kCtlThreads) sh.pslot_used[w] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < n_funded; i += kCtlThreads) {
        const int ps = c.q_pslot[c.act[i]];
        atomicOr(&sh.pslot_used[ps >> 5], 1u << (ps & 31));
    }
    __syncthreads();
    int assigned = 0;
    for (int base = 0; base < c.max_active && assigned < n_fresh; base += kCtlThreads) {
        const int ps = base + threadIdx.x;
        const int freeb = (ps < c.max_active) && !((sh.pslot_used[ps >> 5] >> (ps & 31)) & 1u);
        int tot;
        const int off = blk_excl_scan(freeb, tot, sh);
        if (freeb && assigned + off < n_fresh) c.fresh_pslot[assigned + off] = ps;
        assigned += tot;
    }
    __syncthreads();
    if (assigned < n_fresh) { if (threadIdx.x == 0) report_error(&V.err, ERR_CAPACITY); return; }
    for (int f = threadIdx.x; f < n_fresh; f += kCtlThreads) c.q_pslot[first_fresh_q + f] = c.fresh_pslot[f];
    __syncthreads();

    // rollout slots in issue order
    const int n_iss = V.n_iss;
    int R = 0;
    for (int base = 0; base < n_iss; base += kCtlThreads) {
        const int e = base + threadIdx.x;
        const int cnt = (e < n_iss) ? c.iss_c[e] : 0;
        int tot;
        const int off = blk_excl_scan(cnt, tot, sh);
        if (e < n_iss) {
            const int q = c.iss_q[e];
            const int n_before = c.q_n[q];
            for (int t = 0; t < cnt; ++t) {
                const int slot = R + off + t;
                if (slot >= c.max_seqs) continue;
                const int j = n_before + t;
                int L = c.p_len[(int64_t)q * k + j];
                if (L < 1 || L > K.max_gen) {  // lengths bound the KV cache and the token output
                    report_error(&V.err, ERR_BOUNDS);
                    L = L < 1 ? 1 : K.max_gen;
                }
                c.seq_q[slot] = q;
                c.seq_j[slot] = j;
                c.seq_len[slot] = L;
                c.seq_gen[slot] = 0;
                c.seq_pslot[slot] = c.q_pslot[q];
                c.seq_uid[slot] = (int64_t)q * 64 + j;
            }
        }
        R += tot;
    }
    __syncthreads();
    if (R > c.max_seqs) { if (threadIdx.x == 0) report_error(&V.err, ERR_CAPACITY); return; }
    // first decode step: input = last prompt token at position Lp - 1
    const int nblk = (Lp + K.attn_chunk - 1) / K.attn_chunk;
    const int span = att_span_for((int64_t)R * nblk, K.att_slots, R);
    const int nsplit = (nblk + span - 1) / span;
    int maxL = 0;
    for (int r = threadIdx.x; r < R; r += kCtlThreads) {
        const int q = c.seq_q[r];
        c.row_slot[r] = r;
        c.row_pos[r] = Lp - 1;
        c.row_tok[r] = c.p_tok[(int64_t)q * Lp + Lp - 1];
        c.row_seed[r] = sampler_row_seed(K.sample_seed, c.seq_uid[r], 0);
        c.row_item0[r] = r * nsplit;
        for (int sp = 0; sp < nsplit; ++sp) c.att_items[r * nsplit + sp] = make_int2(r, sp);
        maxL = max(maxL, c.seq_len[r]);
    }
    maxL = blk_max(maxL, sh);
    // KV blocks of the round's rollouts (the previous round's were all freed as its rollouts
    // finished): the prompt's full blocks, shared, then one private block from the free stack
    // for the block holding position Lp - 1 (the prompt's tail is copied into it), in slot order
    {
        const int nsh = shared_blocks(Lp, K.attn_chunk);
        const int top = V.blk_top;
        __syncthreads();
        if (R > top) { if (threadIdx.x == 0) report_error(&V.err, ERR_CAPACITY); return; }
        for (int r = threadIdx.x; r < R; r += kCtlThreads) {
            int32_t *bt = c.blk_tab + (int64_t)r * c.nblk_max;
            const int ps = c.seq_pslot[r];
            for (int j = 0; j < nsh; ++j) bt[j] = ps * c.nsh_max + j;
            bt[nsh] = c.blk_free[top - 1 - r];
            c.new_slots[r] = r;
        }
        if (threadIdx.x == 0) {
            V.blk_top = top - R;
            V.blk_low = min(V.blk_low, top - R);
            V.n_new = R;
        }
    }
    // prefill rows: fresh prompt f, token t < Lp - 1, written into prompt slot fresh_pslot[f]
    const int Lpre = Lp - 1;
    const int pre_rows = n_fresh * Lpre;
    if (pre_rows > c.pre_cap) { if (threadIdx.x == 0) report_error(&V.err, ERR_CAPACITY); return; }
    for (int r = threadIdx.x; r < pre_rows; r += kCtlThreads) {
        const int f = r / Lpre, t = r - f * Lpre;
        const int q = first_fresh_q + f;
        c.pre_slot[r] = c.fresh_pslot[f];
        c.pre_pos[r] = t;
        c.pre_tok[r] = c.p_tok[(int64_t)q * Lp + t];
        c.pre_items[r] = make_int2(r, 0);
        c.pre_item0[r] = r;
    }
    if (threadIdx.x == 0) {
        V.live = R;
        V.att_items = R * nsplit;
        V.att_span = span;
        V.pre_rows = pre_rows;
        V.n_fresh = n_fresh;
        V.round_maxL = maxL;
        V.round_steps = 0;
    }
}

// One round end + allocation (everything but the decode).
static __device__ void ctl_round(const StepConst &K, StepVars &V, const StepPtrs &c, CtlShared &sh) {
    const int k = K.k;
    const int tid = threadIdx.x;
    // ---- 1. apply the finished round's verdicts
    if (V.round >= 0) {
        const int n_iss = V.n_iss;
        long long tok = 0;
        int lmax = 0;
        for (int e = tid; e < n_iss; e += kCtlThreads) {
            const int q = c.iss_q[e], cnt = c.iss_c[e];
            const int n = c.q_n[q];
            int s = c.q_s[q];
            for (int t = 0; t < cnt; ++t) {
                const int j = n + t;
                s += verdict_of(K.reward_seed, q, j, c.p_thr[q]);
                const int L = c.p_len[(int64_t)q * k + j];
                tok += L;
                lmax = max(lmax, L);
            }
            c.q_n[q] = (uint8_t)(n + cnt);
            c.q_s[q] = (uint8_t)s;
        }
        tok = blk_sum64(tok, sh);
        lmax = blk_max(lmax, sh);
        if (tid == 0) {
            V.gen_tokens += tok;
            V.sched_steps += lmax;
            V.rounds_done += 1;
        }
        __syncthreads();
        // ---- 2. DECIDE (Eq. decide) for every active prompt
        const int n_act = V.n_act;
        long long commits = 0;
        for (int i = tid; i < n_act; i += kCtlThreads) {
            const int q = c.act[i];
            const int d = K.warm ? decide_real(c.q_n[q], c.q_s[q], K, c.q_pa[q], c.q_pb[q])
                                 : c.dec_tab[c.q_n[q] * kTabDim + c.q_s[q]];
            if (d == D_COMMIT) { c.q_status[q] = ST_COMMITTED; c.q_round[q] = (int16_t)V.round; ++commits; }
            else if (d == D_ABANDON) { c.q_status[q] = ST_ABANDONED; c.q_round[q] = (int16_t)V.round; }
        }
        commits = blk_sum64(commits, sh);
        __syncthreads();
        const int n_cont = blk_compact(c.act, n_act, c.act_tmp,
                                       [&](int i) { return c.q_status[c.act[i]] == ST_ACTIVE; }, sh);
        for (int i = tid; i < n_cont; i += kCtlThreads) c.act[i] = c.act_tmp[i];
        __syncthreads();
        if (tid == 0) { V.C += commits; V.n_act = n_cont; }
        __syncthreads();
    }
    const int B = K.B;
    const int n_cont = V.n_act;
    // ---- stop once B effective groups are committed
    if (V.C >= B) {
        for (int i = tid; i < n_cont; i += kCtlThreads) c.q_status[c.act[i]] = ST_INCOMPLETE;
        __syncthreads();
        if (tid == 0) { V.n_act = 0; V.n_iss = 0; V.done = 1; }
        __syncthreads();
        return;
    }
    // ---- 3. fund continuing prompts by p_eff priority while the budget allows
    const long long budget = K.N - V.used;
    int n_funded = n_cont;
    if ((long long)n_cont > budget && K.warm) {
        // warm-start priors: p_eff is real, so each continuing prompt counts the prompts ahead
        // of it (higher p_eff, or equal p_eff and lower stream index) over tiles of the keys
        const int take = (int)max(0ll, budget);
        for (int i = tid; i < n_cont; i += kCtlThreads) {
            const int q = c.act[i];
            c.q_key[i] = peff_real(c.q_n[q], c.q_s[q], k, c.q_pa[q], c.q_pb[q]);
        }
        __syncthreads();
        __shared__ double tkey[kCtlThreads];
        __shared__ int tq[kCtlThreads];
        for (int base = 0; base < n_cont; base += kCtlThreads) {
            const int i = base + tid;
            const double ki = i < n_cont ? c.q_key[i] : 0.0;
            const int qi = i < n_cont ? c.act[i] : 0;
            int ahead = 0;
            for (int t0 = 0; t0 < n_cont; t0 += kCtlThreads) {
                __syncthreads();
                if (t0 + tid < n_cont) {
                    tkey[tid] = c.q_key[t0 + tid];
                    tq[tid] = c.act[t0 + tid];
                }
                __syncthreads();
                const int m = min(kCtlThreads, n_cont - t0);
                for (int j = 0; j < m; ++j) ahead += (tkey[j] > ki) || (tkey[j] == ki && tq[j] < qi);
            }
            if (i < n_cont && ahead >= take) c.q_status[qi] = ST_INCOMPLETE;
        }
        __syncthreads();
        n_funded = blk_compact(c.act, n_cont, c.act_tmp,
                               [&](int i) { return c.q_status[c.act[i]] == ST_ACTIVE; }, sh);
        for (int i = tid; i < n_funded; i += kCtlThreads) c.act[i] = c.act_tmp[i];
        __syncthreads();
    } else if ((long long)n_cont > budget) {
        const int take = (int)max(0ll, budget);
        for (int b = tid; b < 2 * kMaxK + 2; b += kCtlThreads) sh.hist[b] = 0;
        __syncthreads();
        for (int i = tid; i < n_cont; i += kCtlThreads) {
            const int q = c.act[i];
            atomicAdd(&sh.hist[c.rank_tab[c.q_n[q] * kTabDim + c.q_s[q]]], 1);
        }
        __syncthreads();
        if (tid == 0) {
            int acc = 0, rstar = 0;
            while (rstar < 2 * kMaxK + 2 && acc + sh.hist[rstar] < take) acc += sh.hist[rstar++];
            sh.bcast[0] = rstar;
            sh.bcast[1] = take - acc;  // how many of rank rstar, in stream order
        }
        __syncthreads();
        const int rstar = sh.bcast[0], need = sh.bcast[1];
        int seen = 0;
        for (int base = 0; base < n_cont; base += kCtlThreads) {
            const int i = base + tid;
            int rk = 1 << 30, q = -1;
            if (i < n_cont) { q = c.act[i]; rk = c.rank_tab[c.q_n[q] * kTabDim + c.q_s[q]]; }
            const int at = (rk == rstar) ? 1 : 0;
            int tot;
            const int off = blk_excl_scan(at, tot, sh);
            if (i < n_cont) {
                const bool fund = rk < rstar || (at && seen + off < need);
                if (!fund) c.q_status[q] = ST_INCOMPLETE;
            }
            seen += tot;
        }
        __syncthreads();
        n_funded = blk_compact(c.act, n_cont, c.act_tmp,
                               [&](int i) { return c.q_status[c.act[i]] == ST_ACTIVE; }, sh);
        for (int i = tid; i < n_funded; i += kCtlThreads) c.act[i] = c.act_tmp[i];
        __syncthreads();
    }
    // ---- 4. refill toward B - |C| with fresh n0-probes
    const long long used_after = V.used + n_funded;
    const long long room = (long long)(B - V.C) - n_funded;
    const long long by_budget = (K.N - used_after) / K.n0;
    const long long by_pool = (long long)K.P - V.cursor;
    const int n_fresh = (int)max(0ll, min(min(room, by_budget), by_pool));
    const int first_fresh = (int)V.cursor;
    if (n_funded + n_fresh > c.max_active) {  // cannot happen when B <= max_active
        if (tid == 0) { report_error(&V.err, ERR_CAPACITY); V.done = 1; }
        __syncthreads();
        return;
    }
    for (int f = tid; f < n_fresh; f += kCtlThreads) {
        const int q = first_fresh + f;
        c.q_status[q] = ST_ACTIVE;
        c.act[n_funded + f] = q;
    }
    const int n_iss = n_funded + n_fresh;
    __syncthreads();
    for (int i = tid; i < n_iss; i += kCtlThreads) {
        c.iss_q[i] = c.act[i];
        c.iss_c[i] = (i < n_funded) ? 1 : K.n0;
    }
    __syncthreads();
    if (tid == 0) {
        V.used = used_after + (long long)n_fresh * K.n0;
        V.drawn += n_fresh;
        V.cursor += n_fresh;
        V.n_act = n_iss;
        V.n_iss = n_iss;
        V.round += 1;
        if (n_iss == 0) V.done = 1;
    }
    __syncthreads();
    if (K.decode && n_iss > 0) ctl_round_setup(K, V, c, sh, n_funded, n_fresh, first_fresh);
    __syncthreads();
}

// ------------------------------------------------------------------------------------------
// Asynchronous per-prompt schedule on the decode engine (Discussion, Limitations (ii): no round
// barrier).  At every decode-step boundary the prompts whose batch in flight finished in the
// step just run (dec_list, from the bookkeeping kernel) are decided as one event: verdicts of
// the batch, DECIDE (Eq. decide) in stream order; after |C| >= B nothing is issued and
// continuing prompts end INCOMPLETE (rollouts in flight still finish and are decided);
// otherwise continuing prompts are funded one rollout each by p_eff rank (ties: stream index)
// while the budget allows, then fresh prompts are drawn in stream order while fewer than
// B - |C| prompts are in flight and a whole n0-probe fits the budget (reserve: also every prompt
// in flight running to k).  New rollouts decode from the next step on; fresh prompts are
// prefilled in between.  The event logic is serial (thread 0): an event holds few prompts.
static __device__ void ctl_async_events(const StepConst &K, StepVars &V, const StepPtrs &c) {
    const int k = K.k, n0 = K.n0, B = K.B, P = K.P;
    const int reserve = K.schedule == 2;
    int ni = 0;
    int64_t used = V.used, resv = V.resv, tokens = V.gen_tokens, C = V.C, cursor = V.cursor, drawn = V.drawn;
    int inflight = V.in_flight, ptop = V.pslot_top;
    bool bad = false, cap = false;
    auto issue = [&](int q, int cnt) {
        const int n = c.q_n[q];
        for (int j = n; j < n + cnt; ++j) {
            const int L = c.p_len[(int64_t)q * k + j];
            if (L < 1 || L > K.max_gen) bad = true;
            tokens += L;
        }
        used += cnt;
        if (reserve) resv += k - (n + cnt);
        c.q_inflight[q] = cnt;
        c.iss_q[ni] = q;
        c.iss_c[ni] = cnt;
        ++ni;
        ++inflight;
    };
    auto free_pslot = [&](int q) { c.pslot_free[ptop++] = c.q_pslot[q]; };
    auto draw = [&]() {
        while (cursor < P && inflight < B - C && used + (reserve ? k : n0) + resv <= K.N) {
            if (ptop <= 0 || ni >= c.max_active) { cap = true; break; }
            const int q = (int)cursor++;
            c.q_status[q] = ST_ACTIVE;
            c.q_pslot[q] = c.pslot_free[--ptop];
            ++drawn;
            issue(q, n0);
        }
    };
    auto key_before = [&](int p2, int q) {  // p2 funded before q: higher p_eff, then lower index
        if (K.warm) {
            const double a = peff_real(c.q_n[p2], c.q_s[p2], k, c.q_pa[p2], c.q_pb[p2]);
            const double b = peff_real(c.q_n[q], c.q_s[q], k, c.q_pa[q], c.q_pb[q]);
            return a > b || (a == b && p2 < q);
        }
        const int rp = c.rank_tab[c.q_n[p2] * kTabDim + c.q_s[p2]], rq = c.rank_tab[c.q_n[q] * kTabDim + c.q_s[q]];
        return rp < rq || (rp == rq && p2 < q);
    };
    if (V.round < 0) {  // the first probes
        V.round = 0;
        draw();
    } else if (V.n_dec > 0) {
        const int nd = V.n_dec;
        for (int i = 1; i < nd; ++i) {  // stream order
            const int q = c.dec_list[i];
            int j = i - 1;
            while (j >= 0 && c.dec_list[j] > q) { c.dec_list[j + 1] = c.dec_list[j]; --j; }
            c.dec_list[j + 1] = q;
        }
        const int ev = V.events++;
        int ncont = 0;
        for (int i = 0; i < nd; ++i) {
            const int q = c.dec_list[i];
            --inflight;
            int n = c.q_n[q], sc = c.q_s[q];
            const int cnt = n == 0 ? n0 : 1;
            for (int j = n; j < n + cnt; ++j) sc += verdict_of(K.reward_seed, q, j, c.p_thr[q]);
            n += cnt;
            c.q_n[q] = (uint8_t)n;
            c.q_s[q] = (uint8_t)sc;
            if (reserve) resv -= k - n;
            const int d = K.warm ? decide_real(n, sc, K, c.q_pa[q], c.q_pb[q]) : c.dec_tab[n * kTabDim + sc];
            if (d == D_COMMIT) {
                c.q_status[q] = ST_COMMITTED;
                c.q_round[q] = (int16_t)min(ev, 32767);
                ++C;
                free_pslot(q);
            } else if (d == D_ABANDON) {
                c.q_status[q] = ST_ABANDONED;
                c.q_round[q] = (int16_t)min(ev, 32767);
                free_pslot(q);
            } else {
                c.act[ncont++] = q;
            }
        }
        if (V.stopped || C >= B) {
            V.stopped = 1;
            for (int i = 0; i < ncont; ++i) {
                c.q_status[c.act[i]] = ST_INCOMPLETE;
                free_pslot(c.act[i]);
            }
        } else {
            for (int i = 1; i < ncont; ++i) {  // priority order (insertion sort: few per event)
                const int q = c.act[i];
                int j = i - 1;
                while (j >= 0 && !key_before(c.act[j], q)) { c.act[j + 1] = c.act[j]; --j; }
                c.act[j + 1] = q;
            }
            for (int i = 0; i < ncont; ++i) {
                const int q = c.act[i];
                if (used + 1 <= K.N) {
                    issue(q, 1);
                } else {
                    c.q_status[q] = ST_INCOMPLETE;
                    free_pslot(q);
                }
            }
            draw();
        }
    }
    if (bad) report_error(&V.err, ERR_BOUNDS);
    if (cap) report_error(&V.err, ERR_CAPACITY);
    V.n_dec = 0;
    V.n_iss = ni;
    V.used = used;
    V.resv = resv;
    V.gen_tokens = tokens;
    V.C = C;
    V.cursor = cursor;
    V.drawn = drawn;
    V.in_flight = inflight;
    V.pslot_top = ptop;
}

// The rollouts issued at this boundary join the live rows (all threads): rollout slots and a
// private KV block from the free stacks, rows appended after the live ones, prefill rows of the
// fresh prompts, then the attention items of every live row.
static __device__ void ctl_async_join(const StepConst &K, StepVars &V, const StepPtrs &c, CtlShared &sh) {
    const int tid = threadIdx.x;
    const int Lp = K.Lp, Lpre = Lp - 1, nsh = shared_blocks(Lp, K.attn_chunk);
    const int n_iss = V.n_iss, live0 = V.live, stop = V.slot_top, btop = V.blk_top;
    int R = 0, nf = 0;
    for (int base = 0; base < n_iss; base += kCtlThreads) {
        const int e = base + tid;
        const int cnt = e < n_iss ? c.iss_c[e] : 0;
        const int q = e < n_iss ? c.iss_q[e] : 0;
        const int fresh = (e < n_iss && c.q_n[q] == 0) ? 1 : 0;
        int tot, ftot;
        const int off = blk_excl_scan(cnt, tot, sh);
        const int foff = blk_excl_scan(fresh, ftot, sh);
        if (e < n_iss) {
            const int ps = c.q_pslot[q];
            for (int t = 0; t < cnt; ++t) {
                const int r = R + off + t;  // new rollout index
                if (r >= stop || r >= btop || live0 + r >= c.max_seqs) continue;  // capacity: reported below
                const int slot = c.slot_free[stop - 1 - r];
                const int j = c.q_n[q] + t;
                c.seq_q[slot] = q;
                c.seq_j[slot] = j;
                c.seq_len[slot] = c.p_len[(int64_t)q * K.k + j];
                c.seq_gen[slot] = 0;
                c.seq_pslot[slot] = ps;
                c.seq_uid[slot] = (int64_t)q * 64 + j;
                int32_t *bt = c.blk_tab + (int64_t)slot * c.nblk_max;
                for (int b = 0; b < nsh; ++b) bt[b] = ps * c.nsh_max + b;
                bt[nsh] = c.blk_free[btop - 1 - r];
                c.new_slots[r] = slot;
                const int row = live0 + r;
                c.row_slot[row] = slot;
                c.row_pos[row] = Lp - 1;
                c.row_tok[row] = c.p_tok[(int64_t)q * Lp + Lp - 1];
                c.row_seed[row] = sampler_row_seed(K.sample_seed, c.seq_uid[slot], 0);
            }
            if (fresh) {
                c.fresh_pslot[nf + foff] = ps;
                c.act_tmp[nf + foff] = q;
            }
        }
        R += tot;
        nf += ftot;
    }
    __syncthreads();
    if (R > stop || R > btop || live0 + R > c.max_seqs) {
        if (tid == 0) report_error(&V.err, ERR_CAPACITY);
        return;
    }
    // prefill rows of the fresh prompts (in the issue order of fresh_pslot)
    const int pre_rows = nf * Lpre;
    if (pre_rows > c.pre_cap) { if (tid == 0) report_error(&V.err, ERR_CAPACITY); return; }
    for (int r = tid; r < pre_rows; r += kCtlThreads) {  // fresh prompt f = act_tmp[f], token t
        const int f = r / Lpre, t = r - f * Lpre;
        c.pre_slot[r] = c.fresh_pslot[f];
        c.pre_pos[r] = t;
        c.pre_tok[r] = c.p_tok[(int64_t)c.act_tmp[f] * Lp + t];
        c.pre_items[r] = make_int2(r, 0);
        c.pre_item0[r] = r;
    }
    __syncthreads();
    const int live = live0 + R;
    // attention items of every live row: splits of `span` KV blocks
    int blocks = 0;
    for (int base = 0; base < live; base += kCtlThreads) {
        const int i = base + tid;
        int tot;
        blk_excl_scan(i < live ? (c.row_pos[i] + K.attn_chunk) / K.attn_chunk : 0, tot, sh);
        blocks += tot;
    }
    const int span = att_span_for(blocks, K.att_slots, live);
    int items = 0;
    for (int base = 0; base < live; base += kCtlThreads) {
        const int i = base + tid;
        const int ns = (i < live) ? ((c.row_pos[i] + K.attn_chunk) / K.attn_chunk + span - 1) / span : 0;
        int tot;
        const int before = blk_excl_scan(ns, tot, sh);
        if (i < live) {
            const int i0 = items + before;
            c.row_item0[i] = i0;
            for (int sp = 0; sp < ns; ++sp) {
                if (i0 + sp < c.att_cap) c.att_items[i0 + sp] = make_int2(i, sp);
                else report_error(&V.err, ERR_CAPACITY);
            }
        }
        items += tot;
    }
    __syncthreads();
    if (tid == 0) {
        V.slot_top = stop - R;
        V.blk_top = btop - R;
        V.blk_low = min(V.blk_low, btop - R);
        V.n_new = R;
        V.live = live;
        V.att_items = min(items, c.att_cap);
        V.att_span = span;
        V.pre_rows = pre_rows;
        V.n_fresh = nf;
    }
}

static __device__ void ctl_async_step(const StepConst &K, StepVars &V, const StepPtrs &c, CtlShared &sh,
                                      const CondHandles &hs, int use_handles) {
    if (threadIdx.x == 0) ctl_async_events(K, V, c);
    __syncthreads();
    if (V.err == 0) ctl_async_join(K, V, c, sh);
    __syncthreads();
    const int done = V.err != 0 || V.live == 0;
    if (done && threadIdx.x == 0) {  // nothing in flight and nothing issued: the step is over
        V.done = 1;
        V.live = 0;
        V.rounds_done = V.events;
        V.sched_steps = V.exec_steps;
    }
    __syncthreads();
    set_conds(hs, !done, !done && V.n_new > 0, use_handles, !done && V.n_fresh > 0);
}

// Per-iteration controller kernel of the step graph.
static __global__ void __launch_bounds__(kCtlThreads, 1)
ctl_kernel(StepPtrs c, CondHandles hs, int use_handles) {
    __shared__ CtlShared sh;
    pdl_wait_prior_grids();
    const StepConst K = *c.kc;
    StepVars &V = *c.v;
    __syncthreads();
    if (threadIdx.x == 0) {
        V.iters += 1;
        // the caller's bound on the loop (sara_set_limits)
        if (K.max_iters > 0 && V.iters > K.max_iters && !V.done) report_error(&V.err, ERR_ITER_BOUND);
    }
    __syncthreads();
    if (V.err != 0 && !V.done) {  // a kernel reported an error: end the step now
        __syncthreads();
        if (threadIdx.x == 0) { V.done = 1; V.live = 0; }
        set_conds(hs, 0, 0, use_handles);
        return;
    }
    if (V.done) { set_conds(hs, 0, 0, use_handles); return; }
    if (K.schedule != 0 && K.decode) {  // asynchronous: an event boundary after every decode step
        if (V.exec_steps > (int64_t)K.N * K.max_gen + 1) {  // bound: every rollout at full length in turn
            if (threadIdx.x == 0) { report_error(&V.err, ERR_ITER_BOUND); V.done = 1; V.live = 0; }
            set_conds(hs, 0, 0, use_handles);
            return;
        }
        ctl_async_step(K, V, c, sh, hs, use_handles);
        return;
    }
    if (V.live > 0) {
        // mid-round: the round may run at most round_maxL decode steps
        const int stop = V.round_steps > V.round_maxL;
        if (stop && threadIdx.x == 0) { report_error(&V.err, ERR_ITER_BOUND); V.done = 1; }
        set_conds(hs, !stop, 0, use_handles);
        return;
    }
    if (K.teacher) {  // teacher forcing runs one prepared round
        if (threadIdx.x == 0) V.done = 1;
        set_conds(hs, 0, 0, use_handles);
        return;
    }
    // a round boundary: bound the number of rounds (each issues >= 1 rollout)
    if (V.rounds_done > K.N + 1) {
        if (threadIdx.x == 0) { report_error(&V.err, ERR_ITER_BOUND); V.done = 1; }
        set_conds(hs, 0, 0, use_handles);
        return;
    }
    ctl_round(K, V, c, sh);
    __syncthreads();
    if (V.err & (ERR_CAPACITY | ERR_BOUNDS)) { if (threadIdx.x == 0) V.done = 1; }
    __syncthreads();
    const int done = V.done;
    if (done) {
        // remaining active prompts end INCOMPLETE
        const int n_act = V.n_act;
        for (int i = threadIdx.x; i < n_act; i += kCtlThreads)
            if (c.q_status[c.act[i]] == ST_ACTIVE) c.q_status[c.act[i]] = ST_INCOMPLETE;
        if (threadIdx.x == 0) { V.live = 0; V.n_act = 0; }
    }
    set_conds(hs, !done, !done && K.decode, use_handles, !done && K.decode && V.n_fresh > 0);
}

// The next step's priors (warm-start carry, App. D): decayed evidence on top of the base
// prior, a' = alpha0 + lambda (a - alpha0 + s), b' = beta0 + lambda (b - beta0 + n - s), with
// (a, b) the prior this step used (the base prior unless warm).
static __global__ void carry_prior_kernel(const StepPtrs c, double lambda, double *a_next, double *b_next) {
    const StepConst &K = *c.kc;
    for (int q = blockIdx.x * blockDim.x + threadIdx.x; q < K.P; q += gridDim.x * blockDim.x) {
        const double a0 = K.a0, b0 = K.b0;
        const double a = K.warm ? c.q_pa[q] : a0, b = K.warm ? c.q_pb[q] : b0;
        const int n = c.q_n[q], s = c.q_s[q];
        // rounded operation by operation (no contraction), as the formula reads
        a_next[q] = __dadd_rn(a0, __dmul_rn(lambda, __dadd_rn(__dsub_rn(a, a0), (double)s)));
        b_next[q] = __dadd_rn(b0, __dmul_rn(lambda, __dadd_rn(__dsub_rn(b, b0), (double)(n - s))));
    }
}

// Reset the step state and build the decision tables (one CTA).
static __global__ void __launch_bounds__(kCtlThreads, 1) ctl_init_kernel(StepPtrs c) {
    pdl_wait_prior_grids();
    const StepConst K = *c.kc;
    StepVars &V = *c.v;
    for (int q = threadIdx.x; q < K.P; q += kCtlThreads) {
        c.q_status[q] = ST_UNDRAWN;
        c.q_n[q] = 0;
        c.q_s[q] = 0;
        c.q_round[q] = -1;
        c.q_pslot[q] = -1;
    }
    ctl_build_tables(K, c);
    // every private KV block free (popped from the top: ids n_shared, n_shared + 1, .. first)
    for (int i = threadIdx.x; i < c.n_priv; i += kCtlThreads) c.blk_free[i] = c.n_shared + c.n_priv - 1 - i;
    if (K.decode) {  // the asynchronous schedule's free rollout and prompt slots, batches in flight
        for (int i = threadIdx.x; i < c.max_seqs; i += kCtlThreads) c.slot_free[i] = c.max_seqs - 1 - i;
        for (int i = threadIdx.x; i < c.max_active; i += kCtlThreads) c.pslot_free[i] = c.max_active - 1 - i;
        for (int q = threadIdx.x; q < K.P; q += kCtlThreads) c.q_inflight[q] = 0;
    }
    if (threadIdx.x == 0) {
        StepVars z;
        memset(&z, 0, sizeof(z));
        z.round = -1;
        z.kt0 = ~0ull;
        z.blk_top = z.blk_low = c.n_priv;
        z.slot_top = c.max_seqs;
        z.pslot_top = c.max_active;
        V = z;
    }
}

}  // namespace sara

namespace sara {

// ------------------------------------------------------------------------------------------
// Asynchronous per-prompt schedule (controller-only handles: decode-step time comes from the
// length table, nothing is decoded).  Algorithm 1 without the round barrier: a prompt is
// decided at the end of the decode step in which its batch in flight (the n0-rollout probe, or
// the one rollout of a continue decision) finishes; a rollout of length L started at step t0
// occupies steps t0 .. t0 + L - 1.  The prompts decided at one step boundary follow the round
// rules as one round: DECIDE (Eq. decide) in stream order, stop issuing once |C| >= B,
// otherwise fund the continuing ones by p_eff rank (ties: stream order) while the budget
// allows (else INCOMPLETE), then draw fresh prompts in stream order while fewer than B - |C|
// are in flight and a whole probe fits the budget; new rollouts start at the next step.  No
// cancellation: after the stop, rollouts in flight finish and their prompts are decided.
// reserve: a fresh prompt is drawn only if the budget covers it and every prompt in flight
// running to k rollouts.  decided_round receives the index of the deciding event (step
// boundary with decisions), capped at 32767.  One thread runs the event loop over a binary
// min-heap of (decision step << 32 | prompt) in dynamic shared memory (prompts in flight
// <= B <= max_active entries).
constexpr int kAsyncMaxInFlight = 8192;

static __global__ void __launch_bounds__(kCtlThreads, 1) ctl_async_kernel(StepPtrs c, int reserve, int heap_cap) {
    extern __shared__ uint64_t heap[];
    pdl_wait_prior_grids();
    if (threadIdx.x != 0) return;
    const StepConst K = *c.kc;
    StepVars &V = *c.v;
    const int k = K.k, n0 = K.n0, B = K.B, P = K.P;
    const int64_t N = K.N;
    int hn = 0;
    int64_t used = 0, tokens = 0, resv = 0, last = -1;
    int C = 0, cursor = 0, drawn = 0, events = 0;
    bool stopped = false, bad = false;

    auto push = [&](uint64_t key) {
        int i = hn++;
        while (i > 0) {
            const int par = (i - 1) >> 1;
            if (heap[par] <= key) break;
            heap[i] = heap[par];
            i = par;
        }
        heap[i] = key;
    };
    auto pop = [&]() -> uint64_t {
        const uint64_t top = heap[0];
        const uint64_t x = heap[--hn];
        int i = 0;
        for (;;) {
            int ch = 2 * i + 1;
            if (ch >= hn) break;
            if (ch + 1 < hn && heap[ch + 1] < heap[ch]) ++ch;
            if (heap[ch] >= x) break;
            heap[i] = heap[ch];
            i = ch;
        }
        if (hn > 0) heap[i] = x;
        return top;
    };
    // issue the next `cnt` rollouts of prompt q, starting at decode step `start`
    auto issue = [&](int q, int cnt, int64_t start) {
        const int n = c.q_n[q];
        int64_t mx = 0;
        for (int j = n; j < n + cnt; ++j) {
            const int L = c.p_len[(int64_t)q * k + j];
            if (L < 1 || L > K.max_gen) bad = true;
            tokens += L;
            mx = max(mx, (int64_t)L);
        }
        used += cnt;
        if (reserve) resv += k - (n + cnt);
        const int64_t fin = start + mx - 1;  // the batch's decision step
        if (hn < heap_cap && fin <= 0xffffffffLL) push(((uint64_t)fin << 32) | (uint32_t)q);
        else bad = true;
    };
    auto draw = [&](int64_t start) {
        while (!bad && cursor < P && hn < B - C && used + (reserve ? k : n0) + resv <= N) {
            const int q = cursor++;
            c.q_status[q] = ST_ACTIVE;
            ++drawn;
            issue(q, n0, start);
        }
    };

    draw(0);
    while (hn > 0 && !bad) {
        const int64_t t = (int64_t)(heap[0] >> 32);
        int ncont = 0;
        const int ev = events++;
        last = t;
        while (hn > 0 && (int64_t)(heap[0] >> 32) == t) {  // ascending stream index within a step
            const int q = (int)(pop() & 0xffffffffu);
            int n = c.q_n[q], s = c.q_s[q];
            const int cnt = n == 0 ? n0 : 1;
            for (int j = n; j < n + cnt; ++j) s += verdict_of(K.reward_seed, q, j, c.p_thr[q]);
            n += cnt;
            c.q_n[q] = (uint8_t)n;
            c.q_s[q] = (uint8_t)s;
            if (reserve) resv -= k - n;
            const int d = K.warm ? decide_real(n, s, K, c.q_pa[q], c.q_pb[q]) : c.dec_tab[n * kTabDim + s];
            if (d == D_COMMIT) {
                c.q_status[q] = ST_COMMITTED;
                c.q_round[q] = (int16_t)min(ev, 32767);
                ++C;
            } else if (d == D_ABANDON) {
                c.q_status[q] = ST_ABANDONED;
                c.q_round[q] = (int16_t)min(ev, 32767);
            } else {
                c.act[ncont++] = q;
            }
        }
        if (stopped || C >= B) {
            stopped = true;
            for (int i = 0; i < ncont; ++i) c.q_status[c.act[i]] = ST_INCOMPLETE;
            continue;
        }
        // continuing prompts by p_eff (the exact rank; with warm-start priors the fp64 value),
        // then stream index (insertion sort: few per event)
        for (int i = 1; i < ncont; ++i) {
            const int q = c.act[i];
            const int rq = K.warm ? 0 : c.rank_tab[c.q_n[q] * kTabDim + c.q_s[q]];
            const double pq = K.warm ? peff_real(c.q_n[q], c.q_s[q], k, c.q_pa[q], c.q_pb[q]) : 0.0;
            int j = i - 1;
            while (j >= 0) {
                const int p2 = c.act[j];
                bool before;
                if (K.warm) {
                    const double pp = peff_real(c.q_n[p2], c.q_s[p2], k, c.q_pa[p2], c.q_pb[p2]);
                    before = pp > pq || (pp == pq && p2 < q);
                } else {
                    const int rp = c.rank_tab[c.q_n[p2] * kTabDim + c.q_s[p2]];
                    before = rp < rq || (rp == rq && p2 < q);
                }
                if (before) break;
                c.act[j + 1] = p2;
                --j;
            }
            c.act[j + 1] = q;
        }
        for (int i = 0; i < ncont; ++i) {
            const int q = c.act[i];
            if (used + 1 <= N) issue(q, 1, t + 1);
            else c.q_status[q] = ST_INCOMPLETE;
        }
        draw(t + 1);
    }
    if (bad) report_error(&V.err, ERR_BOUNDS);
    V.used = used;
    V.gen_tokens = tokens;
    V.drawn = drawn;
    V.sched_steps = last + 1;
    V.rounds_done = events;
    V.live = 0;
    V.done = 1;
}

}  // namespace sara
