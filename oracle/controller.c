/*
 * O1 -- CPU oracle of SARA's round-synchronous rollout allocation.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and
 * bench.py's CPU-baseline leg may load this library.  The product path
 * (paper_2607_26253_gb300/) never calls it, shares no code with it, and fails
 * loudly when its own CUDA library is missing.
 *
 * What it computes (arxiv 2607.26253):
 *   - Beta prior / conjugate posterior (Sec. 3.2): after n rollouts with s
 *     successes, gamma | (n,s) ~ Beta(alpha0 + s, beta0 + n - s).
 *   - Effectiveness predictor p_eff(n,s) (Prop. 1, Eq. peff): 1 if mixed,
 *     else 1 - B(alpha0, beta0+k)/B(alpha0, beta0+n) for s = 0 and the mirror
 *     image for s = n.  At n = 0 both all-fail and all-pass completions are
 *     possible, so p_eff(0,0) = 1 - R_fail - R_pass (the printed formula drops
 *     one term there; the proof of Prop. 1 needs n >= 1).
 *   - DECIDE (Eq. decide): commit if mixed and n >= commit_min; abandon if
 *     n = k (all-same) or p_eff < tau_low (strict, exact); else continue.
 *   - Algorithm 1: probe, then per round decide -> refill -> advance, with the
 *     budget cap N (App. D defaults: commit_min = k, Beta(1,1)).
 *
 * Arithmetic: integer priors only (1 <= alpha0, beta0 <= 8, k <= 64).  For
 * integer a the Beta-function ratio is a finite product,
 *   B(a, b+r) / B(a, b) = prod_{i<a} (b+i) / (b+r+i),
 * so p_eff is an exact fraction; tau_low is the exact rational
 * tau_num / tau_den (the paper states its thresholds as decimals, 0.45 =
 * 9/20), and every comparison is an exact 128-bit integer test.
 *
 * Readings where the paper is silent (each one is listed in the design notes):
 *   - continuing prompts are funded first, in p_eff-descending order (ties by
 *     ascending stream index), one rollout each while used + 1 <= N; a prompt
 *     that cannot be funded becomes INCOMPLETE;
 *   - fresh prompts are then drawn in stream order while the working set is
 *     below B - |C| and a whole n0-probe fits in the budget (no partial probes);
 *   - the step stops once |C| >= B (groups committed in that round are kept);
 *   - every rollout issued in a round completes (no cancellation).
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef unsigned __int128 u128;

enum { ST_UNDRAWN = 0, ST_ACTIVE = 1, ST_COMMITTED = 2, ST_ABANDONED = 3, ST_INCOMPLETE = 4 };
enum { D_CONTINUE = 0, D_COMMIT = 1, D_ABANDON = 2 };
enum {
    C_ROLLOUTS = 0, C_GEN_TOKENS, C_PREFILL_TOKENS, C_DECODE_STEPS, C_ROUNDS, C_COMMITTED,
    C_ABANDONED, C_INCOMPLETE, C_DRAWN, C_NCOUNTERS
};

#define O1_EINVAL (-1)
#define O1_ENOMEM (-2)

/* ---- synthetic reward: SplitMix64 (Steele, Lea, Flood 2014), counter mode ---------------- */
static uint64_t sm64_at(uint64_t seed, uint64_t c) {
    uint64_t z = seed + c * 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* Verdict of rollout j of prompt q: Bernoulli(thr_q / 2^32) from output
 * number q*64 + j + 1 of SplitMix64(reward_seed). */
int o1_verdict(uint64_t reward_seed, int64_t q, int32_t j, uint64_t thr) {
    uint64_t h = sm64_at(reward_seed, (uint64_t)q * 64u + (uint64_t)j + 1u);
    return (h >> 32) < thr ? 1 : 0;
}

void o1_verdicts(int64_t P, int32_t k, const uint64_t *thr, uint64_t reward_seed, uint8_t *out) {
    for (int64_t q = 0; q < P; ++q)
        for (int32_t j = 0; j < k; ++j) out[q * k + j] = (uint8_t)o1_verdict(reward_seed, q, j, thr[q]);
}

/* ---- exact predictor ---------------------------------------------------------------------- */
typedef struct { u128 num, den; } frac;

/* prod_{i<a} (b+i) / (b+r+i) as a fraction: the posterior-predictive probability that the
 * r remaining Bernoulli draws all land on the side whose posterior count is b, when the other
 * side's count is the integer a (Beta identity, App. A). */
static frac same_side_ratio(int a, int b, int r) {
    frac f = {1, 1};
    for (int i = 0; i < a; ++i) {
        f.num *= (u128)(b + i);
        f.den *= (u128)(b + r + i);
    }
    return f;
}

/* p_eff(n, s) of Prop. 1 (with both saturated completions at n = 0). */
static frac peff_exact(int n, int s, int k, int a0, int b0) {
    frac one = {1, 1};
    if (s >= 1 && n - s >= 1) return one;
    int r = k - n;
    if (n == 0) {
        frac rf = same_side_ratio(a0, b0, r); /* all k fail */
        frac rp = same_side_ratio(b0, a0, r); /* all k pass */
        frac p;
        p.den = rf.den * rp.den;
        p.num = p.den - rf.num * rp.den - rp.num * rf.den;
        return p;
    }
    frac R = (s == 0) ? same_side_ratio(a0, b0 + n, r)   /* all-fail prefix */
                      : same_side_ratio(b0, a0 + n, r);  /* all-pass prefix */
    frac p = {R.den - R.num, R.den};
    return p;
}

/* exact x < tau_num / tau_den for x = num/den with den < 2^64 (n >= 1). */
static int frac_below_tau(frac x, int64_t tau_num, int64_t tau_den) {
    return x.num * (u128)tau_den < (u128)tau_num * x.den;
}

/* a > b exactly (both in [0,1]). */
static int frac_greater(frac a, frac b) { return a.num * b.den > b.num * a.den; }

int o1_valid_prior(int k, int a0, int b0) {
    return k >= 2 && k <= 64 && a0 >= 1 && a0 <= 8 && b0 >= 1 && b0 <= 8;
}

/* p_eff as (num, den) split into 64-bit halves, for tests. */
int o1_peff(int n, int s, int k, int a0, int b0, uint64_t out[4]) {
    if (!o1_valid_prior(k, a0, b0) || n < 0 || n > k || s < 0 || s > n) return O1_EINVAL;
    frac p = peff_exact(n, s, k, a0, b0);
    out[0] = (uint64_t)(p.num >> 64); out[1] = (uint64_t)p.num;
    out[2] = (uint64_t)(p.den >> 64); out[3] = (uint64_t)p.den;
    return 0;
}

/* DECIDE(n, s) of Eq. (decide); n >= 1. */
int o1_decide(int n, int s, int k, int64_t tau_num, int64_t tau_den, int commit_min, int a0,
              int b0) {
    if (n < 1 || n > k || s < 0 || s > n) return -1;
    int mixed = (s >= 1) && (n - s >= 1);
    if (mixed) return n >= commit_min ? D_COMMIT : D_CONTINUE;
    if (n >= k) return D_ABANDON;
    return frac_below_tau(peff_exact(n, s, k, a0, b0), tau_num, tau_den) ? D_ABANDON : D_CONTINUE;
}

/* ---- Algorithm 1 -------------------------------------------------------------------------- */
typedef struct { const uint8_t *n, *s; int k, a0, b0; } prio_ctx;
static prio_ctx g_prio;

/* p_eff descending, then stream index ascending. */
static int prio_cmp(const void *pa, const void *pb) {
    int32_t qa = *(const int32_t *)pa, qb = *(const int32_t *)pb;
    frac fa = peff_exact(g_prio.n[qa], g_prio.s[qa], g_prio.k, g_prio.a0, g_prio.b0);
    frac fb = peff_exact(g_prio.n[qb], g_prio.s[qb], g_prio.k, g_prio.a0, g_prio.b0);
    if (frac_greater(fa, fb)) return -1;
    if (frac_greater(fb, fa)) return 1;
    return (qa > qb) - (qa < qb);
}

/*
 * One rollout-collection step.  Inputs: pool of P prompts in stream order with latent
 * thresholds thr[P] and per-rollout lengths[P*k]; verdicts from `verdict_table` ([P*k], 0/1)
 * when non-NULL, else from o1_verdict(reward_seed, q, j, thr[q]).
 * Outputs: status[P], n[P], s[P], decided_round[P] (-1 unless committed/abandoned),
 * counters[C_NCOUNTERS], and optionally issued_per_round[max_rounds].
 */
int o1_collect_step(int32_t P, const uint64_t *thr, const int32_t *lengths,
                    const uint8_t *verdict_table, int32_t prompt_len, int32_t k, int32_t n0,
                    int64_t tau_num, int64_t tau_den, int32_t commit_min, int32_t a0, int32_t b0,
                    int32_t target_B, int64_t N, uint64_t reward_seed, uint8_t *status, uint8_t *n, uint8_t *s,
                    int16_t *decided_round, int64_t *counters, int32_t *issued_per_round,
                    int32_t max_rounds) {
    if (P < 0 || !o1_valid_prior(k, a0, b0) || n0 < 1 || n0 > k || tau_den < 1 ||
        tau_den > 2147483647 || tau_num < 0 || tau_num > tau_den ||
        commit_min < 2 || commit_min > k || target_B < 1 || N < 0 || prompt_len < 1)
        return O1_EINVAL;
    if (!verdict_table && !thr) return O1_EINVAL;

    int32_t *active = (int32_t *)malloc(sizeof(int32_t) * (size_t)(P + 1));
    int32_t *order = (int32_t *)malloc(sizeof(int32_t) * (size_t)(P + 1));
    int32_t *iss_q = (int32_t *)malloc(sizeof(int32_t) * (size_t)(P + 1));
    int32_t *iss_c = (int32_t *)malloc(sizeof(int32_t) * (size_t)(P + 1));
    if (!active || !order || !iss_q || !iss_c) {
        free(active); free(order); free(iss_q); free(iss_c);
        return O1_ENOMEM;
    }
    for (int32_t q = 0; q < P; ++q) {
        status[q] = ST_UNDRAWN; n[q] = 0; s[q] = 0; decided_round[q] = -1;
    }
    for (int c = 0; c < C_NCOUNTERS; ++c) counters[c] = 0;
    if (issued_per_round)
        for (int32_t r = 0; r < max_rounds; ++r) issued_per_round[r] = 0;

    int64_t used = 0;
    int32_t C = 0, cursor = 0, na = 0, ni = 0, round = 0;

    /* Round 0: probe fresh prompts with n0 rollouts each (Alg. 1, first line). */
    while (cursor < P && na < target_B && used + n0 <= N) {
        int32_t q = cursor++;
        status[q] = ST_ACTIVE;
        active[na++] = q;
        iss_q[ni] = q; iss_c[ni] = n0; ++ni;
        used += n0;
        counters[C_DRAWN]++;
    }

    while (ni > 0) {
        /* Execute the round: one batched call over every issued rollout. */
        int32_t issued = 0;
        int64_t maxL = 0;
        for (int32_t e = 0; e < ni; ++e) {
            int32_t q = iss_q[e];
            for (int32_t t = 0; t < iss_c[e]; ++t) {
                int32_t j = n[q];
                int v = verdict_table ? verdict_table[(int64_t)q * k + j]
                                      : o1_verdict(reward_seed, q, j, thr[q]);
                int64_t L = lengths ? lengths[(int64_t)q * k + j] : 0;
                s[q] = (uint8_t)(s[q] + v);
                n[q] = (uint8_t)(n[q] + 1);
                counters[C_GEN_TOKENS] += L;
                if (L > maxL) maxL = L;
                ++issued;
            }
        }
        if (issued_per_round && round < max_rounds) issued_per_round[round] = issued;
        counters[C_DECODE_STEPS] += maxL;
        counters[C_ROUNDS]++;

        /* DECIDE for every active prompt (stream order). */
        int32_t w = 0;
        for (int32_t i = 0; i < na; ++i) {
            int32_t q = active[i];
            int d = o1_decide(n[q], s[q], k, tau_num, tau_den, commit_min, a0, b0);
            if (d == D_COMMIT) {
                status[q] = ST_COMMITTED; decided_round[q] = (int16_t)round; ++C;
            } else if (d == D_ABANDON) {
                status[q] = ST_ABANDONED; decided_round[q] = (int16_t)round;
            } else {
                active[w++] = q;
            }
        }
        na = w;
        ni = 0;
        if (C >= target_B) break;

        /* Advance continuing prompts by one rollout, prioritised by p_eff. */
        memcpy(order, active, sizeof(int32_t) * (size_t)na);
        g_prio.n = n; g_prio.s = s; g_prio.k = k; g_prio.a0 = a0; g_prio.b0 = b0;
        qsort(order, (size_t)na, sizeof(int32_t), prio_cmp);
        for (int32_t i = 0; i < na; ++i) {
            int32_t q = order[i];
            if (used + 1 <= N) {
                iss_q[ni] = q; iss_c[ni] = 1; ++ni;
                used += 1;
            } else {
                status[q] = ST_INCOMPLETE;
            }
        }
        w = 0;
        for (int32_t i = 0; i < na; ++i)
            if (status[active[i]] == ST_ACTIVE) active[w++] = active[i];
        na = w;

        /* Reallocate: fresh prompts toward the remaining need B - |C|. */
        while (cursor < P && na < target_B - C && used + n0 <= N) {
            int32_t q = cursor++;
            status[q] = ST_ACTIVE;
            active[na++] = q;
            iss_q[ni] = q; iss_c[ni] = n0; ++ni;
            used += n0;
            counters[C_DRAWN]++;
        }
        ++round;
    }

    for (int32_t i = 0; i < na; ++i)
        if (status[active[i]] == ST_ACTIVE) status[active[i]] = ST_INCOMPLETE;
    for (int32_t q = 0; q < P; ++q) {
        if (status[q] == ST_COMMITTED) counters[C_COMMITTED]++;
        else if (status[q] == ST_ABANDONED) counters[C_ABANDONED]++;
        else if (status[q] == ST_INCOMPLETE) counters[C_INCOMPLETE]++;
    }
    counters[C_ROLLOUTS] = used;
    counters[C_PREFILL_TOKENS] = counters[C_DRAWN] * (int64_t)(prompt_len - 1);
    free(active); free(order); free(iss_q); free(iss_c);
    return 0;
}
