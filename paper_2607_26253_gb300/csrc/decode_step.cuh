// One decode step of the policy (embedding -> every layer -> lm_head logits) as a single
// persistent, cooperative kernel: one CTA per SM, phases separated
// by release/acquire arrival counters in global memory instead of kernel boundaries.
//
// Why: at decode batch sizes the per-layer work is a few MB of weights per projection, so
// a kernel per projection spends most of its time starting, filling its pipeline and
// draining.  Here the weight stream never stops: the producer warp walks the whole step's
// weight tiles (and the attention phase's KV blocks, which do not depend on this step's
// activations) ahead of the consumers through a ring of 32 KB shared-memory slots, across
// phase boundaries.  Only the small activation operands wait for the previous phase.
//
// GEMM orientation: the activation rows are the MMA's M and 256 weight rows its N, so one
// tcgen05.mma (K = 16) consumes 8 KB of weights (~133 cycles at M = 64 or 128 alike).  The
// activation is a bf16 hi/lo pair (~16 mantissa bits); up to 64 live rows both parts sit in
// one stacked operand and a k-step is one MMA, above that two MMAs (hi, lo) accumulate.
// Rows beyond the live count are don't-care.
//
// Split-K: a phase's (tile, k-chunk) units are cut into equal contiguous ranges over its
// CTAs; each CTA stores its fp32 partial tile with plain stores and the consuming phase
// sums a tile's partials in CTA order (deterministic, no atomics).
//
// Warp roles (352 threads, 11 warps):
//   warp 0   W producer: bulk copies of pre-swizzled weight tiles and KV blocks
//   warp 1   tcgen05 issuer and tensor-memory owner; hands the attention phase's KV tiles
//            to the compute warp group that runs their unit
//   warp 2   X producer: activation chunks, after the phase they come from has completed
//   warps 3..10  compute: GEMM epilogues, attention softmax / merge, residual + RMSNorm +
//                SwiGLU finalisation, embedding, logits
//
// Phases of layer l (counter index 1 + 9l + k):
//   0 QKV   x_g W_qkv^T -> partials        (a subset of the CTAs: few tiles)
//   1 FIN_Q q, k, v = RMSNorm scale + RoPE of the summed partials, fp16, once per row; the
//           new k, v appended to the KV cache
//   2 ATT   softmax(q K^T) V, 128-position KV blocks, online softmax over a split's blocks
//           with warp-level MMAs (mma.sync: N = 8 heads, operands and accumulators in
//           registers; the tcgen05 path's issue / commit / tensor-memory round trips cost more
//           than these products); the last split of a row to finish merges the splits
//   3 O     att W_o^T -> partials           (a subset of the CTAs)
//   4 FIN_O x += sum; x_g = x * g_mlp (bf16 hi/lo, blocked); per-row sum of squares
//   5 GU    x_g W_gu^T -> partials          (gate / up interleaved in 64-row blocks)
//   6 FIN_GU h = silu(r g) * (r u), r = 1/rms(x)  (bf16 hi/lo, blocked)
//   7 DOWN  h W_down^T -> partials
//   8 FIN_D x += sum; x_g = x * g_next; sum of squares
// then lm_head over whole 256-token tiles fused with the Gumbel-max sampler: per (row, tile,
// half-tile) maximum of logit + noise; the logits are stored only under teacher forcing.
//
// Layouts (all chosen so that bulk copies land MMA operands in shared memory in the
// 128-byte-swizzled K-major form the tensor core reads):
//   weights       tiles of 256 rows (the last may have 128): [N/256][K/64][rows][64],
//                 16-byte granule j of row r at granule j ^ (r % 8)
//   activations   [K/64][2 rows16][64] bf16, 8-row groups alternating hi / lo parts, same swizzle
//   KV cache      per (layer, slot, kv head, 128-position block): K as [d/64][128 pos][64 d]
//                 and V transposed as [pos/64][128 d][64 pos], fp16, head dim padded to 128
#pragma once
#include "device_common.cuh"
#include "step_state.cuh"

namespace sara {

constexpr int kMegaThreads = 352;
constexpr int kMegaCThreads = 256;  // compute warps 3..10
constexpr int kWSlots = 4;  // weight / KV ring entries (a power of two: slot = index & 3)
constexpr int kDetailRows = 16;  // profiling builds: rows of 4 detail stamps per CTA
constexpr int kSlotBytes = 32768;
constexpr int kRingBytes = 4 * 32768 + 65536;  // W slots, then the X stages
constexpr int kMaxXStages = 8;
constexpr int kTileN = 256;           // weight rows (output features) per GEMM tile
constexpr int kKVPos = 128;           // positions per KV block (an attention split holds `span` blocks)
constexpr int kKVBlockBytes = 65536;  // K 2 x 16 KB + V^T 2 x 16 KB
constexpr int kMegaMaxSplits = 96;    // splits per row a merge handles (context <= 96 blocks)
constexpr int kPhasesPerLayer = 9;
constexpr int kMaxCtaBlocks = 256;    // attention KV block ids a CTA keeps in shared memory
// phases of a layer (counter index 1 + 9 l + phase)
enum : int { kPhQKV = 0, kPhFinQ = 1, kPhAtt = 2, kPhO = 3, kPhFinO = 4, kPhGU = 5, kPhFinGU = 6, kPhDown = 7,
             kPhFinD = 8 };
__device__ constexpr int kGemmPhases[4] = {kPhQKV, kPhO, kPhGU, kPhDown};
constexpr int kSmallPhaseUnits = 2;   // QKV / O: units per participating CTA
constexpr int kCntStride = 16;        // phase counters 128 bytes apart (one L2 line each)
constexpr uint32_t kTmemCols = 512;
// Attention P tiles (per warp group, two buffers): [8 heads][128 positions] fp16, rows padded
// to 272 bytes so the eight rows of an ldmatrix fall in distinct banks.
constexpr int kAttPRow = 272;
constexpr int kAttPBytes = 8 * kAttPRow;
// Attention probabilities are taken against a running maximum that is re-based only when a
// score exceeds it by more than this (log2 units): P <= 2^8 in fp16, and most blocks skip the
// block maximum and the rescale of the output.
constexpr float kSoftmaxHeadroom = 8.f;

struct MegaParams {
    int layers, d, H, KVH, hd, F, V, Gq, nqkv;
    float eps, scale_log2;
    const uint8_t *w_qkv, *w_o, *w_gu, *w_down, *w_lm;  // blocked weights, layer strides below
    int64_t ls_qkv, ls_o, ls_gu, ls_down;
    const uint16_t *embed;                          // [V][d] bf16
    const uint16_t *attn_norm, *mlp_norm;           // [L][d]
    const uint16_t *final_norm;                     // [d]
    const float2 *rope;                             // [positions][hd/2] (cos, sin)
    uint8_t *kv;                                    // paged KV cache: block id b of layer l, kv head h
    int64_t kv_layer;                               // at kv + l * kv_layer + (b * KVH + h) * 64 KB
    StepPtrs c;
    int rows_cap, rows_cap16;
    int gp_qkv, gp_o;                               // CTAs taking part in the QKV / O projections
    float *x;                                       // [rows_cap][d] residual stream
    uint8_t *xg;                                    // pair-blocked [d/64][2 rows_cap16][64]
    uint8_t *att;                                   // pair-blocked [H*hd/64][2 rows_cap16][64]
    uint8_t *hm;                                    // pair-blocked [F/64][2 rows_cap16][64]
    float *ssqA, *ssqM;                             // [d/64][rows_cap] partial sums of x^2
    float *gpart;                                   // [segments][rows_cap][256] GEMM partial tiles
    uint16_t *qkv16;                                // [rows_cap][nqkv] fp16 q (scaled), k, v of the step
    float *part;                                    // [items][KVH][Gq][hd + 2] attention split partials
    int *att_cnt;                                   // [rows_cap][KVH] split arrival counters
    float *logits;                                  // [rows_cap][V] fp32, written if write_logits
    int write_logits;                               // teacher forcing: store the logits too
    unsigned long long *cnt;                        // phase arrival counters (monotonic), kCntStride apart
    unsigned long long *epoch;                      // launches completed since the reset
    uint64_t *stamps;                               // profiling builds: [cta][phase + 1][4] timestamps
    int n_stamp_ph;
    unsigned long long *ktime;                      // [2]: earliest CTA start, latest CTA end (ns)
};

// Profiling builds (-DSARA_STAMPS): per CTA and phase, when the compute warps arrived (0),
// when the phase's input dependency was observed (1), when the W producer finished issuing
// the phase's copies (2) and when the MMA issuer committed the phase's last MMA (3).
#ifdef SARA_STAMPS
#define MEGA_STAMP(ph, kind)                                                                              \
    do {                                                                                                  \
        if (p.stamps) p.stamps[((size_t)blockIdx.x * p.n_stamp_ph + (ph)) * 4 + (kind)] = globaltimer_ns(); \
    } while (0)
// Detail stamps of one layer (layer 2): the attention and first finalize phases (first unit
// of each CTA, ids 0-15) and the first 12 units of the gate / up GEMM (ids 16-63: W copy
// issued, W slot full and X stage full as seen by the MMA issuer, MMAs committed); the last
// kDetailRows phase slots of the same array (the one before them holds the kernel start).
#define MEGA_DETAIL(i)                                                                                    \
    do {                                                                                                  \
        if (p.stamps)                                                                                     \
            p.stamps[((size_t)blockIdx.x * p.n_stamp_ph + p.n_stamp_ph - kDetailRows + ((i) >> 2)) * 4 + \
                     ((i) & 3)] = globaltimer_ns();                                                       \
    } while (0)
#else
#define MEGA_STAMP(ph, kind) \
    do {                     \
    } while (0)
#define MEGA_DETAIL(i) \
    do {               \
    } while (0)
#endif

struct MegaSmem {
    uint64_t wfull[kWSlots], wempty[kWSlots];
    uint64_t kvready[2][kWSlots];  // attention: ring slot s holds warp group g's next KV tile
    uint64_t xfull[kMaxXStages], xempty[kMaxXStages];
    uint64_t acc_full[2], acc_empty[2];
    uint64_t drain;
    unsigned long long target;  // counter value meaning "every CTA of this launch arrived"
    uint64_t wait_ns;           // bounded-wait limit of this launch
    float p_headroom;           // attention: log2 of how far P may exceed 1 before re-basing
    int stall_idx;              // test hook: the phase counter whose waits never complete (-1: none)
    uint32_t tmem_base;
    int abort;
    int last_flag;
    int rows, rows16, nx, nx_lg, n_items, att_span;  // nx = 2^nx_lg X stages
    float rstd[128];
    // KV block ids: of this CTA's attention blocks (unit i's block j at ablk[aoff[i] + j]), and
    // of each row's current position (ablk_ok = 0: too many to hold, looked up in the table)
    int ablk[kMaxCtaBlocks];
    int aoff[32];
    int rowblk[128];
    int ablk_ok;
    float red[2][4][8], red2[2][4][8];  // per warp group: attention max / sum reductions
    float mw[2][8][kMegaMaxSplits];      // per warp group: split weights of a merge
    float ml[2][8];
    int last_flag2[2];
};

constexpr size_t kMegaSmemBytes =
    1024 + (size_t)kRingBytes + 4 * 4096 + sizeof(MegaSmem);

// ------------------------------------------------------------------------------ layouts
// Pair-blocked activation (a GEMM operand held as bf16 hi + lo parts): per 64-wide k-chunk,
// 2 rows16 rows of 128 B (64 bf16, 128-byte swizzle) in 8-row groups that alternate between
// the hi parts of rows 8g..8g+7 and their lo parts.  Byte offset of the hi part of element
// (r, k); the lo part sits kLoOff bytes after it.  One MMA over the chunk's first 2 R16 rows
// multiplies hi and lo parts at once (rows16 <= 64); with a 2048-byte group stride the hi
// (lo) groups alone form a 128-row operand.
constexpr int kLoOff = 1024;
__host__ __device__ __forceinline__ int64_t xblk_off(int r, int k, int rows16) {
    const int chunk = k >> 6, col = k & 63;
    return ((int64_t)chunk * 2 * rows16 + 16 * (r >> 3) + (r & 7)) * 128 +
           ((((col >> 3) ^ (r & 7)) << 4) | ((col & 7) << 1));
}
// Byte offsets of K(pp, d) and V(pp, d) inside one 128-position KV block.
__host__ __device__ __forceinline__ int kv_k_off(int pp, int d) {
    return (d >> 6) * 16384 + pp * 128 + (((((d & 63) >> 3) ^ (pp & 7)) << 4) | ((d & 7) << 1));
}
__host__ __device__ __forceinline__ int kv_v_off(int pp, int d) {
    const int c = pp & 63;
    return 32768 + (pp >> 6) * 16384 + d * 128 + ((((c >> 3) ^ (d & 7)) << 4) | ((c & 7) << 1));
}
// Byte offset of the (tile t, k-chunk kc) block of a blocked weight matrix [N][K].
__host__ __device__ __forceinline__ int64_t wblk_off(int N, int K, int t, int kc) {
    const int rows = (N - t * kTileN) < kTileN ? (N - t * kTileN) : kTileN;
    return (int64_t)t * kTileN * K * 2 + (int64_t)kc * rows * 128;
}

// ------------------------------------------------------------------------------ waits
// Bounded mbarrier wait that also gives up (returning false) once the CTA is aborting.
__device__ __forceinline__ bool mwait(uint64_t *bar, uint32_t parity, int *err, volatile int *abort, uint64_t limit) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 63u) == 0) {
            if (*abort) return false;
            if (globaltimer_ns() - t0 > limit) {
                report_error(err, ERR_WAIT_TIMEOUT);
                *abort = 1;
                return false;
            }
        }
    }
}

// Spin until a phase counter reaches `target` (acquire loads);
// bounded, gives up on abort or once another CTA reported a timeout.
__device__ __forceinline__ bool spin_counter(const unsigned long long *cnt, unsigned long long target, int *err,
                                             volatile int *abort, uint64_t limit) {
    if (ld_acquire_u64(cnt) >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        __nanosleep(32);
        if (ld_acquire_u64(cnt) >= target) return true;
        if ((it & 15u) == 0) {
            if (*abort) return false;
            if (*(volatile int *)err & ERR_WAIT_TIMEOUT) {
                *abort = 1;
                return false;
            }
            if (globaltimer_ns() - t0 > limit) {
                report_error(err, ERR_WAIT_TIMEOUT);
                *abort = 1;
                return false;
            }
        }
    }
}

// Counter value a wait on phase counter idx needs: every CTA of this launch arrived (the
// test hook makes one counter's target unreachable, so its waits run into the time limit).
__device__ __forceinline__ unsigned long long phase_target(const MegaParams &p, const MegaSmem &S, int idx) {
    return idx == S.stall_idx ? ~0ull : S.target;
}

// ------------------------------------------------------------------------------ phases
struct GemmPh {
    const uint8_t *w;
    int N, K, kch, T, Gp;
    const uint8_t *x;  // pair-blocked operand
    bool whole;  // whole tiles per CTA (lm_head: the argmax of a tile is finished in one CTA)
};

// GEMM phase k (kPhQKV, kPhO, kPhGU, kPhDown) of layer l; l == layers: lm_head.
__device__ __forceinline__ GemmPh gemm_phase(const MegaParams &p, int l, int k) {
    GemmPh g;
    g.whole = false;
    g.Gp = gridDim.x;
    if (l == p.layers) {
        g.w = p.w_lm; g.N = p.V; g.K = p.d; g.x = p.xg; g.whole = true;
    } else if (k == kPhQKV) {
        g.w = p.w_qkv + l * p.ls_qkv; g.N = p.nqkv; g.K = p.d; g.x = p.xg; g.Gp = p.gp_qkv;
    } else if (k == kPhO) {
        g.w = p.w_o + l * p.ls_o; g.N = p.d; g.K = p.H * p.hd; g.x = p.att; g.Gp = p.gp_o;
    } else if (k == kPhGU) {
        g.w = p.w_gu + l * p.ls_gu; g.N = 2 * p.F; g.K = p.d; g.x = p.xg;
    } else {
        g.w = p.w_down + l * p.ls_down; g.N = p.d; g.K = p.F; g.x = p.hm;
    }
    g.kch = g.K / 64;
    g.T = (g.N + kTileN - 1) / kTileN;
    // at most one CTA per unit (tile for lm_head), so every participating CTA holds a
    // non-empty range and the CTAs between a tile's first and last owner all contributed
    g.Gp = min(g.Gp, g.whole ? g.T : g.T * g.kch);
    return g;
}
__device__ __forceinline__ int tile_rows(const GemmPh &g, int t) { return min(kTileN, g.N - kTileN * t); }

// This CTA's (tile, k-chunk) units: an equal contiguous share over the phase's CTAs, or
// (lm_head) a share of whole tiles.
// (Unit counts stay below 2^31 / SMs for every supported shape: 32-bit products suffice.)
__device__ __forceinline__ void gemm_range(const GemmPh &g, int64_t &u0, int64_t &u1) {
    const int c = blockIdx.x;
    if (c >= g.Gp) {
        u0 = u1 = 0;
        return;
    }
    if (g.whole) {
        u0 = (int64_t)(c * g.T / g.Gp) * g.kch;
        u1 = (int64_t)((c + 1) * g.T / g.Gp) * g.kch;
    } else {
        const int U = g.T * g.kch;
        u0 = c * U / g.Gp;
        u1 = (c + 1) * U / g.Gp;
    }
}
// CTA owning unit u when U units are cut into Gp equal contiguous ranges.
__device__ __forceinline__ int unit_owner(int u, int U, int Gp) {
    int c = u * Gp / U;
    while (c + 1 < Gp && (c + 1) * U / Gp <= u) ++c;
    while (c > 0 && c * U / Gp > u) --c;
    return c;
}
// First and last CTA holding a partial of tile t.  CTA c's partial of tile t is segment
// c + t of the partial buffer (distinct for every (c, t) of a phase: ranges are ordered).
__device__ __forceinline__ void tile_ctas(const GemmPh &g, int t, int &ca, int &cb) {
    const int U = g.T * g.kch;
    ca = unit_owner(t * g.kch, U, g.Gp);
    cb = unit_owner((t + 1) * g.kch - 1, U, g.Gp);
}

// Attention unit: one split of one row for one kv head.  Split sp covers the `span` KV
// blocks from block sp * span on: positions [p0, p0 + n) of the row's ctx, in nb blocks.
struct AttUnit {
    int item, kvh, row, sp, ctx, p0, n, nb, nsplit, slot;
    bool last;
};
__device__ __forceinline__ AttUnit att_unit(const MegaParams &p, int64_t a, int span) {
    AttUnit u;
    u.item = (int)(a / p.KVH);
    u.kvh = (int)(a - (int64_t)u.item * p.KVH);
    const int2 it = __ldg(&p.c.att_items[u.item]);
    u.row = it.x;
    u.sp = it.y;
    u.ctx = __ldg(&p.c.row_pos[u.row]) + 1;
    u.p0 = u.sp * span * kKVPos;
    u.n = min(u.ctx - u.p0, span * kKVPos);
    u.nb = (u.n + kKVPos - 1) / kKVPos;
    u.nsplit = ((u.ctx + kKVPos - 1) / kKVPos + span - 1) / span;
    u.last = u.p0 + u.n == u.ctx;
    u.slot = __ldg(&p.c.row_slot[u.row]);
    return u;
}
// Attention units in equal contiguous ranges, counted from the last CTA down: the QKV
// projection runs on the first CTAs, so a small unit count lands on CTAs that are free
// to prefetch during it.
__device__ __forceinline__ void att_range(const MegaParams &p, int n_items, int64_t &a0, int64_t &a1) {
    const int NU = n_items * p.KVH, G = (int)gridDim.x, v = G - 1 - (int)blockIdx.x;
    a0 = v * NU / G;
    a1 = (v + 1) * NU / G;
}
// Address of block id b, kv head h of layer l in the paged KV cache.
__device__ __forceinline__ uint8_t *kv_addr(const MegaParams &p, int l, int b, int h) {
    return p.kv + l * p.kv_layer + ((int64_t)b * p.KVH + h) * kKVBlockBytes;
}
// Block j of this CTA's attention unit ui (= a - a0) in layer l's KV cache.
__device__ __forceinline__ uint8_t *kv_block(const MegaParams &p, const MegaSmem &S, int l, const AttUnit &u, int ui,
                                             int j) {
    const int b = S.ablk_ok ? S.ablk[S.aoff[ui] + j]
                            : __ldg(&p.c.blk_tab[(int64_t)u.slot * p.c.nblk_max + u.p0 / kKVPos + j]);
    return kv_addr(p, l, b, u.kvh);
}

// The KV block ids of this CTA's attention units (one warp, lane i: unit a0 + i), read once
// per launch from the block table into shared memory for the W producer.
__device__ __forceinline__ void fill_att_blocks(const MegaParams &p, MegaSmem &S, int lane) {
    int64_t a0, a1;
    att_range(p, S.n_items, a0, a1);
    const int nu = (int)(a1 - a0);
    bool ok = nu <= 32;
    int nb = 0, off = 0;
    AttUnit u{};
    if (ok) {
        if (lane < nu) {
            u = att_unit(p, a0 + lane, S.att_span);
            nb = u.nb;
        }
        int x = nb;  // inclusive warp scan of the block counts
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        off = x - nb;
        ok = __shfl_sync(0xffffffffu, x, 31) <= kMaxCtaBlocks;
    }
    if (ok && lane < nu) {
        S.aoff[lane] = off;
        const int32_t *src = p.c.blk_tab + (int64_t)u.slot * p.c.nblk_max + u.p0 / kKVPos;
        for (int j0 = 0; j0 < nb; j0 += 8) {  // eight loads in flight
            int v[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) v[q] = j0 + q < nb ? __ldg(src + j0 + q) : 0;
#pragma unroll
            for (int q = 0; q < 8; ++q)
                if (j0 + q < nb) S.ablk[off + j0 + q] = v[q];
        }
    }
    if (lane == 0) S.ablk_ok = ok ? 1 : 0;
    __syncwarp();
}

// ------------------------------------------------------------------------------ W producer
__device__ __forceinline__ void mega_w_producer(const MegaParams &p, MegaSmem &S, uint8_t *sW) {
    volatile int *ab = &S.abort;
    const uint64_t lim = S.wait_ns;
    int *err = &p.c.v->err;
    const uint64_t pol = l2_policy_evict_first();
    constexpr uint32_t nws = kWSlots;
    uint32_t wi = 0;
    bool ok = true;
    auto acquire = [&](uint32_t i) -> bool {
        return i < nws || mwait(&S.wempty[i % nws], ((i / nws) & 1) ^ 1, err, ab, lim);
    };
    for (int l = 0; l <= p.layers && ok; ++l) {
        for (int gp = 0; gp < 4 && ok; ++gp) {
            if (l == p.layers && gp > 0) break;
            const int k = kGemmPhases[gp];
            const GemmPh g = gemm_phase(p, l, k);
            int64_t u0, u1;
            gemm_range(g, u0, u1);
            for (int64_t u = u0; u < u1; ++u, ++wi) {
                if (!acquire(wi)) { ok = false; break; }
                const int s = (int)(wi % nws);
                const int t = (int)(u / g.kch), kc = (int)(u - (int64_t)t * g.kch);
                const uint32_t bytes = (uint32_t)tile_rows(g, t) * 128;
                mbar_arrive_expect_tx(&S.wfull[s], bytes);
                bulk_load(sW + (size_t)s * kSlotBytes, g.w + wblk_off(g.N, g.K, t, kc), bytes, &S.wfull[s], pol);
                if (k == kPhGU && l == min(2, p.layers - 1) && u - u0 < 12) MEGA_DETAIL(16 + (int)(u - u0));
            }
            MEGA_STAMP(1 + kPhasesPerLayer * l + k, 2);
            if (k == 0 && l < p.layers && ok) {
                // the attention phase's KV blocks follow the QKV weights in ring order: unit
                // pairs (one unit per compute warp group), block by block, the K of the pair's
                // units, then their V^T; each one ring entry (K: d < 64 | d >= 64 halves, V^T:
                // positions < 64 | >= 64).  The block holding a row's new position is copied
                // once the q / k / v phase has appended it to the cache.
                int64_t a0, a1;
                att_range(p, S.n_items, a0, a1);
                const int span = S.att_span;
                bool finq_seen = false;
                for (int64_t a = a0; a < a1 && ok; a += 2) {
                    const bool two = a + 1 < a1;
                    const AttUnit ua = att_unit(p, a, span);
                    const AttUnit ub = two ? att_unit(p, a + 1, span) : ua;
                    const int nbb = two ? ub.nb : 0;
                    for (int j = 0; j < max(ua.nb, nbb) && ok; ++j) {
                        for (int kv = 0; kv < 2 && ok; ++kv) {
                            for (int w = 0; w < 2 && ok; ++w) {
                                const AttUnit &u = w ? ub : ua;
                                if (j >= (w ? nbb : ua.nb)) continue;
                                if (kv == 0 && u.last && j == u.nb - 1 && !finq_seen) {
                                    const int fq = 1 + kPhasesPerLayer * l + kPhFinQ;
                                    if (!spin_counter(&p.cnt[fq * kCntStride], phase_target(p, S, fq), err, ab, lim)) {
                                        ok = false;
                                        break;
                                    }
                                    fence_proxy_async_global();
                                    finq_seen = true;
                                }
                                const uint8_t *blk = kv_block(p, S, l, u, (int)(a - a0) + w, j);
                                const int nj = min(kKVPos, u.n - j * kKVPos);
                                if (!acquire(wi)) { ok = false; break; }
                                const int s = (int)(wi % nws);
                                if (kv == 0) {
                                    const uint32_t kb = (uint32_t)(((nj + 7) & ~7) * 128);
                                    mbar_arrive_expect_tx(&S.wfull[s], p.hd > 64 ? 2 * kb : kb);
                                    bulk_load(sW + (size_t)s * kSlotBytes, blk, kb, &S.wfull[s], pol);
                                    if (p.hd > 64)
                                        bulk_load(sW + (size_t)s * kSlotBytes + 16384, blk + 16384, kb, &S.wfull[s], pol);
                                } else {
                                    const uint32_t vb = (uint32_t)(p.hd * 128);
                                    mbar_arrive_expect_tx(&S.wfull[s], nj > 64 ? 2 * vb : vb);
                                    bulk_load(sW + (size_t)s * kSlotBytes, blk + 32768, vb, &S.wfull[s], pol);
                                    if (nj > 64)
                                        bulk_load(sW + (size_t)s * kSlotBytes + 16384, blk + 49152, vb, &S.wfull[s], pol);
                                }
                                ++wi;
                            }
                        }
                    }
                }
                MEGA_STAMP(1 + kPhasesPerLayer * l + kPhAtt, 2);
            }
        }
    }
    if (!ok) {  // every copy already issued lands before the CTA exits
        for (uint32_t s = 0; s < nws && s < wi; ++s) {
            const uint32_t last = ((wi - 1 - s) / nws) * nws + s;
            mbar_wait(&S.wfull[s], (last / nws) & 1, err);
        }
    }
}

// ------------------------------------------------------------------------------ X producer
__device__ __forceinline__ void mega_x_producer(const MegaParams &p, MegaSmem &S, uint8_t *sX) {
    volatile int *ab = &S.abort;
    const uint64_t lim = S.wait_ns;
    int *err = &p.c.v->err;
    const uint64_t pol = l2_policy_evict_last();
    const int NX = S.nx, R16 = S.rows16, nxl = S.nx_lg;
    const uint32_t stage = (uint32_t)R16 * 256;  // hi + lo parts of the live rows' groups
    const int64_t chunk_stride = (int64_t)p.rows_cap16 * 256;
    uint32_t xi = 0;
    bool ok = true;
    for (int l = 0; l <= p.layers && ok; ++l) {
        for (int gp = 0; gp < 4 && ok; ++gp) {
            if (l == p.layers && gp > 0) break;
            const int k = kGemmPhases[gp];
            const GemmPh g = gemm_phase(p, l, k);
            int64_t u0, u1;
            gemm_range(g, u0, u1);
            if (u0 >= u1) continue;
            // the phase this operand comes from (the one before it): FIN_D of l-1 / embedding,
            // ATT, FIN_O, FIN_GU
            const int dep = (l == p.layers || k == 0) ? kPhasesPerLayer * l : 1 + kPhasesPerLayer * l + k - 1;
            if (!spin_counter(&p.cnt[dep * kCntStride], phase_target(p, S, dep), err, ab, lim)) { ok = false; break; }
            MEGA_STAMP(1 + kPhasesPerLayer * l + k, 1);
            fence_proxy_async_global();
            for (int64_t u = u0; u < u1; ++u, ++xi) {
                const int s = (int)(xi & (uint32_t)(NX - 1));
                if (xi >= (uint32_t)NX && !mwait(&S.xempty[s], ((xi >> nxl) & 1) ^ 1, err, ab, lim)) { ok = false; break; }
                const int kc = (int)(u % g.kch);
                mbar_arrive_expect_tx(&S.xfull[s], stage);
                bulk_load(sX + (size_t)s * stage, g.x + kc * chunk_stride, stage, &S.xfull[s], pol);
            }
        }
    }
    if (!ok) {
        for (uint32_t s = 0; s < (uint32_t)NX && s < xi; ++s) {
            const uint32_t last = (((xi - 1 - s) >> nxl) << nxl) + s;
            mbar_wait(&S.xfull[s], (last >> nxl) & 1, err);
        }
    }
}

// ------------------------------------------------------------------------------ MMA issuer
__device__ __forceinline__ void mega_mma(const MegaParams &p, MegaSmem &S, uint8_t *sW, uint8_t *sX, uint8_t *sQ,
                                         uint8_t *sP, uint32_t tmem) {
    volatile int *ab = &S.abort;
    const uint64_t lim = S.wait_ns;
    int *err = &p.c.v->err;
    const int NX = S.nx, R16 = S.rows16, nxl = S.nx_lg;
    const uint32_t stage = (uint32_t)R16 * 256;
    // at most 64 live rows: one MMA per k-step over the stacked hi / lo groups (M = 2 R16
    // rounded up to 64 or 128: the rows past the stage only feed accumulator rows nobody
    // reads); more: the hi and the lo groups as two 128-row operands into one accumulator
    const bool stacked = R16 <= 64;
    uint32_t wi = 0, xi = 0;
    int use0 = 0, use1 = 0, tseg = 0;  // accumulator buffer uses, GEMM tiles so far
    bool ok = true;
    constexpr uint32_t nws = kWSlots;
    auto wslot = [&](uint32_t i) -> uint32_t { return smem_u32(sW + (size_t)(i % nws) * kSlotBytes); };
    auto wwait = [&](uint32_t i) -> bool { return mwait(&S.wfull[i % nws], (i / nws) & 1, err, ab, lim); };
    auto gemm = [&](const GemmPh &g, int64_t u0, int64_t u1, bool det) {
        const int64_t ub = u0;
        for (int64_t u = u0; u < u1 && ok;) {
            const int t = (int)(u / g.kch);
            const int64_t e = min(u1, (int64_t)(t + 1) * g.kch);
            const int a = tseg & 1;  // tiles alternate between two accumulators (epilogue overlaps)
            const int use_a = a ? use1 : use0;
            if (use_a >= 1 && !mwait(&S.acc_empty[a], (use_a - 1) & 1, err, ab, lim)) { ok = false; break; }
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(a * kTileN);
            const uint32_t idg = idesc_bf16_f32(R16 <= 32 ? 64u : 128u, (uint32_t)tile_rows(g, t));
            bool first = true;
            for (; u < e; ++u, ++wi, ++xi) {
                const int xs = (int)(xi & (uint32_t)(NX - 1));
                const bool dj = det && u - ub < 12;
                if (!wwait(wi)) { ok = false; break; }
                if (dj) MEGA_DETAIL(28 + (int)(u - ub));
                if (!mwait(&S.xfull[xs], (xi >> nxl) & 1, err, ab, lim)) { ok = false; break; }
                if (dj) MEGA_DETAIL(40 + (int)(u - ub));
                tc_fence_after();
                const uint32_t aw = wslot(wi), ax = smem_u32(sX + (size_t)xs * stage);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t bd = sdesc_kmajor_sw128(aw + kk * 32);
                    const uint32_t acc = (first && kk == 0) ? 0u : 1u;
                    if (stacked) {
                        tc_mma_bf16(d, sdesc_kmajor_sw128(ax + kk * 32), bd, idg, acc);
                    } else {
                        tc_mma_bf16(d, sdesc_kmajor_sw128(ax + kk * 32, 2048), bd, idg, acc);
                        tc_mma_bf16(d, sdesc_kmajor_sw128(ax + kLoOff + kk * 32, 2048), bd, idg, 1u);
                    }
                }
                first = false;
                tc_commit(&S.wempty[wi % nws]);
                tc_commit(&S.xempty[xs]);
                if (dj) MEGA_DETAIL(52 + (int)(u - ub));
            }
            if (!ok) break;
            tc_commit(&S.acc_full[a]);
            if (a) ++use1; else ++use0;
            ++tseg;
        }
    };
    // The attention phase's ring entries (its KV tiles) are read and released by the compute
    // warp groups.  The issuer is the ring's one in-order observer: it waits for each entry to
    // land and hands it to the group that runs its unit (an arrival on kvready[group][slot]).
    // A group's consecutive uses of a slot are then at most one barrier phase apart (the slot
    // is refilled only after the group released its previous tile there), which a group
    // waiting on the shared wfull barriers directly could not rely on.
    int gi = 0;  // attention units so far (unit i of a phase runs on group (gi + i) & 1)
    auto att_fwd = [&](int64_t a0, int64_t a1) -> bool {
        const int n = (int)(a1 - a0), span = S.att_span;
        for (int i = 0; i < n; i += 2) {
            const bool two = i + 1 < n;
            const int nba = att_unit(p, a0 + i, span).nb, nbb = two ? att_unit(p, a0 + i + 1, span).nb : 0;
            for (int j = 0; j < max(nba, nbb); ++j)
                for (int kv = 0; kv < 2; ++kv)
                    for (int x = 0; x < 2; ++x) {
                        if (j >= (x ? nbb : nba)) continue;
                        if (!wwait(wi)) return false;
                        mbar_arrive(&S.kvready[(gi + i + x) & 1][wi % nws]);
                        ++wi;
                    }
        }
        gi += n;
        return true;
    };
    for (int l = 0; l <= p.layers && ok; ++l) {
        for (int gp = 0; gp < 4 && ok; ++gp) {
            if (l == p.layers && gp > 0) break;
            const int k = kGemmPhases[gp];
            const GemmPh g = gemm_phase(p, l, k);
            int64_t u0, u1;
            gemm_range(g, u0, u1);
            gemm(g, u0, u1, k == kPhGU && l == min(2, p.layers - 1));
            MEGA_STAMP(1 + kPhasesPerLayer * l + k, 3);
            if (k == 0 && l < p.layers && ok) {
                int64_t a0, a1;
                att_range(p, S.n_items, a0, a1);
                if (!att_fwd(a0, a1)) ok = false;
                MEGA_STAMP(1 + kPhasesPerLayer * l + kPhAtt, 3);
            }
        }
    }
    // every MMA issued has retired before tensor memory is released
    tc_commit(&S.drain);
    mbar_wait(&S.drain, 0, err);
}

// ------------------------------------------------------------------------------ compute
__device__ __forceinline__ void store_hilo(uint8_t *base, int64_t off, float v) {
    uint16_t h, l;
    split_bf16(v, h, l);
    *reinterpret_cast<uint16_t *>(base + off) = h;
    *reinterpret_cast<uint16_t *>(base + off + kLoOff) = l;
}


__device__ __forceinline__ void mega_compute(const MegaParams &p, MegaSmem &S, uint8_t *sW, uint8_t *sQ, uint8_t *sP,
                                             uint32_t tmem) {
    volatile int *ab = &S.abort;
    const uint64_t lim = S.wait_ns;
    int *err = &p.c.v->err;
    const int ctid = threadIdx.x - 96;  // 0..255
    const int cw = ctid >> 5, lane = threadIdx.x & 31;
    const int quarter = (threadIdx.x >> 5) & 3;  // tensor-memory lanes 32*quarter ..
    const int half = cw >> 2;                    // warps 3..6 -> 0, 7..10 -> 1
    const int G = gridDim.x, cta = blockIdx.x;
    const int R = S.rows, R16c = p.rows_cap16;
    const int d = p.d, hd = p.hd, Gq = p.Gq;
    const int gw = cta * 8 + cw, nw = G * 8;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    // GEMM accumulator lane -> activation row.  Stacked operand (at most 64 live rows): operand
    // row m holds the hi (lo) part of row 8 (m / 16) + m % 8 for m % 16 < 8 (>= 8); M = 128
    // puts operand row m in lane m, M = 64 (at most 32 rows) in lane 32 (m / 16) + m % 16.
    // The hi and lo accumulators of a row are lanes i and i ^ 8 of one warp (pair sum by a
    // shuffle; the hi lane stores).  Otherwise (M = 128, hi and lo accumulated together) row
    // i is lane i.
    const int R16 = S.rows16;
    const bool pair = R16 <= 64;
    const int my_row = R16 <= 32   ? ((lane & 0x18) == 0 ? quarter * 8 + lane : 1 << 20)
                       : pair      ? ((lane & 8) == 0 ? quarter * 16 + 8 * (lane >> 4) + (lane & 7) : 1 << 20)
                                   : quarter * 32 + lane;
    const bool quarter_live = (R16 <= 32 ? quarter * 8 : pair ? quarter * 16 : quarter * 32) < R;
    uint32_t wring = 0;  // W ring entries of the phases before the current one (the producer's count)
    uint32_t kvpar = 0;  // per ring slot (bit s): parity of this warp group's next kvready wait
    auto kv_wait = [&](uint32_t e) {
        const uint32_t sl = e % kWSlots;
        mwait(&S.kvready[half][sl], (kvpar >> sl) & 1u, err, ab, lim);
        kvpar ^= 1u << sl;
    };
    int gi = 0, cuse0 = 0, cuse1 = 0, tseg = 0;  // accumulator buffer uses, GEMM tiles so far

    // phase arrival: the CTA's writes of this phase (made visible to thread 0 by the barrier)
    // are released to the other CTAs with the counter increment
    // (x_operand: this phase wrote a GEMM operand that bulk copies of other CTAs will read)
    auto arrive = [&](int idx, bool x_operand) {
        if (x_operand) fence_proxy_async_global();
        named_bar_sync(1, kMegaCThreads);
        if (ctid == 0) {
            MEGA_STAMP(idx, 0);
            red_add_release_gpu(&p.cnt[idx * kCntStride], 1ull);
        }
    };
    auto wait_phase = [&](int idx) {
        if (ctid == 0) {
            spin_counter(&p.cnt[idx * kCntStride], phase_target(p, S, idx), err, ab, lim);
            MEGA_STAMP(idx + 1, 1);
        }
        named_bar_sync(1, kMegaCThreads);
    };
    auto load_rstd = [&](const float *ssq) {
        if (ctid < R) {  // every partial load in flight at once (d <= 2048: at most 32)
            float v[32];
#pragma unroll
            for (int t = 0; t < 32; ++t) v[t] = t < d / 64 ? __ldcg(&ssq[(int64_t)t * p.rows_cap + ctid]) : 0.f;
            float s = 0.f;
#pragma unroll
            for (int t = 0; t < 32; ++t) s += v[t];
            S.rstd[ctid] = rsqrtf(s / (float)d + p.eps);
        }
        named_bar_sync(1, kMegaCThreads);
    };
    // this CTA's partial tiles: row my_row, columns [128 half, +128) of the tile
    auto gemm_epi = [&](const GemmPh &g, int64_t u0, int64_t u1) {
        for (int64_t u = u0; u < u1;) {
            const int t = (int)(u / g.kch);
            u = min(u1, (int64_t)(t + 1) * g.kch);
            const int a = tseg & 1;
            mwait(&S.acc_full[a], (a ? cuse1 : cuse0) & 1, err, ab, lim);
            tc_fence_after();
            const int rows_t = tile_rows(g, t);
            if (quarter_live && half * 128 < rows_t) {
                float *dst = p.gpart + ((int64_t)(cta + t) * p.rows_cap + (my_row < R ? my_row : 0)) * kTileN + half * 128;
#pragma unroll 1
                for (int cc = 0; cc < 4; ++cc) {
                    float v[32];
                    tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(a * kTileN + half * 128 + cc * 32), v);
                    if (pair) {
#pragma unroll
                        for (int e = 0; e < 32; ++e) v[e] += __shfl_xor_sync(0xffffffffu, v[e], 8);
                    }
                    if (my_row < R) {
                        float4 *q = reinterpret_cast<float4 *>(dst + cc * 32);
#pragma unroll
                        for (int e = 0; e < 8; ++e) q[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.acc_empty[a]);
            if (a) ++cuse1; else ++cuse0;
            ++tseg;
        }
    };
    // x += (sum of g's partials); x_g = x * gn (blocked hi/lo); per (row, 128-feature
    // block) sum of squares of x.  g == nullptr: x as it is (embedding).
    auto fin_resid = [&](const GemmPh *g, const uint16_t *gn, float *ssq) {
        // unit = (row, 64 features): lane = 2 features; up to 32 contributors' loads in
        // flight per round, summed in CTA order.  Sums of squares per 128 features: the two
        // 64-feature halves of a block are adjacent units of the same warp pass
        const int d64 = d / 64;
        for (int u = gw; u < R * d64; u += nw) {
            const int r = u / d64, h64 = u - r * d64;
            const int f = h64 * 64 + lane * 2;
            // the norm weights load with the residual and the partials (a layer's norm is not
            // in L1, and after the residual's store the load could not move ahead of it)
            const uint32_t gb = __ldg(reinterpret_cast<const unsigned int *>(gn + f));
            float2 x = __ldcg(reinterpret_cast<const float2 *>(p.x + (int64_t)r * d + f));
            if (g) {
                const int gt = f / kTileN, col = f - gt * kTileN;
                int ca, cb;
                tile_ctas(*g, gt, ca, cb);
                float2 s = make_float2(0.f, 0.f);
                for (int c0 = ca; c0 <= cb; c0 += 32) {
                    float2 v[32];
#pragma unroll
                    for (int k = 0; k < 32; ++k)
                        v[k] = c0 + k <= cb ? __ldcg(reinterpret_cast<const float2 *>(
                                                  p.gpart + ((int64_t)(c0 + k + gt) * p.rows_cap + r) * kTileN + col))
                                            : make_float2(0.f, 0.f);
#pragma unroll
                    for (int k = 0; k < 32; ++k) {
                        s.x += v[k].x; s.y += v[k].y;
                    }
                }
                x.x += s.x; x.y += s.y;
                *reinterpret_cast<float2 *>(p.x + (int64_t)r * d + f) = x;
            }
            uint16_t h0, l0, h1, l1;
            split_bf16(x.x * bf16_to_f32(gb & 0xffff), h0, l0);
            split_bf16(x.y * bf16_to_f32(gb >> 16), h1, l1);
            const int64_t off = xblk_off(r, f, R16c);
            *reinterpret_cast<uint32_t *>(p.xg + off) = (uint32_t)h0 | ((uint32_t)h1 << 16);
            *reinterpret_cast<uint32_t *>(p.xg + off + kLoOff) = (uint32_t)l0 | ((uint32_t)l1 << 16);
            const float sq = warp_sum(x.x * x.x + x.y * x.y);
            if (lane == 0) ssq[(int64_t)h64 * p.rows_cap + r] = sq;
        }
    };

    // the KV block of each row's current position (its k, v are appended there every layer)
    if (ctid < R) {
        const int pos = __ldg(&p.c.row_pos[ctid]);
        S.rowblk[ctid] = __ldg(&p.c.blk_tab[(int64_t)__ldg(&p.c.row_slot[ctid]) * p.c.nblk_max + pos / kKVPos]);
    }

    // ---------------------------------------------------------------- embedding
    // (same (row, 64-feature) units and lanes as the finalisation that reads them back)
    for (int u = gw; u < R * (d / 64); u += nw) {
        const int r = u / (d / 64), h64 = u - r * (d / 64);
        int tok = p.c.row_tok[r];
        if (tok < 0 || tok >= p.V) {
            if (lane == 0) report_error(err, ERR_BOUNDS);
            tok = 0;
        }
        const int f = h64 * 64 + lane * 2;
        const uint32_t e = *reinterpret_cast<const uint32_t *>(p.embed + (int64_t)tok * d + f);
        *reinterpret_cast<float2 *>(p.x + (int64_t)r * d + f) = make_float2(bf16_to_f32(e & 0xffff), bf16_to_f32(e >> 16));
    }
    __syncwarp();
    fin_resid(nullptr, p.attn_norm, p.ssqA);
    arrive(0, true);

    for (int l = 0; l < p.layers; ++l) {
        const int base = 1 + kPhasesPerLayer * l;
        int64_t u0, u1;
        const GemmPh gq = gemm_phase(p, l, kPhQKV), go = gemm_phase(p, l, kPhO), gu = gemm_phase(p, l, kPhGU),
                     gdn = gemm_phase(p, l, kPhDown);
        // ------------------------------------------------------------ QKV
        gemm_range(gq, u0, u1);
        wring += (uint32_t)(u1 - u0);
        gemm_epi(gq, u0, u1);
        arrive(base + kPhQKV, false);
        // ------------------------------------------------------------ q, k, v (once per row)
        {
            // unit = (row, head, 64 dims): the head's QKV partials summed in CTA order, times
            // 1/rms; RoPE on q and k; q pre-scaled by log2(e)/sqrt(hd) for the exp2 softmax;
            // fp16 q, k, v for the attention phase; k and v appended to the KV cache at the
            // row's position
            wait_phase(base + kPhQKV);
            const int nh = p.H + 2 * p.KVH, dpu = min(hd, 64), upr = hd / dpu;
            for (int u = gw; u < R * nh * upr; u += nw) {
                const int r = u / (nh * upr), rem = u - r * nh * upr;
                // lanes past the unit's dims (head dim 32) repeat lane 0's loads and store nothing:
                // every lane takes part in the row's sum-of-squares reduction
                const bool live = 2 * lane < dpu;
                const int head = rem / upr, d0 = (rem - head * upr) * dpu + (live ? 2 * lane : 0);
                const bool isq = head < p.H, isk = !isq && head < p.H + p.KVH;
                const int half_hd = hd >> 1;
                const int pd0 = d0 < half_hd ? d0 + half_hd : d0 - half_hd;
                const int f0 = head * hd + d0, t = f0 / kTileN;
                const int col = f0 - t * kTileN, pcol = head * hd + pd0 - t * kTileN;
                int ca, cb;
                tile_ctas(gq, t, ca, cb);
                // the row's sum-of-squares partials and rotation factors load with the first
                // batch of QKV partials
                const float sq = lane < d / 64 ? __ldcg(&p.ssqA[(int64_t)lane * p.rows_cap + r]) : 0.f;
                const int pos = __ldg(&p.c.row_pos[r]);
                float2 c0r = make_float2(1.f, 0.f), c1r = c0r;
                if (isq || isk) {
                    const int fr = d0 < half_hd ? d0 : pd0;
                    c0r = __ldg(&p.rope[(int64_t)pos * half_hd + fr]);
                    c1r = __ldg(&p.rope[(int64_t)pos * half_hd + fr + 1]);
                }
                float2 x = make_float2(0.f, 0.f), xp = x;
                for (int c0 = ca; c0 <= cb; c0 += 16) {  // 16 contributors' loads in flight, CTA order
                    float2 a[16], b2[16];
#pragma unroll
                    for (int k = 0; k < 16; ++k) {
                        const bool ok = c0 + k <= cb;
                        const float *src = p.gpart + ((int64_t)(c0 + k + t) * p.rows_cap + r) * kTileN;
                        a[k] = ok ? __ldcg(reinterpret_cast<const float2 *>(src + col)) : make_float2(0.f, 0.f);
                        b2[k] = (ok && !(head >= p.H + p.KVH)) ? __ldcg(reinterpret_cast<const float2 *>(src + pcol))
                                                               : make_float2(0.f, 0.f);
                    }
#pragma unroll
                    for (int k = 0; k < 16; ++k) {
                        x.x += a[k].x; x.y += a[k].y;
                        xp.x += b2[k].x; xp.y += b2[k].y;
                    }
                }
                const float rs = rsqrtf(warp_sum(sq) / (float)d + p.eps) * (isq ? p.scale_log2 : 1.f);
                if (!live) continue;
                float y0 = x.x, y1 = x.y;
                if (isq || isk) {  // rotate the pairs (i, i + hd/2)
                    if (d0 < half_hd) {
                        y0 = x.x * c0r.x - xp.x * c0r.y;
                        y1 = x.y * c1r.x - xp.y * c1r.y;
                    } else {
                        y0 = x.x * c0r.x + xp.x * c0r.y;
                        y1 = x.y * c1r.x + xp.y * c1r.y;
                    }
                }
                const uint16_t h0 = f32_to_f16_sat(y0 * rs), h1 = f32_to_f16_sat(y1 * rs);
                *reinterpret_cast<uint32_t *>(p.qkv16 + (int64_t)r * p.nqkv + head * hd + d0) =
                    (uint32_t)h0 | ((uint32_t)h1 << 16);
                if (!isq) {  // the new position's k / v into the cache (blocked layout)
                    const int kvh = head - p.H - (isk ? 0 : p.KVH);
                    uint8_t *blk = kv_addr(p, l, S.rowblk[r], kvh);
                    const int pp = pos % kKVPos;
                    if (isk) {
                        *reinterpret_cast<uint32_t *>(blk + kv_k_off(pp, d0)) = (uint32_t)h0 | ((uint32_t)h1 << 16);
                    } else {
                        *reinterpret_cast<uint16_t *>(blk + kv_v_off(pp, d0)) = h0;
                        *reinterpret_cast<uint16_t *>(blk + kv_v_off(pp, d0 + 1)) = h1;
                    }
                }
            }
            arrive(base + kPhFinQ, false);
        }
        // ------------------------------------------------------------ attention
        {
            int64_t a0, a1;
            att_range(p, S.n_items, a0, a1);
            const int n = (int)(a1 - a0);
            wait_phase(base + kPhFinQ);
            const bool det_layer = l == min(2, p.layers - 1);
            if (det_layer && ctid == 0) MEGA_DETAIL(13);
            if (det_layer && ctid == 0) MEGA_DETAIL(14);
#define DETAIL(i)                                       \
    do {                                                \
        if (det_layer && ctid == 0 && i_unit == 0) MEGA_DETAIL(i); \
    } while (0)
            int i_unit = 0;
            DETAIL(0);
            // units alternate between the two warp groups: group h (warps 3..6 / 7..10, named
            // barrier 2 + h) runs the units (gi + i) & 1 == h, each unit: q in registers, then
            // per KV block scores -> probabilities against the running max -> output sum
            // (online softmax over the unit's blocks, warp-level MMAs on the ring's K and V^T
            // tiles, which the group releases), then output / split partial + merge, in order
            const int hb = 2 + half;     // this group's named barrier
            const int ht = ctid & 127;   // thread index within the group
            const int hq = ht >> 5;      // warp within the group
            const int span = S.att_span;
            // ring entries of the phase's KV blocks: per unit pair, block by block, the K of
            // the pair's units, then their V^T (the W producer's order)
            uint32_t wpair = wring;
            uint8_t *pbufs = sQ + half * 2 * kAttPBytes;  // this group's two P buffers
            const int g8 = lane >> 2, t4 = lane & 3;     // mma fragment row / column pair
            const int kst = hd >> 4;                      // k-steps of q.k (16 dims each)
            for (int ip = 0; ip < n; ip += 2) {
                const bool two = ip + 1 < n;
                const AttUnit ua = att_unit(p, a0 + ip, span);
                const int nba = ua.nb, nbb = two ? att_unit(p, a0 + ip + 1, span).nb : 0;
                const int x = ((gi + ip) & 1) == half ? 0 : 1;  // our unit of the pair
                const uint32_t w0 = wpair;
                wpair += 2u * (uint32_t)(nba + nbb);
                if (x == 1 && !two) continue;
                const int i = ip + x;
                const AttUnit u = x ? att_unit(p, a0 + i, span) : ua;
                const int jm = min(nba, nbb);
                auto ent = [&](int j, int kv) -> uint32_t {
                    return j < jm ? w0 + 4u * j + 2u * kv + x : w0 + 4u * jm + 2u * (j - jm) + kv;
                };
                if (half == 0) { i_unit = i; DETAIL(1); }
                // ---- q of the unit's heads as mma B fragments (q^T: k = dim, n = head g8)
                uint32_t qf[8][2];
                {
                    const bool hv = g8 < Gq;
                    const uint16_t *qh = p.qkv16 + (int64_t)u.row * p.nqkv + (u.kvh * Gq + (hv ? g8 : 0)) * hd + 2 * t4;
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks) {
                        const bool ok = hv && ks < kst;
                        qf[ks][0] = ok ? __ldcg(reinterpret_cast<const unsigned int *>(qh + 16 * ks)) : 0u;
                        qf[ks][1] = ok ? __ldcg(reinterpret_cast<const unsigned int *>(qh + 16 * ks + 8)) : 0u;
                    }
                }
                // ---- per block: S^T = K q^T (warp hq: positions 32 hq ..), probabilities
                // against the running max, which is re-based only when a score exceeds it by
                // more than the headroom; P to shared memory; O^T += V^T P^T (warp hq: dims
                // 16 (hq + 4 m)).  Thread (g8, t4) holds heads 2 t4, 2 t4 + 1 throughout.
                float mrun[2] = {-INFINITY, -INFINITY}, lthr[2] = {0.f, 0.f};
                float o[2][4];
#pragma unroll
                for (int m = 0; m < 2; ++m)
#pragma unroll
                    for (int q = 0; q < 4; ++q) o[m][q] = 0.f;
                for (int jb = 0; jb < u.nb; ++jb) {
                    const int nj = min(kKVPos, u.n - jb * kKVPos);
                    const uint32_t ek = ent(jb, 0), ev = ent(jb, 1);
                    kv_wait(ek);
                    if (half == 0 && jb == 0) DETAIL(2);
                    const uint32_t kbase = smem_u32(sW + (size_t)(ek % kWSlots) * kSlotBytes);
                    float sc[2][4];
#pragma unroll
                    for (int m = 0; m < 2; ++m) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) sc[m][q] = 0.f;
                        const int pb0 = 32 * hq + 16 * m;
                        if (pb0 < nj) {  // rows past the copied ones are never read
                            const int pr = pb0 + (lane & 7) + ((lane >> 3) & 1) * 8;  // ldmatrix row of this lane
#pragma unroll
                            for (int ks = 0; ks < 8; ++ks) {
                                if (ks < kst) {
                                    const int dim = 16 * ks + (lane >> 4) * 8;
                                    uint32_t a[4];
                                    ldsm_x4(kbase + (dim >> 6) * 16384 + pr * 128 + ((((dim & 63) >> 3) ^ (pr & 7)) << 4), a);
                                    mma_f16_16816(sc[m], a, qf[ks][0], qf[ks][1]);
                                }
                            }
                        }
                    }
                    // scores: sc[m][q] = s(position 32 hq + 16 m + g8 + 8 (q >> 1), head 2 t4 + (q & 1))
                    uint8_t *pbuf = pbufs + (jb & 1) * kAttPBytes;
                    auto put_p = [&](float (&e)[2][4]) {
#pragma unroll
                        for (int m = 0; m < 2; ++m)
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const int pos = 32 * hq + 16 * m + g8 + 8 * (q >> 1);
                                *reinterpret_cast<uint16_t *>(pbuf + (2 * t4 + (q & 1)) * kAttPRow + 2 * pos) =
                                    f32_to_f16_sat(e[m][q]);
                            }
                    };
                    float e[2][4];
                    bool rebase = jb == 0;
                    if (!rebase) {
                        bool over = false;
#pragma unroll
                        for (int m = 0; m < 2; ++m)
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const bool valid = 32 * hq + 16 * m + g8 + 8 * (q >> 1) < nj;
                                e[m][q] = valid ? exp2f(sc[m][q] - mrun[q & 1]) : 0.f;
                                over |= valid && sc[m][q] - mrun[q & 1] > S.p_headroom;
                            }
                        put_p(e);
                        rebase = named_bar_any(hb, 128, over);
                    }
                    if (rebase) {  // the block's maximum per head joins the running max
                        float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
                        for (int m = 0; m < 2; ++m)
#pragma unroll
                            for (int q = 0; q < 4; ++q)
                                if (32 * hq + 16 * m + g8 + 8 * (q >> 1) < nj) mx[q & 1] = fmaxf(mx[q & 1], sc[m][q]);
#pragma unroll
                        for (int k = 0; k < 2; ++k)
#pragma unroll
                            for (int o2 = 4; o2 < 32; o2 <<= 1) mx[k] = fmaxf(mx[k], __shfl_xor_sync(0xffffffffu, mx[k], o2));
                        if (g8 == 0) {
                            S.red[half][hq][2 * t4] = mx[0];
                            S.red[half][hq][2 * t4 + 1] = mx[1];
                        }
                        named_bar_sync(hb, 128);
                        float alpha[2];
#pragma unroll
                        for (int k = 0; k < 2; ++k) {
                            const int h = 2 * t4 + k;
                            const float mnew = fmaxf(mrun[k], fmaxf(fmaxf(S.red[half][0][h], S.red[half][1][h]),
                                                                    fmaxf(S.red[half][2][h], S.red[half][3][h])));
                            alpha[k] = exp2f(mrun[k] - mnew);  // 0 on the first block
                            mrun[k] = mnew;
                            lthr[k] *= alpha[k];
                        }
#pragma unroll
                        for (int m = 0; m < 2; ++m)
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                o[m][q] *= alpha[q & 1];
                                const bool valid = 32 * hq + 16 * m + g8 + 8 * (q >> 1) < nj;
                                e[m][q] = valid ? exp2f(sc[m][q] - mrun[q & 1]) : 0.f;
                            }
                        put_p(e);
                        named_bar_sync(hb, 128);
                    }
                    // every warp has read the K block: its ring slot goes back to the producer
                    if (ht == 0) mbar_arrive(&S.wempty[ek % kWSlots]);
#pragma unroll
                    for (int m = 0; m < 2; ++m)
#pragma unroll
                        for (int q = 0; q < 4; ++q) lthr[q & 1] += e[m][q];
                    if (half == 0 && jb == 0) DETAIL(3);
                    // ---- O^T += V^T P^T over the block's positions (k-steps of 16)
                    kv_wait(ev);
                    const uint32_t vbase = smem_u32(sW + (size_t)(ev % kWSlots) * kSlotBytes);
                    const uint32_t pbase = smem_u32(pbuf);
                    const int kpv = (nj + 15) >> 4;
#pragma unroll
                    for (int ks = 0; ks < 8; ks += 2) {
                        if (ks < kpv) {
                            uint32_t bq[4];  // P^T fragments of k-steps ks, ks + 1 (rows: heads 0..7)
                            ldsm_x4(pbase + (lane & 7) * kAttPRow + (16 * ks + 8 * (lane >> 3)) * 2, bq);
#pragma unroll
                            for (int m = 0; m < 2; ++m) {
                                const int dr = 16 * (hq + 4 * m) + (lane & 7) + ((lane >> 3) & 1) * 8;  // V^T row (dim)
                                if (16 * (hq + 4 * m) < hd) {
#pragma unroll
                                    for (int kk = 0; kk < 2; ++kk) {
                                        if (ks + kk < kpv) {
                                            const int pos = 16 * (ks + kk) + (lane >> 4) * 8;
                                            uint32_t a[4];
                                            ldsm_x4(vbase + (pos >> 6) * 16384 + dr * 128 + ((((pos & 63) >> 3) ^ (dr & 7)) << 4), a);
                                            mma_f16_16816(o[m], a, bq[2 * kk], bq[2 * kk + 1]);
                                        }
                                    }
                                }
                            }
                        }
                    }
                    named_bar_sync(hb, 128);  // every warp has read the V^T block
                    if (ht == 0) mbar_arrive(&S.wempty[ev % kWSlots]);
                }
                if (half == 0) DETAIL(4);
                // ---- row sums: heads 2 t4, 2 t4 + 1 over the warp (lanes of equal t4), then
                // over the group's warps
                float lrun[2];
                {
#pragma unroll
                    for (int k = 0; k < 2; ++k)
#pragma unroll
                        for (int o2 = 4; o2 < 32; o2 <<= 1) lthr[k] += __shfl_xor_sync(0xffffffffu, lthr[k], o2);
                    if (g8 == 0) {
                        S.red2[half][hq][2 * t4] = lthr[0];
                        S.red2[half][hq][2 * t4 + 1] = lthr[1];
                    }
                    named_bar_sync(hb, 128);
#pragma unroll
                    for (int k = 0; k < 2; ++k) {
                        const int h = 2 * t4 + k;
                        lrun[k] = (S.red2[half][0][h] + S.red2[half][1][h]) + (S.red2[half][2][h] + S.red2[half][3][h]);
                    }
                }
                // ---- output (single split) or partial + split merge.  o[m][q]: O^T(dim
                // 16 (hq + 4 m) + g8 + 8 (q >> 1), head 2 t4 + (q & 1))
                {
                    const int dd = quarter * 32 + lane;  // output dim of this thread in the merge
                    if (u.nsplit == 1) {
#pragma unroll
                        for (int m = 0; m < 2; ++m)
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const int dim = 16 * (hq + 4 * m) + g8 + 8 * (q >> 1), h = 2 * t4 + (q & 1);
                                if (dim < hd && h < Gq)
                                    store_hilo(p.att, xblk_off(u.row, (u.kvh * Gq + h) * hd + dim, R16c),
                                               o[m][q] / lrun[q & 1]);
                            }
                    } else {
                        float *mine = p.part + ((int64_t)u.item * p.KVH + u.kvh) * Gq * (hd + 2);
#pragma unroll
                        for (int m = 0; m < 2; ++m)
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const int dim = 16 * (hq + 4 * m) + g8 + 8 * (q >> 1), h = 2 * t4 + (q & 1);
                                if (dim < hd && h < Gq) mine[h * (hd + 2) + 2 + dim] = o[m][q];
                            }
                        if (hq == 0 && g8 == 0) {
#pragma unroll
                            for (int k = 0; k < 2; ++k) {
                                const int h = 2 * t4 + k;
                                if (h < Gq) {
                                    mine[h * (hd + 2)] = mrun[k];
                                    mine[h * (hd + 2) + 1] = lrun[k];
                                }
                            }
                        }
                        named_bar_sync(hb, 128);
                        if (half == 0) DETAIL(5);
                        if (ht == 0) {  // one acquire-release count: publishes this split, sees the others
                            const int old = atom_add_acq_rel_gpu(&p.att_cnt[u.row * p.KVH + u.kvh], 1);
                            S.last_flag2[half] = old == u.nsplit - 1;
                            if (S.last_flag2[half]) p.att_cnt[u.row * p.KVH + u.kvh] = 0;
                        }
                        named_bar_sync(hb, 128);
                        if (half == 0) DETAIL(6);
                        if (S.last_flag2[half]) {  // merge the row's splits in split order
                            const int ns = min(u.nsplit, kMegaMaxSplits);
                            const int64_t sp_stride = (int64_t)p.KVH * Gq * (hd + 2);
                            const float *pbase = p.part + ((int64_t)__ldg(&p.c.row_item0[u.row]) * p.KVH + u.kvh) * Gq * (hd + 2);
                            // the first four splits' outputs (thread dd: dim dd of every head) load
                            // together with the split weights' inputs: one round trip for both
                            const float *src = pbase + 2 + dd;
                            float vpre[4][8];
#pragma unroll
                            for (int q = 0; q < 4; ++q)
#pragma unroll
                                for (int g = 0; g < 8; ++g)
                                    vpre[q][g] = (dd < hd && g < Gq && q < ns) ? __ldcg(src + q * sp_stride + g * (hd + 2)) : 0.f;
                            // split weights 2^(m_s - M) and the total weight L per head (warp hq: heads hq, hq + 4)
                            for (int g = hq; g < Gq; g += 4) {
                                float ms[3], ls[3];
                                float Mx = -INFINITY;
#pragma unroll
                                for (int q = 0; q < 3; ++q) {
                                    const int sp = lane + 32 * q;
                                    ms[q] = sp < ns ? __ldcg(pbase + sp * sp_stride + g * (hd + 2)) : -INFINITY;
                                    ls[q] = sp < ns ? __ldcg(pbase + sp * sp_stride + g * (hd + 2) + 1) : 0.f;
                                    Mx = fmaxf(Mx, ms[q]);
                                }
#pragma unroll
                                for (int o = 16; o > 0; o >>= 1) Mx = fmaxf(Mx, __shfl_xor_sync(0xffffffffu, Mx, o));
                                float L = 0.f;
#pragma unroll
                                for (int q = 0; q < 3; ++q) {
                                    const int sp = lane + 32 * q;
                                    const float w = sp < ns ? exp2f(ms[q] - Mx) : 0.f;
                                    if (sp < ns) S.mw[half][g][sp] = w;
                                    L += w * ls[q];
                                }
                                L = warp_sum(L);
                                if (lane == 0) S.ml[half][g] = L;
                            }
                            named_bar_sync(hb, 128);
                            if (dd < hd) {  // thread dd: output dim dd of every head
                                float acc[8];
#pragma unroll
                                for (int g = 0; g < 8; ++g) acc[g] = 0.f;
#pragma unroll
                                for (int q = 0; q < 4; ++q)
#pragma unroll
                                    for (int g = 0; g < 8; ++g) acc[g] += (g < Gq && q < ns ? S.mw[half][g][q] : 0.f) * vpre[q][g];
                                for (int s0 = 4; s0 < ns; s0 += 4) {  // the rest, four splits' loads in flight
                                    float v[4][8];
#pragma unroll
                                    for (int q = 0; q < 4; ++q)
#pragma unroll
                                        for (int g = 0; g < 8; ++g)
                                            v[q][g] = (g < Gq && s0 + q < ns) ? __ldcg(src + (s0 + q) * sp_stride + g * (hd + 2)) : 0.f;
#pragma unroll
                                    for (int q = 0; q < 4; ++q)
#pragma unroll
                                        for (int g = 0; g < 8; ++g)
                                            acc[g] += (g < Gq && s0 + q < ns ? S.mw[half][g][s0 + q] : 0.f) * v[q][g];
                                }
#pragma unroll
                                for (int g = 0; g < 8; ++g)
                                    if (g < Gq)
                                        store_hilo(p.att, xblk_off(u.row, (u.kvh * Gq + g) * hd + dd, R16c),
                                                   acc[g] / S.ml[half][g]);
                            }
                        }
                        named_bar_sync(hb, 128);
                        if (half == 0) DETAIL(7);
                    }
                }
            }
            wring = wpair;
            gi += n;
            i_unit = 0;
            DETAIL(8);
            arrive(base + kPhAtt, true);
            DETAIL(9);
#undef DETAIL
        }
        // ------------------------------------------------------------ O projection
        gemm_range(go, u0, u1);
        wring += (uint32_t)(u1 - u0);
        gemm_epi(go, u0, u1);
        arrive(base + kPhO, false);
        // ------------------------------------------------------------ residual, MLP norm input
        wait_phase(base + kPhO);
        if (l == min(2, p.layers - 1) && ctid == 0) MEGA_DETAIL(10);
        fin_resid(&go, p.mlp_norm + (int64_t)l * d, p.ssqM);
        if (l == min(2, p.layers - 1) && ctid == 0) MEGA_DETAIL(11);
        arrive(base + kPhFinO, true);
        if (l == min(2, p.layers - 1) && ctid == 0) MEGA_DETAIL(12);
        // ------------------------------------------------------------ gate / up
        gemm_range(gu, u0, u1);
        wring += (uint32_t)(u1 - u0);
        gemm_epi(gu, u0, u1);
        arrive(base + kPhGU, false);
        // ------------------------------------------------------------ SwiGLU
        {
            wait_phase(base + kPhGU);
            const int fb = p.F / 128;
            // unit = (row, 128 features of h) = one 256-row tile of the gate/up outputs; lane:
            // 4 features, gate at tile column c, up at c + 64 (c = 4 lane, or 128 + 4 lane - 64
            // for the tile's second 64 features).  A warp takes two units per pass with every
            // partial load in flight before the sums (in CTA order).
            const int c0 = (lane < 16) ? 4 * lane : 128 + 4 * lane - 64;
            for (int u = gw; u < R * fb; u += 2 * nw) {
                float4 gs[2], us[2];
                int rr[2], tt[2];
                float sq[2];  // the rows' sum-of-squares partials, loaded with the gate / up partials
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    const int uq = u + q * nw;
                    gs[q] = us[q] = make_float4(0.f, 0.f, 0.f, 0.f);
                    rr[q] = -1;
                    tt[q] = 0;
                    sq[q] = 0.f;
                    if (uq >= R * fb) continue;
                    const int r = uq / fb, t = uq - r * fb;
                    rr[q] = r;
                    tt[q] = t;
                    sq[q] = lane < d / 64 ? __ldcg(&p.ssqM[(int64_t)lane * p.rows_cap + r]) : 0.f;
                    int ca, cb;
                    tile_ctas(gu, t, ca, cb);
                    for (int cq = ca; cq <= cb; cq += 4) {
                        float4 a4[4], b4[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const bool ok = cq + k <= cb;
                            const float *src = p.gpart + ((int64_t)(cq + k + t) * p.rows_cap + r) * kTileN + c0;
                            a4[k] = ok ? __ldcg(reinterpret_cast<const float4 *>(src)) : make_float4(0.f, 0.f, 0.f, 0.f);
                            b4[k] = ok ? __ldcg(reinterpret_cast<const float4 *>(src + 64)) : make_float4(0.f, 0.f, 0.f, 0.f);
                        }
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            gs[q].x += a4[k].x; gs[q].y += a4[k].y; gs[q].z += a4[k].z; gs[q].w += a4[k].w;
                            us[q].x += b4[k].x; us[q].y += b4[k].y; us[q].z += b4[k].z; us[q].w += b4[k].w;
                        }
                    }
                }
                float rsq[2];
#pragma unroll
                for (int q = 0; q < 2; ++q) rsq[q] = rsqrtf(warp_sum(sq[q]) / (float)d + p.eps);
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    if (rr[q] < 0) continue;
                    const float rs = rsq[q];
                    const float gv[4] = {gs[q].x * rs, gs[q].y * rs, gs[q].z * rs, gs[q].w * rs};
                    const float uv[4] = {us[q].x * rs, us[q].y * rs, us[q].z * rs, us[q].w * rs};
                    uint16_t hh[4], hl[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) split_bf16(gv[e] / (1.0f + expf(-gv[e])) * uv[e], hh[e], hl[e]);
                    const int64_t off = xblk_off(rr[q], tt[q] * 128 + 4 * lane, R16c);
                    *reinterpret_cast<uint2 *>(p.hm + off) =
                        make_uint2((uint32_t)hh[0] | ((uint32_t)hh[1] << 16), (uint32_t)hh[2] | ((uint32_t)hh[3] << 16));
                    *reinterpret_cast<uint2 *>(p.hm + off + kLoOff) =
                        make_uint2((uint32_t)hl[0] | ((uint32_t)hl[1] << 16), (uint32_t)hl[2] | ((uint32_t)hl[3] << 16));
                }
            }
            arrive(base + kPhFinGU, true);
        }
        // ------------------------------------------------------------ down
        gemm_range(gdn, u0, u1);
        wring += (uint32_t)(u1 - u0);
        gemm_epi(gdn, u0, u1);
        arrive(base + kPhDown, false);
        // ------------------------------------------------------------ residual, next norm input
        wait_phase(base + kPhDown);
        fin_resid(&gdn, (l + 1 < p.layers) ? p.attn_norm + (int64_t)(l + 1) * d : p.final_norm, p.ssqA);
        arrive(base + kPhFinD, true);
    }

    // ---------------------------------------------------------------- lm_head + Gumbel-max
    // logits = (x_g W_lm^T) / rms(x) for the live rows, fused with the temperature-1 sampler:
    // each thread scans its row's 128 columns of a tile in increasing token order, adds the
    // Gumbel noise g(row key, token) and keeps the first maximum of logit + g; the per (row,
    // tile, half) maxima go to the bookkeeping kernel, which takes the row's argmax (ties to
    // the lowest token id).  Products and sums are rounded separately (no contraction), as
    // the sampler on stored logits would do them.  The logits themselves are written only
    // when requested (teacher forcing).
    {
        wait_phase(kPhasesPerLayer * p.layers);
        load_rstd(p.ssqA);
        const GemmPh g = gemm_phase(p, p.layers, 0);
        int64_t u0, u1;
        gemm_range(g, u0, u1);
        const bool act = my_row < R;
        const float rs = act ? S.rstd[my_row] : 0.f;
        const uint64_t seed = act ? __ldg(&p.c.row_seed[my_row]) : 0ull;
        const int nparts = 2 * g.T;
        float best = -INFINITY;  // running over this thread's tiles (its row and half)
        int bi = 0x7fffffff;
        for (int64_t u = u0; u < u1; u += g.kch) {
            const int t = (int)(u / g.kch);
            const int a = tseg & 1;
            mwait(&S.acc_full[a], (a ? cuse1 : cuse0) & 1, err, ab, lim);
            tc_fence_after();
            if (quarter_live && half * 128 < tile_rows(g, t)) {
                const int n0 = t * kTileN + half * 128;
                float *dst = p.logits + (int64_t)(act ? my_row : 0) * p.V + n0;
                const float best0 = best;  // the maximum over this thread's earlier tiles
#pragma unroll 1
                for (int cc = 0; cc < 4; ++cc) {
                    float v[32];
                    tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(a * kTileN + half * 128 + cc * 32), v);
                    if (pair) {
#pragma unroll
                        for (int e = 0; e < 32; ++e) v[e] += __shfl_xor_sync(0xffffffffu, v[e], 8);
                    }
                    if (act) {
#pragma unroll
                        for (int e = 0; e < 32; ++e) v[e] = __fmul_rn(v[e], rs);
                        if (p.write_logits) {
                            float4 *q = reinterpret_cast<float4 *>(dst + cc * 32);
#pragma unroll
                            for (int e = 0; e < 8; ++e) q[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
                        }
                        // Only tokens whose noise could lift them over the best so far are
                        // evaluated exactly: g(u) increases with u = (top 24 hash bits + 0.5) / 2^24,
                        // so v_e + g(u_e) > best needs u_e > exp(-exp(-(best - max_e v_e))); the
                        // cut is taken 1e-3 lower in g and 4 codes lower in the 24-bit u, far
                        // beyond the rounding of the float evaluation, so no candidate is lost.
                        // `best` runs over all of this thread's tiles: a (tile, half) whose
                        // tokens cannot beat an earlier tile's maximum reports -inf, which the
                        // row's argmax ignores (ties go to the lower token id either way).
                        float vmax = v[0];
#pragma unroll
                        for (int e = 1; e < 32; ++e) vmax = fmaxf(vmax, v[e]);
                        const float ureq = expf(-expf(-(best - vmax - 1e-3f)));  // 0 while best = -inf
                        const float cut = ureq * 16777216.0f - 4.0f;
                        const uint32_t thr = cut > 0.f ? (uint32_t)cut : 0u;
                        const int nb = n0 + cc * 32;
                        uint32_t cand = 0;
#pragma unroll
                        for (int e = 0; e < 32; ++e)
                            cand |= (uint32_t)((uint32_t)(splitmix_at(seed, (uint64_t)(nb + e) + 1) >> 40) >= thr) << e;
                        while (cand) {  // candidates in increasing token order: the first maximum is kept
                            const int e = __ffs(cand) - 1;
                            cand &= cand - 1;
                            float ve = v[0];
#pragma unroll
                            for (int k = 1; k < 32; ++k) ve = (k == e) ? v[k] : ve;
                            const float z = __fadd_rn(ve, gumbel_from_hash(splitmix_at(seed, (uint64_t)(nb + e) + 1)));
                            if (z > best) { best = z; bi = nb + e; }
                        }
                    }
                }
                if (act) {  // this (tile, half)'s maximum if it beats the earlier tiles, else -inf
                    const bool won = best > best0;
                    p.c.arg_val[(int64_t)my_row * nparts + 2 * t + half] = won ? best : -INFINITY;
                    p.c.arg_idx[(int64_t)my_row * nparts + 2 * t + half] = won ? bi : 0x7fffffff;
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.acc_empty[a]);
            if (a) ++cuse1; else ++cuse0;
            ++tseg;
        }
        named_bar_sync(1, kMegaCThreads);
        if (ctid == 0) MEGA_STAMP(1 + kPhasesPerLayer * p.layers, 0);
    }
}

// ------------------------------------------------------------------------------ kernel
__global__ void __launch_bounds__(kMegaThreads, 1) decode_step_kernel(const __grid_constant__ MegaParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t *sW = base;
    uint8_t *sQ = sW + kRingBytes;
    uint8_t *sP = sQ + 8192;
    MegaSmem &S = *reinterpret_cast<MegaSmem *>(sP + 8192);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    StepVars *V = p.c.v;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kWSlots; ++s) {
            mbar_init(&S.wfull[s], 1);
            mbar_init(&S.wempty[s], 1);
            mbar_init(&S.kvready[0][s], 1);
            mbar_init(&S.kvready[1][s], 1);
        }
        for (int s = 0; s < kMaxXStages; ++s) { mbar_init(&S.xfull[s], 1); mbar_init(&S.xempty[s], 1); }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&S.acc_full[a], 1);
            mbar_init(&S.acc_empty[a], 8);
        }
        mbar_init(&S.drain, 1);
        const int live = *(volatile int *)&V->live;
        const int rows = max(0, min(live, p.rows_cap));
        S.rows = rows;
        S.rows16 = max(16, (rows + 15) & ~15);
        // X stages: the largest power of two (at most kMaxXStages) that fits after the W slots
        {
            const int fit = min(kMaxXStages, (kRingBytes - kWSlots * kSlotBytes) / (S.rows16 * 256));
            int lg = 0;
            while ((2 << lg) <= fit) ++lg;
            S.nx = 1 << lg;
            S.nx_lg = lg;
        }
        S.n_items = *(volatile int *)&V->att_items;
        S.att_span = max(1, *(volatile int *)&V->att_span);
        S.target = (*(volatile unsigned long long *)p.epoch + 1ull) * gridDim.x;
        // failure limits of this call (sara_set_limits): read at run time, not baked into the graph
        const int64_t wl = p.c.kc->wait_ns;
        S.wait_ns = wl > 0 ? (uint64_t)wl : kWaitLimitNs;
        S.stall_idx = p.c.kc->stall_plus1 - 1;
        S.p_headroom = p.c.kc->eager_softmax ? 0.f : kSoftmaxHeadroom;
        S.abort = (*(volatile int *)&V->err & ERR_WAIT_TIMEOUT) != 0;
        S.last_flag = 0;
        fence_mbar_init();
    }
    if (threadIdx.x == 0) MEGA_STAMP(p.n_stamp_ph - kDetailRows - 1, 0);  // kernel start
    const uint64_t t_start = globaltimer_ns();
    if (warp == 1) {
        tmem_alloc(&S.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    uint8_t *sX = sW + (size_t)kWSlots * kSlotBytes;
    const bool run = !S.abort && S.rows > 0;
    if (run) {
        if (warp == 0) {
            fill_att_blocks(p, S, lane);
            if (lane == 0) mega_w_producer(p, S, sW);
        } else if (warp == 1) {
            if (lane == 0) mega_mma(p, S, sW, sX, sQ, sP, tmem);
        } else if (warp == 2) {
            if (lane == 0) mega_x_producer(p, S, sX);
        } else {
            mega_compute(p, S, sW, sQ, sP, tmem);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
    // every CTA read the epoch before any CTA could pass the first phase; the last phase's
    // wait in CTA 0 therefore happens after all reads
    if (run && threadIdx.x == 0 && blockIdx.x == 0) atomicAdd(p.epoch, 1ull);
    // launch duration for the step's kernel-time total (the bookkeeping kernel folds it in)
    if (run && threadIdx.x == 0 && p.ktime) {
        atomicMin(&p.ktime[0], (unsigned long long)t_start);
        atomicMax(&p.ktime[1], (unsigned long long)globaltimer_ns());
    }
}

// ------------------------------------------------------------------------------ layout kernels
// Row-major W [N][K] (bf16) -> blocked tiles of 256 rows (the last may have fewer): block
// (t, kc) holds rows [256 t, ..) x columns [64 kc, +64), 16-byte granule j of row r stored at
// granule j ^ (r % 8).  N must be a multiple of 128 and K of 64.
static __global__ void block_weights_kernel(const uint16_t *src, uint8_t *dst, int N, int K) {
    const int gpr = K / 8;
    const int64_t total = (int64_t)N * gpr;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int n = (int)(e / gpr), j = (int)(e - (int64_t)n * gpr);
        const int t = n / kTileN, r = n - t * kTileN;
        const uint4 v = *reinterpret_cast<const uint4 *>(src + (int64_t)n * K + (int64_t)j * 8);
        *reinterpret_cast<uint4 *>(dst + wblk_off(N, K, t, j >> 3) + (int64_t)r * 128 + (((j & 7) ^ (r & 7)) << 4)) = v;
    }
}

// KV set-up of the rollouts that join, from the prefill's row-major prompt KV ([2][n_kv][cap_p]
// [hd] per prompt slot and layer, positions < Lp - 1): (a) every fresh prompt's full blocks
// (positions < nsh * 128), which its rollouts share; (b) every new rollout's private block
// holding position Lp - 1 (slots new_slots[0 .. n_new)), filled with the prompt's tail positions
// nsh * 128 .. Lp - 2.  One thread per K granule (8 dims of a position) or V granule (8
// positions of a dim).
static __global__ void prompt_blocks_kernel(const uint16_t *pkv, uint8_t *kv, const StepPtrs c, int layers, int n_kv,
                                            int hd, int cap_p, int64_t kv_layer, int max_active) {
    pdl_wait_prior_grids();
    pdl_allow_dependents();
    const int n_new = c.v->n_new, n_fresh = c.v->n_fresh;
    const int Lp = c.kc->Lp, Lpre = Lp - 1;
    const int nsh = shared_blocks(Lp, kKVPos);
    const int gk = hd / 8;
    // per (layer, kv head) plane: K granules npos * gk, then V granules ceil(npos / 8) * hd
    const int na = nsh * kKVPos, nt = Lpre - na;  // positions of a shared plane / of a tail plane
    const int64_t per_a = (int64_t)na * gk + (int64_t)(na / 8) * hd;
    const int64_t per_b = (int64_t)nt * gk + (int64_t)((nt + 7) / 8) * hd;
    const int64_t tot_a = (int64_t)n_fresh * layers * n_kv * per_a;
    const int64_t total = tot_a + (int64_t)n_new * layers * n_kv * per_b;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        int64_t rem;
        int owner, npos, p0;  // owner: fresh prompt f or rollout slot s; positions [p0, p0 + npos)
        int64_t per;
        if (e < tot_a) {
            rem = e;
            per = per_a;
            npos = na;
            p0 = 0;
        } else {
            rem = e - tot_a;
            per = per_b;
            npos = nt;
            p0 = na;
        }
        const int64_t per_owner = (int64_t)layers * n_kv * per;
        owner = (int)(rem / per_owner);
        rem -= (int64_t)owner * per_owner;
        const int l = (int)(rem / ((int64_t)n_kv * per));
        rem -= (int64_t)l * n_kv * per;
        const int kvh = (int)(rem / per);
        rem -= (int64_t)kvh * per;
        const bool shared = e < tot_a;
        const int slot = shared ? 0 : c.new_slots[owner];
        const int ps = shared ? c.fresh_pslot[owner] : c.seq_pslot[slot];
        const uint16_t *kplane = pkv + (((int64_t)l * max_active + ps) * 2 * n_kv + kvh) * cap_p * hd;
        const uint16_t *vplane = kplane + (int64_t)n_kv * cap_p * hd;
        const int nk = npos * gk;
        int pos, dd = 0;
        bool isk = rem < nk;
        if (isk) {
            pos = p0 + (int)(rem / gk);
            dd = (int)(rem - (int64_t)(pos - p0) * gk) * 8;
        } else {
            rem -= nk;
            pos = p0 + (int)(rem / hd) * 8;
            dd = (int)(rem - (int64_t)((pos - p0) / 8) * hd);
        }
        const int b = pos / kKVPos;
        const int blk = shared ? ps * c.nsh_max + b : c.blk_tab[(int64_t)slot * c.nblk_max + b];
        uint8_t *dst = kv + l * kv_layer + ((int64_t)blk * n_kv + kvh) * kKVBlockBytes;
        if (isk) {
            const uint4 v = *reinterpret_cast<const uint4 *>(kplane + (int64_t)pos * hd + dd);
            *reinterpret_cast<uint4 *>(dst + kv_k_off(pos % kKVPos, dd)) = v;
        } else {
            uint32_t w[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int pa = pos + 2 * q;
                const uint32_t x = pa < Lpre ? vplane[(int64_t)pa * hd + dd] : 0u;
                const uint32_t y = pa + 1 < Lpre ? vplane[(int64_t)(pa + 1) * hd + dd] : 0u;
                w[q] = x | (y << 16);
            }
            *reinterpret_cast<uint4 *>(dst + kv_v_off(pos % kKVPos, dd)) = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

}  // namespace sara
