// One decode step of the policy (embedding -> every layer -> lm_head with fused Gumbel-max
// partials) as a single persistent, cooperative kernel: one CTA per SM, phases separated
// by release/acquire arrival counters in global memory instead of kernel boundaries.
//
// Why: at decode batch sizes the per-layer work is a few MB of weights per projection, so
// a kernel per projection spends most of its time starting, filling its pipeline and
// draining.  Here the weight stream never stops: the producer warp walks the whole step's
// weight tiles (and the attention phase's KV blocks, which do not depend on this step's
// activations) ahead of the consumers through an 8-slot shared-memory ring, across phase
// boundaries.  Only the small activation operands wait for the previous phase.
//
// Warp roles (352 threads, 11 warps):
//   warp 0   W producer: 16 KB bulk copies of pre-swizzled weight tiles and KV blocks
//   warp 1   tcgen05 issuer and tensor-memory owner
//   warp 2   X producer: activation chunks, after the phase they come from has completed
//   warps 3..10  compute: GEMM epilogues (fixed-point folds), attention softmax / merge,
//                residual + RMSNorm + SwiGLU finalisation, embedding, sampling partials
//
// Phases of layer l (counter index 1 + 8l + k):
//   0 QKV   x_g W_qkv^T          -> accQ (64-bit fixed point, atomic fold over k-splits)
//   1 ATT   q, k, v = RMSNorm scale + RoPE of accQ; new k, v appended to the KV cache;
//           softmax(q K^T) V on the tensor cores per 128-position split; split merge
//   2 O     att W_o^T            -> accO
//   3 FIN_O x += accO; x_g = x * g_mlp (bf16 hi/lo, blocked); per-row sum of squares
//   4 GU    x_g W_gu^T           -> accGU (gate / up interleaved in 64-row blocks)
//   5 FIN_GU h = silu(r g) * (r u), r = 1/rms(x)  (bf16 hi/lo, blocked)
//   6 DOWN  h W_down^T           -> accD
//   7 FIN_D x += accD; x_g = x * g_next; sum of squares
// then lm_head over whole 128-token tiles with the Gumbel-max partial argmax per tile.
//
// Layouts (all chosen so that one bulk copy lands an MMA operand in shared memory in the
// 128-byte-swizzled K-major form the tensor core reads):
//   weights       [N/128][K/64] blocks of 128 rows x 64 elements (16 KB), swizzled
//   activations   [K/64][rows16][64] bf16 (hi and lo planes), swizzled per 8-row atom
//   KV cache      per (layer, slot, kv head, 128-position block): K as [d/64][128 pos][64 d]
//                 and V transposed as [pos/64][128 d][64 pos], fp16, head dim padded to 128
#pragma once
#include "device_common.cuh"
#include "step_state.cuh"

namespace sara {

constexpr int kMegaThreads = 352;
constexpr int kMegaCThreads = 256;  // compute warps 3..10
constexpr int kWSlots = 8;
constexpr int kSlotBytes = 16384;
constexpr int kXRingBytes = 65536;
constexpr int kMaxXStages = 8;
constexpr int kKVPos = 128;           // positions per KV block and per attention split
constexpr int kKVBlockBytes = 65536;  // K 2 x 16 KB + V^T 2 x 16 KB
constexpr int kMegaMaxSplits = 96;
constexpr int kPhasesPerLayer = 8;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemS = 256;  // attention scores, 2 buffers x 16 columns
constexpr uint32_t kTmemO = 288;  // attention output, 2 buffers x 16 columns
constexpr float kFix = 4294967296.0f;                 // 2^32
constexpr float kUnfix = 2.3283064365386963e-10f;     // 2^-32

struct MegaParams {
    int layers, d, H, KVH, hd, F, V, Gq, nqkv;
    float eps, scale_log2;
    const uint8_t *w_qkv, *w_o, *w_gu, *w_down, *w_lm;  // blocked weights, layer strides below
    int64_t ls_qkv, ls_o, ls_gu, ls_down;
    const uint16_t *embed;                          // [V][d] bf16
    const uint16_t *attn_norm, *mlp_norm;           // [L][d]
    const uint16_t *final_norm;                     // [d]
    const float2 *rope;                             // [positions][hd/2] (cos, sin)
    uint8_t *kv;                                    // blocked KV cache
    int64_t kv_layer, kv_slot;                      // bytes
    int kv_nblk;                                    // 128-position blocks per (slot, kv head)
    StepPtrs c;
    int rows_cap, rows_cap16;
    float *x;                                       // [rows_cap][d] residual stream
    uint8_t *xg_hi, *xg_lo;                         // blocked [d/64][rows_cap16][64]
    uint8_t *att_hi, *att_lo;                       // blocked [H*hd/64][rows_cap16][64]
    uint8_t *h_hi, *h_lo;                           // blocked [F/64][rows_cap16][64]
    float *ssqA, *ssqM;                             // [d/128][rows_cap] partial sums of x^2
    unsigned long long *accQ, *accO, *accGU, *accD; // [rows_cap][N] fixed point, zero between uses
    float *part;                                    // [items][KVH][Gq][hd + 2] split partials
    int *att_cnt;                                   // [rows_cap][KVH] split arrival counters
    float *logits;                                  // optional [rows][V] fp32
    float *arg_val;                                 // [rows][V/128] partial max
    int *arg_idx;                                   //   and its token
    unsigned long long *cnt;                        // phase arrival counters (monotonic)
    unsigned long long *epoch;                      // launches completed since the reset
};

struct MegaSmem {
    uint64_t wfull[kWSlots], wempty[kWSlots];
    uint64_t xfull[kMaxXStages], xempty[kMaxXStages];
    uint64_t acc_full[2], acc_empty[2];
    uint64_t q_ready[2], s_full[2], p_ready[2], o_full[2];
    uint64_t drain;
    unsigned long long target;  // counter value meaning "every CTA of this launch arrived"
    uint32_t tmem_base;
    int abort;
    int last_flag;
    int rows, rows16, nx, n_items;
    float rstd[128];
    unsigned long long seed[128];
    float att_m[2][8], att_l[2][8];
    float red[4][8];
    float mw[8][kMegaMaxSplits];
    float ml[8];
    float lm_v[2][4][32];
    int lm_i[2][4][32];
};

constexpr size_t kMegaSmemBytes =
    1024 + (size_t)kWSlots * kSlotBytes + kXRingBytes + 4 * 4096 + sizeof(MegaSmem);

// ------------------------------------------------------------------------------ layouts
// Byte offset of element (r, k) of a blocked activation plane with rows16 rows per chunk.
__host__ __device__ __forceinline__ int64_t xblk_off(int r, int k, int rows16) {
    const int chunk = k >> 6, col = k & 63;
    return ((int64_t)chunk * rows16 + r) * 128 + ((((col >> 3) ^ (r & 7)) << 4) | ((col & 7) << 1));
}
// Byte offsets of K(pp, d) and V(pp, d) inside one 128-position KV block.
__host__ __device__ __forceinline__ int kv_k_off(int pp, int d) {
    return (d >> 6) * 16384 + pp * 128 + (((((d & 63) >> 3) ^ (pp & 7)) << 4) | ((d & 7) << 1));
}
__host__ __device__ __forceinline__ int kv_v_off(int pp, int d) {
    const int c = pp & 63;
    return 32768 + (pp >> 6) * 16384 + d * 128 + ((((c >> 3) ^ (d & 7)) << 4) | ((c & 7) << 1));
}

// ------------------------------------------------------------------------------ waits
// Bounded mbarrier wait that also gives up (returning false) once the CTA is aborting.
__device__ __forceinline__ bool mwait(uint64_t *bar, uint32_t parity, int *err, volatile int *abort) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 63u) == 0) {
            if (*abort) return false;
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                report_error(err, ERR_WAIT_TIMEOUT);
                *abort = 1;
                return false;
            }
        }
    }
}

// Spin until a phase counter reaches `target` (acquire); bounded, gives up on abort or once
// another CTA reported a timeout.
__device__ __forceinline__ bool spin_counter(const unsigned long long *cnt, unsigned long long target, int *err,
                                             volatile int *abort) {
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
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                report_error(err, ERR_WAIT_TIMEOUT);
                *abort = 1;
                return false;
            }
        }
    }
}

// ------------------------------------------------------------------------------ phases
struct GemmPh {
    const uint8_t *w;
    int m_tiles, kch;
    const uint8_t *xhi, *xlo;
    unsigned long long *acc;
    int ld;
};

// GEMM phase k (0 QKV, 2 O, 4 GU, 6 DOWN) of layer l; l == layers: lm_head.
__device__ __forceinline__ GemmPh gemm_phase(const MegaParams &p, int l, int k) {
    GemmPh g;
    if (l == p.layers) {
        g.w = p.w_lm; g.m_tiles = p.V / 128; g.kch = p.d / 64; g.xhi = p.xg_hi; g.xlo = p.xg_lo; g.acc = nullptr;
        g.ld = p.V;
        return g;
    }
    switch (k) {
        case 0:
            g.w = p.w_qkv + l * p.ls_qkv; g.m_tiles = p.nqkv / 128; g.kch = p.d / 64;
            g.xhi = p.xg_hi; g.xlo = p.xg_lo; g.acc = p.accQ; g.ld = p.nqkv;
            break;
        case 2:
            g.w = p.w_o + l * p.ls_o; g.m_tiles = p.d / 128; g.kch = p.H * p.hd / 64;
            g.xhi = p.att_hi; g.xlo = p.att_lo; g.acc = p.accO; g.ld = p.d;
            break;
        case 4:
            g.w = p.w_gu + l * p.ls_gu; g.m_tiles = 2 * p.F / 128; g.kch = p.d / 64;
            g.xhi = p.xg_hi; g.xlo = p.xg_lo; g.acc = p.accGU; g.ld = 2 * p.F;
            break;
        default:
            g.w = p.w_down + l * p.ls_down; g.m_tiles = p.d / 128; g.kch = p.F / 64;
            g.xhi = p.h_hi; g.xlo = p.h_lo; g.acc = p.accD; g.ld = p.d;
            break;
    }
    return g;
}

// This CTA's (tile, k-chunk) units: an equal share of the whole GEMM, or (lm_head) of
// whole tiles so that every tile's argmax is finished by one CTA.
__device__ __forceinline__ void gemm_range(const GemmPh &g, bool whole, int64_t &u0, int64_t &u1) {
    const int G = gridDim.x, c = blockIdx.x;
    if (whole) {
        u0 = (int64_t)c * g.m_tiles / G * g.kch;
        u1 = (int64_t)(c + 1) * g.m_tiles / G * g.kch;
    } else {
        const int64_t U = (int64_t)g.m_tiles * g.kch;
        u0 = (int64_t)c * U / G;
        u1 = (int64_t)(c + 1) * U / G;
    }
}

struct AttUnit {
    int item, kvh, row, sp, ctx, p0, n, nsplit, slot;
    bool last;
};
__device__ __forceinline__ AttUnit att_unit(const MegaParams &p, int64_t a) {
    AttUnit u;
    u.item = (int)(a / p.KVH);
    u.kvh = (int)(a - (int64_t)u.item * p.KVH);
    const int2 it = p.c.att_items[u.item];
    u.row = it.x;
    u.sp = it.y;
    u.ctx = p.c.row_pos[u.row] + 1;
    u.p0 = u.sp * kKVPos;
    u.n = min(u.ctx - u.p0, kKVPos);
    u.nsplit = (u.ctx + kKVPos - 1) / kKVPos;
    u.last = u.p0 + u.n == u.ctx;
    u.slot = p.c.row_slot[u.row];
    return u;
}
__device__ __forceinline__ void att_range(const MegaParams &p, int n_items, int64_t &a0, int64_t &a1) {
    const int64_t NU = (int64_t)n_items * p.KVH;
    a0 = (int64_t)blockIdx.x * NU / gridDim.x;
    a1 = (int64_t)(blockIdx.x + 1) * NU / gridDim.x;
}
__device__ __forceinline__ uint8_t *kv_block(const MegaParams &p, int l, const AttUnit &u) {
    return p.kv + l * p.kv_layer + (int64_t)u.slot * p.kv_slot + ((int64_t)u.kvh * p.kv_nblk + u.sp) * kKVBlockBytes;
}
// Bytes of the four ring slots of one attention unit: K (d < 64), K (d >= 64), V^T (positions
// < 64), V^T (positions >= 64).  Zero = slot not needed (arrive without data).
__device__ __forceinline__ uint32_t att_slot_bytes(const MegaParams &p, const AttUnit &u, int q) {
    if (q < 2) return (q * 64 < p.hd) ? (uint32_t)(((u.n + 7) & ~7) * 128) : 0u;
    return (q == 2 || u.n > 64) ? (uint32_t)(p.hd * 128) : 0u;
}

// ------------------------------------------------------------------------------ W producer
__device__ __forceinline__ void mega_w_producer(const MegaParams &p, MegaSmem &S, uint8_t *sW) {
    volatile int *ab = &S.abort;
    int *err = &p.c.v->err;
    const uint64_t pol = l2_policy_evict_first();
    uint32_t wi = 0;
    bool ok = true;
    auto slot = [&](uint32_t i) -> int { return (int)(i % kWSlots); };
    auto acquire = [&](uint32_t i) -> bool {
        return i < kWSlots || mwait(&S.wempty[slot(i)], ((i / kWSlots) & 1) ^ 1, err, ab);
    };
    auto gemm = [&](const GemmPh &g, int64_t u0, int64_t u1) {
        for (int64_t u = u0; u < u1 && ok; ++u, ++wi) {
            if (!acquire(wi)) { ok = false; break; }
            const int s = slot(wi);
            mbar_arrive_expect_tx(&S.wfull[s], kSlotBytes);
            bulk_load(sW + (size_t)s * kSlotBytes, g.w + u * kSlotBytes, kSlotBytes, &S.wfull[s], pol);
        }
    };
    for (int l = 0; l <= p.layers && ok; ++l) {
        for (int k = 0; k < kPhasesPerLayer && ok; k += 2) {
            if (l == p.layers && k > 0) break;
            const GemmPh g = gemm_phase(p, l, k);
            int64_t u0, u1;
            gemm_range(g, l == p.layers, u0, u1);
            gemm(g, u0, u1);
            if (k == 0 && l < p.layers) {
                // the attention phase's KV blocks follow the QKV weights in ring order
                int64_t a0, a1;
                att_range(p, S.n_items, a0, a1);
                for (int64_t a = a0; a < a1 && ok; ++a) {
                    const AttUnit u = att_unit(p, a);
                    const uint8_t *blk = kv_block(p, l, u);
                    for (int q = 0; q < 4; ++q, ++wi) {
                        if (!acquire(wi)) { ok = false; break; }
                        const int s = slot(wi);
                        const uint32_t bytes = att_slot_bytes(p, u, q);
                        if (bytes) {
                            mbar_arrive_expect_tx(&S.wfull[s], bytes);
                            bulk_load(sW + (size_t)s * kSlotBytes, blk + q * 16384, bytes, &S.wfull[s], pol);
                        } else {
                            mbar_arrive(&S.wfull[s]);
                        }
                    }
                }
            }
        }
    }
    if (!ok) {  // every copy already issued lands before the CTA exits
        for (uint32_t s = 0; s < kWSlots && s < wi; ++s) {
            const uint32_t last = ((wi - 1 - s) / kWSlots) * kWSlots + s;
            mbar_wait(&S.wfull[s], (last / kWSlots) & 1, err);
        }
    }
}

// ------------------------------------------------------------------------------ X producer
__device__ __forceinline__ void mega_x_producer(const MegaParams &p, MegaSmem &S, uint8_t *sX) {
    volatile int *ab = &S.abort;
    int *err = &p.c.v->err;
    const uint64_t pol = l2_policy_evict_last();
    const int NX = S.nx, R16 = S.rows16;
    const uint32_t plane = (uint32_t)R16 * 128, stage = 2 * plane;
    const int64_t chunk_stride = (int64_t)p.rows_cap16 * 128;
    uint32_t xi = 0;
    bool ok = true;
    for (int l = 0; l <= p.layers && ok; ++l) {
        for (int k = 0; k < kPhasesPerLayer && ok; k += 2) {
            if (l == p.layers && k > 0) break;
            const GemmPh g = gemm_phase(p, l, k);
            int64_t u0, u1;
            gemm_range(g, l == p.layers, u0, u1);
            if (u0 >= u1) continue;
            // the phase this operand comes from: FIN_D of l-1 / embedding, ATT, FIN_O, FIN_GU
            const int dep = (l == p.layers) ? kPhasesPerLayer * l : (k == 0 ? kPhasesPerLayer * l : 1 + 8 * l + k - 1);
            if (!spin_counter(&p.cnt[dep], S.target, err, ab)) { ok = false; break; }
            fence_proxy_async_global();
            for (int64_t u = u0; u < u1; ++u, ++xi) {
                const int s = (int)(xi % NX);
                if (xi >= (uint32_t)NX && !mwait(&S.xempty[s], ((xi / NX) & 1) ^ 1, err, ab)) { ok = false; break; }
                const int kc = (int)(u % g.kch);
                mbar_arrive_expect_tx(&S.xfull[s], stage);
                uint8_t *dst = sX + (size_t)s * stage;
                bulk_load(dst, g.xhi + kc * chunk_stride, plane, &S.xfull[s], pol);
                bulk_load(dst + plane, g.xlo + kc * chunk_stride, plane, &S.xfull[s], pol);
            }
        }
    }
    if (!ok) {
        for (uint32_t s = 0; s < (uint32_t)NX && s < xi; ++s) {
            const uint32_t last = ((xi - 1 - s) / NX) * NX + s;
            mbar_wait(&S.xfull[s], (last / NX) & 1, err);
        }
    }
}

// ------------------------------------------------------------------------------ MMA issuer
__device__ __forceinline__ void mega_mma(const MegaParams &p, MegaSmem &S, uint8_t *sW, uint8_t *sX, uint8_t *sQ,
                                         uint8_t *sP, uint32_t tmem) {
    volatile int *ab = &S.abort;
    int *err = &p.c.v->err;
    const int NX = S.nx, R16 = S.rows16;
    const uint32_t plane = (uint32_t)R16 * 128, stage = 2 * plane;
    const uint32_t idg = idesc_bf16_f32(128, (uint32_t)R16);
    const uint32_t ida = idesc_f16_f32(128, 16);
    uint32_t wi = 0, xi = 0;
    int seg = 0, gi = 0;
    bool ok = true;
    auto wslot = [&](uint32_t i) -> uint32_t { return smem_u32(sW + (size_t)(i % kWSlots) * kSlotBytes); };
    auto wwait = [&](uint32_t i) -> bool { return mwait(&S.wfull[i % kWSlots], (i / kWSlots) & 1, err, ab); };
    auto gemm = [&](const GemmPh &g, int64_t u0, int64_t u1) {
        for (int64_t u = u0; u < u1 && ok;) {
            const int tile = (int)(u / g.kch);
            const int64_t e = min(u1, (int64_t)(tile + 1) * g.kch);
            const int a = seg & 1;
            if (seg >= 2 && !mwait(&S.acc_empty[a], ((seg >> 1) - 1) & 1, err, ab)) { ok = false; break; }
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(a * 128);
            bool first = true;
            for (; u < e; ++u, ++wi, ++xi) {
                const int xs = (int)(xi % NX);
                if (!wwait(wi) || !mwait(&S.xfull[xs], (xi / NX) & 1, err, ab)) { ok = false; break; }
                tc_fence_after();
                const uint32_t aw = wslot(wi), ax = smem_u32(sX + (size_t)xs * stage);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t ad = sdesc_kmajor_sw128(aw + kk * 32);
                    tc_mma_bf16(d, ad, sdesc_kmajor_sw128(ax + kk * 32), idg, (first && kk == 0) ? 0u : 1u);
                    tc_mma_bf16(d, ad, sdesc_kmajor_sw128(ax + plane + kk * 32), idg, 1u);
                }
                first = false;
                tc_commit(&S.wempty[wi % kWSlots]);
                tc_commit(&S.xempty[xs]);
            }
            if (!ok) break;
            tc_commit(&S.acc_full[a]);
            ++seg;
        }
    };
    auto att = [&](int64_t a0, int64_t a1) {
        const int n = (int)(a1 - a0);
        const uint32_t wb = wi;
        for (int i = 0; i <= n && ok; ++i) {
            if (i < n) {  // scores S = K q^T of unit i
                const int g = gi + i, b = g & 1;
                const uint32_t w0 = wb + 4 * i;
                if (!mwait(&S.q_ready[b], (g >> 1) & 1, err, ab) || !wwait(w0) || !wwait(w0 + 1)) { ok = false; break; }
                tc_fence_after();
                const uint32_t dS = tmem + kTmemS + 16 * b, qb = smem_u32(sQ + 4096 * b);
                for (int ks = 0; ks < p.hd / 16; ++ks)
                    tc_mma_bf16(dS, sdesc_kmajor_sw128(wslot(w0 + (ks >> 2)) + (ks & 3) * 32),
                                sdesc_kmajor_sw128(qb + (ks >> 2) * 2048 + (ks & 3) * 32), ida, ks > 0 ? 1u : 0u);
                tc_commit(&S.s_full[b]);
                tc_commit(&S.wempty[w0 % kWSlots]);
                tc_commit(&S.wempty[(w0 + 1) % kWSlots]);
            }
            if (i >= 1) {  // output O^T = V^T P^T of unit i - 1
                const int g = gi + i - 1, b = g & 1;
                const uint32_t w0 = wb + 4 * (i - 1);
                const AttUnit u = att_unit(p, a0 + i - 1);
                if (!mwait(&S.p_ready[b], (g >> 1) & 1, err, ab) || !wwait(w0 + 2) || !wwait(w0 + 3)) { ok = false; break; }
                tc_fence_after();
                const uint32_t dO = tmem + kTmemO + 16 * b, pb = smem_u32(sP + 4096 * b);
                const int ksteps = (u.n + 15) >> 4;
                for (int ks = 0; ks < ksteps; ++ks)
                    tc_mma_bf16(dO, sdesc_kmajor_sw128(wslot(w0 + 2 + (ks >> 2)) + (ks & 3) * 32),
                                sdesc_kmajor_sw128(pb + (ks >> 2) * 2048 + (ks & 3) * 32), ida, ks > 0 ? 1u : 0u);
                tc_commit(&S.o_full[b]);
                tc_commit(&S.wempty[(w0 + 2) % kWSlots]);
                tc_commit(&S.wempty[(w0 + 3) % kWSlots]);
            }
        }
        wi = wb + 4 * n;
        gi += n;
    };
    for (int l = 0; l <= p.layers && ok; ++l) {
        for (int k = 0; k < kPhasesPerLayer && ok; k += 2) {
            if (l == p.layers && k > 0) break;
            const GemmPh g = gemm_phase(p, l, k);
            int64_t u0, u1;
            gemm_range(g, l == p.layers, u0, u1);
            gemm(g, u0, u1);
            if (k == 0 && l < p.layers && ok) {
                int64_t a0, a1;
                att_range(p, S.n_items, a0, a1);
                att(a0, a1);
            }
        }
    }
    // every MMA issued has retired before tensor memory is released
    tc_commit(&S.drain);
    mbar_wait(&S.drain, 0, err);
}

// ------------------------------------------------------------------------------ compute
__device__ __forceinline__ void store_hilo(uint8_t *hi, uint8_t *lo, int64_t off, float v) {
    uint16_t h, l;
    split_bf16(v, h, l);
    *reinterpret_cast<uint16_t *>(hi + off) = h;
    *reinterpret_cast<uint16_t *>(lo + off) = l;
}

__device__ __forceinline__ float unfix(unsigned long long v) { return (float)(long long)v * kUnfix; }

// 8 consecutive head dims (granule j) of one head of accQ, RMSNorm-scaled by `scale`, with
// the rotary embedding (pairs i, i + hd/2) when `rot`.
__device__ __forceinline__ void head_granule(const unsigned long long *src, int j, int hd, const float2 *cs, bool rot,
                                             float scale, float (&y)[8]) {
    const int d0 = j * 8, half = hd >> 1;
    const ulonglong2 *a = reinterpret_cast<const ulonglong2 *>(src + d0);
    float x[8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const ulonglong2 t = __ldcg(a + e);
        x[2 * e] = unfix(t.x);
        x[2 * e + 1] = unfix(t.y);
    }
    if (!rot) {
#pragma unroll
        for (int e = 0; e < 8; ++e) y[e] = x[e] * scale;
        return;
    }
    const bool low = d0 < half;
    const int pd0 = low ? d0 + half : d0 - half;
    const ulonglong2 *b = reinterpret_cast<const ulonglong2 *>(src + pd0);
    float xp[8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const ulonglong2 t = __ldcg(b + e);
        xp[2 * e] = unfix(t.x);
        xp[2 * e + 1] = unfix(t.y);
    }
    const int f0 = low ? d0 : pd0;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float2 r = __ldg(&cs[f0 + e]);
        y[e] = (low ? (x[e] * r.x - xp[e] * r.y) : (x[e] * r.x + xp[e] * r.y)) * scale;
    }
}

__device__ __forceinline__ uint4 pack_f16x8(const float (&y)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e)
        w[e] = (uint32_t)f32_to_f16_sat(y[2 * e]) | ((uint32_t)f32_to_f16_sat(y[2 * e + 1]) << 16);
    return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ void argmax_combine(float &v, int &i, float ov, int oi) {
    if (ov > v || (ov == v && oi < i)) { v = ov; i = oi; }
}

__device__ __forceinline__ void mega_compute(const MegaParams &p, MegaSmem &S, uint8_t *sW, uint8_t *sQ, uint8_t *sP,
                                             uint32_t tmem) {
    volatile int *ab = &S.abort;
    int *err = &p.c.v->err;
    const int ctid = threadIdx.x - 96;  // 0..255
    const int cw = ctid >> 5, lane = threadIdx.x & 31;
    const int quarter = (threadIdx.x >> 5) & 3;  // tensor-memory lanes 32*quarter ..
    const int half = cw >> 2;                    // warps 3..6 -> 0, 7..10 -> 1
    const int G = gridDim.x, cta = blockIdx.x;
    const int R = S.rows, R16c = p.rows_cap16;
    const int d = p.d, dt = d / 128, hd = p.hd, Gq = p.Gq;
    const int gw = cta * 8 + cw, nw = G * 8;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    uint32_t wi = 0;
    int seg = 0, gi = 0;

    auto arrive = [&](int idx) {
        fence_proxy_async_global();
        __threadfence();
        named_bar_sync(1, kMegaCThreads);
        if (ctid == 0) {
            __threadfence();
            atomicAdd(&p.cnt[idx], 1ull);
        }
    };
    auto wait_phase = [&](int idx) {
        if (ctid == 0) spin_counter(&p.cnt[idx], S.target, err, ab);
        named_bar_sync(1, kMegaCThreads);
    };
    auto load_rstd = [&](const float *ssq) {
        if (ctid < R) {
            float s = 0.f;
            for (int t = 0; t < dt; ++t) s += __ldcg(&ssq[(int64_t)t * p.rows_cap + ctid]);
            S.rstd[ctid] = rsqrtf(s / (float)d + p.eps);
        }
        named_bar_sync(1, kMegaCThreads);
    };
    // fixed-point fold of this CTA's partial tile sums (every k-split adds into acc)
    auto gemm_epi = [&](const GemmPh &g, int64_t u0, int64_t u1) {
        for (int64_t u = u0; u < u1;) {
            const int tile = (int)(u / g.kch);
            u = min(u1, (int64_t)(tile + 1) * g.kch);
            const int a = seg & 1;
            mwait(&S.acc_full[a], (seg >> 1) & 1, err, ab);
            tc_fence_after();
            const int n = tile * 128 + quarter * 32 + lane;
            for (int cc = half; cc * 32 < R; cc += 2) {
                float v[32];
                tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(a * 128 + cc * 32), v);
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const int r = cc * 32 + j;
                    if (r < R) atomicAdd(&g.acc[(int64_t)r * g.ld + n], (unsigned long long)__float2ll_rn(v[j] * kFix));
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.acc_empty[a]);
            ++seg;
        }
    };
    // x += acc; x_g = x * gw (blocked hi/lo); per (row, 128-feature block) sum of squares
    auto fin_resid = [&](unsigned long long *acc, const uint16_t *gn, float *ssq) {
        for (int u = gw; u < R * dt; u += nw) {
            const int r = u / dt, t = u - r * dt;
            const int f = t * 128 + lane * 4;
            float4 x = __ldcg(reinterpret_cast<const float4 *>(p.x + (int64_t)r * d + f));
            if (acc) {
                ulonglong2 *ap = reinterpret_cast<ulonglong2 *>(acc + (int64_t)r * d + f);
                const ulonglong2 a0 = __ldcg(ap), a1 = __ldcg(ap + 1);
                x.x += unfix(a0.x); x.y += unfix(a0.y); x.z += unfix(a1.x); x.w += unfix(a1.y);
                ap[0] = make_ulonglong2(0ull, 0ull);
                ap[1] = make_ulonglong2(0ull, 0ull);
                *reinterpret_cast<float4 *>(p.x + (int64_t)r * d + f) = x;
            }
            const uint2 gb = *reinterpret_cast<const uint2 *>(gn + f);
            const float g0 = bf16_to_f32(gb.x & 0xffff), g1 = bf16_to_f32(gb.x >> 16);
            const float g2 = bf16_to_f32(gb.y & 0xffff), g3 = bf16_to_f32(gb.y >> 16);
            uint16_t h[4], lo[4];
            split_bf16(x.x * g0, h[0], lo[0]);
            split_bf16(x.y * g1, h[1], lo[1]);
            split_bf16(x.z * g2, h[2], lo[2]);
            split_bf16(x.w * g3, h[3], lo[3]);
            const int64_t off = xblk_off(r, f, R16c);
            *reinterpret_cast<uint2 *>(p.xg_hi + off) =
                make_uint2((uint32_t)h[0] | ((uint32_t)h[1] << 16), (uint32_t)h[2] | ((uint32_t)h[3] << 16));
            *reinterpret_cast<uint2 *>(p.xg_lo + off) =
                make_uint2((uint32_t)lo[0] | ((uint32_t)lo[1] << 16), (uint32_t)lo[2] | ((uint32_t)lo[3] << 16));
            const float s = warp_sum(x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w);
            if (lane == 0) ssq[(int64_t)t * p.rows_cap + r] = s;
        }
    };

    // ---------------------------------------------------------------- embedding
    for (int u = gw; u < R * dt; u += nw) {
        const int r = u / dt, t = u - r * dt;
        int tok = p.c.row_tok[r];
        if (tok < 0 || tok >= p.V) {
            if (lane == 0) report_error(err, ERR_BOUNDS);
            tok = 0;
        }
        const int f = t * 128 + lane * 4;
        const uint2 e = *reinterpret_cast<const uint2 *>(p.embed + (int64_t)tok * d + f);
        const float4 x = make_float4(bf16_to_f32(e.x & 0xffff), bf16_to_f32(e.x >> 16), bf16_to_f32(e.y & 0xffff),
                                     bf16_to_f32(e.y >> 16));
        *reinterpret_cast<float4 *>(p.x + (int64_t)r * d + f) = x;
    }
    __syncwarp();
    fin_resid(nullptr, p.attn_norm, p.ssqA);
    arrive(0);

    for (int l = 0; l < p.layers; ++l) {
        const int base = 1 + kPhasesPerLayer * l;
        int64_t u0, u1;
        // ------------------------------------------------------------ QKV
        {
            const GemmPh g = gemm_phase(p, l, 0);
            gemm_range(g, false, u0, u1);
            gemm_epi(g, u0, u1);
            wi += (uint32_t)(u1 - u0);
            arrive(base + 0);
        }
        // ------------------------------------------------------------ attention
        {
            wait_phase(base + 0);
            load_rstd(p.ssqA);
            int64_t a0, a1;
            att_range(p, S.n_items, a0, a1);
            const int n = (int)(a1 - a0);
            const uint32_t wb = wi;
            const float2 *rope = p.rope;
            // warps 3..6 run the attention units; warps 7..10 wait at the phase arrival
            for (int i = 0; half == 0 && i < n + 2; ++i) {
                if (i < n) {  // q tile of unit i (+ the new position's k, v on the last split)
                    const AttUnit u = att_unit(p, a0 + i);
                    const int b = (gi + i) & 1;
                    const float rs = S.rstd[u.row];
                    const float2 *cs = rope + (int64_t)(u.ctx - 1) * (hd / 2);
                    const int g = ctid >> 4, j = ctid & 15;  // rows 0..7 (score columns 8..15 unused)
                    uint4 pk = make_uint4(0, 0, 0, 0);
                    if (g < Gq && j * 8 < hd) {
                        float y[8];
                        head_granule(p.accQ + (int64_t)u.row * p.nqkv + (u.kvh * Gq + g) * hd, j, hd, cs, true,
                                     rs * p.scale_log2, y);
                        pk = pack_f16x8(y);
                    }
                    *reinterpret_cast<uint4 *>(sQ + 4096 * b + (j >> 3) * 2048 + g * 128 + (((j & 7) ^ (g & 7)) << 4)) = pk;
                    if (u.last && ctid < 32) {
                        const int jj = ctid & 15;
                        const bool isv = ctid >= 16;
                        if (jj * 8 < hd) {
                            const uint32_t w0 = wb + 4 * i;
                            const int pp = u.ctx - 1 - u.p0;
                            const int head = p.H + (isv ? p.KVH : 0) + u.kvh;
                            float y[8];
                            head_granule(p.accQ + (int64_t)u.row * p.nqkv + head * hd, jj, hd, cs, !isv, rs, y);
                            uint8_t *gblk = kv_block(p, l, u);
                            if (!isv) {
                                const uint4 kp = pack_f16x8(y);
                                const int off = kv_k_off(pp, jj * 8);
                                *reinterpret_cast<uint4 *>(gblk + off) = kp;
                                const uint32_t ws = w0 + (jj >> 3);
                                mwait(&S.wfull[ws % kWSlots], (ws / kWSlots) & 1, err, ab);
                                *reinterpret_cast<uint4 *>(sW + (size_t)(ws % kWSlots) * kSlotBytes + (off & 16383)) = kp;
                            } else {
                                const uint32_t ws = w0 + 2 + (pp >> 6);
                                mwait(&S.wfull[ws % kWSlots], (ws / kWSlots) & 1, err, ab);
                                uint8_t *sv = sW + (size_t)(ws % kWSlots) * kSlotBytes;
#pragma unroll
                                for (int e = 0; e < 8; ++e) {
                                    const uint16_t hv = f32_to_f16_sat(y[e]);
                                    const int off = kv_v_off(pp, jj * 8 + e);
                                    *reinterpret_cast<uint16_t *>(gblk + off) = hv;
                                    *reinterpret_cast<uint16_t *>(sv + (off & 16383)) = hv;
                                }
                            }
                        }
                    }
                    fence_proxy_async_smem();
                    named_bar_sync(2, 128);
                    if (ctid == 0) mbar_arrive(&S.q_ready[b]);
                }
                if (i >= 1 && i <= n) {  // softmax of unit i - 1 -> P
                    const AttUnit u = att_unit(p, a0 + i - 1);
                    const int g1 = gi + i - 1, b = g1 & 1;
                    mwait(&S.s_full[b], (g1 >> 1) & 1, err, ab);
                    tc_fence_after();
                    float sv[8];
                    tmem_ld_32x32b_x8(tmem + lane_base + kTmemS + 16 * b, sv);
                    const int pos = quarter * 32 + lane;
                    const bool valid = pos < u.n;
                    float M[8];
#pragma unroll
                    for (int g = 0; g < 8; ++g) {
                        sv[g] = valid ? sv[g] : -INFINITY;
                        float m = sv[g];
#pragma unroll
                        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
                        if (lane == 0) S.red[quarter][g] = m;
                    }
                    named_bar_sync(2, 128);
#pragma unroll
                    for (int g = 0; g < 8; ++g)
                        M[g] = fmaxf(fmaxf(S.red[0][g], S.red[1][g]), fmaxf(S.red[2][g], S.red[3][g]));
                    named_bar_sync(2, 128);
                    uint8_t *pb = sP + 4096 * b + (pos >> 6) * 2048;
                    const int pc = pos & 63;
#pragma unroll
                    for (int g = 0; g < 8; ++g) {
                        const float e = valid ? exp2f(sv[g] - M[g]) : 0.f;
                        *reinterpret_cast<uint16_t *>(pb + g * 128 + ((((pc >> 3) ^ (g & 7)) << 4) | ((pc & 7) << 1))) =
                            f32_to_f16_sat(e);
                        const float s = warp_sum(e);
                        if (lane == 0) S.red[quarter][g] = s;
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    named_bar_sync(2, 128);
                    if (ctid < 8) {
                        float mc = M[0];
#pragma unroll
                        for (int g = 1; g < 8; ++g) mc = (ctid == g) ? M[g] : mc;
                        S.att_m[b][ctid] = mc;
                        S.att_l[b][ctid] = S.red[0][ctid] + S.red[1][ctid] + S.red[2][ctid] + S.red[3][ctid];
                    }
                    named_bar_sync(2, 128);
                    if (ctid == 0) mbar_arrive(&S.p_ready[b]);
                }
                if (i >= 2) {  // output of unit i - 2
                    const AttUnit u = att_unit(p, a0 + i - 2);
                    const int g2 = gi + i - 2, b = g2 & 1;
                    mwait(&S.o_full[b], (g2 >> 1) & 1, err, ab);
                    tc_fence_after();
                    float ov[8];
                    tmem_ld_32x32b_x8(tmem + lane_base + kTmemO + 16 * b, ov);
                    tc_fence_before();
                    const int dd = quarter * 32 + lane;
                    if (u.nsplit == 1) {
                        if (dd < hd) {
#pragma unroll
                            for (int g = 0; g < 8; ++g)
                                if (g < Gq)
                                    store_hilo(p.att_hi, p.att_lo, xblk_off(u.row, (u.kvh * Gq + g) * hd + dd, R16c),
                                               ov[g] / S.att_l[b][g]);
                        }
                    } else {
                        float *mine = p.part + ((int64_t)u.item * p.KVH + u.kvh) * Gq * (hd + 2);
                        if (dd < hd) {
#pragma unroll
                            for (int g = 0; g < 8; ++g)
                                if (g < Gq) mine[g * (hd + 2) + 2 + dd] = ov[g];
                        }
                        if (ctid < Gq) {
                            mine[ctid * (hd + 2)] = S.att_m[b][ctid];
                            mine[ctid * (hd + 2) + 1] = S.att_l[b][ctid];
                        }
                        __threadfence();
                        named_bar_sync(2, 128);
                        if (ctid == 0) {
                            const int old = atomicAdd(&p.att_cnt[u.row * p.KVH + u.kvh], 1);
                            S.last_flag = old == u.nsplit - 1;
                            if (S.last_flag) p.att_cnt[u.row * p.KVH + u.kvh] = 0;
                        }
                        named_bar_sync(2, 128);
                        if (S.last_flag) {  // merge the row's splits in split order
                            __threadfence();
                            const int ns = min(u.nsplit, kMegaMaxSplits);
                            const int64_t sp_stride = (int64_t)p.KVH * Gq * (hd + 2);
                            const float *pbase = p.part + ((int64_t)p.c.row_item0[u.row] * p.KVH + u.kvh) * Gq * (hd + 2);
                            for (int g = cw; g < Gq; g += 4) {
                                float Mx = -INFINITY;
                                for (int s = lane; s < ns; s += 32) Mx = fmaxf(Mx, __ldcg(pbase + s * sp_stride + g * (hd + 2)));
#pragma unroll
                                for (int o = 16; o > 0; o >>= 1) Mx = fmaxf(Mx, __shfl_xor_sync(0xffffffffu, Mx, o));
                                float L = 0.f;
                                for (int s = lane; s < ns; s += 32) {
                                    const float ms = __ldcg(pbase + s * sp_stride + g * (hd + 2));
                                    const float w = exp2f(ms - Mx);
                                    S.mw[g][s] = w;
                                    L += w * __ldcg(pbase + s * sp_stride + g * (hd + 2) + 1);
                                }
                                L = warp_sum(L);
                                if (lane == 0) S.ml[g] = L;
                            }
                            named_bar_sync(2, 128);
                            for (int e = ctid; e < Gq * hd; e += 128) {
                                const int g = e / hd, de = e - g * hd;
                                const float *src = pbase + g * (hd + 2) + 2 + de;
                                float acc = 0.f;
#pragma unroll 4
                                for (int s = 0; s < ns; ++s) acc += S.mw[g][s] * __ldcg(src + s * sp_stride);
                                store_hilo(p.att_hi, p.att_lo, xblk_off(u.row, (u.kvh * Gq + g) * hd + de, R16c),
                                           acc / S.ml[g]);
                            }
                        }
                        named_bar_sync(2, 128);
                    }
                }
            }
            wi = wb + 4 * n;
            gi += n;
            arrive(base + 1);
        }
        // ------------------------------------------------------------ O projection
        {
            const GemmPh g = gemm_phase(p, l, 2);
            gemm_range(g, false, u0, u1);
            gemm_epi(g, u0, u1);
            wi += (uint32_t)(u1 - u0);
            arrive(base + 2);
        }
        // ------------------------------------------------------------ residual, MLP norm input
        {
            wait_phase(base + 2);
            fin_resid(p.accO, p.mlp_norm + (int64_t)l * d, p.ssqM);
            // accQ is no longer read by anyone: clear the live rows for the next layer
            const int64_t nz = (int64_t)R * p.nqkv / 2;
            ulonglong2 *q2 = reinterpret_cast<ulonglong2 *>(p.accQ);
            for (int64_t e = (int64_t)cta * kMegaCThreads + ctid; e < nz; e += (int64_t)G * kMegaCThreads)
                q2[e] = make_ulonglong2(0ull, 0ull);
            arrive(base + 3);
        }
        // ------------------------------------------------------------ gate / up
        {
            const GemmPh g = gemm_phase(p, l, 4);
            gemm_range(g, false, u0, u1);
            gemm_epi(g, u0, u1);
            wi += (uint32_t)(u1 - u0);
            arrive(base + 4);
        }
        // ------------------------------------------------------------ SwiGLU
        {
            wait_phase(base + 4);
            load_rstd(p.ssqM);
            const int fb = p.F / 64;
            for (int u = gw; u < R * fb; u += nw) {
                const int r = u / fb, jb = u - r * fb;
                const float rs = S.rstd[r];
                unsigned long long *gp = p.accGU + (int64_t)r * 2 * p.F + jb * 128 + 2 * lane;
                ulonglong2 *g2 = reinterpret_cast<ulonglong2 *>(gp);
                ulonglong2 *u2 = reinterpret_cast<ulonglong2 *>(gp + 64);
                const ulonglong2 ga = __ldcg(g2), ua = __ldcg(u2);
                *g2 = make_ulonglong2(0ull, 0ull);
                *u2 = make_ulonglong2(0ull, 0ull);
                const float gv0 = unfix(ga.x) * rs, gv1 = unfix(ga.y) * rs;
                const float uv0 = unfix(ua.x) * rs, uv1 = unfix(ua.y) * rs;
                const float h0 = gv0 / (1.0f + expf(-gv0)) * uv0, h1 = gv1 / (1.0f + expf(-gv1)) * uv1;
                uint16_t a0h, a0l, a1h, a1l;
                split_bf16(h0, a0h, a0l);
                split_bf16(h1, a1h, a1l);
                const int64_t off = xblk_off(r, jb * 64 + 2 * lane, R16c);
                *reinterpret_cast<uint32_t *>(p.h_hi + off) = (uint32_t)a0h | ((uint32_t)a1h << 16);
                *reinterpret_cast<uint32_t *>(p.h_lo + off) = (uint32_t)a0l | ((uint32_t)a1l << 16);
            }
            arrive(base + 5);
        }
        // ------------------------------------------------------------ down
        {
            const GemmPh g = gemm_phase(p, l, 6);
            gemm_range(g, false, u0, u1);
            gemm_epi(g, u0, u1);
            wi += (uint32_t)(u1 - u0);
            arrive(base + 6);
        }
        // ------------------------------------------------------------ residual, next norm input
        {
            wait_phase(base + 6);
            const uint16_t *gn = (l + 1 < p.layers) ? p.attn_norm + (int64_t)(l + 1) * d : p.final_norm;
            fin_resid(p.accD, gn, p.ssqA);
            arrive(base + 7);
        }
    }

    // ---------------------------------------------------------------- lm_head + Gumbel-max
    {
        wait_phase(kPhasesPerLayer * p.layers);
        load_rstd(p.ssqA);
        if (ctid < R) S.seed[ctid] = p.c.row_seed[ctid];
        named_bar_sync(1, kMegaCThreads);
        const GemmPh g = gemm_phase(p, p.layers, 0);
        int64_t u0, u1;
        gemm_range(g, true, u0, u1);
        const int ntiles = p.V / 128;
        for (int64_t u = u0; u < u1; u += g.kch) {
            const int tile = (int)(u / g.kch);
            const int a = seg & 1;
            mwait(&S.acc_full[a], (seg >> 1) & 1, err, ab);
            tc_fence_after();
            const int n = tile * 128 + quarter * 32 + lane;
            for (int cc = half; cc * 32 < R; cc += 2) {
                float v[32];
                int id[32];
                tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(a * 128 + cc * 32), v);
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const int r = cc * 32 + j;
                    float z = -INFINITY;
                    if (r < R) {
                        z = v[j] * S.rstd[r];
                        if (p.logits) p.logits[(int64_t)r * p.V + n] = z;
                        z += gumbel_from_hash(splitmix_at(S.seed[r], (uint64_t)n + 1));
                    }
                    v[j] = z;
                    id[j] = n;
                }
                // transpose-reduce: after the five steps lane l holds the argmax of column l
#pragma unroll
                for (int s = 16; s >= 1; s >>= 1) {
                    const bool up = (lane & s) != 0;
#pragma unroll
                    for (int k = 0; k < s; ++k) {
                        const float sendv = up ? v[k] : v[k + s];
                        const int sendi = up ? id[k] : id[k + s];
                        const float rv = __shfl_xor_sync(0xffffffffu, sendv, s);
                        const int ri = __shfl_xor_sync(0xffffffffu, sendi, s);
                        float kv = up ? v[k + s] : v[k];
                        int ki = up ? id[k + s] : id[k];
                        argmax_combine(kv, ki, rv, ri);
                        v[k] = kv;
                        id[k] = ki;
                    }
                }
                S.lm_v[half][quarter][lane] = v[0];
                S.lm_i[half][quarter][lane] = id[0];
                named_bar_sync(2 + half, 128);
                if ((ctid & 127) < 32) {
                    const int j = ctid & 31;
                    float bv = S.lm_v[half][0][j];
                    int bi = S.lm_i[half][0][j];
                    for (int q = 1; q < 4; ++q) argmax_combine(bv, bi, S.lm_v[half][q][j], S.lm_i[half][q][j]);
                    const int r = cc * 32 + j;
                    if (r < R) {
                        p.arg_val[(int64_t)r * ntiles + tile] = bv;
                        p.arg_idx[(int64_t)r * ntiles + tile] = bi;
                    }
                }
                named_bar_sync(2 + half, 128);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.acc_empty[a]);
            ++seg;
        }
    }
}

// ------------------------------------------------------------------------------ kernel
__global__ void __launch_bounds__(kMegaThreads, 1) decode_step_kernel(const __grid_constant__ MegaParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t *sW = base;
    uint8_t *sX = sW + (size_t)kWSlots * kSlotBytes;
    uint8_t *sQ = sX + kXRingBytes;
    uint8_t *sP = sQ + 8192;
    MegaSmem &S = *reinterpret_cast<MegaSmem *>(sP + 8192);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    StepVars *V = p.c.v;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kWSlots; ++s) { mbar_init(&S.wfull[s], 1); mbar_init(&S.wempty[s], 1); }
        for (int s = 0; s < kMaxXStages; ++s) { mbar_init(&S.xfull[s], 1); mbar_init(&S.xempty[s], 1); }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&S.acc_full[a], 1);
            mbar_init(&S.acc_empty[a], 8);
            mbar_init(&S.q_ready[a], 1);
            mbar_init(&S.s_full[a], 1);
            mbar_init(&S.p_ready[a], 1);
            mbar_init(&S.o_full[a], 1);
        }
        mbar_init(&S.drain, 1);
        const int live = *(volatile int *)&V->live;
        const int rows = max(0, min(live, p.rows_cap));
        S.rows = rows;
        S.rows16 = max(16, (rows + 15) & ~15);
        S.nx = min(kMaxXStages, kXRingBytes / (S.rows16 * 256));
        S.n_items = *(volatile int *)&V->att_items;
        S.target = (*(volatile unsigned long long *)p.epoch + 1ull) * gridDim.x;
        S.abort = (*(volatile int *)&V->err & ERR_WAIT_TIMEOUT) != 0;
        S.last_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&S.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    const bool run = !S.abort && S.rows > 0;
    if (run) {
        if (warp == 0) {
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
}

// ------------------------------------------------------------------------------ layout kernels
// Row-major W [N][K] (bf16) -> blocked tiles: tile (n/128, k/64) is 128 rows of 128 bytes,
// 16-byte granule j of row r stored at granule j ^ (r % 8).
static __global__ void block_weights_kernel(const uint16_t *src, uint8_t *dst, int N, int K) {
    const int gpr = K / 8, kch = K / 64;
    const int64_t total = (int64_t)N * gpr;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int n = (int)(e / gpr), j = (int)(e - (int64_t)n * gpr);
        const int r = n & 127;
        const uint4 v = *reinterpret_cast<const uint4 *>(src + (int64_t)n * K + (int64_t)j * 8);
        *reinterpret_cast<uint4 *>(dst + (((int64_t)(n >> 7) * kch + (j >> 3)) * 128 + r) * 128 + (((j & 7) ^ (r & 7)) << 4)) =
            v;
    }
}

// Copy every layer's prompt KV (positions < Lp - 1, row-major [2][n_kv][cap_p][hd] per prompt
// slot) into rollout slot s < live in the blocked decode layout (run once at a round start).
// One thread per K granule (8 dims of a position) or per V granule (8 positions of a dim).
static __global__ void kv_fanout_kernel(const uint16_t *pkv, uint8_t *kv, const StepPtrs c, int layers, int n_kv,
                                        int hd, int cap_p, int64_t kv_layer, int64_t kv_slot, int nblk,
                                        int max_active) {
    pdl_wait_prior_grids();
    pdl_allow_dependents();
    const int live = c.v->live;
    const int Lpre = c.kc->Lp - 1;
    const int gk = hd / 8;
    const int64_t nk = (int64_t)Lpre * gk;
    const int64_t nv = (int64_t)((Lpre + 7) / 8) * hd;
    const int64_t per = nk + nv;
    const int64_t total = (int64_t)layers * live * n_kv * per;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        int64_t rem = e;
        const int64_t per_layer = (int64_t)live * n_kv * per;
        const int l = (int)(rem / per_layer);
        rem -= l * per_layer;
        const int s = (int)(rem / ((int64_t)n_kv * per));
        rem -= (int64_t)s * n_kv * per;
        const int kvh = (int)(rem / per);
        rem -= (int64_t)kvh * per;
        const int ps = c.seq_pslot[s];
        const uint16_t *kplane = pkv + (((int64_t)l * max_active + ps) * 2 * n_kv + kvh) * cap_p * hd;
        const uint16_t *vplane = kplane + (int64_t)n_kv * cap_p * hd;
        uint8_t *dst = kv + l * kv_layer + (int64_t)s * kv_slot + (int64_t)kvh * nblk * kKVBlockBytes;
        if (rem < nk) {
            const int pos = (int)(rem / gk), j = (int)(rem - (int64_t)pos * gk);
            const uint4 v = *reinterpret_cast<const uint4 *>(kplane + (int64_t)pos * hd + j * 8);
            *reinterpret_cast<uint4 *>(dst + (int64_t)(pos / kKVPos) * kKVBlockBytes + kv_k_off(pos % kKVPos, j * 8)) = v;
        } else {
            rem -= nk;
            const int pg = (int)(rem / hd), dd = (int)(rem - (int64_t)pg * hd);
            uint32_t w[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int p0 = pg * 8 + 2 * q;
                const uint32_t a = p0 < Lpre ? vplane[(int64_t)p0 * hd + dd] : 0u;
                const uint32_t b = p0 + 1 < Lpre ? vplane[(int64_t)(p0 + 1) * hd + dd] : 0u;
                w[q] = a | (b << 16);
            }
            const int pos = pg * 8;
            *reinterpret_cast<uint4 *>(dst + (int64_t)(pos / kKVPos) * kKVBlockBytes + kv_v_off(pos % kKVPos, dd)) =
                make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

}  // namespace sara
