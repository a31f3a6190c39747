// Projection GEMM of the prefill path on sm_103a:
//     Y[r][n] = sum_c X[r][c] * W[n][c]        (X: activations, W: a linear layer's weight)
// computed "swap-AB" on the 5th-generation tensor core: the weight tile is the MMA's A
// operand (M = 128 output features), the activation rows are B (N = rows rounded up to
// 16, <= 128), the fp32 accumulator lives in tensor memory.  Activations arrive as a bf16
// pair hi + lo (hi = bf16(x), lo = bf16(x - hi)); both are multiplied with the same weight
// tile into the same accumulator, so the product keeps ~16 mantissa bits of x at the cost of
// one extra MMA per weight tile (the GEMM is weight-bandwidth bound).  Operands are staged in shared
// memory by TMA (128-byte swizzle) through a multi-stage mbarrier pipeline; one elected
// thread issues tcgen05.mma; four epilogue warps read the accumulator with tcgen05.ld.
//
// Work split: stream-K.  The (tile, k-chunk) units of the whole GEMM are cut into
// gridDim.x equal contiguous ranges, so every SM streams the same number of weight bytes.
// A tile whose k-chunks span several CTAs is folded into a 64-bit fixed-point accumulator
// (value * 2^32) with fire-and-forget integer atomic adds -- integer addition is
// associative, so the sum does not depend on arrival order -- and the CTA that arrives
// last (a per-tile counter, no spinning) reads it once, clears it, and runs the epilogue.
//
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = MMA issuer + tensor-memory
// owner, warps 2..5 = epilogue (warp w reads tensor-memory lanes 32*(w%4) .. +31).
//
// In decode mode (one row tile) the producer streams the first pipeline stages of weights
// before waiting on the preceding grid (programmatic dependent launch), so weight reads
// overlap the previous kernel's tail.
#pragma once
#include "device_common.cuh"

namespace sara {

enum EpiKind : int {
    EPI_F32 = 0,     // Y fp32 [rows][ld]
    EPI_QKV = 1,     // RMSNorm scale, RoPE on q/k, q -> q_out (fp16), k/v -> KV cache (fp16)
    EPI_RESID = 2,   // x += Y; xg = x * g_next as a bf16 hi/lo pair; per-tile sum of squares of x
    EPI_SWIGLU = 3,  // RMSNorm scale; tile = 64 gate rows + 64 up rows -> h = silu(g) * u (hi/lo)
};

constexpr int kGemmThreads = 192;
constexpr int kGemmStages = 4;
constexpr int kTileM = 128;       // weight rows per tile (MMA M)
constexpr int kTileK = 64;        // reduction elements per pipeline stage (128 B of bf16)
constexpr int kTileR = 128;       // activation rows per tile (max MMA N here)
constexpr int kXBoxRows = 32;     // activation rows per TMA box
constexpr int kWStageBytes = kTileM * kTileK * 2;   // 16 KB
constexpr int kXStageBytes = kTileR * kTileK * 2;   // 16 KB
constexpr int kEpiLd = 33;                          // padded fp32 row of the exchange tile

struct GemmParams {
    int m_tiles, k_chunks;
    int rows_cap;              // rows of the activation tensor map
    const int *rows_dev;       // device count of valid rows (nullptr -> rows_fixed)
    int rows_fixed;
    int decode;                // 1: a single row tile, weights prefetched before the PDL wait
    const uint8_t *w_blk;      // non-null: W stored as pre-swizzled 256-row tiles (bulk copies, wblk128_off)
    int has_lo;                // 1: the activation's lo part (second tensor map) is multiplied too
    unsigned long long *ws_acc;  // [gridDim.x][kTileR * kTileM] fixed-point tile sums, zero between launches
    int *ws_cnt;               // [tiles] arrival counters, zero between launches
    int *err;
    // outputs / epilogue inputs
    float *y_f32; int ld;      // EPI_F32 output; row stride
    const float *ssq;          // [ssq_tiles][rows_cap] per-128-feature partial sums of x^2
    int ssq_tiles; float inv_dim; float eps;
    uint16_t *q_out;           // EPI_QKV: [rows][n_heads * head_dim] fp16
    int n_heads, n_kv, head_dim;
    const float2 *rope;        // [positions][head_dim / 2] (cos, sin)
    const int *row_pos;        // [rows] position of the row's token
    const int *row_slot;       // [rows] KV slot of the row
    uint16_t *kv;              // KV cache of this layer: slot s at kv + s * kv_slot_stride,
    int64_t kv_slot_stride;    //   laid out [2][n_kv][kv_cap][head_dim]
    int kv_cap;
    float *x_f32;              // EPI_RESID residual stream [rows][ld]
    uint16_t *xg_out;          // EPI_RESID x * g_next, bf16 hi [rows][ld]
    uint16_t *xg_lo;           //   and bf16 lo
    const uint16_t *g_next;    // EPI_RESID next RMSNorm weight [ld]
    float *ssq_out;            // EPI_RESID [m_tiles][rows_cap]
    uint16_t *h_out;           // EPI_SWIGLU [rows][ld] bf16 hi
    uint16_t *h_lo;            //   and bf16 lo
    uint64_t *stamps;          // optional [gridDim.x][16] phase timestamps (profiling builds)
};

struct GemmSmem {
    uint64_t full[kGemmStages];
    uint64_t empty[kGemmStages];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort_flag;
    int last_flag;
    int epi_abort;      // set by an epilogue warp whose bounded wait gave up
    int epi_decision;   // uniform abort decision of the epilogue warps
    int skip;           // an earlier kernel of the step reported an error: do nothing
    float inv_rms[kTileR];
    int row_pos[kTileR];               // per-row metadata of the tile being finished
    int row_slot[kTileR];
    float xch[kTileM * kEpiLd];        // exchange tile: 128 features x 32 columns
};

constexpr size_t kGemmSmemBytes =
    1024 /* alignment slack */ + (size_t)kGemmStages * (kWStageBytes + 2 * kXStageBytes) + sizeof(GemmSmem);

// Stream-K partition: CTA c owns units [unit_begin(c), unit_begin(c+1)).
__device__ __forceinline__ int64_t unit_begin(int c, int64_t U, int G) { return (int64_t)c * U / G; }
__device__ __forceinline__ int cta_of_unit(int64_t u, int64_t U, int G) {
    int c = (int)((u * G) / U);
    while (c + 1 < G && unit_begin(c + 1, U, G) <= u) ++c;
    while (c > 0 && unit_begin(c, U, G) > u) --c;
    return c;
}
#ifdef SARA_STAMPS
#define GEMM_STAMP(i) do { if (p.stamps) p.stamps[(size_t)blockIdx.x * 16 + (i)] = globaltimer_ns(); } while (0)
#else
#define GEMM_STAMP(i) do { } while (0)
#endif
__device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

// Byte offset of the 128 x 64 weight sub-tile (m_tile, kc) of a weight [Nout][K] stored as
// pre-swizzled tiles of 256 rows (the last may have 128): tile t = m_tile / 2 holds, for
// each k-chunk, its rows at a 128-byte pitch, so the two 128-row halves are 16 KB apart.
__device__ __forceinline__ int64_t wblk128_off(int Nout, int K, int m_tile, int kc) {
    const int t = m_tile >> 1;
    const int rows = min(256, Nout - 256 * t);
    return (int64_t)t * 256 * K * 2 + (int64_t)kc * rows * 128 + (m_tile & 1) * 16384;
}


template <int EPI>
__device__ __forceinline__ void gemm_epilogue_chunk(const GemmParams &p, GemmSmem &S, float (&v)[32], int m_tile,
                                                    int r_base, int c0, int rows_in_tile, int mrow, int etid) {
    const int n = m_tile * kTileM + mrow;  // output feature
    const int ncols = min(32, rows_in_tile - c0);
    if constexpr (EPI == EPI_F32) {
#pragma unroll
        for (int c = 0; c < 32; ++c)
            if (c < ncols) p.y_f32[(int64_t)(r_base + c0 + c) * p.ld + n] = v[c];
    } else {
        if constexpr (EPI == EPI_QKV || EPI == EPI_SWIGLU) {
#pragma unroll
            for (int c = 0; c < 32; ++c) v[c] *= S.inv_rms[c0 + c];
        }
        if constexpr (EPI == EPI_RESID) {
            const float g = bf16_to_f32(p.g_next[n]);
            float xo[32];
#pragma unroll
            for (int c = 0; c < 32; ++c)  // every load before any store (the stores may alias)
                xo[c] = (c < ncols) ? __ldcg(&p.x_f32[(int64_t)(r_base + c0 + c) * p.ld + n]) : 0.f;
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                if (c < ncols) {
                    const int64_t idx = (int64_t)(r_base + c0 + c) * p.ld + n;
                    const float x = xo[c] + v[c];
                    p.x_f32[idx] = x;
                    uint16_t hi, lo;
                    split_bf16(x * g, hi, lo);
                    p.xg_out[idx] = hi;
                    p.xg_lo[idx] = lo;
                    v[c] = x * x;
                }
            }
        }
        // stage the chunk in shared memory for the cross-feature exchanges / reductions
#pragma unroll
        for (int c = 0; c < 32; ++c) S.xch[mrow * kEpiLd + c] = v[c];
        named_bar_sync(1, 128);
        if constexpr (EPI == EPI_QKV) {
            const int hd = p.head_dim, half = hd >> 1;
            const int head = n / hd, i = n - head * hd;
            const int partner = (i < half) ? mrow + half : mrow - half;
            const int fi = (i < half) ? i : i - half;
            const int nq = p.n_heads, nkv = p.n_kv;
            const bool rot = head < nq + nkv;  // q or k: rotate the pair (i, i + hd/2)
            float2 cs[32];
#pragma unroll
            for (int c = 0; c < 32; ++c)  // every table load before any store
                cs[c] = (rot && c < ncols) ? __ldg(&p.rope[(int64_t)S.row_pos[c0 + c] * half + fi]) : make_float2(1.f, 0.f);
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                if (c < ncols) {
                    const int r = r_base + c0 + c;
                    float y = v[c];
                    if (rot) {
                        const float o = S.xch[partner * kEpiLd + c];
                        y = (i < half) ? (y * cs[c].x - o * cs[c].y) : (y * cs[c].x + o * cs[c].y);
                    }
                    if (head < nq) {
                        p.q_out[(int64_t)r * (nq * hd) + n] = f32_to_f16_sat(y);
                    } else {
                        const int isv = head >= nq + nkv;
                        const int kvh = head - nq - isv * nkv;
                        uint16_t *dst = p.kv + (int64_t)S.row_slot[c0 + c] * p.kv_slot_stride +
                                        ((int64_t)(isv * nkv + kvh) * p.kv_cap + S.row_pos[c0 + c]) * hd + i;
                        *dst = f32_to_f16_sat(y);
                    }
                }
            }
        } else if constexpr (EPI == EPI_SWIGLU) {
            if (mrow < 64) {
                const int f = m_tile * 64 + mrow;
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    if (c < ncols) {
                        const float g = v[c], u = S.xch[(mrow + 64) * kEpiLd + c];
                        const float h = g / (1.0f + expf(-g)) * u;
                        uint16_t hi, lo;
                        split_bf16(h, hi, lo);
                        p.h_out[(int64_t)(r_base + c0 + c) * p.ld + f] = hi;
                        p.h_lo[(int64_t)(r_base + c0 + c) * p.ld + f] = lo;
                    }
                }
            }
        } else if constexpr (EPI == EPI_RESID) {
            // thread etid reduces column c = etid / 4 over features [32 * (etid % 4), +32)
            const int c = etid >> 2, part = etid & 3;
            float s = 0.f;
            for (int f = 0; f < 32; ++f) s += S.xch[(part * 32 + f) * kEpiLd + c];
            s += __shfl_xor_sync(0xffffffffu, s, 1);
            s += __shfl_xor_sync(0xffffffffu, s, 2);
            if (part == 0 && c < ncols) p.ssq_out[(int64_t)m_tile * p.rows_cap + r_base + c0 + c] = s;
        }
        named_bar_sync(1, 128);  // xch reused by the next chunk
    }
}

template <int EPI>
__global__ void __launch_bounds__(kGemmThreads, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
               const __grid_constant__ CUtensorMap tmXlo, GemmParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t *sW = base;
    uint8_t *sX = base + (size_t)kGemmStages * kWStageBytes;
    uint8_t *sXlo = sX + (size_t)kGemmStages * kXStageBytes;
    GemmSmem &S = *reinterpret_cast<GemmSmem *>(sXlo + (size_t)kGemmStages * kXStageBytes);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int G = gridDim.x, cta = blockIdx.x;

    if (threadIdx.x == 0) {
        GEMM_STAMP(0);
        for (int s = 0; s < kGemmStages; ++s) { mbar_init(&S.full[s], 1); mbar_init(&S.empty[s], 1); }
        for (int a = 0; a < 2; ++a) { mbar_init(&S.acc_full[a], 1); mbar_init(&S.acc_empty[a], 4); }
        mbar_init(&S.drain, 1);
        S.abort_flag = 0;
        S.epi_abort = 0;
        S.skip = (p.err != nullptr) && (*(volatile int *)p.err != 0);
        fence_mbar_init();
        if (!p.w_blk) prefetch_tensormap(&tmW);
        prefetch_tensormap(&tmX);
        if (p.has_lo) prefetch_tensormap(&tmXlo);
    }
    if (warp == 1) { tmem_alloc(&S.tmem_base, 256); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    if (threadIdx.x == 0) GEMM_STAMP(1);

    // Let the next kernel in the stream start its own weight prefetch.
    pdl_allow_dependents();

    const int m_tiles = p.m_tiles, kch = p.k_chunks;
    // In decode mode the row count does not change the partition (one row tile).
    int rows = 0, r_tiles = 1;
    if (!p.decode) {
        pdl_wait_prior_grids();
        rows = p.rows_dev ? min(*p.rows_dev, p.rows_cap) : p.rows_fixed;
        r_tiles = (rows + kTileR - 1) / kTileR;
    }
    const int64_t U = (int64_t)m_tiles * r_tiles * kch;
    const int64_t u0 = S.skip ? 0 : unit_begin(cta, U, G);
    const int64_t u1 = S.skip ? 0 : unit_begin(cta + 1, U, G);

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (p.decode) {
            if (lane == 0) {
                // weights of the first stages before the dependency wait
                const int64_t n_pre = min64(kGemmStages, u1 - u0);
                for (int64_t i = 0; i < n_pre; ++i) {
                    const int64_t u = u0 + i;
                    const int tile = (int)(u / kch), kc = (int)(u % kch);
                    const int m_tile = tile % m_tiles;
                    mbar_expect_tx(&S.full[i], (uint32_t)kWStageBytes);
                    if (p.w_blk)
                        bulk_load(sW + i * kWStageBytes, p.w_blk + wblk128_off(m_tiles * kTileM, kch * kTileK, m_tile, kc),
                                  kWStageBytes, &S.full[i], l2_policy_evict_first());
                    else
                        tma_load_2d(sW + i * kWStageBytes, &tmW, &S.full[i], kc * kTileK, m_tile * kTileM,
                                    l2_policy_evict_first());
                }
            }
            pdl_wait_prior_grids();
            rows = p.rows_dev ? min(*p.rows_dev, p.rows_cap) : p.rows_fixed;
        }
        if (lane == 0) {
            const uint64_t pol_w = l2_policy_evict_first(), pol_x = l2_policy_evict_last();
            const int64_t n_pre = p.decode ? min64(kGemmStages, u1 - u0) : 0;
            int64_t i = 0;
            for (int64_t u = u0; u < u1; ++u, ++i) {
                const int s = (int)(i % kGemmStages);
                const uint32_t ph = (uint32_t)((i / kGemmStages) & 1);
                if (i >= kGemmStages && !mbar_wait(&S.empty[s], ph ^ 1, p.err)) { S.abort_flag = 1; break; }
                if (*(volatile int *)&S.abort_flag) break;
                const int tile = (int)(u / kch), kc = (int)(u % kch);
                const int m_tile = tile % m_tiles, r_tile = tile / m_tiles;
                const int rin = min(kTileR, max(rows - r_tile * kTileR, 0));
                const int nbox = max(1, (rin + kXBoxRows - 1) / kXBoxRows);
                const uint32_t xbytes = (uint32_t)(nbox * kXBoxRows * kTileK * 2) * (p.has_lo ? 2u : 1u);
                if (i >= n_pre) {
                    mbar_arrive_expect_tx(&S.full[s], (uint32_t)kWStageBytes + xbytes);
                    if (p.w_blk)
                        bulk_load(sW + (size_t)s * kWStageBytes,
                                  p.w_blk + wblk128_off(m_tiles * kTileM, kch * kTileK, m_tile, kc), kWStageBytes,
                                  &S.full[s], pol_w);
                    else
                        tma_load_2d(sW + (size_t)s * kWStageBytes, &tmW, &S.full[s], kc * kTileK, m_tile * kTileM,
                                    pol_w);
                } else {
                    mbar_arrive_expect_tx(&S.full[s], xbytes);
                }
                for (int b = 0; b < nbox; ++b) {
                    tma_load_2d(sX + (size_t)s * kXStageBytes + b * kXBoxRows * kTileK * 2, &tmX, &S.full[s],
                                kc * kTileK, r_tile * kTileR + b * kXBoxRows, pol_x);
                    if (p.has_lo)
                        tma_load_2d(sXlo + (size_t)s * kXStageBytes + b * kXBoxRows * kTileK * 2, &tmXlo, &S.full[s],
                                    kc * kTileK, r_tile * kTileR + b * kXBoxRows, pol_x);
                }
            }
            // On abort, the last load issued on every stage lands before the CTA exits.
            if (*(volatile int *)&S.abort_flag) {
                const int64_t issued = i;
                for (int s = 0; s < kGemmStages && s < issued; ++s) {
                    const int64_t last = ((issued - 1 - s) / kGemmStages) * kGemmStages + s;
                    mbar_wait(&S.full[s], (uint32_t)((last / kGemmStages) & 1), p.err);
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (p.decode) {
            pdl_wait_prior_grids();
            rows = p.rows_dev ? min(*p.rows_dev, p.rows_cap) : p.rows_fixed;
        }
        if (lane == 0) {
            int64_t i = 0;
            int seg = 0;
            for (int64_t u = u0; u < u1; ++seg) {
                const int tile = (int)(u / kch);
                const int64_t seg_end = min64(u1, (int64_t)(tile + 1) * kch);
                const int r_tile = tile / m_tiles;
                const int rin = min(kTileR, max(rows - r_tile * kTileR, 0));
                const uint32_t N = (uint32_t)max(16, (rin + 15) & ~15);
                const uint32_t idesc = idesc_bf16_f32(128, N);
                const int a = seg & 1;
                if (seg >= 2 && !mbar_wait(&S.acc_empty[a], (uint32_t)(((seg >> 1) - 1) & 1), p.err)) {
                    S.abort_flag = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(a * kTileR);
                bool first = true;
                for (; u < seg_end; ++u, ++i) {
                    const int s = (int)(i % kGemmStages);
                    if (!mbar_wait(&S.full[s], (uint32_t)((i / kGemmStages) & 1), p.err) ||
                        *(volatile int *)&S.abort_flag) {
                        S.abort_flag = 1;
                        break;
                    }
                    tc_fence_after();
                    if (i == 0) GEMM_STAMP(2);
                    const uint32_t aw = smem_u32(sW + (size_t)s * kWStageBytes);
                    const uint32_t ax = smem_u32(sX + (size_t)s * kXStageBytes);
                    const uint32_t axl = smem_u32(sXlo + (size_t)s * kXStageBytes);
#pragma unroll
                    for (int kk = 0; kk < kTileK / 16; ++kk) {
                        const uint64_t adesc = sdesc_kmajor_sw128(aw + kk * 32);
                        tc_mma_bf16(d, adesc, sdesc_kmajor_sw128(ax + kk * 32), idesc, (first && kk == 0) ? 0u : 1u);
                        if (p.has_lo) tc_mma_bf16(d, adesc, sdesc_kmajor_sw128(axl + kk * 32), idesc, 1u);
                    }
                    first = false;
                    tc_commit(&S.empty[s]);
                }
                if (*(volatile int *)&S.abort_flag) break;
                tc_commit(&S.acc_full[a]);
            }
            GEMM_STAMP(3);
            // every MMA this thread issued has retired before tensor memory is released
            tc_commit(&S.drain);
            mbar_wait(&S.drain, 0, p.err);
        }
    } else {
        // ------------------------------------------------------------ epilogue (warps 2..5)
        pdl_wait_prior_grids();
        if (p.decode) rows = p.rows_dev ? min(*p.rows_dev, p.rows_cap) : p.rows_fixed;
        const int quarter = warp & 3;
        const int mrow = quarter * 32 + lane;
        const int etid = threadIdx.x - 64;  // 0..127
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        // Per-row values (1/rms, position, KV slot) staged once per tile: in
        // decode mode every tile has the same rows, so they are loaded once, while the
        // mainloop streams weights.
        int staged_rbase = -1;
        auto stage_rows = [&](int r_base, int rin) {
            if constexpr (EPI == EPI_QKV || EPI == EPI_SWIGLU) {
                if (etid < rin) {
                    const int r = r_base + etid;
                    float part[16];
#pragma unroll
                    for (int t = 0; t < 16; ++t)
                        part[t] = (t < p.ssq_tiles) ? __ldcg(&p.ssq[(int64_t)t * p.rows_cap + r]) : 0.f;
                    float s = 0.f;
#pragma unroll
                    for (int t = 0; t < 16; ++t) s += part[t];
                    for (int t = 16; t < p.ssq_tiles; ++t) s += __ldcg(&p.ssq[(int64_t)t * p.rows_cap + r]);
                    S.inv_rms[etid] = rsqrtf(s * p.inv_dim + p.eps);
                    if constexpr (EPI == EPI_QKV) {
                        S.row_pos[etid] = p.row_pos[r];
                        S.row_slot[etid] = p.row_slot[r];
                    }
                } else {
                    S.inv_rms[etid] = 0.f;
                    S.row_pos[etid] = 0;
                    S.row_slot[etid] = 0;
                }
                named_bar_sync(1, 128);
            }
        };
        if (p.decode && u0 < u1) {
            stage_rows(0, min(kTileR, rows));
            staged_rbase = 0;
        }
        int seg = 0;
        for (int64_t u = u0; u < u1; ++seg) {
            const int tile = (int)(u / kch);
            const int kc_first = (int)(u % kch);
            const int64_t seg_end = min64(u1, (int64_t)(tile + 1) * kch);
            const int kc_last = (int)((seg_end - 1) % kch);
            u = seg_end;
            const int m_tile = tile % m_tiles, r_tile = tile / m_tiles;
            const int r_base = r_tile * kTileR;
            const int rin = min(kTileR, max(rows - r_base, 0));
            const int a = seg & 1;
            // every epilogue warp takes the same abort decision, so none is left in a named barrier
            const bool ok = mbar_wait(&S.acc_full[a], (uint32_t)((seg >> 1) & 1), p.err);
            if (!ok && lane == 0) atomicOr(&S.epi_abort, 1);
            named_bar_sync(1, 128);
            if (etid == 0) S.epi_decision = S.epi_abort | *(volatile int *)&S.abort_flag;
            named_bar_sync(1, 128);
            if (S.epi_decision) {
                S.abort_flag = 1;
                break;
            }
            tc_fence_after();
            if (seg == 0 && etid == 0) GEMM_STAMP(4);
            const bool whole = (kc_first == 0) && (kc_last == kch - 1);
            bool do_epi = whole;
            int c_a = cta, c_b = cta;
            if (!whole) {
                // fold this CTA's share into the tile's fixed-point sum; the last arrival finishes
                c_a = cta_of_unit((int64_t)tile * kch, U, G);
                c_b = cta_of_unit((int64_t)(tile + 1) * kch - 1, U, G);
                unsigned long long *acc = p.ws_acc + (size_t)c_a * (kTileR * kTileM);
                for (int c0 = 0; c0 < rin; c0 += 32) {
                    float v[32];
                    tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(a * kTileR + c0), v);
#pragma unroll
                    for (int c = 0; c < 32; ++c)
                        if (c0 + c < rin)
                            atomicAdd(&acc[(c0 + c) * kTileM + mrow],
                                      (unsigned long long)__float2ll_rn(v[c] * 4294967296.0f));
                }
                if (etid == 0) GEMM_STAMP(8);
                __threadfence();
                named_bar_sync(1, 128);
                if (etid == 0) GEMM_STAMP(9);
                if (etid == 0) {
                    int nseg = 0;
                    for (int c = c_a; c <= c_b; ++c) nseg += unit_begin(c, U, G) < unit_begin(c + 1, U, G);
                    const int old = atomicAdd(&p.ws_cnt[tile], 1);
                    S.last_flag = (old == nseg - 1);
                    if (S.last_flag) p.ws_cnt[tile] = 0;
                }
                named_bar_sync(1, 128);
                do_epi = S.last_flag != 0;
                __threadfence();
            }
            if (do_epi) {
                if (staged_rbase != r_base) {
                    stage_rows(r_base, rin);
                    staged_rbase = r_base;
                }
                for (int c0 = 0; c0 < rin; c0 += 32) {
                    float v[32];
                    if (whole) {
                        tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(a * kTileR + c0), v);
                    } else {
                        unsigned long long *acc = p.ws_acc + (size_t)c_a * (kTileR * kTileM);
#pragma unroll
                        for (int c = 0; c < 32; ++c) {
                            const size_t idx = (size_t)(c0 + c) * kTileM + mrow;
                            v[c] = (float)(long long)__ldcg(&acc[idx]) * 2.3283064365386963e-10f;  // 2^-32
                            if (c0 + c < rin) acc[idx] = 0ull;
                        }
                    }
                    if (etid == 0) GEMM_STAMP(10);
                    gemm_epilogue_chunk<EPI>(p, S, v, m_tile, r_base, c0, rin, mrow, etid);
                    if (etid == 0) GEMM_STAMP(11);
                }
            }
            // release the accumulator buffer
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&S.acc_empty[a]);
        }
    }

    if (threadIdx.x == 64) GEMM_STAMP(6);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, 256);
    if (threadIdx.x == 32) GEMM_STAMP(7);
}

}  // namespace sara
