// Host engine behind include/sara.h: device memory layout, weight packing (pre-swizzled
// 16 KB tiles), the step graph (a conditional WHILE loop whose body is controller ->
// [round start: prefill + prompt-KV fan-out] -> persistent decode-step kernel ->
// sampling/bookkeeping), and the C ABI.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <string>
#include <vector>

#include "../../include/sara.h"
#include "attention.cuh"
#include "controller.cuh"
#include "decode_step.cuh"
#include "gemm_tc.cuh"
#include "host_util.h"
#include "step_kernels.cuh"

using namespace sara;

namespace {

constexpr int kDecodeChunk = 128;  // decode attention positions per split

struct DeviceBuf {
    std::vector<void *> ptrs;
    ~DeviceBuf() {
        for (void *p : ptrs) cudaFree(p);
    }
    template <typename T>
    T *alloc(size_t count, bool zero = true) {
        void *p = nullptr;
        const size_t bytes = std::max<size_t>(count * sizeof(T), 256);
        if (cudaMalloc(&p, bytes) != cudaSuccess)
            throw SaraError(SARA_ENOMEM, "cudaMalloc of " + std::to_string(bytes) + " bytes failed");
        ptrs.push_back(p);
        if (zero) CK(cudaMemset(p, 0, bytes));
        return static_cast<T *>(p);
    }
};

struct Acts {  // activation buffers of the prefill rows (row-major, TMA operands)
    int rows_cap = 0;
    float *x_f32 = nullptr;
    // GEMM operands as bf16 hi/lo pairs; q is fp16
    uint16_t *xg = nullptr, *xg_lo = nullptr, *q = nullptr, *att = nullptr, *att_lo = nullptr, *h = nullptr,
             *h_lo = nullptr;
    float *ssq_a = nullptr, *ssq_m = nullptr;
    CUtensorMap tm_xg{}, tm_xg_lo{}, tm_att{}, tm_att_lo{}, tm_h{}, tm_h_lo{};
};

}  // namespace

struct sara_handle {
    sara_model_cfg cfg{};
    cudaStream_t stream = nullptr;
    int device = 0, sms = 0;
    bool has_model = false;
    bool use_graph = true, use_pdl = true;
    std::string err;
    DeviceBuf mem;
    // weights: embedding row-major, projections as pre-swizzled 16 KB tiles (all layers
    // of one kind contiguous), norms [layers][d]
    uint16_t *embed = nullptr, *final_norm = nullptr, *norm_attn = nullptr, *norm_mlp = nullptr;
    uint8_t *wb_qkv = nullptr, *wb_o = nullptr, *wb_gu = nullptr, *wb_down = nullptr, *wb_lm = nullptr;
    int64_t ls_qkv = 0, ls_o = 0, ls_gu = 0, ls_down = 0;
    // KV caches: rollout slots in the blocked decode layout, prompt slots row-major
    uint8_t *kv_seq = nullptr;  // paged KV pool: [layer][block id][kv head] 64 KB blocks
    uint16_t *kv_pr = nullptr;
    int cap_s = 0, cap_p = 0;
    int64_t kv_seq_layer = 0, kv_pr_layer = 0, kv_pr_slot = 0;
    float2 *rope = nullptr;
    Acts pre;
    // decode-step activations (blocked operands) and phase counters
    int rows_cap16 = 0;
    float *dx = nullptr, *ssqA = nullptr, *ssqM = nullptr;
    uint8_t *xg = nullptr, *att = nullptr, *hm = nullptr;  // pair-blocked GEMM operands of the decode step
    float *gpart = nullptr;  // GEMM partial tiles of the decode step
    uint16_t *qkv16 = nullptr;  // the step's q (scaled), k, v in fp16
    int gp_qkv = 0, gp_o = 0;
    unsigned long long *phase_cnt = nullptr;  // [1 + 8 layers + 1] then the epoch
    int n_phase_cnt = 0;
    int pre_cap = 0, att_cap = 0;
    // workspaces
    unsigned long long *gemm_acc = nullptr;
    int *gemm_cnt = nullptr;
    float *attn_part = nullptr;
    int *attn_cnt = nullptr;
    float *lm_val = nullptr;
    int *lm_idx = nullptr;
    // step state
    StepConst *kc = nullptr;
    StepVars *vars = nullptr;
    StepPtrs ptrs{};
    int32_t *p_tok = nullptr, *p_len = nullptr;
    uint64_t *p_thr = nullptr;
    int32_t *gen_tok = nullptr;
    float *logit_buf = nullptr;  // [max_seqs][vocab] logits of the decode step's live rows
    // teacher forcing staging (allocated on first use)
    int32_t *forced = nullptr, *sampled_out = nullptr;
    int64_t *uid_dev = nullptr;
    size_t forced_cap = 0;
    uint64_t *stamps = nullptr;  // profiling builds: per-CTA phase timestamps of GEMM launches
    double *prior_next = nullptr;  // [2][max_prompts] warm-start priors of the next step
    // failure limits (sara_set_limits): bounded-wait limit, loop bound, stalled phase counter
    uint64_t wait_ns = 0;
    int32_t max_iters = 0, stall_idx = -1, eager_softmax = 0;
    // graph
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    cudaStream_t cap_stream = nullptr, cap_stream2 = nullptr;
    cudaEvent_t ev0 = nullptr, ev1 = nullptr;

    ~sara_handle() {
        if (exec) cudaGraphExecDestroy(exec);
        if (graph) cudaGraphDestroy(graph);
        if (cap_stream) cudaStreamDestroy(cap_stream);
        if (cap_stream2) cudaStreamDestroy(cap_stream2);
        if (ev0) cudaEventDestroy(ev0);
        if (ev1) cudaEventDestroy(ev1);
    }
};

namespace {

thread_local std::string g_create_error;

// ------------------------------------------------------------------------ launches
void set_kernel_attrs() {
    static bool done = false;
    if (done) return;
    CK(cudaFuncSetAttribute(gemm_tc_kernel<EPI_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmemBytes));
    CK(cudaFuncSetAttribute(gemm_tc_kernel<EPI_QKV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmemBytes));
    CK(cudaFuncSetAttribute(gemm_tc_kernel<EPI_RESID>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmemBytes));
    CK(cudaFuncSetAttribute(gemm_tc_kernel<EPI_SWIGLU>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmemBytes));
    CK(cudaFuncSetAttribute(decode_step_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMegaSmemBytes));
    done = true;
}

template <typename Kern, typename... Args>
void launch_ex(cudaStream_t s, bool pdl, bool coop, dim3 grid, dim3 block, size_t smem, Kern kern, Args... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    unsigned n = 0;
    if (pdl) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    if (coop) {  // every CTA resident at once (the decode step's CTAs wait on one another)
        attr[n].id = cudaLaunchAttributeCooperative;
        attr[n].val.cooperative = 1;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    CK(cudaLaunchKernelEx(&cfg, kern, args...));
}
template <typename Kern, typename... Args>
void launch(cudaStream_t s, bool pdl, dim3 grid, dim3 block, size_t smem, Kern kern, Args... args) {
    launch_ex(s, pdl, false, grid, block, smem, kern, args...);
}

// Grid of a decode GEMM: one whole tile per CTA when the tile count nearly fills the SMs
// (no split reduction at all), else one CTA per SM with the stream-K split.
int gemm_grid(int sms, int tiles, bool decode) {
#ifdef SARA_STAMPS
    if (const char *e = getenv("SARA_GEMM_GRID")) return std::max(1, std::min(sms, atoi(e)));  // profiling sweeps
#endif
    if (decode && tiles <= sms && tiles * 20 >= sms * 17) return tiles;
    return sms;
}

template <int EPI>
void launch_gemm(cudaStream_t s, bool pdl, int grid, const CUtensorMap &tw, const CUtensorMap &tx,
                 const CUtensorMap &tx_lo, GemmParams p) {
    grid = gemm_grid(grid, p.m_tiles, p.decode != 0);
    p.has_lo = 1;
    launch(s, pdl, dim3(grid), dim3(kGemmThreads), kGemmSmemBytes, gemm_tc_kernel<EPI>, tw, tx, tx_lo, p);
}

template <int HD>
void launch_attention_hd(cudaStream_t s, bool pdl, dim3 grid, int G, const AttnParams &p) {
    switch (G) {
        case 1: launch(s, pdl, grid, dim3(kAttnThreads), 0, attn_rows_kernel<HD, 1>, p); break;
        case 2: launch(s, pdl, grid, dim3(kAttnThreads), 0, attn_rows_kernel<HD, 2>, p); break;
        case 4: launch(s, pdl, grid, dim3(kAttnThreads), 0, attn_rows_kernel<HD, 4>, p); break;
        case 6: launch(s, pdl, grid, dim3(kAttnThreads), 0, attn_rows_kernel<HD, 6>, p); break;
        case 8: launch(s, pdl, grid, dim3(kAttnThreads), 0, attn_rows_kernel<HD, 8>, p); break;
        default: throw SaraError(SARA_EINVAL, "n_heads / n_kv_heads must be 1, 2, 4, 6 or 8");
    }
}

void launch_attention(cudaStream_t s, bool pdl, int sms, int hd, const AttnParams &p) {
    dim3 grid(std::max(1, (sms * 4) / std::max(1, p.n_kv)), p.n_kv);
    const int G = p.n_heads / p.n_kv;
    switch (hd) {
        case 32: launch_attention_hd<32>(s, pdl, grid, G, p); break;
        case 64: launch_attention_hd<64>(s, pdl, grid, G, p); break;
        case 128: launch_attention_hd<128>(s, pdl, grid, G, p); break;
        default: throw SaraError(SARA_EINVAL, "head_dim must be 32, 64 or 128");
    }
}

GemmParams gemm_base(const sara_handle &h, int m_tiles, int k_chunks, const Acts &A, const int *rows_dev) {
    GemmParams p{};
    p.m_tiles = m_tiles;
    p.k_chunks = k_chunks;
    p.rows_cap = A.rows_cap;
    p.rows_dev = rows_dev;
    p.decode = 0;
    p.ws_acc = h.gemm_acc;
    p.ws_cnt = h.gemm_cnt;
    p.err = &h.vars->err;
    p.ssq_tiles = h.cfg.d_model / 128;
    p.inv_dim = 1.0f / (float)h.cfg.d_model;
    p.eps = h.cfg.rms_eps;
    p.stamps = h.stamps;
    return p;
}

enum Kern { K_QKV = 1, K_ATTN = 2, K_OPROJ = 3, K_GATEUP = 4, K_DOWN = 5 };

// Launch one projection / attention kernel of layer l over the prefill rows (one row per
// fresh prompt token, KV = the prompt slots).  Weights are read from the blocked tiles.
void enqueue_prefill_kernel(sara_handle &h, cudaStream_t s, int which, int l, bool pdl) {
    const sara_model_cfg &m = h.cfg;
    const StepPtrs &c = h.ptrs;
    Acts &A = h.pre;
    const int *rows_dev = &h.vars->pre_rows;
    const int d = m.d_model, H = m.n_heads, KVH = m.n_kv_heads, hd = m.head_dim, F = m.ffn;
    const int G = h.sms;
    const bool last = l == m.layers - 1;
    uint16_t *kv_l = h.kv_pr + l * h.kv_pr_layer;
    switch (which) {
        case K_QKV: {
            GemmParams p = gemm_base(h, (H + 2 * KVH) * hd / 128, d / 64, A, rows_dev);
            p.w_blk = h.wb_qkv + l * h.ls_qkv;
            p.ssq = A.ssq_a;
            p.q_out = A.q;
            p.n_heads = H;
            p.n_kv = KVH;
            p.head_dim = hd;
            p.rope = h.rope;
            p.row_pos = c.pre_pos;
            p.row_slot = c.pre_slot;
            p.kv = kv_l;
            p.kv_slot_stride = h.kv_pr_slot;
            p.kv_cap = h.cap_p;
            launch_gemm<EPI_QKV>(s, pdl, G, A.tm_xg, A.tm_xg, A.tm_xg_lo, p);
            break;
        }
        case K_ATTN: {
            AttnParams a{};
            a.q = A.q;
            a.out = A.att;
            a.out_lo = A.att_lo;
            a.kv = kv_l;
            a.slot_stride = h.kv_pr_slot;
            a.cap = h.cap_p;
            a.row_slot = c.pre_slot;
            a.row_pos = c.pre_pos;
            a.items = c.pre_items;
            a.n_items_dev = &h.vars->pre_rows;
            a.row_item0 = c.pre_item0;
            a.n_heads = H;
            a.n_kv = KVH;
            a.chunk = h.cap_p;  // one split per row
            a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)hd));
            a.part = h.attn_part;
            a.cnt = h.attn_cnt;
            a.err = &h.vars->err;
            a.stamps = h.stamps;
            launch_attention(s, pdl, h.sms, hd, a);
            break;
        }
        case K_OPROJ: {
            GemmParams p = gemm_base(h, d / 128, H * hd / 64, A, rows_dev);
            p.w_blk = h.wb_o + l * h.ls_o;
            p.x_f32 = A.x_f32;
            p.xg_out = A.xg;
            p.xg_lo = A.xg_lo;
            p.g_next = h.norm_mlp + (size_t)l * d;
            p.ssq_out = A.ssq_m;
            p.ld = d;
            launch_gemm<EPI_RESID>(s, pdl, G, A.tm_att, A.tm_att, A.tm_att_lo, p);
            break;
        }
        case K_GATEUP: {
            GemmParams p = gemm_base(h, 2 * F / 128, d / 64, A, rows_dev);
            p.w_blk = h.wb_gu + l * h.ls_gu;
            p.ssq = A.ssq_m;
            p.h_out = A.h;
            p.h_lo = A.h_lo;
            p.ld = F;
            launch_gemm<EPI_SWIGLU>(s, pdl, G, A.tm_xg, A.tm_xg, A.tm_xg_lo, p);
            break;
        }
        case K_DOWN: {
            GemmParams p = gemm_base(h, d / 128, F / 64, A, rows_dev);
            p.w_blk = h.wb_down + l * h.ls_down;
            p.x_f32 = A.x_f32;
            p.xg_out = A.xg;
            p.xg_lo = A.xg_lo;
            p.g_next = last ? h.final_norm : h.norm_attn + (size_t)(l + 1) * d;
            p.ssq_out = A.ssq_a;
            p.ld = d;
            launch_gemm<EPI_RESID>(s, pdl, G, A.tm_h, A.tm_h, A.tm_h_lo, p);
            break;
        }
        default: throw SaraError(SARA_EINVAL, "unknown kernel id");
    }
}

MegaParams mega_params(const sara_handle &h) {
    const sara_model_cfg &m = h.cfg;
    MegaParams p{};
    p.layers = m.layers;
    p.d = m.d_model;
    p.H = m.n_heads;
    p.KVH = m.n_kv_heads;
    p.hd = m.head_dim;
    p.F = m.ffn;
    p.V = m.vocab;
    p.Gq = m.n_heads / m.n_kv_heads;
    p.nqkv = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim;
    p.eps = m.rms_eps;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)m.head_dim));
    p.w_qkv = h.wb_qkv;
    p.w_o = h.wb_o;
    p.w_gu = h.wb_gu;
    p.w_down = h.wb_down;
    p.w_lm = h.wb_lm;
    p.ls_qkv = h.ls_qkv;
    p.ls_o = h.ls_o;
    p.ls_gu = h.ls_gu;
    p.ls_down = h.ls_down;
    p.embed = h.embed;
    p.attn_norm = h.norm_attn;
    p.mlp_norm = h.norm_mlp;
    p.final_norm = h.final_norm;
    p.rope = h.rope;
    p.kv = h.kv_seq;
    p.kv_layer = h.kv_seq_layer;
    p.c = h.ptrs;
    p.rows_cap = m.max_seqs;
    p.rows_cap16 = h.rows_cap16;
    p.x = h.dx;
    p.xg = h.xg;
    p.att = h.att;
    p.hm = h.hm;
    p.ssqA = h.ssqA;
    p.ssqM = h.ssqM;
    p.gpart = h.gpart;
    p.qkv16 = h.qkv16;
    p.gp_qkv = h.gp_qkv;
    p.gp_o = h.gp_o;
    p.part = h.attn_part;
    p.att_cnt = h.attn_cnt;
    p.logits = h.logit_buf;
    p.write_logits = 0;
    p.cnt = h.phase_cnt;
    p.epoch = h.phase_cnt + (size_t)h.n_phase_cnt * kCntStride;
    p.stamps = h.stamps;
    p.n_stamp_ph = h.n_phase_cnt + 1 + kDetailRows;  // phases, kernel start, detail stamps
    p.ktime = &h.vars->kt0;
    return p;
}

// One decode step over the live rows: the persistent decode-step kernel (embedding, every
// layer, lm_head with the fused Gumbel-max maxima) followed by the sampling finish and
// bookkeeping kernel.  write_logits: also store the fp32 logits (teacher forcing).
void enqueue_decode_step(sara_handle &h, cudaStream_t s, bool write_logits = false) {
    MegaParams mp = mega_params(h);
    mp.write_logits = write_logits ? 1 : 0;
    launch_ex(s, false, true, dim3(h.sms), dim3(kMegaThreads), kMegaSmemBytes, decode_step_kernel, mp);
    launch(s, false, dim3(h.cfg.max_seqs), dim3(256), 0, sample_finish_kernel, h.ptrs, h.cfg.vocab);
}

// Prefill of the fresh prompts of a round: embedding, every layer up to the last layer's
// K/V (the prompt's last hidden state is not needed: its last token is the rollouts' first
// decode row).
void enqueue_prefill(sara_handle &h, cudaStream_t s, bool pdl) {
    const sara_model_cfg &m = h.cfg;
    const StepPtrs &c = h.ptrs;
    Acts &A = h.pre;
    launch(s, false, dim3(A.rows_cap), dim3(128), 0, embed_kernel, (const uint16_t *)h.embed,
           (const uint16_t *)h.norm_attn, (const int *)&h.vars->pre_rows, (const int *)c.pre_tok, m.d_model,
           A.rows_cap, m.vocab, A.x_f32, A.xg, A.xg_lo, A.ssq_a, &h.vars->err);
    for (int l = 0; l < m.layers; ++l) {
        enqueue_prefill_kernel(h, s, K_QKV, l, pdl);
        if (l == m.layers - 1) break;
        enqueue_prefill_kernel(h, s, K_ATTN, l, pdl);
        enqueue_prefill_kernel(h, s, K_OPROJ, l, pdl);
        enqueue_prefill_kernel(h, s, K_GATEUP, l, pdl);
        enqueue_prefill_kernel(h, s, K_DOWN, l, pdl);
    }
}

void enqueue_prompt_blocks(sara_handle &h, cudaStream_t s, bool pdl, const StepPtrs &c) {
    const sara_model_cfg &m = h.cfg;
    launch(s, pdl, dim3(h.sms * 8), dim3(256), 0, prompt_blocks_kernel, (const uint16_t *)h.kv_pr, h.kv_seq, c,
           m.layers, m.n_kv_heads, m.head_dim, h.cap_p, h.kv_seq_layer, m.max_active);
}


// ------------------------------------------------------------------------ graph
void build_graph(sara_handle &h) {
    const bool pdl = h.use_pdl;
    CK(cudaGraphCreate(&h.graph, 0));
    CondHandles hs{};
    CK(cudaGraphConditionalHandleCreate(&hs.h[0], h.graph, 1, cudaGraphCondAssignDefault));
    cudaGraphNodeParams wp{};
    wp.type = cudaGraphNodeTypeConditional;
    wp.conditional.handle = hs.h[0];
    wp.conditional.type = cudaGraphCondTypeWhile;
    wp.conditional.size = 1;
    cudaGraphNode_t wnode;
    CK(cudaGraphAddNode(&wnode, h.graph, nullptr, nullptr, 0, &wp));
    cudaGraph_t body = wp.conditional.phGraph_out[0];
    if (h.has_model) {
        CK(cudaGraphConditionalHandleCreate(&hs.h[1], body, 0, cudaGraphCondAssignDefault));
        CK(cudaGraphConditionalHandleCreate(&hs.h[2], body, 0, cudaGraphCondAssignDefault));
    }
    cudaStream_t cs = h.cap_stream;
    CK(cudaStreamBeginCaptureToGraph(cs, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
    launch(cs, false, dim3(1), dim3(kCtlThreads), 0, ctl_kernel, h.ptrs, hs, h.has_model ? 3 : 1);
    if (h.has_model) {
        // IF(fresh prompts) { prefill }, then IF(new rollouts) { KV blocks of the new rollouts }
        auto add_if = [&](cudaGraphConditionalHandle hc, const std::function<void(cudaStream_t)> &fill) {
            cudaStreamCaptureStatus st;
            cudaGraph_t capg;
            const cudaGraphNode_t *deps = nullptr;
            size_t ndeps = 0;
            CK(cudaStreamGetCaptureInfo(cs, &st, nullptr, &capg, &deps, nullptr, &ndeps));
            std::vector<cudaGraphNode_t> dv(deps, deps + ndeps);
            cudaGraphNodeParams ip{};
            ip.type = cudaGraphNodeTypeConditional;
            ip.conditional.handle = hc;
            ip.conditional.type = cudaGraphCondTypeIf;
            ip.conditional.size = 1;
            cudaGraphNode_t inode;
            CK(cudaGraphAddNode(&inode, capg, dv.data(), nullptr, dv.size(), &ip));
            CK(cudaStreamUpdateCaptureDependencies(cs, &inode, nullptr, 1, cudaStreamSetCaptureDependencies));
            cudaGraph_t ibody = ip.conditional.phGraph_out[0];
            CK(cudaStreamBeginCaptureToGraph(h.cap_stream2, ibody, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
            fill(h.cap_stream2);
            cudaGraph_t ib2;
            CK(cudaStreamEndCapture(h.cap_stream2, &ib2));
        };
        add_if(hs.h[2], [&](cudaStream_t st) { enqueue_prefill(h, st, pdl); });
        add_if(hs.h[1], [&](cudaStream_t st) { enqueue_prompt_blocks(h, st, pdl, h.ptrs); });
        enqueue_decode_step(h, cs);
    }
    cudaGraph_t b2;
    CK(cudaStreamEndCapture(cs, &b2));
    CK(cudaGraphInstantiate(&h.exec, h.graph, 0));
}

// Host-driven loop (debugging, SARA_GRAPH=0): the same kernels as the graph body, one
// iteration at a time, with the round-start branch decided on the host.
void run_host_loop(sara_handle &h, int schedule) {
    cudaStream_t s = h.stream;
    StepVars v{};
    for (;;) {
        launch(s, false, dim3(1), dim3(kCtlThreads), 0, ctl_kernel, h.ptrs, CondHandles{}, 0);
        CK(cudaMemcpyAsync(&v, h.vars, sizeof(v), cudaMemcpyDeviceToHost, s));
        CK(cudaStreamSynchronize(s));
        if (v.done || v.err) break;
        if (!h.has_model) continue;
        const bool joins = schedule != 0 ? v.n_new > 0 : (v.round_steps == 0 && v.live > 0);
        if (joins) {
            if (v.n_fresh > 0) enqueue_prefill(h, s, h.use_pdl);
            enqueue_prompt_blocks(h, s, h.use_pdl, h.ptrs);
        }
        enqueue_decode_step(h, s);
    }
}

// ------------------------------------------------------------------------ weights

// Copy a row-major bf16 matrix [N][K] (host or device) into blocked 16 KB tiles at dst,
// through the device staging buffer tmp.
void block_matrix(cudaStream_t s, const void *src, bool on_device, uint16_t *tmp, uint8_t *dst, int N, int K) {
    CK(cudaMemcpyAsync(tmp, src, (size_t)N * K * 2, on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
    launch(s, false, dim3(1024), dim3(256), 0, block_weights_kernel, (const uint16_t *)tmp, dst, N, K);
}

void load_weights(sara_handle &h, const sara_weights *w) {
    const sara_model_cfg &m = h.cfg;
    const int d = m.d_model, H = m.n_heads, KVH = m.n_kv_heads, hd = m.head_dim, F = m.ffn, V = m.vocab, L = m.layers;
    const bool dev = w->on_device != 0;
    cudaStream_t s = h.stream;
    if (!w->embed || !w->lm_head || !w->final_norm || !w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo ||
        !w->mlp_norm || !w->wgate || !w->wup || !w->wdown)
        throw SaraError(SARA_EINVAL, "a weight pointer is NULL");
    for (int l = 0; l < L; ++l)
        if (!w->attn_norm[l] || !w->wq[l] || !w->wk[l] || !w->wv[l] || !w->wo[l] || !w->mlp_norm[l] || !w->wgate[l] ||
            !w->wup[l] || !w->wdown[l])
            throw SaraError(SARA_EINVAL, "a per-layer weight pointer is NULL");
    const cudaMemcpyKind kind = dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    const int nqkv = (H + 2 * KVH) * hd;
    h.ls_qkv = (int64_t)nqkv * d * 2;
    h.ls_o = (int64_t)d * H * hd * 2;
    h.ls_gu = (int64_t)2 * F * d * 2;
    h.ls_down = (int64_t)d * F * 2;
    h.embed = h.mem.alloc<uint16_t>((size_t)V * d, false);
    h.final_norm = h.mem.alloc<uint16_t>(d, false);
    h.norm_attn = h.mem.alloc<uint16_t>((size_t)L * d, false);
    h.norm_mlp = h.mem.alloc<uint16_t>((size_t)L * d, false);
    h.wb_qkv = h.mem.alloc<uint8_t>((size_t)L * h.ls_qkv, false);
    h.wb_o = h.mem.alloc<uint8_t>((size_t)L * h.ls_o, false);
    h.wb_gu = h.mem.alloc<uint8_t>((size_t)L * h.ls_gu, false);
    h.wb_down = h.mem.alloc<uint8_t>((size_t)L * h.ls_down, false);
    h.wb_lm = h.mem.alloc<uint8_t>((size_t)V * d * 2, false);
    CK(cudaMemcpyAsync(h.embed, w->embed, (size_t)V * d * 2, kind, s));
    CK(cudaMemcpyAsync(h.final_norm, w->final_norm, (size_t)d * 2, kind, s));
    // staging buffer for one row-major matrix, freed when loading is done
    const size_t stage = std::max({(size_t)V * d, (size_t)nqkv * d, (size_t)2 * F * d, (size_t)d * H * hd});
    uint16_t *tmp = nullptr;
    if (cudaMalloc(&tmp, stage * 2) != cudaSuccess) throw SaraError(SARA_ENOMEM, "cudaMalloc of the weight staging buffer failed");
    try {
        block_matrix(s, w->lm_head, dev, tmp, h.wb_lm, V, d);
        for (int l = 0; l < L; ++l) {
            CK(cudaMemcpyAsync(h.norm_attn + (size_t)l * d, w->attn_norm[l], (size_t)d * 2, kind, s));
            CK(cudaMemcpyAsync(h.norm_mlp + (size_t)l * d, w->mlp_norm[l], (size_t)d * 2, kind, s));
            // fused q|k|v rows
            CK(cudaMemcpyAsync(tmp, w->wq[l], (size_t)H * hd * d * 2, kind, s));
            CK(cudaMemcpyAsync(tmp + (size_t)H * hd * d, w->wk[l], (size_t)KVH * hd * d * 2, kind, s));
            CK(cudaMemcpyAsync(tmp + (size_t)(H + KVH) * hd * d, w->wv[l], (size_t)KVH * hd * d * 2, kind, s));
            launch(s, false, dim3(1024), dim3(256), 0, block_weights_kernel, (const uint16_t *)tmp,
                   h.wb_qkv + l * h.ls_qkv, nqkv, d);
            block_matrix(s, w->wo[l], dev, tmp, h.wb_o + l * h.ls_o, d, H * hd);
            // gate/up interleaved in blocks of 64 rows: [g 0..63, u 0..63, g 64..127, u 64..127, ...]
            CK(cudaMemcpy2DAsync(tmp, (size_t)128 * d * 2, w->wgate[l], (size_t)64 * d * 2, (size_t)64 * d * 2, F / 64,
                                 kind, s));
            CK(cudaMemcpy2DAsync(tmp + (size_t)64 * d, (size_t)128 * d * 2, w->wup[l], (size_t)64 * d * 2,
                                 (size_t)64 * d * 2, F / 64, kind, s));
            launch(s, false, dim3(1024), dim3(256), 0, block_weights_kernel, (const uint16_t *)tmp,
                   h.wb_gu + l * h.ls_gu, 2 * F, d);
            block_matrix(s, w->wdown[l], dev, tmp, h.wb_down + l * h.ls_down, d, F);
        }
        CK(cudaStreamSynchronize(s));
    } catch (...) {
        cudaStreamSynchronize(s);
        cudaFree(tmp);
        throw;
    }
    CK(cudaFree(tmp));
}

void alloc_acts(sara_handle &h, Acts &A, int rows) {
    const sara_model_cfg &m = h.cfg;
    A.rows_cap = rows;
    const int d = m.d_model, Hhd = m.n_heads * m.head_dim;
    A.x_f32 = h.mem.alloc<float>((size_t)rows * d);
    A.xg = h.mem.alloc<uint16_t>((size_t)rows * d);
    A.xg_lo = h.mem.alloc<uint16_t>((size_t)rows * d);
    A.q = h.mem.alloc<uint16_t>((size_t)rows * Hhd);
    A.att = h.mem.alloc<uint16_t>((size_t)rows * Hhd);
    A.att_lo = h.mem.alloc<uint16_t>((size_t)rows * Hhd);
    A.h = h.mem.alloc<uint16_t>((size_t)rows * m.ffn);
    A.h_lo = h.mem.alloc<uint16_t>((size_t)rows * m.ffn);
    A.ssq_a = h.mem.alloc<float>((size_t)(d / 128) * rows);
    A.ssq_m = h.mem.alloc<float>((size_t)(d / 128) * rows);
}

// Decode-step buffers: residual stream, blocked hi/lo operands (rows padded to 16), the
// GEMM partial tiles and the phase counters.
void alloc_decode(sara_handle &h) {
    const sara_model_cfg &m = h.cfg;
    const int S = m.max_seqs, d = m.d_model, Hhd = m.n_heads * m.head_dim, F = m.ffn;
    const int nqkv = (m.n_heads + 2 * m.n_kv_heads) * m.head_dim;
    h.rows_cap16 = (S + 15) & ~15;
    const size_t R16 = h.rows_cap16;
    h.dx = h.mem.alloc<float>((size_t)S * d);
    h.xg = h.mem.alloc<uint8_t>(R16 * d * 4);
    h.att = h.mem.alloc<uint8_t>(R16 * Hhd * 4);
    h.hm = h.mem.alloc<uint8_t>(R16 * F * 4);
    h.ssqA = h.mem.alloc<float>((size_t)(d / 64) * S);
    h.ssqM = h.mem.alloc<float>((size_t)(d / 64) * S);
    // partial tiles: one segment per (CTA, tile) pair of a phase, at most CTAs + tiles - 1
    const int tmax = std::max({nqkv, d, 2 * F}) / kTileN + 1;
    h.gpart = h.mem.alloc<float>((size_t)(h.sms + tmax) * S * kTileN, false);
    h.qkv16 = h.mem.alloc<uint16_t>((size_t)S * nqkv, false);
    // the QKV and O projections are spread over few CTAs (each about one ring of weights)
    auto small = [&](int N, int K) {
        const int units = ((N + kTileN - 1) / kTileN) * (K / 64);
        return std::max(1, std::min(h.sms, units / kSmallPhaseUnits));
    };
    h.gp_qkv = small(nqkv, d);
    h.gp_o = small(d, Hhd);
    h.n_phase_cnt = 1 + kPhasesPerLayer * m.layers + 1;
    h.phase_cnt = h.mem.alloc<unsigned long long>(((size_t)h.n_phase_cnt + 1) * kCntStride);
}

// Phase counters and split counters back to zero (start of every call: a step that failed
// part-way may have left them anywhere).
// Decode attention units run at once per kv head: one per compute warp group (two per SM).
int att_slots(const sara_handle &h) {
    const int kvh = h.has_model ? std::max(1, h.cfg.n_kv_heads) : 1;
    return std::max(1, 2 * h.sms / kvh);
}

void reset_decode_state(sara_handle &h, cudaStream_t s) {
    const sara_model_cfg &m = h.cfg;
    CK(cudaMemsetAsync(h.phase_cnt, 0, ((size_t)h.n_phase_cnt + 1) * kCntStride * 8, s));
    CK(cudaMemsetAsync(h.attn_cnt, 0, (size_t)m.max_seqs * m.n_kv_heads * 4, s));
}

void make_tensor_maps(sara_handle &h) {
    const sara_model_cfg &m = h.cfg;
    const int d = m.d_model, H = m.n_heads, hd = m.head_dim, F = m.ffn;
    Acts *A = &h.pre;
    A->tm_xg = make_tmap_bf16(A->xg, d, A->rows_cap, kTileK, kXBoxRows);
    A->tm_xg_lo = make_tmap_bf16(A->xg_lo, d, A->rows_cap, kTileK, kXBoxRows);
    A->tm_att = make_tmap_bf16(A->att, H * hd, A->rows_cap, kTileK, kXBoxRows);
    A->tm_att_lo = make_tmap_bf16(A->att_lo, H * hd, A->rows_cap, kTileK, kXBoxRows);
    A->tm_h = make_tmap_bf16(A->h, F, A->rows_cap, kTileK, kXBoxRows);
    A->tm_h_lo = make_tmap_bf16(A->h_lo, F, A->rows_cap, kTileK, kXBoxRows);
}

void validate_cfg(const sara_model_cfg &m) {
    auto bad = [](const char *msg) { throw SaraError(SARA_EINVAL, msg); };
    if (m.max_prompts < 1 || m.max_active < 1 || m.max_k < 2 || m.max_k > kMaxK) bad("capacities out of range (max_k 2..64)");
    if (m.max_active > 8192) bad("max_active must be <= 8192");
    if (m.layers < 0) bad("layers < 0");
    if (m.layers == 0) return;
    if (m.d_model % 128 || m.d_model < 128 || m.d_model > 2048) bad("d_model must be a multiple of 128 in [128, 2048]");
    if (m.head_dim != 32 && m.head_dim != 64 && m.head_dim != 128) bad("head_dim must be 32, 64 or 128");
    if (m.n_kv_heads < 1 || m.n_heads % m.n_kv_heads)
        bad("n_heads must be a multiple of n_kv_heads");
    {
        const int G = m.n_heads / m.n_kv_heads;
        if (G != 1 && G != 2 && G != 4 && G != 6 && G != 8) bad("n_heads / n_kv_heads must be 1, 2, 4, 6 or 8");
    }
    if ((m.max_prompt_len + m.max_gen_len + kDecodeChunk - 1) / kDecodeChunk > kAttnMaxSplits)
        bad("max_prompt_len + max_gen_len exceeds the attention split capacity (96 x 128 positions)");
    if ((m.n_heads * m.head_dim) % 128 || ((m.n_heads + 2 * m.n_kv_heads) * m.head_dim) % 128)
        bad("head dims must tile by 128");
    if (m.ffn % 64 || m.ffn < 64) bad("ffn must be a multiple of 64");
    if (m.vocab % 128 || m.vocab < 128) bad("vocab must be a multiple of 128");
    if (m.max_seqs < 1 || m.max_seqs > kTileR) bad("max_seqs must be 1..128");
    if (m.max_prompt_len < 2 || m.max_gen_len < 1) bad("max_prompt_len >= 2 and max_gen_len >= 1 required");
    if (m.kv_blocks < 0) bad("kv_blocks < 0");
    if (!(m.rms_eps > 0.f) || !(m.rope_theta > 0.f)) bad("rms_eps and rope_theta must be positive");
}

void create_impl(sara_handle &h, const sara_model_cfg *cfgp, const sara_weights *w, void *stream) {
    if (!cfgp) throw SaraError(SARA_EINVAL, "cfg is NULL");
    h.cfg = *cfgp;
    sara_model_cfg &m = h.cfg;
    validate_cfg(m);
    h.has_model = m.layers > 0;
    if (h.has_model && !w) throw SaraError(SARA_EINVAL, "weights are NULL");
    h.stream = static_cast<cudaStream_t>(stream);
    CK(cudaGetDevice(&h.device));
    CK(cudaDeviceGetAttribute(&h.sms, cudaDevAttrMultiProcessorCount, h.device));
    int major = 0;
    CK(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, h.device));
    if (major != 10) throw SaraError(SARA_EDEVICE, "this library is built for sm_103a (GB300)");
    set_kernel_attrs();
    CK(cudaStreamCreateWithFlags(&h.cap_stream, cudaStreamNonBlocking));
    CK(cudaStreamCreateWithFlags(&h.cap_stream2, cudaStreamNonBlocking));
    CK(cudaEventCreate(&h.ev0));
    CK(cudaEventCreate(&h.ev1));

    const int P = m.max_prompts, Bc = m.max_active, K = m.max_k;
    h.kc = h.mem.alloc<StepConst>(1);
    h.vars = h.mem.alloc<StepVars>(1);
    StepPtrs &c = h.ptrs;
    c.kc = h.kc;
    c.v = h.vars;
    h.p_thr = h.mem.alloc<uint64_t>(P);
    h.p_len = h.mem.alloc<int32_t>((size_t)P * K);
    c.p_thr = h.p_thr;
    c.p_len = h.p_len;
    c.q_status = h.mem.alloc<uint8_t>(P);
    c.q_n = h.mem.alloc<uint8_t>(P);
    c.q_pa = h.mem.alloc<double>(P);
    c.q_pb = h.mem.alloc<double>(P);
    c.q_key = h.mem.alloc<double>((size_t)Bc + 1);
    h.prior_next = h.mem.alloc<double>((size_t)2 * P);
    c.q_s = h.mem.alloc<uint8_t>(P);
    c.q_round = h.mem.alloc<int16_t>(P);
    c.q_pslot = h.mem.alloc<int32_t>(P);
    c.act = h.mem.alloc<int32_t>(Bc + 1);
    c.act_tmp = h.mem.alloc<int32_t>(Bc + 1);
    c.iss_q = h.mem.alloc<int32_t>(Bc + 1);
    c.iss_c = h.mem.alloc<int32_t>(Bc + 1);
    c.fresh_pslot = h.mem.alloc<int32_t>(Bc + 1);
    c.dec_tab = h.mem.alloc<uint8_t>(kTabDim * kTabDim);
    c.rank_tab = h.mem.alloc<uint8_t>(kTabDim * kTabDim);
    c.max_active = Bc;
    if (h.has_model) {
        const int S = m.max_seqs, d = m.d_model, KVH = m.n_kv_heads, hd = m.head_dim;
        h.p_tok = h.mem.alloc<int32_t>((size_t)P * m.max_prompt_len);
        c.p_tok = h.p_tok;
        c.seq_q = h.mem.alloc<int32_t>(S);
        c.seq_j = h.mem.alloc<int32_t>(S);
        c.seq_len = h.mem.alloc<int32_t>(S);
        c.seq_gen = h.mem.alloc<int32_t>(S);
        c.seq_pslot = h.mem.alloc<int32_t>(S);
        c.seq_uid = h.mem.alloc<int64_t>(S);
        c.row_slot = h.mem.alloc<int32_t>(S);
        c.row_pos = h.mem.alloc<int32_t>(S);
        c.row_tok = h.mem.alloc<int32_t>(S);
        c.row_item0 = h.mem.alloc<int32_t>(S);
        c.row_seed = h.mem.alloc<uint64_t>(S);
        c.sampled = h.mem.alloc<int32_t>(S);
        h.cap_p = m.max_prompt_len;
        h.cap_s = m.max_prompt_len + m.max_gen_len;
        h.att_cap = S * ((h.cap_s + kDecodeChunk - 1) / kDecodeChunk);
        c.att_items = h.mem.alloc<int2>(h.att_cap);
        c.att_cap = h.att_cap;
        h.pre_cap = std::min(Bc, S) * (m.max_prompt_len - 1);
        c.pre_cap = h.pre_cap;
        c.pre_slot = h.mem.alloc<int32_t>(h.pre_cap);
        c.pre_pos = h.mem.alloc<int32_t>(h.pre_cap);
        c.pre_tok = h.mem.alloc<int32_t>(h.pre_cap);
        c.pre_item0 = h.mem.alloc<int32_t>(h.pre_cap);
        c.pre_items = h.mem.alloc<int2>(h.pre_cap);
        c.max_seqs = S;
        h.gen_tok = h.mem.alloc<int32_t>((size_t)P * K * m.max_gen_len, false);
        c.gen_tok = h.gen_tok;
        // Paged KV cache of 128-position blocks in the decode layout (64 KB per block and kv
        // head, zero-filled so padded head dims read as 0): the prompts' full blocks (shared by
        // their rollouts), then the rollouts' private blocks, handed out as positions are
        // reached and returned when a rollout finishes.  Prompt slots row-major
        // [layer][pslot][2][kv][cap_p][hd] (the prefill's own layout).
        c.nblk_max = (h.cap_s + kKVPos - 1) / kKVPos;
        c.nsh_max = shared_blocks(m.max_prompt_len, kKVPos);
        c.n_shared = Bc * c.nsh_max;
        c.n_priv = m.kv_blocks > 0 ? m.kv_blocks : S * ((m.max_gen_len + kKVPos - 1) / kKVPos + 2);
        c.blk_tab = h.mem.alloc<int32_t>((size_t)S * c.nblk_max);
        c.blk_free = h.mem.alloc<int32_t>((size_t)c.n_priv);
        c.new_slots = h.mem.alloc<int32_t>((size_t)S);
        c.q_inflight = h.mem.alloc<int32_t>((size_t)P);
        c.dec_list = h.mem.alloc<int32_t>((size_t)std::max(Bc, S) + 1);
        c.slot_free = h.mem.alloc<int32_t>((size_t)S);
        c.pslot_free = h.mem.alloc<int32_t>((size_t)Bc);
        h.kv_seq_layer = (int64_t)(c.n_shared + c.n_priv) * KVH * kKVBlockBytes;
        h.kv_pr_slot = 2LL * KVH * h.cap_p * hd;
        h.kv_pr_layer = h.kv_pr_slot * Bc;
        h.kv_seq = h.mem.alloc<uint8_t>((size_t)h.kv_seq_layer * m.layers);
        h.kv_pr = h.mem.alloc<uint16_t>((size_t)h.kv_pr_layer * m.layers);
        // rotary table: angle = pos * theta^(-2i/hd), computed in double
        std::vector<float2> rope((size_t)h.cap_s * (hd / 2));
        for (int pos = 0; pos < h.cap_s; ++pos)
            for (int i = 0; i < hd / 2; ++i) {
                const double a = (double)pos * std::pow((double)m.rope_theta, -2.0 * i / hd);
                rope[(size_t)pos * (hd / 2) + i] = make_float2((float)std::cos(a), (float)std::sin(a));
            }
        h.rope = h.mem.alloc<float2>(rope.size(), false);
        CK(cudaMemcpy(h.rope, rope.data(), rope.size() * sizeof(float2), cudaMemcpyHostToDevice));
        alloc_acts(h, h.pre, h.pre_cap);
        alloc_decode(h);
        // GEMM stream-K workspace: one fixed-point tile sum per CTA + per-tile counters (zeroed)
        h.gemm_acc = h.mem.alloc<unsigned long long>((size_t)h.sms * kTileR * kTileM);
        const int max_m = std::max({(m.n_heads + 2 * KVH) * hd, d, 2 * m.ffn, m.vocab}) / 128;
        h.gemm_cnt = h.mem.alloc<int>((size_t)max_m * ((h.pre_cap + kTileR - 1) / kTileR + 1));
        const int Gq = m.n_heads / KVH;
        h.attn_part = h.mem.alloc<float>((size_t)h.att_cap * KVH * Gq * (hd + 2), false);
        h.attn_cnt = h.mem.alloc<int>((size_t)S * KVH);
        // the lm_head epilogue's sampler maxima: [rows][2 per 256-token tile]
        c.lm_tiles = (m.vocab + kTileN - 1) / kTileN;
        h.lm_val = h.mem.alloc<float>((size_t)S * 2 * c.lm_tiles, false);
        h.lm_idx = h.mem.alloc<int>((size_t)S * 2 * c.lm_tiles, false);
        h.logit_buf = h.mem.alloc<float>((size_t)S * m.vocab, false);
        c.arg_val = h.lm_val;
        c.arg_idx = h.lm_idx;
        load_weights(h, w);
        make_tensor_maps(h);
    }
    const char *eg = getenv("SARA_GRAPH");
    const char *ep = getenv("SARA_PDL");
    h.use_graph = !(eg && eg[0] == '0');
    h.use_pdl = !(ep && ep[0] == '0');
    if (h.use_graph) build_graph(h);
    CK(cudaStreamSynchronize(h.stream));
}

void check_step_error(const StepVars &v) {
    if (v.err & ERR_WAIT_TIMEOUT) throw SaraError(SARA_ETIMEOUT, "a bounded device wait timed out");
    if (v.err & ERR_ITER_BOUND) throw SaraError(SARA_ETIMEOUT, "the step exceeded its iteration bound");
    if (v.err & ERR_CAPACITY) throw SaraError(SARA_ENOMEM, "a round exceeded the handle's capacities");
    if (v.err & ERR_BOUNDS) throw SaraError(SARA_EINVAL, "a token id or rollout length was out of range");
    if (v.err) throw SaraError(SARA_EDEVICE, "device consistency check failed (err=" + std::to_string(v.err) + ")");
}

void collect_impl(sara_handle &h, const sara_prompts *pr, int64_t N, int32_t k, int32_t n0, const sara_thresholds *t,
                  uint64_t reward_seed, sara_result *out) {
    const sara_model_cfg &m = h.cfg;
    if (!pr || !t || !out) throw SaraError(SARA_EINVAL, "NULL argument");
    const int P = pr->n_prompts, Lp = pr->prompt_len;
    if (P < 0 || P > m.max_prompts) throw SaraError(SARA_ENOMEM, "n_prompts exceeds max_prompts");
    if (k < 2 || k > std::min(kMaxK, m.max_k)) throw SaraError(SARA_EINVAL, "k out of range");
    if (n0 < 1 || n0 > k) throw SaraError(SARA_EINVAL, "n0 out of range");
    if (N < 0) throw SaraError(SARA_EINVAL, "N < 0");
    if (t->tau_den < 1 || t->tau_den > 2147483647LL || t->tau_num < 0 || t->tau_num > t->tau_den)
        throw SaraError(SARA_EINVAL, "tau_low must be num/den in [0, 1] with 0 < den < 2^31");
    const int cm = t->commit_min == 0 ? k : t->commit_min;
    if (cm < 2 || cm > k) throw SaraError(SARA_EINVAL, "commit_min out of range");
    if (t->alpha0 < 1 || t->alpha0 > 8 || t->beta0 < 1 || t->beta0 > 8)
        throw SaraError(SARA_EINVAL, "prior out of range (1..8)");
    if (t->target_B < 1 || t->target_B > m.max_active) throw SaraError(SARA_EINVAL, "target_B out of range");
    if (P > 0 && (!pr->p_threshold || !pr->lengths)) throw SaraError(SARA_EINVAL, "p_threshold / lengths are NULL");
    if (t->schedule < 0 || t->schedule > 2) throw SaraError(SARA_EINVAL, "schedule must be 0, 1 or 2");
    const bool warm = pr->prior_a != nullptr || pr->prior_b != nullptr;
    if (warm && (!pr->prior_a || !pr->prior_b)) throw SaraError(SARA_EINVAL, "prior_a and prior_b go together");
    if (!(t->decay >= 0.0 && t->decay <= 1.0)) throw SaraError(SARA_EINVAL, "decay must be in [0, 1]");
    if (warm && !pr->on_device) {
        for (int q = 0; q < P; ++q)
            if (!(pr->prior_a[q] > 0.0 && pr->prior_b[q] > 0.0 && pr->prior_a[q] < 1e12 && pr->prior_b[q] < 1e12))
                throw SaraError(SARA_EINVAL, "warm-start priors must be positive and finite");
    }
    if (h.has_model) {
        if (Lp < 2 || Lp > m.max_prompt_len) throw SaraError(SARA_EINVAL, "prompt_len out of range");
        if (P > 0 && !pr->tokens) throw SaraError(SARA_EINVAL, "tokens are NULL");
        if ((int64_t)t->target_B * n0 > m.max_seqs) throw SaraError(SARA_ENOMEM, "target_B * n0 exceeds max_seqs");
    } else if (Lp < 1) {
        throw SaraError(SARA_EINVAL, "prompt_len < 1");
    }
    // host-resident inputs are validated here; device-resident ones by the kernels (error word)
    if (!pr->on_device && h.has_model) {
        for (int64_t i = 0; i < (int64_t)P * k; ++i)
            if (pr->lengths[i] < 1 || pr->lengths[i] > m.max_gen_len)
                throw SaraError(SARA_EINVAL, "a rollout length is outside [1, max_gen_len]");
        for (int64_t i = 0; i < (int64_t)P * Lp; ++i)
            if (pr->tokens[i] < 0 || pr->tokens[i] >= m.vocab)
                throw SaraError(SARA_EINVAL, "a prompt token id is outside [0, vocab)");
    }
    cudaStream_t s = h.stream;
    const cudaMemcpyKind kin = pr->on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    StepConst K{};
    K.P = P; K.Lp = Lp; K.k = k; K.n0 = n0; K.commit_min = cm; K.a0 = t->alpha0; K.b0 = t->beta0; K.B = t->target_B;
    K.N = N; K.tau_num = t->tau_num; K.tau_den = t->tau_den;
    K.reward_seed = reward_seed; K.sample_seed = t->sample_seed;
    K.decode = h.has_model ? 1 : 0;
    K.teacher = 0;
    K.max_gen = m.max_gen_len;
    K.attn_chunk = kDecodeChunk;
    K.att_slots = att_slots(h);
    K.max_iters = h.max_iters;
    K.stall_plus1 = h.stall_idx + 1;
    K.wait_ns = (int64_t)h.wait_ns;
    K.eager_softmax = h.eager_softmax;
    K.tau_f = (double)t->tau_num / (double)t->tau_den;
    K.warm = warm ? 1 : 0;
    K.schedule = t->schedule;

    CK(cudaMemcpyAsync(h.kc, &K, sizeof(K), cudaMemcpyHostToDevice, s));
    if (P > 0) {
        CK(cudaMemcpyAsync(h.p_thr, pr->p_threshold, (size_t)P * 8, kin, s));
        CK(cudaMemcpyAsync(h.p_len, pr->lengths, (size_t)P * k * 4, kin, s));
        if (h.has_model) CK(cudaMemcpyAsync(h.p_tok, pr->tokens, (size_t)P * Lp * 4, kin, s));
        if (warm) {
            CK(cudaMemcpyAsync(h.ptrs.q_pa, pr->prior_a, (size_t)P * 8, kin, s));
            CK(cudaMemcpyAsync(h.ptrs.q_pb, pr->prior_b, (size_t)P * 8, kin, s));
        }
    }
    // device time of the step: from here (inputs on the device) to the end of its last kernel
    CK(cudaEventRecord(h.ev0, s));
    if (h.has_model) reset_decode_state(h, s);
    launch(s, false, dim3(1), dim3(kCtlThreads), 0, ctl_init_kernel, h.ptrs);
    if (t->schedule != 0 && !h.has_model) {  // asynchronous schedule without decode: one event-loop kernel
        const int cap = std::min(m.max_active, kAsyncMaxInFlight);
        const size_t smem = (size_t)cap * sizeof(uint64_t);
        CK(cudaFuncSetAttribute(ctl_async_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        launch(s, false, dim3(1), dim3(kCtlThreads), smem, ctl_async_kernel, h.ptrs, t->schedule == 2 ? 1 : 0, cap);
    } else if (h.use_graph) {
        CK(cudaGraphLaunch(h.exec, s));
    } else {
        run_host_loop(h, t->schedule);
    }
    if (P > 0 && (out->prior_a_next || out->prior_b_next))
        launch(s, false, dim3((P + 255) / 256), dim3(256), 0, carry_prior_kernel, h.ptrs, t->decay, h.prior_next,
               h.prior_next + P);
    CK(cudaEventRecord(h.ev1, s));
    // results (one device -> host read per call)
    StepVars v{};
    const cudaMemcpyKind kout = out->on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
    CK(cudaMemcpyAsync(&v, h.vars, sizeof(v), cudaMemcpyDeviceToHost, s));
    std::vector<uint8_t> st(P);
    if (P > 0) {
        CK(cudaMemcpyAsync(st.data(), h.ptrs.q_status, P, cudaMemcpyDeviceToHost, s));
        if (out->status) CK(cudaMemcpyAsync(out->status, h.ptrs.q_status, P, kout, s));
        if (out->n) CK(cudaMemcpyAsync(out->n, h.ptrs.q_n, P, kout, s));
        if (out->s) CK(cudaMemcpyAsync(out->s, h.ptrs.q_s, P, kout, s));
        if (out->decided_round) CK(cudaMemcpyAsync(out->decided_round, h.ptrs.q_round, (size_t)P * 2, kout, s));
        if (out->prior_a_next) CK(cudaMemcpyAsync(out->prior_a_next, h.prior_next, (size_t)P * 8, kout, s));
        if (out->prior_b_next) CK(cudaMemcpyAsync(out->prior_b_next, h.prior_next + P, (size_t)P * 8, kout, s));
        if (out->tokens && h.has_model)
            CK(cudaMemcpyAsync(out->tokens, h.gen_tok, (size_t)P * k * m.max_gen_len * 4, kout, s));
    }
    CK(cudaStreamSynchronize(s));
    check_step_error(v);
    float ms = 0.f;
    CK(cudaEventElapsedTime(&ms, h.ev0, h.ev1));
    out->rollouts = v.used;
    out->gen_tokens = v.gen_tokens;
    out->prefill_tokens = v.drawn * (int64_t)(Lp - 1);
    out->decode_steps = h.has_model ? v.exec_steps : v.sched_steps;
    out->rounds = v.rounds_done;
    out->prompts_drawn = v.drawn;
    out->committed = out->abandoned = out->incomplete = 0;
    for (int q = 0; q < P; ++q) {
        out->committed += st[q] == ST_COMMITTED;
        out->abandoned += st[q] == ST_ABANDONED;
        out->incomplete += st[q] == ST_INCOMPLETE;
    }
    out->device_ms = ms;
    out->decode_kernel_ms = (double)v.kernel_ns * 1e-6;
    out->kv_blocks_peak = h.has_model ? (int64_t)(h.ptrs.n_priv - v.blk_low) : 0;
    if (h.has_model && v.exec_steps != v.sched_steps)
        throw SaraError(SARA_EDEVICE, "decode steps run (" + std::to_string(v.exec_steps) +
                                          ") differ from the schedule (" + std::to_string(v.sched_steps) + ")");
}

void teacher_impl(sara_handle &h, int n, int Lp, const int32_t *prompts, int T, const int32_t *forced,
                  const int64_t *uid, uint64_t sample_seed, float *logits, int32_t *sampled, int on_device) {
    const sara_model_cfg &m = h.cfg;
    if (!h.has_model) throw SaraError(SARA_EINVAL, "teacher forcing needs a model");
    if (n < 1 || n > std::min(m.max_seqs, m.max_active)) throw SaraError(SARA_EINVAL, "n_seq out of range");
    if (Lp < 2 || Lp > m.max_prompt_len || T < 1 || T > m.max_gen_len)
        throw SaraError(SARA_EINVAL, "prompt_len / T out of range");
    if (!prompts || !forced || !uid || !logits) throw SaraError(SARA_EINVAL, "NULL argument");
    if (!on_device) {
        for (int64_t i = 0; i < (int64_t)n * Lp; ++i)
            if (prompts[i] < 0 || prompts[i] >= m.vocab) throw SaraError(SARA_EINVAL, "a prompt token id is outside [0, vocab)");
        for (int64_t i = 0; i < (int64_t)n * T; ++i)
            if (forced[i] < 0 || forced[i] >= m.vocab) throw SaraError(SARA_EINVAL, "a forced token id is outside [0, vocab)");
    }
    cudaStream_t s = h.stream;
    const cudaMemcpyKind kin = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    const cudaMemcpyKind kout = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
    if ((size_t)n * T > h.forced_cap) {
        h.forced_cap = (size_t)n * T;
        h.forced = h.mem.alloc<int32_t>(h.forced_cap, false);
        h.sampled_out = h.mem.alloc<int32_t>(h.forced_cap, false);
    }
    if (!h.uid_dev) h.uid_dev = h.mem.alloc<int64_t>(m.max_seqs, false);
    StepConst K{};
    K.P = n; K.Lp = Lp; K.k = 2; K.n0 = 1; K.commit_min = 2; K.a0 = 1; K.b0 = 1; K.B = n; K.N = n;
    K.tau_num = 0; K.tau_den = 1; K.sample_seed = sample_seed; K.decode = 1; K.teacher = 1; K.T_forced = T;
    K.max_gen = m.max_gen_len; K.attn_chunk = kDecodeChunk; K.att_slots = att_slots(h);
    CK(cudaMemcpyAsync(h.kc, &K, sizeof(K), cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(h.p_tok, prompts, (size_t)n * Lp * 4, kin, s));
    CK(cudaMemcpyAsync(h.forced, forced, (size_t)n * T * 4, kin, s));
    CK(cudaMemcpyAsync(h.uid_dev, uid, (size_t)n * 8, kin, s));
    StepPtrs c = h.ptrs;  // the teacher's copy carries the forced-token buffers
    c.forced = h.forced;
    c.sampled_out = h.sampled_out;
    const StepPtrs saved = h.ptrs;
    h.ptrs = c;
    try {
        reset_decode_state(h, s);
        launch(s, false, dim3(1), dim3(kCtlThreads), 0, teacher_setup_kernel, c, n, (const int64_t *)h.uid_dev);
        enqueue_prefill(h, s, false);
        enqueue_prompt_blocks(h, s, false, c);
        for (int step = 0; step < T; ++step) {
            enqueue_decode_step(h, s, true);
            // rows stay in rollout order for all T steps (every rollout has length T)
            CK(cudaMemcpy2DAsync(logits + (size_t)step * m.vocab, (size_t)T * m.vocab * 4, h.logit_buf,
                                 (size_t)m.vocab * 4, (size_t)m.vocab * 4, n, kout, s));
        }
    } catch (...) {
        h.ptrs = saved;
        throw;
    }
    h.ptrs = saved;
    if (sampled) CK(cudaMemcpyAsync(sampled, h.sampled_out, (size_t)n * T * 4, kout, s));
    StepVars v{};
    CK(cudaMemcpyAsync(&v, h.vars, sizeof(v), cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
    check_step_error(v);
    if (v.live != 0 || v.exec_steps != T) throw SaraError(SARA_EDEVICE, "teacher forcing ran an unexpected number of steps");
}

#ifdef SARA_STAMPS
// Phase timeline of the last decode-step launch (profiling builds): for each phase kind,
// averaged over the middle layers, the time from the previous phase's completion (last CTA
// arrived) to this one's, the median delay until CTAs observed the dependency, and how far
// ahead of the previous phase's completion the W producer had issued this phase's copies.
void print_stamps(sara_handle &h, int rows, int ctx) {
    const int NP = h.n_phase_cnt + 1 + kDetailRows, G = h.sms, L = h.cfg.layers;
    std::vector<uint64_t> st((size_t)G * NP * 4);
    CK(cudaMemcpy(st.data(), h.stamps, st.size() * 8, cudaMemcpyDeviceToHost));
    auto at = [&](int c, int ph, int k) { return st[((size_t)c * NP + ph) * 4 + k]; };
    uint64_t t0 = ~0ull;
    for (int c = 0; c < G; ++c) t0 = std::min(t0, at(c, NP - kDetailRows - 1, 0));
    auto stat = [&](int ph, int k, bool mx) {
        std::vector<double> v;
        for (int c = 0; c < G; ++c)
            if (at(c, ph, k) >= t0) v.push_back((double)(at(c, ph, k) - t0) * 1e-3);
        if (v.empty()) return -1.0;
        std::sort(v.begin(), v.end());
        return mx ? v.back() : v[v.size() / 2];
    };
    const int NPH = 1 + kPhasesPerLayer * L + 1;
    std::vector<double> done(NPH);
    for (int ph = 0; ph < NPH; ++ph) done[ph] = stat(ph, 0, true);
    fprintf(stderr, "rows %d ctx %d: start->embed done %.2f us, lm_head done at %.2f us\n", rows, ctx, done[0],
            done[NPH - 1]);
    const char *names[kPhasesPerLayer] = {"QKV", "FIN_Q", "ATT", "O", "FIN_O", "GU", "FIN_GU", "DOWN", "FIN_D"};
    const int l0 = L > 4 ? 2 : 0, l1 = L > 4 ? L - 2 : L;
    for (int k = 0; k < kPhasesPerLayer; ++k) {
        double span = 0, obs = 0, wahead = 0, mma = 0;
        int n = 0;
        for (int l = l0; l < l1; ++l) {
            const int ph = 1 + kPhasesPerLayer * l + k;
            span += done[ph] - done[ph - 1];
            obs += stat(ph, 1, false) - done[ph - 1];
            wahead += done[ph - 1] - stat(ph, 2, false);
            mma += stat(ph, 3, false) - done[ph - 1];
            ++n;
        }
        fprintf(stderr, "  %-6s span %7.2f us  dep seen +%6.2f  W issued %+7.2f before  MMA done +%6.2f\n", names[k],
                span / n, obs / n, wahead / n, mma / n);
    }
    fprintf(stderr, "  LM     span %7.2f us\n", done[NPH - 1] - done[NPH - 2]);
    // detail stamps (layer 2): median over CTAs relative to the QKV phase's completion
    const int lq = std::min(2, L - 1);
    const double ref = done[1 + kPhasesPerLayer * lq];
    const char *dn[15] = {"att start", "q built", "S ready", "P ready", "O ready", "partial out", "split count",
                          "merged", "units done", "att arrived", "fin_o start", "fin_o work", "fin_o arrived",
                          "att dep seen", "att rstd"};
    for (int i = 0; i < 15; ++i) {
        std::vector<double> v;
        for (int c = 0; c < G; ++c) {
            const uint64_t x = at(c, NP - kDetailRows + i / 4, i % 4);
            if (x >= t0) v.push_back((double)(x - t0) * 1e-3 - ref);
        }
        std::sort(v.begin(), v.end());
        if (!v.empty())
            fprintf(stderr, "    %-14s n=%3zu  med %+7.2f  max %+7.2f us\n", dn[i], v.size(), v[v.size() / 2], v.back());
    }
    // gate / up units of layer 2 (medians over CTAs, relative to FIN_O's completion)
    const double ref_fo = done[1 + kPhasesPerLayer * lq + kPhFinO];
    fprintf(stderr, "    GU unit: W issued / W full / X full / MMA committed (us after FIN_O)\n");
    for (int j = 0; j < 12; ++j) {
        double med[4];
        int nn = 0;
        for (int kind = 0; kind < 4; ++kind) {
            std::vector<double> v;
            const int i = 16 + 12 * kind + j;
            for (int c = 0; c < G; ++c) {
                const uint64_t x = at(c, NP - kDetailRows + i / 4, i % 4);
                if (x >= t0) v.push_back((double)(x - t0) * 1e-3 - ref_fo);
            }
            std::sort(v.begin(), v.end());
            med[kind] = v.empty() ? 0.0 : v[v.size() / 2];
            nn = std::max(nn, (int)v.size());
        }
        fprintf(stderr, "      %2d n=%3d  %+7.2f %+7.2f %+7.2f %+7.2f\n", j, nn, med[0], med[1], med[2], med[3]);
    }
}
#endif

// Profiling hook: `rows` live rollouts at context `ctx` (synthetic row state), `iters`
// launches of the whole decode step (kernel 0: decode-step kernel + sampling/bookkeeping,
// positions advance) or of the decode-step kernel alone (kernel 1, positions fixed), timed
// with CUDA events on the handle's stream around a captured graph after two warm-up launches.
void profile_impl(sara_handle &h, int which, int rows, int ctx, int iters, double *ms) {
    const sara_model_cfg &m = h.cfg;
    if (!h.has_model) throw SaraError(SARA_EINVAL, "profiling needs a model");
    if (which < 0 || which > 1) throw SaraError(SARA_EINVAL, "unknown kernel id (0 = decode step, 1 = decode-step kernel)");
    if (rows < 1 || rows > m.max_seqs || iters < 1 || !ms) throw SaraError(SARA_EINVAL, "rows / iters out of range");
    const int steps = which == 0 ? 2 * iters + 2 : 0;  // the whole step advances positions
    if (ctx < 2 || ctx + steps + 1 > h.cap_s || steps + 1 > m.max_gen_len) throw SaraError(SARA_EINVAL, "ctx out of range");
    cudaStream_t s = h.stream;
    StepConst K{};
    K.P = 1; K.Lp = ctx; K.k = 2; K.n0 = 1; K.commit_min = 2; K.a0 = 1; K.b0 = 1; K.B = 1; K.N = 1;
    K.tau_num = 0; K.tau_den = 1; K.decode = 1; K.max_gen = m.max_gen_len; K.attn_chunk = kDecodeChunk;
    K.att_slots = att_slots(h);
    const int nblk = (ctx + kDecodeChunk - 1) / kDecodeChunk;
    const int span = att_span_for((int64_t)rows * nblk, K.att_slots, rows);
    const int nsplit = (nblk + span - 1) / span;
    std::vector<int> slot(rows), pos(rows, ctx - 1), tok(rows, 0), item0(rows), zero(rows, 0), len(rows, m.max_gen_len);
    std::vector<uint64_t> seed(rows);
    std::vector<int64_t> uid(rows);
    std::vector<int2> items;
    for (int r = 0; r < rows; ++r) {
        slot[r] = r;
        item0[r] = r * nsplit;
        seed[r] = 0x9E3779B97F4A7C15ull * (r + 1);
        uid[r] = r;
        for (int sp = 0; sp < nsplit; ++sp) items.push_back(make_int2(r, sp));
    }
    const StepPtrs &c = h.ptrs;
    // KV blocks: row r's blocks of positions < ctx are private ids (wrapping round the pool if
    // it is smaller: the values read are then another row's, which only timing sees); later
    // blocks come from a full free stack
    std::vector<int32_t> bt((size_t)rows * c.nblk_max, c.n_shared), fr(c.n_priv);
    for (int r = 0; r < rows; ++r)
        for (int j = 0; j < nblk; ++j) bt[(size_t)r * c.nblk_max + j] = c.n_shared + (r * nblk + j) % c.n_priv;
    for (int i = 0; i < c.n_priv; ++i) fr[i] = c.n_shared + c.n_priv - 1 - i;
    StepVars v{};
    v.kt0 = ~0ull;
    v.live = rows;
    v.att_items = rows * nsplit;
    v.att_span = span;
    v.round_maxL = 1 << 30;
    v.blk_top = v.blk_low = c.n_priv;
    reset_decode_state(h, s);
    CK(cudaMemcpyAsync(c.blk_tab, bt.data(), bt.size() * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.blk_free, fr.data(), fr.size() * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(h.kc, &K, sizeof(K), cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(h.vars, &v, sizeof(v), cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.row_slot, slot.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.row_pos, pos.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.row_tok, tok.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.row_item0, item0.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.row_seed, seed.data(), rows * 8, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.att_items, items.data(), items.size() * sizeof(int2), cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.seq_q, zero.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.seq_j, zero.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.seq_gen, zero.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.seq_len, len.data(), rows * 4, cudaMemcpyHostToDevice, s));
    CK(cudaMemcpyAsync(c.seq_uid, uid.data(), rows * 8, cudaMemcpyHostToDevice, s));
#ifdef SARA_STAMPS
    const size_t nst = (size_t)h.sms * (h.n_phase_cnt + 1 + kDetailRows) * 4;
    if (!h.stamps) h.stamps = h.mem.alloc<uint64_t>(nst);
#endif
    CK(cudaStreamSynchronize(s));
    auto one = [&](cudaStream_t st) {
        if (which == 0) {
            enqueue_decode_step(h, st);
        } else {
            launch_ex(st, false, true, dim3(h.sms), dim3(kMegaThreads), kMegaSmemBytes, decode_step_kernel,
                      mega_params(h));
        }
    };
    one(s);
    one(s);
    CK(cudaStreamSynchronize(s));
    // time the launches from a captured graph, so host launch cost is not measured
    cudaGraph_t g = nullptr;
    cudaGraphExec_t ge = nullptr;
    CK(cudaStreamBeginCapture(h.cap_stream, cudaStreamCaptureModeRelaxed));
    for (int i = 0; i < iters; ++i) one(h.cap_stream);
    CK(cudaStreamEndCapture(h.cap_stream, &g));
    CK(cudaGraphInstantiate(&ge, g, 0));
    CK(cudaGraphLaunch(ge, s));  // warm the graph
    CK(cudaStreamSynchronize(s));
    CK(cudaEventRecord(h.ev0, s));
    CK(cudaGraphLaunch(ge, s));
    CK(cudaEventRecord(h.ev1, s));
    CK(cudaStreamSynchronize(s));
    cudaGraphExecDestroy(ge);
    cudaGraphDestroy(g);
    float t = 0.f;
    CK(cudaEventElapsedTime(&t, h.ev0, h.ev1));
    CK(cudaMemcpy(&v, h.vars, sizeof(v), cudaMemcpyDeviceToHost));
    check_step_error(v);
    *ms = (double)t / iters;
#ifdef SARA_STAMPS
    if (which == 1) print_stamps(h, rows, ctx);
#endif
}

int guard(sara_handle *h, const std::function<void()> &fn) {
    try {
        fn();
        return SARA_OK;
    } catch (const SaraError &e) {
        if (h) h->err = e.what(); else g_create_error = e.what();
        return e.code;
    } catch (const std::exception &e) {
        if (h) h->err = e.what(); else g_create_error = e.what();
        return SARA_EDEVICE;
    }
}

}  // namespace

extern "C" {

int sara_create(const sara_model_cfg *cfg, const sara_weights *weights, void *stream, sara_handle **out) {
    if (!out) {
        g_create_error = "out is NULL";
        return SARA_EINVAL;
    }
    *out = nullptr;
    sara_handle *h = nullptr;
    try {
        h = new sara_handle();
    } catch (...) {
        g_create_error = "host allocation failed";
        return SARA_ENOMEM;
    }
    const int rc = guard(nullptr, [&] { create_impl(*h, cfg, weights, stream); });
    if (rc != SARA_OK) {
        delete h;
        return rc;
    }
    g_create_error.clear();
    *out = h;
    return SARA_OK;
}

int sara_collect_step(sara_handle *h, const sara_prompts *prompts, int64_t N, int32_t k, int32_t n0,
                      const sara_thresholds *thr, uint64_t reward_seed, sara_result *out) {
    if (!h) return SARA_EINVAL;
    return guard(h, [&] { collect_impl(*h, prompts, N, k, n0, thr, reward_seed, out); });
}

int sara_teacher_force(sara_handle *h, int32_t n_seq, int32_t prompt_len, const int32_t *prompts, int32_t T,
                       const int32_t *forced, const int64_t *uid, uint64_t sample_seed, float *logits,
                       int32_t *sampled, int32_t on_device) {
    if (!h) return SARA_EINVAL;
    return guard(h, [&] {
        teacher_impl(*h, n_seq, prompt_len, prompts, T, forced, uid, sample_seed, logits, sampled, on_device);
    });
}

int sara_profile(sara_handle *h, int32_t kernel, int32_t rows, int32_t ctx, int32_t iters, double *ms_per_launch) {
    if (!h) return SARA_EINVAL;
    return guard(h, [&] { profile_impl(*h, kernel, rows, ctx, iters, ms_per_launch); });
}

int sara_set_limits(sara_handle *h, const sara_limits *lim) {
    if (!h || !lim) return SARA_EINVAL;
    if (lim->wait_limit_ns < 0 || lim->max_loop_iters < 0 || lim->stall_phase < -1 ||
        (lim->eager_softmax != 0 && lim->eager_softmax != 1) || lim->reserved != 0 ||
        (h->has_model && lim->stall_phase >= h->n_phase_cnt)) {
        h->err = "limits out of range";
        return SARA_EINVAL;
    }
    h->wait_ns = (uint64_t)lim->wait_limit_ns;
    h->max_iters = lim->max_loop_iters;
    h->stall_idx = lim->stall_phase;
    h->eager_softmax = lim->eager_softmax;
    return SARA_OK;
}

int sara_abi_version(void) { return SARA_ABI_VERSION; }

const char *sara_last_error(const sara_handle *h) { return h ? h->err.c_str() : g_create_error.c_str(); }

void sara_destroy(sara_handle *h) {
    if (!h) return;
    cudaStreamSynchronize(h->stream);
    delete h;
}

}  // extern "C"
