// Host engine behind include/sara.h: device memory layout, weight packing, TMA descriptors,
// the step graph (a conditional WHILE loop whose body is controller -> [round start:
// prefill + prompt-KV fan-out] -> decode step -> sampling/bookkeeping), and the C ABI.
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

struct Acts {  // activation buffers of one row set (decode or prefill)
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
    // weights
    uint16_t *embed = nullptr, *lm_head = nullptr, *final_norm = nullptr;
    std::vector<uint16_t *> attn_norm, mlp_norm, w_qkv, w_o, w_gu, w_down;
    std::vector<CUtensorMap> tm_qkv, tm_o, tm_gu, tm_down;
    CUtensorMap tm_lm{};
    // KV caches
    uint16_t *kv_seq = nullptr, *kv_pr = nullptr;
    int cap_s = 0, cap_p = 0;
    int64_t kv_seq_layer = 0, kv_seq_slot = 0, kv_pr_layer = 0, kv_pr_slot = 0;
    float2 *rope = nullptr;
    Acts dec, pre;
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
    // teacher forcing staging (allocated on first use)
    float *logit_stage = nullptr;
    int32_t *forced = nullptr, *sampled_out = nullptr;
    int64_t *uid_dev = nullptr;
    size_t forced_cap = 0;
    uint64_t *stamps = nullptr;  // profiling builds: per-CTA phase timestamps of GEMM launches
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
    CK(cudaFuncSetAttribute(gemm_tc_kernel<EPI_LMHEAD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmemBytes));
    done = true;
}

template <typename Kern, typename... Args>
void launch(cudaStream_t s, bool pdl, dim3 grid, dim3 block, size_t smem, Kern kern, Args... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    CK(cudaLaunchKernelEx(&cfg, kern, args...));
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

GemmParams gemm_base(const sara_handle &h, int m_tiles, int k_chunks, const Acts &A, const int *rows_dev, bool decode) {
    GemmParams p{};
    p.m_tiles = m_tiles;
    p.k_chunks = k_chunks;
    p.rows_cap = A.rows_cap;
    p.rows_dev = rows_dev;
    p.decode = decode ? 1 : 0;
    p.ws_acc = h.gemm_acc;
    p.ws_cnt = h.gemm_cnt;
    p.err = &h.vars->err;
    p.ssq_tiles = h.cfg.d_model / 128;
    p.inv_dim = 1.0f / (float)h.cfg.d_model;
    p.eps = h.cfg.rms_eps;
    p.stamps = h.stamps;
    return p;
}

enum Kern { K_QKV = 1, K_ATTN = 2, K_OPROJ = 3, K_GATEUP = 4, K_DOWN = 5, K_LMHEAD = 6 };

// Launch one projection / attention kernel of layer l for a row set (decode: live rollouts,
// KV = rollout slots; prefill: fresh prompt tokens, KV = prompt slots).
void enqueue_kernel(sara_handle &h, cudaStream_t s, bool decode, int which, int l, bool pdl, float *logits_stage) {
    const sara_model_cfg &m = h.cfg;
    const StepPtrs &c = h.ptrs;
    Acts &A = decode ? h.dec : h.pre;
    const int *rows_dev = decode ? &h.vars->live : &h.vars->pre_rows;
    const int d = m.d_model, H = m.n_heads, KVH = m.n_kv_heads, hd = m.head_dim, F = m.ffn;
    const int G = h.sms;
    const bool last = l == m.layers - 1;
    uint16_t *kv_l = decode ? h.kv_seq + l * h.kv_seq_layer : h.kv_pr + l * h.kv_pr_layer;
    switch (which) {
        case K_QKV: {
            GemmParams p = gemm_base(h, (H + 2 * KVH) * hd / 128, d / 64, A, rows_dev, decode);
            p.ssq = A.ssq_a;
            p.q_out = A.q;
            p.n_heads = H;
            p.n_kv = KVH;
            p.head_dim = hd;
            p.rope = h.rope;
            p.row_pos = decode ? c.row_pos : c.pre_pos;
            p.row_slot = decode ? c.row_slot : c.pre_slot;
            p.kv = kv_l;
            p.kv_slot_stride = decode ? h.kv_seq_slot : h.kv_pr_slot;
            p.kv_cap = decode ? h.cap_s : h.cap_p;
            launch_gemm<EPI_QKV>(s, pdl, G, h.tm_qkv[l], A.tm_xg, A.tm_xg_lo, p);
            break;
        }
        case K_ATTN: {
            AttnParams a{};
            a.q = A.q;
            a.out = A.att;
            a.out_lo = A.att_lo;
            a.kv = kv_l;
            a.slot_stride = decode ? h.kv_seq_slot : h.kv_pr_slot;
            a.cap = decode ? h.cap_s : h.cap_p;
            a.row_slot = decode ? c.row_slot : c.pre_slot;
            a.row_pos = decode ? c.row_pos : c.pre_pos;
            a.items = decode ? c.att_items : c.pre_items;
            a.n_items_dev = decode ? &h.vars->att_items : &h.vars->pre_rows;
            a.row_item0 = decode ? c.row_item0 : c.pre_item0;
            a.n_heads = H;
            a.n_kv = KVH;
            a.chunk = decode ? kDecodeChunk : h.cap_p;  // prefill: one split per row
            a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)hd));
            a.part = h.attn_part;
            a.cnt = h.attn_cnt;
            a.err = &h.vars->err;
            a.stamps = h.stamps;
            launch_attention(s, pdl, h.sms, hd, a);
            break;
        }
        case K_OPROJ: {
            GemmParams p = gemm_base(h, d / 128, H * hd / 64, A, rows_dev, decode);
            p.x_f32 = A.x_f32;
            p.xg_out = A.xg;
            p.xg_lo = A.xg_lo;
            p.g_next = h.mlp_norm[l];
            p.ssq_out = A.ssq_m;
            p.ld = d;
            launch_gemm<EPI_RESID>(s, pdl, G, h.tm_o[l], A.tm_att, A.tm_att_lo, p);
            break;
        }
        case K_GATEUP: {
            GemmParams p = gemm_base(h, 2 * F / 128, d / 64, A, rows_dev, decode);
            p.ssq = A.ssq_m;
            p.h_out = A.h;
            p.h_lo = A.h_lo;
            p.ld = F;
            launch_gemm<EPI_SWIGLU>(s, pdl, G, h.tm_gu[l], A.tm_xg, A.tm_xg_lo, p);
            break;
        }
        case K_DOWN: {
            GemmParams p = gemm_base(h, d / 128, F / 64, A, rows_dev, decode);
            p.x_f32 = A.x_f32;
            p.xg_out = A.xg;
            p.xg_lo = A.xg_lo;
            p.g_next = last ? h.final_norm : h.attn_norm[l + 1];
            p.ssq_out = A.ssq_a;
            p.ld = d;
            launch_gemm<EPI_RESID>(s, pdl, G, h.tm_down[l], A.tm_h, A.tm_h_lo, p);
            break;
        }
        case K_LMHEAD: {
            GemmParams p = gemm_base(h, m.vocab / 128, d / 64, A, rows_dev, true);
            p.ssq = A.ssq_a;
            p.y_f32 = logits_stage;
            p.ld = m.vocab;
            p.row_seed = c.row_seed;
            p.arg_val = h.lm_val;
            p.arg_idx = h.lm_idx;
            launch_gemm<EPI_LMHEAD>(s, pdl, G, h.tm_lm, A.tm_xg, A.tm_xg_lo, p);
            break;
        }
        default: throw SaraError(SARA_EINVAL, "unknown kernel id");
    }
}

// One forward pass over a row set: embedding, every layer, and (decode) lm_head with fused
// sampling followed by the step bookkeeping.  Prefill stops after the last layer's K/V.
// The first kernel of the sequence is launched without PDL.
void enqueue_forward(sara_handle &h, cudaStream_t s, bool decode, bool pdl, float *logits_stage) {
    const sara_model_cfg &m = h.cfg;
    const StepPtrs &c = h.ptrs;
    Acts &A = decode ? h.dec : h.pre;
    const int *rows_dev = decode ? &h.vars->live : &h.vars->pre_rows;
    launch(s, false, dim3(A.rows_cap), dim3(128), 0, embed_kernel, (const uint16_t *)h.embed,
           (const uint16_t *)h.attn_norm[0], rows_dev, decode ? (const int *)c.row_tok : (const int *)c.pre_tok,
           m.d_model, A.rows_cap, m.vocab, A.x_f32, A.xg, A.xg_lo, A.ssq_a, &h.vars->err);
    for (int l = 0; l < m.layers; ++l) {
        enqueue_kernel(h, s, decode, K_QKV, l, pdl, nullptr);
        if (!decode && l == m.layers - 1) break;  // the prompt's last hidden state is not needed
        enqueue_kernel(h, s, decode, K_ATTN, l, pdl, nullptr);
        enqueue_kernel(h, s, decode, K_OPROJ, l, pdl, nullptr);
        enqueue_kernel(h, s, decode, K_GATEUP, l, pdl, nullptr);
        enqueue_kernel(h, s, decode, K_DOWN, l, pdl, nullptr);
    }
    if (!decode) return;
    enqueue_kernel(h, s, true, K_LMHEAD, m.layers - 1, pdl, logits_stage);
    launch(s, pdl, dim3(A.rows_cap), dim3(256), 0, sample_finish_kernel, c);
}

void enqueue_kv_fanout(sara_handle &h, cudaStream_t s, bool pdl, const StepPtrs &c) {
    const sara_model_cfg &m = h.cfg;
    launch(s, pdl, dim3(h.sms * 8), dim3(256), 0, kv_fanout_kernel, (const uint16_t *)h.kv_pr, h.kv_seq, c, m.layers,
           m.n_kv_heads, m.head_dim, h.cap_p, h.cap_s, m.max_active, m.max_seqs);
}

void enqueue_round_start(sara_handle &h, cudaStream_t s, bool pdl) {
    enqueue_forward(h, s, false, pdl, nullptr);
    enqueue_kv_fanout(h, s, pdl, h.ptrs);
}

// ------------------------------------------------------------------------ graph
void build_graph(sara_handle &h) {
    const bool pdl = h.use_pdl;
    CK(cudaGraphCreate(&h.graph, 0));
    cudaGraphConditionalHandle h_loop;
    CK(cudaGraphConditionalHandleCreate(&h_loop, h.graph, 1, cudaGraphCondAssignDefault));
    cudaGraphNodeParams wp{};
    wp.type = cudaGraphNodeTypeConditional;
    wp.conditional.handle = h_loop;
    wp.conditional.type = cudaGraphCondTypeWhile;
    wp.conditional.size = 1;
    cudaGraphNode_t wnode;
    CK(cudaGraphAddNode(&wnode, h.graph, nullptr, nullptr, 0, &wp));
    cudaGraph_t body = wp.conditional.phGraph_out[0];
    cudaGraphConditionalHandle h_round = 0;
    if (h.has_model) CK(cudaGraphConditionalHandleCreate(&h_round, body, 0, cudaGraphCondAssignDefault));

    cudaStream_t cs = h.cap_stream;
    CK(cudaStreamBeginCaptureToGraph(cs, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
    launch(cs, false, dim3(1), dim3(kCtlThreads), 0, ctl_kernel, h.ptrs, h_loop, h_round, h.has_model ? 3 : 1);
    if (h.has_model) {
        cudaStreamCaptureStatus st;
        cudaGraph_t capg;
        const cudaGraphNode_t *deps = nullptr;
        size_t ndeps = 0;
        CK(cudaStreamGetCaptureInfo(cs, &st, nullptr, &capg, &deps, nullptr, &ndeps));
        std::vector<cudaGraphNode_t> dv(deps, deps + ndeps);
        cudaGraphNodeParams ip{};
        ip.type = cudaGraphNodeTypeConditional;
        ip.conditional.handle = h_round;
        ip.conditional.type = cudaGraphCondTypeIf;
        ip.conditional.size = 1;
        cudaGraphNode_t inode;
        CK(cudaGraphAddNode(&inode, capg, dv.data(), nullptr, dv.size(), &ip));
        CK(cudaStreamUpdateCaptureDependencies(cs, &inode, nullptr, 1, cudaStreamSetCaptureDependencies));
        cudaGraph_t ibody = ip.conditional.phGraph_out[0];
        CK(cudaStreamBeginCaptureToGraph(h.cap_stream2, ibody, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
        enqueue_round_start(h, h.cap_stream2, pdl);
        cudaGraph_t ib2;
        CK(cudaStreamEndCapture(h.cap_stream2, &ib2));
        enqueue_forward(h, cs, true, pdl, nullptr);
    }
    cudaGraph_t b2;
    CK(cudaStreamEndCapture(cs, &b2));
    CK(cudaGraphInstantiate(&h.exec, h.graph, 0));
}

// Host-driven loop (debugging, SARA_GRAPH=0): the same kernels as the graph body, one
// iteration at a time, with the round-start branch decided on the host.
void run_host_loop(sara_handle &h) {
    cudaStream_t s = h.stream;
    StepVars v{};
    for (;;) {
        launch(s, false, dim3(1), dim3(kCtlThreads), 0, ctl_kernel, h.ptrs, (cudaGraphConditionalHandle)0,
               (cudaGraphConditionalHandle)0, 0);
        CK(cudaMemcpyAsync(&v, h.vars, sizeof(v), cudaMemcpyDeviceToHost, s));
        CK(cudaStreamSynchronize(s));
        if (v.done || v.err) break;
        if (!h.has_model) continue;
        if (v.round_steps == 0 && v.live > 0) enqueue_round_start(h, s, h.use_pdl);
        enqueue_forward(h, s, true, h.use_pdl, nullptr);
    }
}

// ------------------------------------------------------------------------ weights
void upload(const void *src, void *dst, size_t bytes, bool on_device, cudaStream_t s) {
    CK(cudaMemcpyAsync(dst, src, bytes, on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
}

void load_weights(sara_handle &h, const sara_weights *w) {
    const sara_model_cfg &m = h.cfg;
    const int d = m.d_model, H = m.n_heads, KVH = m.n_kv_heads, hd = m.head_dim, F = m.ffn, V = m.vocab;
    const bool dev = w->on_device != 0;
    cudaStream_t s = h.stream;
    if (!w->embed || !w->lm_head || !w->final_norm || !w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo ||
        !w->mlp_norm || !w->wgate || !w->wup || !w->wdown)
        throw SaraError(SARA_EINVAL, "a weight pointer is NULL");
    h.embed = h.mem.alloc<uint16_t>((size_t)V * d, false);
    h.lm_head = h.mem.alloc<uint16_t>((size_t)V * d, false);
    h.final_norm = h.mem.alloc<uint16_t>(d, false);
    upload(w->embed, h.embed, (size_t)V * d * 2, dev, s);
    upload(w->lm_head, h.lm_head, (size_t)V * d * 2, dev, s);
    upload(w->final_norm, h.final_norm, (size_t)d * 2, dev, s);
    const size_t qkv = (size_t)(H + 2 * KVH) * hd * d;
    const cudaMemcpyKind kind = dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    for (int l = 0; l < m.layers; ++l) {
        if (!w->attn_norm[l] || !w->wq[l] || !w->wk[l] || !w->wv[l] || !w->wo[l] || !w->mlp_norm[l] || !w->wgate[l] ||
            !w->wup[l] || !w->wdown[l])
            throw SaraError(SARA_EINVAL, "a per-layer weight pointer is NULL");
        uint16_t *an = h.mem.alloc<uint16_t>(d, false), *mn = h.mem.alloc<uint16_t>(d, false);
        upload(w->attn_norm[l], an, (size_t)d * 2, dev, s);
        upload(w->mlp_norm[l], mn, (size_t)d * 2, dev, s);
        // fused q|k|v rows
        uint16_t *wqkv = h.mem.alloc<uint16_t>(qkv, false);
        upload(w->wq[l], wqkv, (size_t)H * hd * d * 2, dev, s);
        upload(w->wk[l], wqkv + (size_t)H * hd * d, (size_t)KVH * hd * d * 2, dev, s);
        upload(w->wv[l], wqkv + (size_t)(H + KVH) * hd * d, (size_t)KVH * hd * d * 2, dev, s);
        uint16_t *wo = h.mem.alloc<uint16_t>((size_t)d * H * hd, false);
        upload(w->wo[l], wo, (size_t)d * H * hd * 2, dev, s);
        // gate/up interleaved in blocks of 64 rows: [g 0..63, u 0..63, g 64..127, u 64..127, ...]
        uint16_t *wgu = h.mem.alloc<uint16_t>((size_t)2 * F * d, false);
        CK(cudaMemcpy2DAsync(wgu, (size_t)128 * d * 2, w->wgate[l], (size_t)64 * d * 2, (size_t)64 * d * 2, F / 64,
                             kind, s));
        CK(cudaMemcpy2DAsync(wgu + (size_t)64 * d, (size_t)128 * d * 2, w->wup[l], (size_t)64 * d * 2,
                             (size_t)64 * d * 2, F / 64, kind, s));
        uint16_t *wd = h.mem.alloc<uint16_t>((size_t)d * F, false);
        upload(w->wdown[l], wd, (size_t)d * F * 2, dev, s);
        h.attn_norm.push_back(an);
        h.mlp_norm.push_back(mn);
        h.w_qkv.push_back(wqkv);
        h.w_o.push_back(wo);
        h.w_gu.push_back(wgu);
        h.w_down.push_back(wd);
    }
    CK(cudaStreamSynchronize(s));
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

void make_tensor_maps(sara_handle &h) {
    const sara_model_cfg &m = h.cfg;
    const int d = m.d_model, H = m.n_heads, KVH = m.n_kv_heads, hd = m.head_dim, F = m.ffn;
    for (int l = 0; l < m.layers; ++l) {
        h.tm_qkv.push_back(make_tmap_bf16(h.w_qkv[l], d, (H + 2 * KVH) * hd, kTileK, kTileM));
        h.tm_o.push_back(make_tmap_bf16(h.w_o[l], H * hd, d, kTileK, kTileM));
        h.tm_gu.push_back(make_tmap_bf16(h.w_gu[l], d, 2 * F, kTileK, kTileM));
        h.tm_down.push_back(make_tmap_bf16(h.w_down[l], F, d, kTileK, kTileM));
    }
    h.tm_lm = make_tmap_bf16(h.lm_head, d, m.vocab, kTileK, kTileM);
    for (Acts *A : {&h.dec, &h.pre}) {
        A->tm_xg = make_tmap_bf16(A->xg, d, A->rows_cap, kTileK, kXBoxRows);
        A->tm_xg_lo = make_tmap_bf16(A->xg_lo, d, A->rows_cap, kTileK, kXBoxRows);
        A->tm_att = make_tmap_bf16(A->att, H * hd, A->rows_cap, kTileK, kXBoxRows);
        A->tm_att_lo = make_tmap_bf16(A->att_lo, H * hd, A->rows_cap, kTileK, kXBoxRows);
        A->tm_h = make_tmap_bf16(A->h, F, A->rows_cap, kTileK, kXBoxRows);
        A->tm_h_lo = make_tmap_bf16(A->h_lo, F, A->rows_cap, kTileK, kXBoxRows);
    }
}

void validate_cfg(const sara_model_cfg &m) {
    auto bad = [](const char *msg) { throw SaraError(SARA_EINVAL, msg); };
    if (m.max_prompts < 1 || m.max_active < 1 || m.max_k < 2 || m.max_k > kMaxK) bad("capacities out of range (max_k 2..64)");
    if (m.max_active > 8192) bad("max_active must be <= 8192");
    if (m.layers < 0) bad("layers < 0");
    if (m.layers == 0) return;
    if (m.d_model % 128 || m.d_model < 128) bad("d_model must be a positive multiple of 128");
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
        // KV caches: rollout slots [layer][slot][2][kv][cap_s][hd], prompt slots [layer][pslot][2][kv][cap_p][hd]
        h.kv_seq_slot = 2LL * KVH * h.cap_s * hd;
        h.kv_seq_layer = h.kv_seq_slot * S;
        h.kv_pr_slot = 2LL * KVH * h.cap_p * hd;
        h.kv_pr_layer = h.kv_pr_slot * Bc;
        h.kv_seq = h.mem.alloc<uint16_t>((size_t)h.kv_seq_layer * m.layers);
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
        alloc_acts(h, h.dec, S);
        alloc_acts(h, h.pre, h.pre_cap);
        // GEMM stream-K workspace: one fixed-point tile sum per CTA + per-tile counters (zeroed)
        h.gemm_acc = h.mem.alloc<unsigned long long>((size_t)h.sms * kTileR * kTileM);
        const int max_m = std::max({(m.n_heads + 2 * KVH) * hd, d, 2 * m.ffn, m.vocab}) / 128;
        h.gemm_cnt = h.mem.alloc<int>((size_t)max_m * ((h.pre_cap + kTileR - 1) / kTileR + 1));
        const int Gq = m.n_heads / KVH;
        h.attn_part = h.mem.alloc<float>((size_t)h.att_cap * KVH * Gq * (hd + 2), false);
        h.attn_cnt = h.mem.alloc<int>((size_t)S * KVH);
        c.lm_tiles = m.vocab / 128;
        h.lm_val = h.mem.alloc<float>((size_t)S * c.lm_tiles, false);
        h.lm_idx = h.mem.alloc<int>((size_t)S * c.lm_tiles, false);
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

    CK(cudaEventRecord(h.ev0, s));
    CK(cudaMemcpyAsync(h.kc, &K, sizeof(K), cudaMemcpyHostToDevice, s));
    if (P > 0) {
        CK(cudaMemcpyAsync(h.p_thr, pr->p_threshold, (size_t)P * 8, kin, s));
        CK(cudaMemcpyAsync(h.p_len, pr->lengths, (size_t)P * k * 4, kin, s));
        if (h.has_model) CK(cudaMemcpyAsync(h.p_tok, pr->tokens, (size_t)P * Lp * 4, kin, s));
    }
    launch(s, false, dim3(1), dim3(kCtlThreads), 0, ctl_init_kernel, h.ptrs);
    if (h.use_graph) CK(cudaGraphLaunch(h.exec, s));
    else run_host_loop(h);
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
        if (out->tokens && h.has_model)
            CK(cudaMemcpyAsync(out->tokens, h.gen_tok, (size_t)P * k * m.max_gen_len * 4, kout, s));
    }
    CK(cudaEventRecord(h.ev1, s));
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
    if (!h.logit_stage) h.logit_stage = h.mem.alloc<float>((size_t)m.max_seqs * m.vocab, false);
    if ((size_t)n * T > h.forced_cap) {
        h.forced_cap = (size_t)n * T;
        h.forced = h.mem.alloc<int32_t>(h.forced_cap, false);
        h.sampled_out = h.mem.alloc<int32_t>(h.forced_cap, false);
    }
    if (!h.uid_dev) h.uid_dev = h.mem.alloc<int64_t>(m.max_seqs, false);
    StepConst K{};
    K.P = n; K.Lp = Lp; K.k = 2; K.n0 = 1; K.commit_min = 2; K.a0 = 1; K.b0 = 1; K.B = n; K.N = n;
    K.tau_num = 0; K.tau_den = 1; K.sample_seed = sample_seed; K.decode = 1; K.teacher = 1; K.T_forced = T;
    K.max_gen = m.max_gen_len; K.attn_chunk = kDecodeChunk;
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
        launch(s, false, dim3(1), dim3(kCtlThreads), 0, teacher_setup_kernel, c, n, (const int64_t *)h.uid_dev);
        enqueue_forward(h, s, false, false, nullptr);
        enqueue_kv_fanout(h, s, false, c);
        for (int step = 0; step < T; ++step) {
            enqueue_forward(h, s, true, false, h.logit_stage);
            // rows stay in rollout order for all T steps (every rollout has length T)
            CK(cudaMemcpy2DAsync(logits + (size_t)step * m.vocab, (size_t)T * m.vocab * 4, h.logit_stage,
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

// Profiling hook: `rows` live rollouts at context `ctx` (synthetic row state), `iters` launches
// of one kernel of layer 0 (or of the whole eager decode step, kernel 0) timed with CUDA
// events on the handle's stream after two warm-up launches.
void profile_impl(sara_handle &h, int which, int rows, int ctx, int iters, double *ms) {
    const sara_model_cfg &m = h.cfg;
    if (!h.has_model) throw SaraError(SARA_EINVAL, "profiling needs a model");
    if (which < 0 || which > K_LMHEAD) throw SaraError(SARA_EINVAL, "unknown kernel id");
    if (rows < 1 || rows > m.max_seqs || iters < 1 || !ms) throw SaraError(SARA_EINVAL, "rows / iters out of range");
    const int steps = which == 0 ? 2 * iters + 2 : 0;  // the whole step advances positions
    if (ctx < 2 || ctx + steps + 1 > h.cap_s || steps + 1 > m.max_gen_len) throw SaraError(SARA_EINVAL, "ctx out of range");
    cudaStream_t s = h.stream;
    StepConst K{};
    K.P = 1; K.Lp = ctx; K.k = 2; K.n0 = 1; K.commit_min = 2; K.a0 = 1; K.b0 = 1; K.B = 1; K.N = 1;
    K.tau_num = 0; K.tau_den = 1; K.decode = 1; K.max_gen = m.max_gen_len; K.attn_chunk = kDecodeChunk;
    const int nsplit = (ctx + kDecodeChunk - 1) / kDecodeChunk;
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
    StepVars v{};
    v.live = rows;
    v.att_items = rows * nsplit;
    v.round_maxL = 1 << 30;
    const StepPtrs &c = h.ptrs;
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
    if (!h.stamps) h.stamps = h.mem.alloc<uint64_t>((size_t)h.sms * 16);
    CK(cudaMemsetAsync(h.stamps, 0, (size_t)h.sms * 16 * 8, s));
#endif
    CK(cudaStreamSynchronize(s));
    auto one = [&](cudaStream_t st) {
        if (which == 0) enqueue_forward(h, st, true, h.use_pdl, nullptr);
        else enqueue_kernel(h, st, true, which, 0, h.use_pdl, nullptr);
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
    if (h.stamps && which != 0) {  // phase breakdown of the last launch, relative to the earliest entry
        std::vector<uint64_t> st((size_t)h.sms * 16);
        CK(cudaMemcpy(st.data(), h.stamps, st.size() * 8, cudaMemcpyDeviceToHost));
        uint64_t t0 = ~0ull;
        for (int c = 0; c < h.sms; ++c) t0 = std::min(t0, st[(size_t)c * 16]);
        for (int i = 0; i < 16; ++i) {
            std::vector<double> d;
            for (int c = 0; c < h.sms; ++c)
                if (st[(size_t)c * 16 + i]) d.push_back((double)(st[(size_t)c * 16 + i] - t0) * 1e-3);
            std::sort(d.begin(), d.end());
            if (!d.empty())
                fprintf(stderr, "stamp %d: n=%zu min %.2f med %.2f max %.2f us\n", i, d.size(), d.front(), d[d.size() / 2],
                        d.back());
        }
    }
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

const char *sara_last_error(const sara_handle *h) { return h ? h->err.c_str() : g_create_error.c_str(); }

void sara_destroy(sara_handle *h) {
    if (!h) return;
    cudaStreamSynchronize(h->stream);
    delete h;
}

}  // extern "C"
