// Kernel-level entry points of include/sara.h on caller-provided device buffers: the
// prefill's projection GEMM and attention kernels, and a one-CTA-per-row Gumbel-max sampler
// (the decode step's sampling rule).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <string>
#include <vector>

#include "../../include/sara.h"
#include "attention.cuh"
#include "gemm_tc.cuh"
#include "host_util.h"
#include "step_kernels.cuh"

using namespace sara;

namespace {

int sm_count() {
    int dev = 0, sms = 0;
    CK(cudaGetDevice(&dev));
    CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    return sms;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct GemmWs {
    size_t part_bytes, cnt_bytes;
};
GemmWs gemm_ws_layout(int Nout, int sms) {
    GemmWs w;
    w.part_bytes = align_up((size_t)sms * kTileR * kTileM * sizeof(unsigned long long), 256);
    w.cnt_bytes = align_up((size_t)(Nout / kTileM) * sizeof(int), 256);
    return w;
}

template <int HD>
void launch_g(dim3 grid, int G, cudaStream_t s, const AttnParams &a) {
    switch (G) {
        case 1: attn_rows_kernel<HD, 1><<<grid, kAttnThreads, 0, s>>>(a); break;
        case 2: attn_rows_kernel<HD, 2><<<grid, kAttnThreads, 0, s>>>(a); break;
        case 4: attn_rows_kernel<HD, 4><<<grid, kAttnThreads, 0, s>>>(a); break;
        case 6: attn_rows_kernel<HD, 6><<<grid, kAttnThreads, 0, s>>>(a); break;
        default: attn_rows_kernel<HD, 8><<<grid, kAttnThreads, 0, s>>>(a); break;
    }
}

template <typename F>
int op_guard(F fn) {
    try {
        fn();
        return SARA_OK;
    } catch (const SaraError &e) {
        return e.code;
    } catch (...) {
        return SARA_EDEVICE;
    }
}

}  // namespace

extern "C" {

size_t sara_gemm_workspace_bytes(int32_t R, int32_t Nout, int32_t K) {
    (void)R;
    (void)K;
    if (Nout <= 0) return 0;
    int sms = 0;
    try {
        sms = sm_count();
    } catch (...) {
        return 0;
    }
    const GemmWs w = gemm_ws_layout(Nout, sms);
    return w.part_bytes + w.cnt_bytes;
}

int sara_gemm_bf16(const uint16_t *X, const uint16_t *W, float *Y, int32_t R, int32_t Nout, int32_t K, void *workspace,
                   size_t workspace_bytes, void *stream) {
    if (!X || !W || !Y || !workspace) return SARA_EINVAL;
    if (R < 1 || R > kTileR || Nout < kTileM || Nout % kTileM || K < kTileK || K % kTileK) return SARA_EINVAL;
    if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(W)) & 15) return SARA_EINVAL;
    return op_guard([&] {
        const int sms = sm_count();
        const GemmWs w = gemm_ws_layout(Nout, sms);
        if (workspace_bytes < w.part_bytes + w.cnt_bytes) throw SaraError(SARA_EINVAL, "workspace too small");
        CK(cudaFuncSetAttribute(gemm_tc_kernel<EPI_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmemBytes));
        const CUtensorMap tw = make_tmap_bf16(W, K, Nout, kTileK, kTileM);
        const CUtensorMap tx = make_tmap_bf16(X, K, R, kTileK, kXBoxRows);
        GemmParams p{};
        p.m_tiles = Nout / kTileM;
        p.k_chunks = K / kTileK;
        p.rows_cap = R;
        p.rows_dev = nullptr;
        p.rows_fixed = R;
        p.decode = 1;
        p.ws_acc = reinterpret_cast<unsigned long long *>(workspace);
        p.ws_cnt = reinterpret_cast<int *>(reinterpret_cast<uint8_t *>(workspace) + w.part_bytes);
        p.err = nullptr;
        p.y_f32 = Y;
        p.ld = Nout;
        gemm_tc_kernel<EPI_F32><<<sms, kGemmThreads, kGemmSmemBytes, static_cast<cudaStream_t>(stream)>>>(tw, tx, tx, p);
        CK(cudaGetLastError());
    });
}

size_t sara_attention_workspace_bytes(int32_t b, int32_t n_heads, int32_t head_dim, int32_t max_ctx) {
    if (b < 1 || n_heads < 1 || head_dim < 1 || max_ctx < 1) return 0;
    const size_t splits = (size_t)(max_ctx + 127) / 128;
    const size_t items = (size_t)b * splits;
    // partials (<= items * n_heads * (hd + 2) floats), counters [b][n_kv], items, 3 row arrays
    return align_up(items * n_heads * (head_dim + 2) * sizeof(float), 256) +
           align_up((size_t)b * n_heads * sizeof(int), 256) + align_up(items * sizeof(int2), 256) +
           align_up((size_t)b * sizeof(int) * 3, 256);
}

int sara_attention_decode(const uint16_t *q, const uint16_t *kv, int64_t kv_stride, const int32_t *ctx, uint16_t *out,
                          int32_t b, int32_t n_heads, int32_t n_kv_heads, int32_t head_dim, int32_t cap,
                          int32_t max_ctx, void *workspace, size_t workspace_bytes, void *stream) {
    if (!q || !kv || !ctx || !out || !workspace) return SARA_EINVAL;
    if (b < 1 || n_kv_heads < 1 || n_heads % n_kv_heads || n_heads / n_kv_heads > kAttnMaxG) return SARA_EINVAL;
    if (head_dim != 32 && head_dim != 64 && head_dim != 128) return SARA_EINVAL;
    if (max_ctx < 1 || max_ctx > cap || (max_ctx + 127) / 128 > kAttnMaxSplits) return SARA_EINVAL;
    return op_guard([&] {
        if (workspace_bytes < sara_attention_workspace_bytes(b, n_heads, head_dim, max_ctx))
            throw SaraError(SARA_EINVAL, "workspace too small");
        cudaStream_t s = static_cast<cudaStream_t>(stream);
        const size_t splits = (size_t)(max_ctx + 127) / 128;
        const size_t items_cap = (size_t)b * splits;
        uint8_t *ws = reinterpret_cast<uint8_t *>(workspace);
        float *part = reinterpret_cast<float *>(ws);
        ws += align_up(items_cap * n_heads * (head_dim + 2) * sizeof(float), 256);
        int *cnt = reinterpret_cast<int *>(ws);
        ws += align_up((size_t)b * n_heads * sizeof(int), 256);
        int2 *items = reinterpret_cast<int2 *>(ws);
        ws += align_up(items_cap * sizeof(int2), 256);
        int *row_pos = reinterpret_cast<int *>(ws);
        int *row_item0 = row_pos + b;
        int *row_slot = row_item0 + b;  // row i reads KV slot i
        // work items (row, split) from the context lengths, built on the host
        std::vector<int> hctx(b), hpos(b), hi0(b), slots(b);
        CK(cudaMemcpyAsync(hctx.data(), ctx, b * sizeof(int), cudaMemcpyDeviceToHost, s));
        CK(cudaStreamSynchronize(s));
        std::vector<int2> hitems;
        for (int i = 0; i < b; ++i) {
            if (hctx[i] < 1 || hctx[i] > max_ctx) throw SaraError(SARA_EINVAL, "ctx out of range");
            hpos[i] = hctx[i] - 1;
            hi0[i] = (int)hitems.size();
            slots[i] = i;
            for (int sp = 0; sp < (hctx[i] + 127) / 128; ++sp) hitems.push_back(make_int2(i, sp));
        }
        CK(cudaMemcpyAsync(items, hitems.data(), hitems.size() * sizeof(int2), cudaMemcpyHostToDevice, s));
        CK(cudaMemcpyAsync(row_pos, hpos.data(), b * sizeof(int), cudaMemcpyHostToDevice, s));
        CK(cudaMemcpyAsync(row_item0, hi0.data(), b * sizeof(int), cudaMemcpyHostToDevice, s));
        CK(cudaMemcpyAsync(row_slot, slots.data(), b * sizeof(int), cudaMemcpyHostToDevice, s));
        AttnParams a{};
        a.q = q;
        a.out = out;
        a.kv = kv;
        a.slot_stride = kv_stride;
        a.cap = cap;
        a.row_slot = row_slot;
        a.row_pos = row_pos;
        a.items = items;
        a.n_items_dev = nullptr;
        a.n_items_fixed = (int)hitems.size();
        a.row_item0 = row_item0;
        a.n_heads = n_heads;
        a.n_kv = n_kv_heads;
        a.chunk = 128;
        a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)head_dim));
        a.part = part;
        a.cnt = cnt;
        a.err = nullptr;
        const int sms = sm_count();
        dim3 grid(std::max(1, sms * 4 / n_kv_heads), n_kv_heads);
        const int G = n_heads / n_kv_heads;
        if (G != 1 && G != 2 && G != 4 && G != 6 && G != 8) throw SaraError(SARA_EINVAL, "query group must be 1, 2, 4, 6 or 8");
        if (head_dim == 32) launch_g<32>(grid, G, s, a);
        else if (head_dim == 64) launch_g<64>(grid, G, s, a);
        else launch_g<128>(grid, G, s, a);
        CK(cudaGetLastError());
        CK(cudaStreamSynchronize(s));  // the host vectors above back in-flight copies
    });
}

int sara_sample(const float *logits, int32_t R, int32_t V, uint64_t sample_seed, const int64_t *uid, const int32_t *t,
                int32_t *token, void *stream) {
    if (!logits || !uid || !t || !token || R < 1 || V < 1) return SARA_EINVAL;
    return op_guard([&] {
        sample_rows_kernel<<<R, 256, 0, static_cast<cudaStream_t>(stream)>>>(logits, V, sample_seed, uid, t, token);
        CK(cudaGetLastError());
    });
}

}  // extern "C"
