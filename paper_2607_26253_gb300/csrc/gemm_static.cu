// A variant of the projection-GEMM entry point for callers that cannot allocate device
// memory: the stream-K scratch lives in a fixed array compiled into the library instead
// of a caller-provided workspace.  Same kernel as sara_gemm_bf16, at most kStaticCtas CTAs.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "../../include/sara.h"
#include "gemm_tc.cuh"
#include "host_util.h"

using namespace sara;

namespace {

constexpr int kStaticCtas = 64;      // CTAs of one call (stream-K slots in the scratch)
constexpr int kStaticTiles = 2048;   // output tiles of 128 features: Nout <= 262,144
constexpr size_t kAccElems = (size_t)kStaticCtas * kTileR * kTileM;  // 8 MiB of 64-bit sums
constexpr size_t kMaxDevices = 64;

// File-scope scratch, resident on every GPU that loads the library until the process
// exits: fixed-point tile sums, then per-tile arrival counters.  In host code this name is
// only a stand-in for the device array; its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned long long g_static_acc[kAccElems];
static __device__ __align__(256) int g_static_cnt[kStaticTiles];

struct DeviceScratch {
    unsigned long long *acc = nullptr;
    int *cnt = nullptr;
    bool ready = false;
};
DeviceScratch g_scratch[kMaxDevices];
std::mutex g_scratch_mu;

// Device addresses of the scratch for the current device, looked up once per device.
DeviceScratch scratch_for_current_device() {
    int dev = 0;
    CK(cudaGetDevice(&dev));
    if (dev < 0 || (size_t)dev >= kMaxDevices) throw SaraError(SARA_EINVAL, "device index out of range");
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    DeviceScratch &d = g_scratch[dev];
    if (!d.ready) {
        void *a = nullptr, *c = nullptr;
        CK(cudaGetSymbolAddress(&a, g_static_acc));
        CK(cudaGetSymbolAddress(&c, g_static_cnt));
        d.acc = static_cast<unsigned long long *>(a);
        d.cnt = static_cast<int *>(c);
        CK(cudaFuncSetAttribute(gemm_tc_kernel<EPI_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kGemmSmemBytes));
        d.ready = true;
    }
    return d;
}

}  // namespace

extern "C" {

int sara_gemm_bf16_static(const uint16_t *X, const uint16_t *W, float *Y, int32_t R, int32_t Nout, int32_t K,
                          void *stream) {
    if (!X || !W || !Y) return SARA_EINVAL;
    if (R < 1 || R > kTileR || Nout < kTileM || Nout % kTileM || K < kTileK || K % kTileK) return SARA_EINVAL;
    if (Nout / kTileM > kStaticTiles) return SARA_EINVAL;  // beyond the scratch's tile counters
    if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(W)) & 15) return SARA_EINVAL;
    try {
        const DeviceScratch d = scratch_for_current_device();
        int dev = 0, sms = 0;
        CK(cudaGetDevice(&dev));
        CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
        const int grid = std::min(sms, kStaticCtas);
        cudaStream_t s = static_cast<cudaStream_t>(stream);
        // the scratch keeps the previous call's contents: clear what this call's sums start from
        CK(cudaMemsetAsync(d.cnt, 0, (size_t)(Nout / kTileM) * sizeof(int), s));
        CK(cudaMemsetAsync(d.acc, 0, (size_t)grid * kTileR * kTileM * sizeof(unsigned long long), s));
        const CUtensorMap tw = make_tmap_bf16(W, K, Nout, kTileK, kTileM);
        const CUtensorMap tx = make_tmap_bf16(X, K, R, kTileK, kXBoxRows);
        GemmParams p{};
        p.m_tiles = Nout / kTileM;
        p.k_chunks = K / kTileK;
        p.rows_cap = R;
        p.rows_dev = nullptr;
        p.rows_fixed = R;
        p.decode = 1;
        p.ws_acc = d.acc;
        p.ws_cnt = d.cnt;
        p.err = nullptr;
        p.y_f32 = Y;
        p.ld = Nout;
        gemm_tc_kernel<EPI_F32><<<grid, kGemmThreads, kGemmSmemBytes, s>>>(tw, tx, tx, p);
        CK(cudaGetLastError());
        return SARA_OK;
    } catch (const SaraError &e) {
        return e.code;
    } catch (...) {
        return SARA_EDEVICE;
    }
}

}  // extern "C"
