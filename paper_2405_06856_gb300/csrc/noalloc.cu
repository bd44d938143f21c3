// aladdin_score_noalloc: candidate x worker scoring that allocates nothing.
//
// For callers that must not reach a device allocator while they schedule:
// processes whose device memory is reserved up front by another allocator (a
// serving engine that owns the whole KV-cache pool and leaves nothing for a
// cudaMalloc to take), or real-time loops that cannot afford the allocator's
// latency or its implicit device synchronisation. aladdin_score grows private
// scratch buffers (the sorted candidate records, the predicted-length
// histogram and the per-candidate argbest keys) with cudaMalloc and stages
// host arrays through device copies. This entry point uses one file-scope
// device array instead, so every buffer it touches exists from the moment the
// library is loaded on a device, and it accepts device (or managed) pointers of
// the cluster's GPU only.
//
// The array holds the scratch of up to NOALLOC_MAX_CAND candidates. Every GPU
// that loads the library keeps it until the process exits. All calls share
// it: calls that overlap on the GPU (two streams, or two clusters on the same
// device) race on it and must be serialized by the caller. What must start
// from zero (the histogram) is cleared on every call; the argbest keys are
// rewritten on every call.
//
// Set-up, once per device, on the first call with that device current: the
// array's device address (in host code the symbol is only a host-side
// handle) and the loading of every scoring kernel with its launch
// configuration, so that later calls reach neither the module loader nor a
// device query. The address belongs to the device's primary context:
// cudaDeviceReset while the library is in use is not supported (it also
// invalidates every cluster's device memory).
#include <mutex>

#include "../../include/aladdin.h"
#include "aladdin_host.h"

namespace {

constexpr int NOALLOC_MAX_CAND = ALADDIN_NOALLOC_MAX_CAND;
constexpr size_t REC_BYTES = (size_t)NOALLOC_MAX_CAND * aladdin::CAND_REC_F4 * 16;  // sorted records
constexpr size_t HIST_BYTES = ((size_t)(65536 + 2) * 4 + 255) / 256 * 256;  // K <= 65536
constexpr size_t BEST_BYTES = (size_t)NOALLOC_MAX_CAND * 4;
constexpr size_t SCRATCH_BYTES = REC_BYTES + HIST_BYTES + BEST_BYTES;

__device__ __align__(256) unsigned char g_score_scratch[SCRATCH_BYTES];

// Device address of g_score_scratch per device ordinal, looked up once with
// that device current (in host code the symbol is only a host-side handle).
constexpr int MAX_DEVICES = 64;
std::mutex g_mu;
void* g_scratch[MAX_DEVICES] = {};

int scratch_address(int device, void** out)
{
    if (device < 0 || device >= MAX_DEVICES) return ALADDIN_ERR_ARG;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch[device]) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_score_scratch);
        if (e == cudaSuccess) e = aladdin::prepare_score_kernels();
        if (e != cudaSuccess || !p) {
            cudaGetLastError();
            return ALADDIN_ERR_CUDA;
        }
        g_scratch[device] = p;
    }
    *out = g_scratch[device];
    return ALADDIN_OK;
}

// Device memory of `device`, or managed memory (which any device may reach).
bool on_device(const void* p, int device)
{
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (a.type == cudaMemoryTypeManaged) return true;
    return a.type == cudaMemoryTypeDevice && a.device == device;
}

}  // namespace

extern "C" int aladdin_score_noalloc(aladdin_cluster* cl, int32_t n_cand, const int32_t* in,
                                     const int32_t* pred, const float* wait_ms, uint8_t* flags,
                                     float* margin, int32_t* argbest)
try {
    aladdin::ClusterView v;
    if (!cl || n_cand < 0) return ALADDIN_ERR_ARG;
    int rc = aladdin::cluster_view(cl, &v);
    if (rc) return rc;
    if (n_cand > NOALLOC_MAX_CAND) return ALADDIN_ERR_SCRATCH;
    if (n_cand == 0) return ALADDIN_OK;
    if (!in || !pred) return ALADDIN_ERR_ARG;
    const void* ptrs[6] = {in, pred, wait_ms, flags, margin, argbest};
    for (const void* p : ptrs)
        if (p && !on_device(p, v.device)) return ALADDIN_ERR_ARG;
    if (cudaSetDevice(v.device) != cudaSuccess) {
        cudaGetLastError();
        return ALADDIN_ERR_CUDA;
    }
    void* base = nullptr;
    if ((rc = scratch_address(v.device, &base))) return rc;
    unsigned char* b = static_cast<unsigned char*>(base);
    aladdin::ScoreBuffers B;
    B.sorted = reinterpret_cast<float4*>(b);
    B.hist = reinterpret_cast<int32_t*>(b + REC_BYTES);
    B.best = reinterpret_cast<unsigned int*>(b + REC_BYTES + HIST_BYTES);
    const cudaError_t e = aladdin::launch_score(v.dp, v.dev, n_cand, in, pred, wait_ms, flags, margin,
                                                argbest, nullptr, nullptr, B, v.round_open, v.stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return ALADDIN_ERR_CUDA;
    }
    return ALADDIN_OK;
} catch (...) {
    return ALADDIN_ERR_NOMEM;  // a host allocation or thread start failed
}
