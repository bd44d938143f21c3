// K2: per-worker projection tables (one warp per worker) and the
// capacity_norm ranking of workers used by Algorithm 1.
#include "aladdin_host.h"

namespace aladdin {

constexpr int BUILD_WARPS = 4;

template <int E>
__global__ void __launch_bounds__(BUILD_WARPS * 32)
k_build(DevParams P, ClusterDev C, const int32_t* __restrict__ list, int count)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    BuildSmem<E>* sm = reinterpret_cast<BuildSmem<E>*>(smraw);
    const int warp = threadIdx.x >> 5;
    const int idx = blockIdx.x * BUILD_WARPS + warp;
    if (idx >= count) return;  // whole warp leaves together
    const int w = list ? list[idx] : idx;
    build_table<E>(P, C, w, sm[warp]);
}

template <int E>
static cudaError_t build_e(const DevParams& P, const ClusterDev& C, const int32_t* list, int count,
                           cudaStream_t st)
{
    if (count <= 0) return cudaSuccess;
    const size_t smem = sizeof(BuildSmem<E>) * BUILD_WARPS;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_build<E>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
    }
    const int blocks = (count + BUILD_WARPS - 1) / BUILD_WARPS;
    k_build<E><<<blocks, BUILD_WARPS * 32, smem, st>>>(P, C, list, count);
    return cudaGetLastError();
}

cudaError_t launch_build(const DevParams& P, const ClusterDev& C, const int32_t* list, int count,
                         cudaStream_t st)
{
    switch (lanes_per_worker(C.cap)) {
    case 1: return build_e<1>(P, C, list, count, st);
    case 2: return build_e<2>(P, C, list, count, st);
    case 4: return build_e<4>(P, C, list, count, st);
    case 8: return build_e<8>(P, C, list, count, st);
    case 16: return build_e<16>(P, C, list, count, st);
    default: return cudaErrorInvalidValue;
    }
}

// rank[w] = number of workers ordered before w: larger key, or equal key and
// smaller index (a stable descending sort). Keys are tiled through shared
// memory; O(W^2) comparisons, each thread one worker.
constexpr int RANK_TILE = 256;

__global__ void __launch_bounds__(RANK_TILE) k_rank(ClusterDev C)
{
    __shared__ double ks[RANK_TILE];
    const int w = blockIdx.x * RANK_TILE + threadIdx.x;
    const double kw = w < C.W ? C.key[w] : 0.0;
    int cnt = 0;
    for (int t0 = 0; t0 < C.W; t0 += RANK_TILE) {
        const int v = t0 + threadIdx.x;
        ks[threadIdx.x] = v < C.W ? C.key[v] : -2.0;
        __syncthreads();
        const int lim = min(RANK_TILE, C.W - t0);
        for (int i = 0; i < lim; ++i) {
            const double kv = ks[i];
            const int vi = t0 + i;
            cnt += (kv > kw) || (kv == kw && vi < w);
        }
        __syncthreads();
    }
    if (w < C.W) {
        C.rank[w] = cnt;
        C.order[cnt] = w;
        C.wrec[w].w = __int_as_float(cnt);
    }
}

cudaError_t launch_rank(const ClusterDev& C, cudaStream_t st)
{
    const int blocks = (C.W + RANK_TILE - 1) / RANK_TILE;
    k_rank<<<blocks, RANK_TILE, 0, st>>>(C);
    return cudaGetLastError();
}

}  // namespace aladdin
