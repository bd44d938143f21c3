// Demand statistics of a request trace for the worker-configuration model
// (Sec. 4.1, Eq. max throughput): the KV demand m_r and the context l_ave of
// a running request, averaged over every decode iteration of every request
// (the footprint vector w of (e): a request (l_in, l_pred) holds l_in + s
// context tokens in its s-th iteration). The sums are exact integers:
// sum_q r_q and sum_q (r_q l_in,q + r_q (r_q + 1) / 2), one grid-stride pass,
// warp sums, one 64-bit atomic per warp.
#include "aladdin_host.h"

namespace aladdin {

constexpr int TD_THREADS = 256;

__global__ void __launch_bounds__(TD_THREADS)
k_trace_demand(const int32_t* __restrict__ in, const int32_t* __restrict__ pred, long long n,
               unsigned long long* sums)
{
    unsigned long long s_it = 0, s_ctx = 0;
    for (long long q = (long long)blockIdx.x * TD_THREADS + threadIdx.x; q < n;
         q += (long long)gridDim.x * TD_THREADS) {
        const unsigned long long r = (unsigned)pred[q];
        const unsigned long long a = (unsigned)in[q];
        s_it += r;
        s_ctx += r * a + r * (r + 1ull) / 2ull;
    }
    s_it = warp_reduce(s_it, OpAdd<unsigned long long>());
    s_ctx = warp_reduce(s_ctx, OpAdd<unsigned long long>());
    if ((threadIdx.x & 31) == 0) {
        if (s_it) atomicAdd(&sums[0], s_it);
        if (s_ctx) atomicAdd(&sums[1], s_ctx);
    }
}

cudaError_t launch_trace_demand(const int32_t* in, const int32_t* pred, long long n,
                                unsigned long long* sums, cudaStream_t st)
{
    cudaError_t e = cudaMemsetAsync(sums, 0, 2 * sizeof(unsigned long long), st);
    if (e != cudaSuccess || n == 0) return e;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    const long long need = (n + TD_THREADS - 1) / TD_THREADS;
    const int blocks = (int)(need < 4ll * sms ? need : 4ll * sms);
    k_trace_demand<<<blocks, TD_THREADS, 0, st>>>(in, pred, n, sums);
    return cudaGetLastError();
}

}  // namespace aladdin
