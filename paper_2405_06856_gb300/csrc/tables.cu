// K2: per-worker projection tables (one warp per worker) and the
// capacity_norm ranking of workers used by Algorithm 1.
#include "aladdin_host.h"

namespace aladdin {

constexpr int BUILD_WARPS = 4;

// One warp packs worker w's requests from CSR arrays into its slots: a worker
// whose request count exceeds the slots is replaced by a single invalid
// request, so that the table builder marks it infeasible and records the
// error (bit 2). Returns the worker's request count (every lane).
__device__ __forceinline__ int pack_worker(const DevParams& P, const ClusterDev& C,
                                           const PackSrc& S, int w)
{
    const int lane = threadIdx.x & 31;
    const int a = S.off[w], b = S.off[w + 1];
    const long long base = (long long)w * C.cap;
    int n = b - a;
    const bool over = n < 0 || n > C.cap;
    if (over) n = 0;
    for (int q = lane; q < n; q += 32) {
        const long long dst = base + q;
        const int g = S.gen[a + q];
        const int32_t pr = S.pred[a + q];
        C.in[dst] = S.in[a + q];
        C.gen[dst] = g;
        C.pred[dst] = pr;
        C.real[dst] = pr;  // exact predictions
        // without a history every request has used exactly its budget: no slack
        const double td = S.tdec ? (double)S.tdec[a + q] : P.thetad * P.T_decd * (double)g;
        C.tdec[dst] = td;
        C.bank[dst] = S.tdec ? banked_slack(P, g, td) : 0.0f;
        C.pend[dst] = 0;
    }
    if (lane == 0) {
        if (over) {
            C.in[base] = -1;
            C.gen[base] = 0;
            C.pred[base] = 1;
            C.real[base] = 1;
            C.tdec[base] = 0.0;
            C.bank[base] = 0.0f;
            C.pend[base] = 0;
            atomicOr(C.err, 2u);
        }
        C.n[w] = over ? 1 : n;
    }
    __syncwarp();  // the slots are visible to the warp's build
    return over ? 1 : n;
}

// The banked decode slack of every slot from its l_out and t^dec (after the
// host wrote the slots: creation, host loads, restore).
__global__ void k_bank(DevParams P, ClusterDev C)
{
    const long long slots = (long long)C.W * C.cap;
    for (long long s = (long long)blockIdx.x * blockDim.x + threadIdx.x; s < slots;
         s += (long long)gridDim.x * blockDim.x)
        C.bank[s] = banked_slack(P, C.gen[s], C.tdec[s]);
}

cudaError_t launch_bank(const DevParams& P, const ClusterDev& C, cudaStream_t st)
{
    const long long slots = (long long)C.W * C.cap;
    const long long nb = (slots + 255) / 256;
    k_bank<<<(int)(nb < 4096 ? nb : 4096), 256, 0, st>>>(P, C);
    return cudaGetLastError();
}

template <int E>
__global__ void __launch_bounds__(BUILD_WARPS * 32)
k_build(DevParams P, ClusterDev C, const int32_t* __restrict__ list, int count, PackSrc S)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    BuildSmem<E>* sm = reinterpret_cast<BuildSmem<E>*>(smraw);
    const int warp = threadIdx.x >> 5;
    const int idx = blockIdx.x * BUILD_WARPS + warp;
    if (idx >= count) return;  // whole warp leaves together
    const int w = list ? list[idx] : idx;
    if (S.off) pack_worker(P, C, S, w);
    build_table<E>(P, C, w, sm[warp]);
}

// Workers of a cluster with b_cap > 128 slots usually hold far fewer
// requests than slots. The build runs as a cascade: a 128-element warp build
// for every worker that fits (fewer registers, a quarter of the sorting work
// of a 512-slot build), the full-capacity build only for the workers that do
// not, listed on the device by the first pass.
constexpr int E_LO = 4;

template <int E>
__global__ void __launch_bounds__(BUILD_WARPS * 32)
k_build_lo(DevParams P, ClusterDev C, int count, int32_t* __restrict__ ovf, int* __restrict__ novf,
           PackSrc S)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    BuildSmem<E>* sm = reinterpret_cast<BuildSmem<E>*>(smraw);
    const int warp = threadIdx.x >> 5;
    const int w = blockIdx.x * BUILD_WARPS + warp;
    if (w >= count) return;
    const int n = S.off ? pack_worker(P, C, S, w) : C.n[w];
    if (n > 32 * E) {  // warp-uniform
        if ((threadIdx.x & 31) == 0) ovf[atomicAdd(novf, 1)] = w;
        return;
    }
    build_table<E>(P, C, w, sm[warp]);
}

// A grid of at most OVF_BLOCKS CTAs whose warps take the listed workers in
// turn: usually the list is empty, and a small grid costs less to launch.
constexpr int OVF_BLOCKS = 256;

template <int E>
__global__ void __launch_bounds__(BUILD_WARPS * 32)
k_build_ovf(DevParams P, ClusterDev C, const int32_t* __restrict__ ovf, const int* __restrict__ novf)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    BuildSmem<E>* sm = reinterpret_cast<BuildSmem<E>*>(smraw);
    const int warp = threadIdx.x >> 5;
    const int n = *novf;
    for (int idx = blockIdx.x * BUILD_WARPS + warp; idx < n; idx += gridDim.x * BUILD_WARPS)
        build_table<E>(P, C, ovf[idx], sm[warp]);
}

// Tables of 1,024 slots: one CTA of NW cooperating warps per worker (a
// single warp cannot hold 32 elements per lane in registers). The workers are
// `list[0..count)` with count read on the device (count_dev) or given.
template <int EW, int NW>
__global__ void __launch_bounds__(NW * 32)
k_build_coop(DevParams P, ClusterDev C, const int32_t* __restrict__ list, int count,
             const int* __restrict__ count_dev)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    BuildSmem<EW, NW>& sm = *reinterpret_cast<BuildSmem<EW, NW>*>(smraw);
    const int n = count_dev ? *count_dev : count;
    if ((int)blockIdx.x >= n) return;  // CTA-uniform
    const int w = list ? list[blockIdx.x] : (int)blockIdx.x;
    build_table_fit<EW, NW>(P, C, w, C.n[w], reinterpret_cast<unsigned char*>(&sm));
}

template <auto Kern>
static cudaError_t allow_smem(size_t smem)
{
    return smem > 48 * 1024 ? allow_max_smem<Kern>() : cudaSuccess;
}

constexpr int COOP_NW = 8;

template <int E>
static cudaError_t build_e(const DevParams& P, const ClusterDev& C, const int32_t* list, int count,
                           cudaStream_t st, const PackSrc& S)
{
    if (count <= 0) return cudaSuccess;
    const int blocks = (count + BUILD_WARPS - 1) / BUILD_WARPS;
    cudaError_t e;
    if constexpr (E > 16) {
        constexpr int EW = E / COOP_NW;
        const size_t sc = sizeof(BuildSmem<EW, COOP_NW>);
        if ((e = allow_smem<k_build_coop<EW, COOP_NW>>(sc)) != cudaSuccess) return e;
        if (list) {
            k_build_coop<EW, COOP_NW><<<count, COOP_NW * 32, sc, st>>>(P, C, list, count, nullptr);
            return cudaGetLastError();
        }
        const size_t slo = sizeof(BuildSmem<E_LO>) * BUILD_WARPS;
        if ((e = allow_smem<k_build_lo<E_LO>>(slo)) != cudaSuccess) return e;
        if ((e = cudaMemsetAsync(C.novf, 0, sizeof(int), st)) != cudaSuccess) return e;
        k_build_lo<E_LO><<<blocks, BUILD_WARPS * 32, slo, st>>>(P, C, count, C.ovf, C.novf, S);
        k_build_coop<EW, COOP_NW><<<count, COOP_NW * 32, sc, st>>>(P, C, C.ovf, 0, C.novf);
        return cudaGetLastError();
    } else {
        if (E > E_LO && !list) {
            constexpr int EL = E > E_LO ? E_LO : E;
            const size_t slo = sizeof(BuildSmem<EL>) * BUILD_WARPS;
            const size_t shi = sizeof(BuildSmem<E>) * BUILD_WARPS;
            if ((e = allow_smem<k_build_lo<EL>>(slo)) != cudaSuccess) return e;
            if ((e = allow_smem<k_build_ovf<E>>(shi)) != cudaSuccess) return e;
            if ((e = cudaMemsetAsync(C.novf, 0, sizeof(int), st)) != cudaSuccess) return e;
            k_build_lo<EL><<<blocks, BUILD_WARPS * 32, slo, st>>>(P, C, count, C.ovf, C.novf, S);
            k_build_ovf<E><<<blocks < OVF_BLOCKS ? blocks : OVF_BLOCKS, BUILD_WARPS * 32, shi, st>>>(
                P, C, C.ovf, C.novf);
            return cudaGetLastError();
        }
        const size_t smem = sizeof(BuildSmem<E>) * BUILD_WARPS;
        if ((e = allow_smem<k_build<E>>(smem)) != cudaSuccess) return e;
        k_build<E><<<blocks, BUILD_WARPS * 32, smem, st>>>(P, C, list, count, S);
        return cudaGetLastError();
    }
}

cudaError_t launch_build(const DevParams& P, const ClusterDev& C, const int32_t* list, int count,
                         cudaStream_t st, const PackSrc* src)
{
    PackSrc S{};
    if (src) {
        if (list) return cudaErrorInvalidValue;  // packing covers every worker
        S = *src;
    }
    switch (lanes_per_worker(C.cap)) {
    case 1: return build_e<1>(P, C, list, count, st, S);
    case 2: return build_e<2>(P, C, list, count, st, S);
    case 4: return build_e<4>(P, C, list, count, st, S);
    case 8: return build_e<8>(P, C, list, count, st, S);
    case 16: return build_e<16>(P, C, list, count, st, S);
    case 32: return build_e<32>(P, C, list, count, st, S);
    default: return cudaErrorInvalidValue;
    }
}

// rank(w) = number of workers ordered before w: larger key, or equal key and
// smaller index (a stable descending sort by capacity_norm). The capacity_norm
// keys stay below 2^63 (a non-negative double's bits plus one, or an integer
// sum of squares below 2^57).
//
// From 8,192 to 24,576 workers: a sort in two launches. k_rank_sort sorts
// each chunk of 1,024 consecutive workers in a CTA (a bitonic network over
// (key, index), one element a thread: the exchanges across warps through
// shared memory, the ones within a warp by shuffles). k_rank_merge then places
// every element, a thread each: its position in its own chunk plus, for every
// other chunk, the number of that chunk's keys ahead of it, found by a binary
// search over the chunk's sorted keys (all W keys are copied into each merge
// CTA's shared memory). Workers of a chunk to the left have smaller indices,
// so their equal keys count as ahead; those of a chunk to the right do not.
// Below 8,192 workers (where the all-pairs count is faster: 6.8 against 13.4
// us at 4,096 workers under ncu; 17.7 against 16.8 at 8,192, 60 against 24 at
// 16,384) and above 24,576 (where the keys no longer fit one CTA's shared
// memory), k_rank_count counts for each worker the keys ahead of it directly
// (all pairs).
constexpr int RANK_S = 1024;                    // workers a chunk (threads a CTA)
constexpr int RANK_MERGE_MAX = 24 * RANK_S;     // keys the merge holds in shared memory
#ifndef ALADDIN_RANK_SORT_MIN
#define ALADDIN_RANK_SORT_MIN 8192
#endif
constexpr int RANK_SORT_MIN = ALADDIN_RANK_SORT_MIN;  // fewer workers: the all-pairs count

// a comes before b
__device__ __forceinline__ bool rank_before(unsigned long long ka, int ia, unsigned long long kb,
                                            int ib)
{
    return ka > kb || (ka == kb && ia < ib);
}

__global__ void __launch_bounds__(RANK_S) k_rank_sort(ClusterDev C)
{
    __shared__ unsigned long long xk[RANK_S];
    __shared__ int xi[RANK_S];
    const int t = threadIdx.x, W = C.W;
    const int w = blockIdx.x * RANK_S + t;
    // padding sorts after every worker (key 0, indices above W - 1)
    unsigned long long k = w < W ? C.key[w] : 0ull;
    int i = w;
    for (int size = 2; size <= RANK_S; size <<= 1) {
        const bool up = (t & size) == 0;  // this block of the network sorts "before" first
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            unsigned long long pk;
            int pi;
            if (stride >= 32) {
                xk[t] = k;
                xi[t] = i;
                __syncthreads();
                pk = xk[t ^ stride];
                pi = xi[t ^ stride];
                __syncthreads();
            } else {
                pk = __shfl_xor_sync(FULL, k, stride);
                pi = __shfl_xor_sync(FULL, i, stride);
            }
            // the lower position of the pair keeps the element that comes
            // first (in an "up" block), the upper one the other
            const bool lower = (t & stride) == 0;
            const bool mine_first = rank_before(k, i, pk, pi);
            if (mine_first != (lower == up)) {
                k = pk;
                i = pi;
            }
        }
    }
    C.rk[w] = k;
    C.ri[w] = i;
}

// Number of keys of the descending run ks[0, n) that are >= key (ge) or > key.
__device__ __forceinline__ int rank_count_ahead(const unsigned long long* ks, int n,
                                                unsigned long long key, bool ge)
{
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        const unsigned long long v = ks[mid];
        if (ge ? v >= key : v > key) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

constexpr int RANK_MT = 256;  // threads of a merge CTA (a quarter of a chunk's elements)

__global__ void __launch_bounds__(RANK_MT) k_rank_merge(ClusterDev C)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    unsigned long long* ks = reinterpret_cast<unsigned long long*>(smraw);
    const int W = C.W;
    const int nchunks = (W + RANK_S - 1) / RANK_S;
    const ulonglong2* src = reinterpret_cast<const ulonglong2*>(C.rk);
    ulonglong2* dst = reinterpret_cast<ulonglong2*>(ks);
    // eight loads in flight a thread (the copy is latency-bound otherwise)
    const int n2 = nchunks * RANK_S / 2;  // key pairs
    for (int p0 = threadIdx.x; p0 < n2; p0 += 8 * RANK_MT) {
        ulonglong2 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            if (p0 + u * RANK_MT < n2) v[u] = __ldg(&src[p0 + u * RANK_MT]);
#pragma unroll
        for (int u = 0; u < 8; ++u)
            if (p0 + u * RANK_MT < n2) dst[p0 + u * RANK_MT] = v[u];
    }
    __syncthreads();
    const int e = blockIdx.x * RANK_MT + threadIdx.x;  // sorted position overall
    const int c = e / RANK_S, t = e % RANK_S;
    const int n_c = min(RANK_S, W - c * RANK_S);  // workers of this chunk (a prefix of it)
    if (t >= n_c) return;
    const unsigned long long key = ks[c * RANK_S + t];
    int r = t;
    for (int c2 = 0; c2 < nchunks; ++c2) {
        if (c2 == c) continue;
        const int n2 = min(RANK_S, W - c2 * RANK_S);
        r += rank_count_ahead(ks + c2 * RANK_S, n2, key, c2 < c);
    }
    const int w = C.ri[c * RANK_S + t];
    C.order[r] = w;
    C.wrec[w].w = __int_as_float(r);
}

// All pairs, for clusters beyond RANK_MERGE_MAX workers: a CTA of 32 warps
// ranks 32 workers (a lane each); its warps split the keys, staged in shared
// memory a chunk at a time and read two at a time as broadcasts. Keys left of
// the worker's block count when >= its key, keys right of it when >, only the
// block's own 32 keys take the full test; the comparison is the sign of the
// 64-bit difference.
constexpr int RANK_WARPS = 32;
constexpr int RANK_CHUNK = 4096;  // keys staged at a time (32 KB)

// -1 if x < y, else 0 (keys below 2^63: the difference does not overflow)
__device__ __forceinline__ int neg_if_lt(unsigned long long x, unsigned long long y)
{
    return (int)((long long)(x - y) >> 63);
}

__global__ void __launch_bounds__(RANK_WARPS * 32) k_rank_count(ClusterDev C)
{
    __shared__ __align__(16) unsigned long long ks[RANK_CHUNK];
    __shared__ int part[RANK_WARPS][33];
    const int lane = threadIdx.x & 31, q = threadIdx.x >> 5;
    const int b0 = blockIdx.x * 32, w = b0 + lane;
    const int W = C.W;
    const unsigned long long kw = w < W ? C.key[w] : 0ull;
    int cnt = 0;
    for (int v0 = 0; v0 < W; v0 += RANK_CHUNK) {
        const int lim = min(RANK_CHUNK, W - v0);
        __syncthreads();
        for (int i = threadIdx.x; i < lim; i += RANK_WARPS * 32) ks[i] = __ldg(&C.key[v0 + i]);
        __syncthreads();
        // this warp's share of the chunk, [j0, j1) in worker indexes, an even
        // number of keys except at the chunk's end
        const int per = ((lim + RANK_WARPS - 1) / RANK_WARPS + 1) & ~1;
        const int j0 = v0 + min(lim, q * per), j1 = v0 + min(lim, (q + 1) * per);
        const int l0 = min(j1, max(j0, b0)), l1 = max(j0, min(j1, b0 + 32));
        if (l0 == j1 && ((j1 - j0) & 1) == 0) {  // all left of the block: pairs
            const ulonglong2* k2 = reinterpret_cast<const ulonglong2*>(ks + (j0 - v0));
            int lt = 0;  // minus the keys below the worker's
#pragma unroll 8
            for (int s = 0; s < (j1 - j0) / 2; ++s) {
                const ulonglong2 kv = k2[s];
                lt += neg_if_lt(kv.x, kw) + neg_if_lt(kv.y, kw);
            }
            cnt += (j1 - j0) + lt;
        } else if (l0 == j0 && l1 == j0 && ((j1 - j0) & 1) == 0) {  // all right: pairs
            const ulonglong2* k2 = reinterpret_cast<const ulonglong2*>(ks + (j0 - v0));
#pragma unroll 8
            for (int s = 0; s < (j1 - j0) / 2; ++s) {
                const ulonglong2 kv = k2[s];
                cnt -= neg_if_lt(kw, kv.x) + neg_if_lt(kw, kv.y);
            }
        } else {
            for (int j = j0; j < l0; ++j) cnt += ks[j - v0] >= kw;
            for (int j = l0; j < l1; ++j) {
                const unsigned long long kv = ks[j - v0];
                cnt += (kv > kw) || (kv == kw && j < w);
            }
            for (int j = l1; j < j1; ++j) cnt += ks[j - v0] > kw;
        }
    }
    part[q][lane] = cnt;
    __syncthreads();
    if (q == 0) {
        int r = 0;
#pragma unroll 8
        for (int k = 0; k < RANK_WARPS; ++k) r += part[k][lane];
        if (w < W) {
            C.order[r] = w;
            C.wrec[w].w = __int_as_float(r);
        }
    }
}

cudaError_t launch_rank(const ClusterDev& C, cudaStream_t st)
{
    if (C.W <= 0) return cudaSuccess;
    const int nchunks = (C.W + RANK_S - 1) / RANK_S;
    if (C.W > RANK_MERGE_MAX || C.W < RANK_SORT_MIN) {
        k_rank_count<<<(C.W + 31) / 32, RANK_WARPS * 32, 0, st>>>(C);
        return cudaGetLastError();
    }
    k_rank_sort<<<nchunks, RANK_S, 0, st>>>(C);
    const size_t smem = sizeof(unsigned long long) * (size_t)nchunks * RANK_S;
    cudaError_t e = allow_smem<k_rank_merge>(smem);
    if (e != cudaSuccess) return e;
    k_rank_merge<<<nchunks * (RANK_S / RANK_MT), RANK_MT, smem, st>>>(C);
    return cudaGetLastError();
}

}  // namespace aladdin
