// A best-fit round under distributed grouped scheduling (Appendix A): the
// requests are dealt to G groups round-robin and every group places its own
// requests on its own workers (w = g mod G), so the groups are independent
// schedulers. On the GPU they run side by side: CTA g runs group g's chain
// of Algorithm 1 (candidates in index order, each on the feasible worker of
// its group with the largest capacity_norm, lowest index on ties), touching
// only its own workers, so the CTAs share nothing. Per candidate every
// thread evaluates a strided share of the group's workers from their table
// rows, a block reduction picks the winner, and the build warps append the
// request and rebuild that worker's table before the group's next candidate.
// A group whose chosen worker has no free slot stops there (status -2); the
// other groups go on.
#include "aladdin_host.h"

namespace aladdin {

constexpr int GR_THREADS = 512;
constexpr int GR_WARPS = GR_THREADS / 32;

template <int EW, int NW>
struct GroupSmem {
    BuildSmem<EW, NW> build;
    unsigned long long bk[GR_WARPS];
    int bw[GR_WARPS];
    int win;
};

// (key, worker): larger key, then lower index; w < 0 is "none".
__device__ __forceinline__ void gr_better(unsigned long long& bk, int& bw, unsigned long long k,
                                          int w)
{
    if (w >= 0 && (bw < 0 || k > bk || (k == bk && w < bw))) {
        bk = k;
        bw = w;
    }
}

template <int EW, int NW>
__global__ void __launch_bounds__(GR_THREADS) k_round_grp(DevParams P, ClusterDev C, RoundIO io)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    GroupSmem<EW, NW>& sm = *reinterpret_cast<GroupSmem<EW, NW>*>(smraw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int G = P.groups, g = blockIdx.x, W = C.W;
    const int n = io.n_cand;
    // the group's first candidate: (rid0 + c) mod G == g
    const int c0 = (int)((((long long)g - io.rid0 % G) % G + G) % G);
    bool stopped = false;
    for (int c = c0; c < n; c += G) {
        if (stopped) {  // CTA-uniform
            if (tid == 0) io.placement[c] = -1;
            continue;
        }
        const int32_t a = io.in[c], r = io.pred[c];
        const double wd = io.wait ? (double)io.wait[c] : 0.0;
        const CandRec cr = make_cand(P, a, r, (float)wd, c);
        if (!cr.valid) {
            if (tid == 0) io.placement[c] = -2;  // ALADDIN_INVALID
            continue;
        }
        unsigned long long bk = 0ull;
        int bw = -1;
        for (int w = g + tid * G; w < W; w += GR_THREADS * G) {
            const long long rb = (long long)w * C.rows;
            const int p = find_row<false>(C.tab, rb, C.R[w], cr.ri);
            const float4* t = C.tab + (rb + p) * ROW_F4;
            float m;
            const unsigned f =
                eval_pair_mode(P.approx != 0, t[0], t[1], C.tab2[rb + p], C.wrec[w],
                               P.approx ? C.wapx[w] : make_float2(0.0f, 0.0f), cr, m);
            if (f == 15u) gr_better(bk, bw, C.key[w], w);
        }
#pragma unroll
        for (int d = 16; d > 0; d >>= 1) {
            const unsigned long long ok = __shfl_xor_sync(FULL, bk, d);
            const int ow = __shfl_xor_sync(FULL, bw, d);
            gr_better(bk, bw, ok, ow);
        }
        if (lane == 0) {
            sm.bk[warp] = bk;
            sm.bw[warp] = bw;
        }
        __syncthreads();
        if (warp == 0) {
            bk = lane < GR_WARPS ? sm.bk[lane] : 0ull;
            bw = lane < GR_WARPS ? sm.bw[lane] : -1;
#pragma unroll
            for (int d = 16; d > 0; d >>= 1) {
                const unsigned long long ok = __shfl_xor_sync(FULL, bk, d);
                const int ow = __shfl_xor_sync(FULL, bw, d);
                gr_better(bk, bw, ok, ow);
            }
            if (lane == 0) sm.win = bw;
        }
        __syncthreads();
        const int win = sm.win;
        if (win >= 0 && C.n[win] >= C.cap) {  // no free slot: the group stops
            if (tid == 0) {
                *io.status = -2;  // ALADDIN_ERR_CAPACITY
                io.placement[c] = -1;
            }
            stopped = true;
            __syncthreads();
            continue;
        }
        if (win >= 0 && warp < NW) {
            if (tid == 0) {
                const long long sl = (long long)win * C.cap + C.n[win];
                C.in[sl] = a;
                C.gen[sl] = 0;
                C.pred[sl] = r;
                C.real[sl] = r;
                C.tdec[sl] = 0.0;
                C.pend[sl] = 1;
                C.wait[sl] = wd;
                C.n[win] += 1;
            }
            group_sync<NW>();
            if constexpr (NW == 1)
                build_table<EW>(P, C, win, sm.build);
            else
                build_table_fit<EW, NW>(P, C, win, C.n[win],
                                        reinterpret_cast<unsigned char*>(&sm.build));
        }
        if (tid == 0) io.placement[c] = win;  // -1: no feasible worker in the group
        __syncthreads();
    }
}

template <int EW, int NW>
static cudaError_t round_grp_e(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                               cudaStream_t st)
{
    const size_t smem = sizeof(GroupSmem<EW, NW>);
    if (smem > 48 * 1024) {
        const cudaError_t e = allow_max_smem<k_round_grp<EW, NW>>();
        if (e != cudaSuccess) return e;
    }
    k_round_grp<EW, NW><<<P.groups, GR_THREADS, smem, st>>>(P, C, io);
    return cudaGetLastError();
}

cudaError_t launch_round_groups(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                                cudaStream_t st)
{
    switch (lanes_per_worker(C.cap)) {  // rebuilds as in the re-balancing kernel
    case 1: return round_grp_e<1, 1>(P, C, io, st);
    case 2: return round_grp_e<2, 1>(P, C, io, st);
    case 4: return round_grp_e<4, 1>(P, C, io, st);
    case 8: return round_grp_e<4, 2>(P, C, io, st);
    case 16: return round_grp_e<4, 4>(P, C, io, st);
    case 32: return round_grp_e<4, 8>(P, C, io, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace aladdin
