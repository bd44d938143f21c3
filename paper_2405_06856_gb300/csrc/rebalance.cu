// Algorithm 2 (Sec. 4.3, re-balancing with prediction error): after a
// placement round and before it executes, the round's requests on workers
// whose running requests outgrew their predictions (error e > 0) move to
// workers whose requests finished early (e < 0).
//
// Worker i's error e_i = k2 l^e_i + c2 b^e_i is its output-length and
// batch-size error (l^e, b^e) measured along the normal of Eq. input limit's
// boundary k2 l + c2 b = T_dec - c3; |e_i| / sqrt(k2^2 + c2^2) is the distance
// of the error line through (l^e_i, b^e_i) to the origin, the quantity the
// algorithm minimises summed over workers. Moving request j (predicted output
// l_j) from x to y moves d_j = k2 l_j + c2 of error from x to y.
//
// The round is a sequential chain (each move changes two workers' errors
// and tables), so one CTA runs it, like the single-CTA placement round: per
// candidate on an over-utilized worker, every thread scores a strided share
// of the under-utilized workers (feasibility in O(1) from the table row, then
// the gain), a block reduction picks the largest gain (then the larger
// capacity_norm key, then the lower index), and the build warps move the
// request and rebuild both workers' tables. Error arithmetic is fp64 with
// explicitly rounded operations, in the oracle's order.
#include "aladdin_host.h"

namespace aladdin {

constexpr int RB_THREADS = 512;
constexpr int RB_WARPS = RB_THREADS / 32;

template <int EW, int NW>
struct RebalSmem {
    BuildSmem<EW, NW> build;
    double bg[RB_WARPS];
    unsigned long long bk[RB_WARPS];
    int bw[RB_WARPS];
    double part[RB_WARPS];
    int win;
    int q;
};

// (g, k, w) better than (bg, bk, bw): larger gain, then larger key, then
// lower index; w < 0 is "none".
__device__ __forceinline__ bool rb_better(double g, unsigned long long k, int w, double bg,
                                          unsigned long long bk, int bw)
{
    if (w < 0) return false;
    if (bw < 0) return true;
    if (g != bg) return g > bg;
    if (k != bk) return k > bk;
    return w < bw;
}

__device__ __forceinline__ void rb_reduce_warp(double& g, unsigned long long& k, int& w)
{
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
        const double og = __shfl_xor_sync(FULL, g, d);
        const unsigned long long ok = __shfl_xor_sync(FULL, k, d);
        const int ow = __shfl_xor_sync(FULL, w, d);
        if (rb_better(og, ok, ow, g, k, w)) {
            g = og;
            k = ok;
            w = ow;
        }
    }
}

template <int NT>
__device__ __forceinline__ double rb_block_sum(double v, double* part)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_reduce(v, OpAdd<double>());
    __syncthreads();
    if (lane == 0) part[warp] = v;
    __syncthreads();
    double s = 0.0;
    for (int i = 0; i < NT / 32; ++i) s = __dadd_rn(s, part[i]);
    return s;
}

template <int EW, int NW>
__device__ __forceinline__ void rb_build(const DevParams& P, const ClusterDev& C, int w,
                                         RebalSmem<EW, NW>& sm)
{
    if constexpr (NW == 1)
        build_table<EW>(P, C, w, sm.build);
    else
        build_table_fit<EW, NW>(P, C, w, C.n[w], reinterpret_cast<unsigned char*>(&sm.build));
}

template <int EW, int NW>
__global__ void __launch_bounds__(RB_THREADS) k_rebalance(DevParams P, ClusterDev C, RoundIO io,
                                                          int* moves, double* obj)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    RebalSmem<EW, NW>& sm = *reinterpret_cast<RebalSmem<EW, NW>*>(smraw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int W = C.W;
    if (io.sim && *io.status != 0) return;  // the simulation halted: no round ran
    const int n_cand = io.sim ? *io.sim_n : io.n_cand;

    // errors e_w = k2 l^e + c2 b^e and their summed distance
    double s0 = 0.0;
    for (int w = tid; w < W; w += RB_THREADS) {
        const double e =
            __dadd_rn(__dmul_rn(P.k2d, (double)C.le[w]), __dmul_rn(P.c2d, (double)C.be[w]));
        C.err_e[w] = e;
        s0 = __dadd_rn(s0, fabs(e));
    }
    const double before = rb_block_sum<RB_THREADS>(s0, sm.part);  // ends with a barrier
    int nmov = 0;

    for (int c = 0; c < n_cand; ++c) {
        const int x = io.sim ? io.sim_pl[c] : io.placement[c];
        if (x < 0) continue;  // uniform
        const double ex = C.err_e[x];
        if (!(ex > 0.0)) continue;
        int32_t a, r;
        double wd;
        long long rid = io.rid0 + c;
        if (io.sim) {
            const long long tix = io.sim_tix[c];
            rid = tix;
            a = io.tin[tix];
            r = io.tpred[tix];
            wd = io.t_now - io.t_arr[tix];
        } else {
            a = io.in[c];
            r = io.pred[c];
            wd = io.wait ? (double)io.wait[c] : 0.0;
        }
        const CandRec cr = make_cand(P, a, r, (float)wd, c);
        if (!cr.valid) continue;
        const double d = __dadd_rn(__dmul_rn(P.k2d, (double)r), P.c2d);
        const int G = P.groups;
        const int grp = G > 1 ? (int)(rid % G) : 0;  // moves stay in the request's group
        double bg = 0.0;
        unsigned long long bk = 0ull;
        int bw = -1;
        for (int y = tid; y < W; y += RB_THREADS) {
            const double ey = C.err_e[y];
            if (y == x || !(ey < 0.0) || C.n[y] >= C.cap || (G > 1 && y % G != grp)) continue;
            const double g = __dsub_rn(__dsub_rn(__dsub_rn(ex, ey), fabs(__dsub_rn(ex, d))),
                                       fabs(__dadd_rn(ey, d)));
            if (!(g > 0.0)) continue;
            const unsigned long long ky = C.key[y];
            if (!rb_better(g, ky, y, bg, bk, bw)) continue;
            const long long rb = (long long)y * C.rows;
            const int p = find_row<false>(C.tab, rb, C.R[y], cr.ri);
            const float4* t = C.tab + (rb + p) * ROW_F4;
            float m;
            const unsigned f =
                eval_pair_mode(P.approx != 0, t[0], t[1], C.tab2[rb + p], C.wrec[y],
                               P.approx ? C.wapx[y] : make_float2(0.0f, 0.0f), cr, m);
            if (f == 15u) {
                bg = g;
                bk = ky;
                bw = y;
            }
        }
        rb_reduce_warp(bg, bk, bw);
        if (lane == 0) {
            sm.bg[warp] = bg;
            sm.bk[warp] = bk;
            sm.bw[warp] = bw;
        }
        __syncthreads();
        if (warp == 0) {
            bg = lane < RB_WARPS ? sm.bg[lane] : 0.0;
            bk = lane < RB_WARPS ? sm.bk[lane] : 0ull;
            bw = lane < RB_WARPS ? sm.bw[lane] : -1;
            rb_reduce_warp(bg, bk, bw);
            if (lane == 0) sm.win = bw;
        }
        __syncthreads();
        const int y = sm.win;
        if (y < 0) continue;  // uniform
        if (warp < NW) {
            if (tid == 0) {
                // the request's pending slot on x: the last one with its values
                int q = -1;
                const long long bx = (long long)x * C.cap;
                for (int k = C.n[x] - 1; k >= 0 && q < 0; --k) {
                    const long long sl = bx + k;
                    if (C.pend[sl] && C.in[sl] == a && C.pred[sl] == r && C.wait[sl] == wd) q = k;
                }
                sm.q = q;
            }
            group_sync<NW>();
            const int q = sm.q;
            if (q >= 0) {
                int32_t rl = r;
                if (tid == 0) {
                    const long long bx = (long long)x * C.cap;
                    const long long sl = bx + q, last = bx + C.n[x] - 1;
                    rl = C.real[sl];
                    C.in[sl] = C.in[last];
                    C.gen[sl] = C.gen[last];
                    C.pred[sl] = C.pred[last];
                    C.real[sl] = C.real[last];
                    C.tdec[sl] = C.tdec[last];
                    C.bank[sl] = C.bank[last];
                    C.pend[sl] = C.pend[last];
                    C.wait[sl] = C.wait[last];
                    C.n[x] -= 1;
                }
                group_sync<NW>();
                rb_build<EW, NW>(P, C, x, sm);
                group_sync<NW>();
                if (tid == 0) {
                    const long long sl = (long long)y * C.cap + C.n[y];
                    C.in[sl] = a;
                    C.gen[sl] = 0;
                    C.pred[sl] = r;
                    C.real[sl] = rl;
                    C.tdec[sl] = 0.0;
                    C.pend[sl] = 1;
                    C.wait[sl] = wd;
                    C.n[y] += 1;
                }
                group_sync<NW>();
                rb_build<EW, NW>(P, C, y, sm);
                if (tid == 0) {
                    C.err_e[x] = __dsub_rn(ex, d);
                    C.err_e[y] = __dadd_rn(C.err_e[y], d);
                    if (io.sim) io.sim_pl[c] = y;
                    else io.placement[c] = y;
                    nmov += 1;
                }
            }
        }
        __syncthreads();
    }
    double s1 = 0.0;
    for (int w = tid; w < W; w += RB_THREADS) s1 = __dadd_rn(s1, fabs(C.err_e[w]));
    const double after = rb_block_sum<RB_THREADS>(s1, sm.part);
    if (tid == 0) {
        if (moves) *moves += nmov;
        if (obj) {
            const double norm = sqrt(__dadd_rn(__dmul_rn(P.k2d, P.k2d), __dmul_rn(P.c2d, P.c2d)));
            obj[0] = before / norm;
            obj[1] = after / norm;
        }
    }
}

template <int EW, int NW>
static cudaError_t rebalance_e(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                               int* moves, double* obj, cudaStream_t st)
{
    const size_t smem = sizeof(RebalSmem<EW, NW>);
    if (smem > 48 * 1024) {
        const cudaError_t e = allow_max_smem<k_rebalance<EW, NW>>();
        if (e != cudaSuccess) return e;
    }
    k_rebalance<EW, NW><<<1, RB_THREADS, smem, st>>>(P, C, io, moves, obj);
    return cudaGetLastError();
}

cudaError_t launch_rebalance(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                             int* moves, double* obj, cudaStream_t st)
{
    switch (lanes_per_worker(C.cap)) {
    case 1: return rebalance_e<1, 1>(P, C, io, moves, obj, st);
    case 2: return rebalance_e<2, 1>(P, C, io, moves, obj, st);
    case 4: return rebalance_e<4, 1>(P, C, io, moves, obj, st);
    // above 128 slots the rebuild is cooperative (4 elements a lane, so that a
    // thread of the 512-thread CTA stays within its 128 registers)
    case 8: return rebalance_e<4, 2>(P, C, io, moves, obj, st);
    case 16: return rebalance_e<4, 4>(P, C, io, moves, obj, st);
    case 32: return rebalance_e<4, 8>(P, C, io, moves, obj, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace aladdin
