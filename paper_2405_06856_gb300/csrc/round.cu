// K4: one greedy best-fit placement round (Algorithm 1).
//
// Candidates are placed in index (arrival) order; candidate c+1 sees the state
// left by candidate c, so the round is a sequential chain. One CTA runs the
// whole chain: for each candidate all threads evaluate the workers
// (strided), a block reduction picks the feasible worker of largest
// capacity_norm (lowest index on ties), and warp 0 appends the request to that
// worker and rebuilds only that worker's table and key before the next
// candidate. In trace mode (fleet simulation) the candidates are the waiting
// requests followed by the heartbeat's arrivals; unplaced requests that can
// still meet their TTFT stay in the waiting list, the others fail.
#include "aladdin_host.h"

namespace aladdin {

constexpr int ROUND_THREADS = 512;
constexpr int ROUND_WARPS = ROUND_THREADS / 32;

template <int E>
struct RoundSmem {
    BuildSmem<E> build;
    unsigned long long bk[ROUND_WARPS];
    int bw[ROUND_WARPS];
    int winner;
    int stop;
};

__device__ __forceinline__ void better(unsigned long long& bk, int& bw, unsigned long long ok, int ow)
{
    if (ow != 0x7fffffff && (bw == 0x7fffffff || ok > bk || (ok == bk && ow < bw))) {
        bk = ok;
        bw = ow;
    }
}

template <int E>
__global__ void __launch_bounds__(ROUND_THREADS) k_round(DevParams P, ClusterDev C, RoundIO io)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    RoundSmem<E>& sm = *reinterpret_cast<RoundSmem<E>*>(smraw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_wait0 = io.sim ? *io.n_wait : 0;
    const int n_cand = io.sim ? n_wait0 + (int)(io.arr_end - io.arr_begin) : io.n_cand;
    int keep = 0;  // thread 0: new waiting-list length
    if (tid == 0) sm.stop = (io.sim && *io.status != 0) ? 1 : 0;
    __syncthreads();
    if (sm.stop) return;

    for (int c = 0; c < n_cand; ++c) {
        long long tix = 0;
        int32_t a, r;
        double wd;
        if (io.sim) {
            tix = c < n_wait0 ? io.wl[c] : io.arr_begin + (c - n_wait0);
            a = io.tin[tix];
            r = io.tpred[tix];
            wd = io.t_now - io.t_arr[tix];
        } else {
            a = io.in[c];
            r = io.pred[c];
            wd = io.wait ? (double)io.wait[c] : 0.0;
        }
        const CandRec cr = make_cand(P, a, r, (float)wd, c);
        int winner = -2;
        if (cr.valid) {
            unsigned long long bk = 0ull;
            int bw = 0x7fffffff;
            for (int w = tid; w < C.W; w += ROUND_THREADS) {
                const long long rb = (long long)w * C.rows;
                const int p = find_row<false>(C.tab, rb, C.R[w], cr.ri);
                const float4* t = C.tab + (rb + p) * ROW_F4;
                float m;
                const unsigned f = eval_pair(t[0], t[1], C.tab2[rb + p], C.wrec[w], cr, m);
                if (f == 15u) better(bk, bw, C.key[w], w);
            }
#pragma unroll
            for (int d = 16; d > 0; d >>= 1) {
                const unsigned long long ok = __shfl_xor_sync(FULL, bk, d);
                const int ow = __shfl_xor_sync(FULL, bw, d);
                better(bk, bw, ok, ow);
            }
            if (lane == 0) {
                sm.bk[warp] = bk;
                sm.bw[warp] = bw;
            }
            __syncthreads();
            if (warp == 0) {
                bk = lane < ROUND_WARPS ? sm.bk[lane] : 0ull;
                bw = lane < ROUND_WARPS ? sm.bw[lane] : 0x7fffffff;
#pragma unroll
                for (int d = 16; d > 0; d >>= 1) {
                    const unsigned long long ok = __shfl_xor_sync(FULL, bk, d);
                    const int ow = __shfl_xor_sync(FULL, bw, d);
                    better(bk, bw, ok, ow);
                }
                if (lane == 0) sm.winner = bw == 0x7fffffff ? -1 : bw;
            }
            __syncthreads();
            winner = sm.winner;
        }
        if (winner >= 0) {
            if (warp == 0) {
                const int nw = C.n[winner];
                const int full = nw >= C.cap;
                if (!full && lane == 0) {
                    const long long slot = (long long)winner * C.cap + nw;
                    C.in[slot] = a;
                    C.gen[slot] = 0;
                    C.pred[slot] = r;
                    C.tdec[slot] = 0.0;
                    C.pend[slot] = 1;
                    C.wait[slot] = wd;
                    C.n[winner] = nw + 1;
                }
                __syncwarp();
                if (!full) {
                    build_table<E>(P, C, winner, sm.build);
                } else if (lane == 0) {
                    *io.status = -2;  // ALADDIN_ERR_CAPACITY
                    sm.stop = 1;
                }
            }
        }
        if (tid == 0 && !sm.stop) {
            if (!io.sim) {
                io.placement[c] = winner;
            } else if (winner >= 0) {
                io.counters[1] += 1;
            } else {
                const double tau_alone = C.scaled[0] * (P.k1d * (double)a + P.c1d);
                if (winner == -2 || wd + io.H + tau_alone > P.T_pred) io.counters[0] += 1;
                else io.wl[keep++] = tix;
            }
        }
        __syncthreads();
        if (sm.stop) {
            if (tid == 0 && !io.sim)
                for (int k = c; k < n_cand; ++k) io.placement[k] = -1;
            break;
        }
    }
    if (tid == 0 && io.sim && !sm.stop) {
        *io.n_wait = keep;
        if (io.stop_at_fail && io.counters[0] > 0) {
            *io.status = 1;
            io.counters[2] = (unsigned long long)io.hb;
        }
    }
}

template <int E>
static cudaError_t round_e(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                           cudaStream_t st)
{
    const size_t smem = sizeof(RoundSmem<E>);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_round<E>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
    }
    k_round<E><<<1, ROUND_THREADS, smem, st>>>(P, C, io);
    return cudaGetLastError();
}

cudaError_t launch_round(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                         cudaStream_t st)
{
    switch (lanes_per_worker(C.cap)) {
    case 1: return round_e<1>(P, C, io, st);
    case 2: return round_e<2>(P, C, io, st);
    case 4: return round_e<4>(P, C, io, st);
    case 8: return round_e<8>(P, C, io, st);
    case 16: return round_e<16>(P, C, io, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace aladdin
