// Placement rounds of the load-balancing baselines the paper compares
// Algorithm 1 with (Sec. 6.1 baselines, Sec. 6.4 simulations): join the
// shortest queue (JSQ) and the power of two choices (Po2). Neither tests
// feasibility; a placement that breaks an SLO shows up when the workers
// execute (the violations counted by k_advance).
//
// The round is a sequential chain (each placement changes the counts the
// next one reads), so one CTA runs it with the per-worker request counts in
// shared memory. JSQ: per candidate, a block-wide argmin of (count, index);
// Po2: two SplitMix64 draws and one comparison by thread 0. Thread 0 appends
// the request to the chosen worker's next free slot as a pending request of
// the round (prefill at the worker's next boundary, gen = 0).
#include "aladdin.h"
#include "aladdin_host.h"

namespace aladdin {

constexpr int Q_THREADS = 1024;
constexpr int Q_WARPS = Q_THREADS / 32;
constexpr int Q_SMEM_MAX_W = 49152;  // workers whose counts fit in shared memory (192 KB)

// SplitMix64 (G. Steele, D. Lea, C. Flood, "Fast splittable pseudorandom
// number generators", OOPSLA 2014): output n >= 1 of the stream seeded with s
// is the mixing function applied to s + n * 0x9E3779B97F4A7C15 (mod 2^64).
__device__ __forceinline__ unsigned long long splitmix64(unsigned long long s,
                                                         unsigned long long n)
{
    unsigned long long z = s + n * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// Worker of draw k (0 or 1) for request id rid: output 2 rid + k + 1, its
// upper 32 bits scaled to [0, W).
__device__ __forceinline__ int po2_draw(unsigned long long seed, long long rid, int k, int W)
{
    const unsigned long long x =
        splitmix64(seed, 2ull * (unsigned long long)rid + (unsigned long long)k + 1ull);
    return (int)(((x >> 32) * (unsigned long long)W) >> 32);
}

__global__ void __launch_bounds__(Q_THREADS) k_round_queue(DevParams P, ClusterDev C, RoundIO io,
                                                           int shared_counts)
{
    extern __shared__ int cnt_s[];
    __shared__ unsigned long long red[Q_WARPS];
    __shared__ int s_stop;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int W = C.W;
    if (tid == 0) s_stop = (io.sim && *io.status != 0) ? 1 : 0;
    __syncthreads();
    if (s_stop) return;
    int* cnt = shared_counts ? cnt_s : C.n;
    if (shared_counts) {
        for (int w = tid; w < W; w += Q_THREADS) cnt_s[w] = C.n[w];
        __syncthreads();
    }
    // every waiting request was placed or failed in its own round: no list
    const int n_cand = io.sim ? (int)(io.arr_end - io.arr_begin) : io.n_cand;
    const bool jsq = P.policy == ALADDIN_POLICY_JSQ;

    for (int c = 0; c < n_cand; ++c) {
        long long tix;
        int32_t a, r;
        double wd;
        if (io.sim) {
            tix = io.arr_begin + c;
            a = io.tin[tix];
            r = io.tpred[tix];
            wd = io.t_now - io.t_arr[tix];
        } else {
            tix = io.rid0 + c;
            a = io.in[c];
            r = io.pred[c];
            wd = io.wait ? (double)io.wait[c] : 0.0;
        }
        const bool valid0 = a >= 0 && r >= 1 && (long long)a + r <= (long long)P.K && wd >= 0.0 &&
                            wd <= 3.0e38;
        // grouped scheduling: group g = id mod G owns workers g, g + G, ...
        const int G = P.groups;
        const int grp = G > 1 ? (int)(tix % G) : 0;
        const int Wg = W > grp ? (W - grp + G - 1) / G : 0;
        const bool valid = valid0 && Wg > 0;
        int choice = -1;
        if (valid && jsq) {
            // smallest (count, index): counts < 2^31, indexes < 2^31
            unsigned long long best = ~0ull;
            for (int w = grp + tid * G; w < W; w += Q_THREADS * G) {
                const unsigned long long k =
                    ((unsigned long long)(unsigned)cnt[w] << 32) | (unsigned)w;
                best = k < best ? k : best;
            }
            best = warp_reduce(best, OpMin<unsigned long long>());
            if (lane == 0) red[warp] = best;
            __syncthreads();
            if (warp == 0) {
                best = red[lane];
                best = warp_reduce(best, OpMin<unsigned long long>());
                __syncwarp();
                if (lane == 0) red[0] = best;
            }
            __syncthreads();
            choice = (int)(red[0] & 0xffffffffull);
        }
        if (tid == 0) {
            if (valid && !jsq) {
                const int w1 = grp + G * po2_draw(P.seed, tix, 0, Wg);
                const int w2 = grp + G * po2_draw(P.seed, tix, 1, Wg);
                choice = cnt[w2] < cnt[w1] ? w2 : w1;
            }
            if (!valid0) {
                if (io.sim) io.counters[0] += 1;
                else io.placement[c] = -2;  // ALADDIN_INVALID
            } else if (!valid || cnt[choice] >= C.cap) {  // no worker in the group, or full
                if (io.sim) {
                    io.counters[0] += 1;  // no free slot: the request fails
                } else {
                    *io.status = -2;  // ALADDIN_ERR_CAPACITY
                    for (int k = c; k < n_cand; ++k) io.placement[k] = -1;
                    s_stop = 1;
                }
            } else {
                const int nw = cnt[choice];
                const long long slot = (long long)choice * C.cap + nw;
                C.in[slot] = a;
                C.gen[slot] = 0;
                C.pred[slot] = r;
                C.real[slot] = io.sim && io.treal ? io.treal[tix] : r;
                C.tdec[slot] = 0.0;
                C.pend[slot] = 1;
                C.wait[slot] = wd;
                cnt[choice] = nw + 1;
                if (io.sim) io.counters[1] += 1;
                else io.placement[c] = choice;
            }
        }
        __syncthreads();
        if (s_stop) break;
    }
    if (shared_counts)
        for (int w = tid; w < W; w += Q_THREADS) C.n[w] = cnt_s[w];
    if (tid == 0 && io.sim) {
        *io.n_wait = 0;
        if (io.stop_at_fail && io.counters[0] > 0) {
            *io.status = 1;
            io.counters[2] = (unsigned long long)io.hb;
        }
    }
}

cudaError_t launch_round_queue(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                               cudaStream_t st)
{
    const int shared = C.W <= Q_SMEM_MAX_W ? 1 : 0;
    const size_t smem = shared ? sizeof(int) * (size_t)C.W : 0;
    if (smem > 48 * 1024) {
        const cudaError_t e = allow_max_smem<k_round_queue>();
        if (e != cudaSuccess) return e;
    }
    k_round_queue<<<1, Q_THREADS, smem, st>>>(P, C, io, shared);
    return cudaGetLastError();
}

}  // namespace aladdin
