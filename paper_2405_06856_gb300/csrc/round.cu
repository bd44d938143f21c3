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
// still meet their TTFT stay in the waiting list, the others fail (on a
// decode instance every unplaced request fails).
#include "round_common.cuh"

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
    const int c_begin = (!io.sim && io.c_first) ? *io.c_first : 0;
    int keep = 0;  // thread 0: new waiting-list length
    if (tid == 0) sm.stop = ((io.sim && *io.status != 0) || c_begin >= n_cand) ? 1 : 0;
    __syncthreads();
    if (sm.stop) return;

    for (int c = c_begin; c < n_cand; ++c) {
        long long tix = 0;
        int32_t a, r, rl;
        double wd;
        if (io.sim) {
            tix = c < n_wait0 ? io.wl[c] : io.arr_begin + (c - n_wait0);
            a = io.tin[tix];
            r = io.tpred[tix];
            rl = io.treal ? io.treal[tix] : r;
            wd = io.t_now - io.t_arr[tix];
        } else {
            a = io.in[c];
            r = io.pred[c];
            rl = r;
            wd = io.wait ? (double)io.wait[c] : 0.0;
        }
        const CandRec cr = make_cand(P, a, r, (float)wd, c);
        // grouped scheduling: the request's group places on its own workers
        const int G = P.groups;
        const int grp = G > 1 ? (int)((io.sim ? tix : io.rid0 + c) % G) : 0;
        int winner = -2;
        if (cr.valid) {
            unsigned long long bk = 0ull;
            int bw = 0x7fffffff;
            for (int w = tid; w < C.W; w += ROUND_THREADS) {
                if (G > 1 && w % G != grp) continue;
                const long long rb = (long long)w * C.rows;
                const int p = find_row<false>(C.tab, rb, C.R[w], cr.ri);
                const float4* t = C.tab + (rb + p) * ROW_F4;
                float m;
                const unsigned f =
                    eval_pair_mode(P.approx != 0, t[0], t[1], C.tab2[rb + p], C.wrec[w],
                                   P.approx ? C.wapx[w] : make_float2(0.0f, 0.0f), cr, m);
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
                    C.real[slot] = rl;
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
            if (io.sim && io.sim_pl) {
                io.sim_pl[c] = winner;
                io.sim_tix[c] = tix;
            }
            if (!io.sim) {
                io.placement[c] = winner;
            } else if (winner >= 0) {
                io.counters[1] += 1;
            } else {
                const double tau_alone = C.scaled[0] * (P.k1d * (double)a + P.c1d);
                // a decode instance has no TTFT budget to absorb a wait
                if (winner == -2 || P.decode || wd + io.H + tau_alone > P.T_pred)
                    io.counters[0] += 1;
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
        if (io.sim_n) *io.sim_n = n_cand;
        *io.n_wait = keep;
        if (io.stop_at_fail && io.counters[0] > 0) {
            *io.status = 1;
            io.counters[2] = (unsigned long long)io.hb;
        }
    }
}

// ---------------------------------------------------------------------------
// Sliced round: the workers are split into contiguous slices, one per CTA of a
// cooperative grid (one CTA when they fit). Each CTA keeps its slice's
// breakpoints (16-bit rho_{p+1} of rows 0..R-1), request counts, worker
// records and keys in shared memory, so locating a candidate's row is a
// shared-memory search and one global load of the row.
//
// Candidate c is committed lazily: its winner's request is appended, and the
// winner's table rebuilt, by warp 0 of the owning CTA at the start of step
// c + 1, which evaluates candidate c + 1 against that worker inside the
// rebuild while the other warps evaluate it against the rest of the slice.
// A step ends with one CTA barrier after which every warp reduces the warp
// bests itself; with several CTAs the CTA bests are exchanged through global
// memory behind one grid barrier (an arrival counter polled with a bounded
// wait) and a second CTA barrier.
// The winner's table is rebuilt by NW cooperating warps (EW element rows per
// lane, E = EW NW), chosen so that the rebuild's latency stays low and its
// registers within the 128 a thread of a 512-thread CTA has.
constexpr int R2_THREADS = 512;
constexpr int R2_WARPS = R2_THREADS / 32;
struct R2Args {
    DevParams P;
    ClusterDev C;
    RoundIO io;
    int G;                          // CTAs
    int slice;                      // workers per CTA
    int rc;                         // breakpoint rows per worker held in shared memory
    ulonglong2* xrec;               // [2][G] per CTA (two parities): best key, its
                                    // worker (NONE: none; bit 30: full)
    unsigned int* arrive;           // grid arrival counter, zero at launch
};

template <int E>
struct R2Smem {
    BuildSmem<R2Split<E>::EW, R2Split<E>::NW> build;
    unsigned long long bk[2][R2_WARPS];
    int bw[2][R2_WARPS];
    int bf[2][R2_WARPS];
    int gwin[2];
    int stop;
};

__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v)
{
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p)
{
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

template <int E>
__global__ void __launch_bounds__(R2_THREADS, 1) k_round2(R2Args A)
{
    constexpr int NW = R2Split<E>::NW, EW = R2Split<E>::EW;
    // the winner's previous sorted order is current: insert its new key
    constexpr bool NW_INSERT = NW > 1;
    extern __shared__ __align__(16) unsigned char smraw[];
    R2Smem<E>& sm = *reinterpret_cast<R2Smem<E>*>(smraw);
    const int cap = A.C.cap;
    unsigned char* tail = smraw + ((sizeof(R2Smem<E>) + 15) / 16) * 16;
    float4* wrec_s = reinterpret_cast<float4*>(tail);
    unsigned long long* key_s = reinterpret_cast<unsigned long long*>(wrec_s + A.slice);
    int* R_s = reinterpret_cast<int*>(key_s + A.slice);
    int* n_s = R_s + A.slice;
    unsigned short* rho = reinterpret_cast<unsigned short*>(n_s + A.slice);

    const DevParams& P = A.P;
    const ClusterDev& C = A.C;
    const RoundIO& io = A.io;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // direct mode after the incremental round: the candidates before c_begin
    // are placed already (every CTA reads the same value)
    const int c_begin = (!io.sim && io.c_first) ? *io.c_first : 0;
    if (!io.sim && c_begin >= io.n_cand) return;
    const int g = blockIdx.x;
    const int w_lo = g * A.slice;
    const int nloc = max(0, min(C.W, w_lo + A.slice) - w_lo);

    // slice state into shared memory
    for (int lw = tid; lw < nloc; lw += R2_THREADS) {
        const int w = w_lo + lw;
        R_s[lw] = C.R[w];
        n_s[lw] = C.n[w];
        wrec_s[lw] = C.wrec[w];
        key_s[lw] = C.key[w];
    }
    __syncthreads();
    const int rc = A.rc;
    const int rs = rc + R2_RHO_PAD;  // per-worker stride: an odd number of words
    for (int k = tid; k < nloc * rc; k += R2_THREADS) {
        const int lw = k / rc, q = k - lw * rc;
        if (q < R_s[lw])
            rho[lw * rs + q] = (unsigned short)(
                __float_as_int(C.tab[((long long)(w_lo + lw) * C.rows + q) * ROW_F4].x) - 1);
    }
    if (tid == 0) sm.stop = (io.sim && *io.status != 0) ? 1 : 0;
    __syncthreads();
    if (sm.stop) return;

    const int n_wait0 = io.sim ? *io.n_wait : 0;
    const int n_cand = io.sim ? n_wait0 + (int)(io.arr_end - io.arr_begin) : io.n_cand;
    int keep = 0;        // CTA 0 thread 0: new waiting-list length
    int pend_w = -1;     // this slice's winner of the previous step, not yet appended
    bool pend_small = false;  // its new count fits the 4-warp rebuild
    int32_t pa = 0, pr = 0, prl = 0;
    double pwd = 0.0;    // its request

    auto append = [&](int w) {  // rebuild group: commit the owed request to w
        if (tid == 0) {
            const int lw = w - w_lo;
            const int nw = n_s[lw];
            const long long slot = (long long)w * C.cap + nw;
            C.in[slot] = pa;
            C.gen[slot] = 0;
            C.pred[slot] = pr;
            C.real[slot] = prl;
            C.tdec[slot] = 0.0;
            C.pend[slot] = 1;
            C.wait[slot] = pwd;
            C.n[w] = nw + 1;
            n_s[lw] = nw + 1;
        }
    };
    // Flags a worker of n requests carries with its evaluation through the
    // reductions and the exchange: 1 no free slot, 2 its count after taking
    // the candidate fits the 4-warp rebuild.
    auto flag_bits = [&](int n) { return (n >= cap ? 1 : 0) | (n + 1 <= 128 ? 2 : 0); };
    // Rebuild group of worker w's table after the append: NW warps, or (small)
    // 4 warps with one element a lane when its new count fits 128: fewer
    // cross-warp steps, and the other warps evaluate the next candidate
    // meanwhile. small comes from the reduced winner flags, so every thread
    // of the CTA takes the same branch (and the same barrier).
    auto rebuild = [&](int w, bool small, const CandRec* cand) -> unsigned {
        const int lw = w - w_lo;
        SliceCache sc{rho + (long long)lw * rs, rc, &R_s[lw], &wrec_s[lw], &key_s[lw]};
        append(w);
        if constexpr (NW > 4) {
            if (small) {
                group_sync<4>();
                return build_table_fit<1, 4, true>(P, C, w, n_s[lw],
                                                   reinterpret_cast<unsigned char*>(&sm.build),
                                                   &sc, cand);
            }
        }
        group_sync<NW>();
        return build_table_fit<EW, NW, NW_INSERT>(P, C, w, n_s[lw],
                                                  reinterpret_cast<unsigned char*>(&sm.build), &sc,
                                                  cand);
    };

    for (int c = c_begin; c < n_cand; ++c) {
        const int par = c & 1;
        long long tix = 0;
        int32_t a, r, rl;
        double wd;
        if (io.sim) {
            tix = c < n_wait0 ? io.wl[c] : io.arr_begin + (c - n_wait0);
            a = io.tin[tix];
            r = io.tpred[tix];
            rl = io.treal ? io.treal[tix] : r;
            wd = io.t_now - io.t_arr[tix];
        } else {
            a = io.in[c];
            r = io.pred[c];
            rl = r;
            wd = io.wait ? (double)io.wait[c] : 0.0;
        }
        const CandRec cr = make_cand(P, a, r, (float)wd, c);
        // grouped scheduling: the request's group places on its own workers
        const int G = P.groups;
        const int grp = G > 1 ? (int)((io.sim ? tix : io.rid0 + c) % G) : 0;
        unsigned long long bk = 0ull;
        int bw = NONE, bf = 0;
        const bool rebuilding = pend_w >= 0;
        const int nwr = rebuilding && NW > 4 && pend_small ? 4 : NW;  // rebuild warps
        if (rebuilding && warp < nwr) {
            const unsigned f = rebuild(pend_w, nwr == 4 && NW > 4, cr.valid ? &cr : nullptr);
            const int lw = pend_w - w_lo;
            if (tid == 0 && cr.valid && f == 15u && (G <= 1 || pend_w % G == grp))
                bk = key_s[lw], bw = pend_w, bf = flag_bits(n_s[lw]);
        } else if (cr.valid) {
            const int first = rebuilding ? tid - 32 * nwr : tid;
            const int stride = rebuilding ? R2_THREADS - 32 * nwr : R2_THREADS;
            for (int lw = first; lw < nloc; lw += stride) {
                const int w = w_lo + lw;
                if (w == pend_w || (G > 1 && w % G != grp)) continue;
                const long long rb = (long long)w * C.rows;
                const int p = r2_find(rho + (long long)lw * rs, R_s[lw], rc, cr.ri, C.tab, rb);
                const long long row = rb + p;
                const float4* t = C.tab + row * ROW_F4;
                float m;
                const unsigned f =
                    eval_pair_mode(P.approx != 0, t[0], t[1], C.tab2[row], wrec_s[lw],
                                   P.approx ? C.wapx[w] : make_float2(0.0f, 0.0f), cr, m);
                if (f == 15u) better_f(bk, bw, bf, key_s[lw], w, flag_bits(n_s[lw]));
            }
        }
        reduce_f(bk, bw, bf);
        if (lane == 0) {
            sm.bk[par][warp] = bk;
            sm.bw[par][warp] = bw;
            sm.bf[par][warp] = bf;
        }
        __syncthreads();
        // every warp reduces the warp bests itself
        bk = lane < R2_WARPS ? sm.bk[par][lane] : 0ull;
        bw = lane < R2_WARPS ? sm.bw[par][lane] : NONE;
        bf = lane < R2_WARPS ? sm.bf[par][lane] : 0;
        reduce_f(bk, bw, bf);  // every lane ends with the CTA best
        if (A.G > 1) {
            if (warp == 0) {
                if (lane == 0) {
                    const int xi = bw == NONE ? NONE : (bw | (bf << 29));
                    A.xrec[par * A.G + g] = make_ulonglong2(bk, (unsigned long long)(unsigned)xi);
                    red_release_add(A.arrive, 1u);  // orders the store before it
                }
                // every lane acquires the counter, so its loads below see the
                // other CTAs' entries
                const unsigned target =
                    (unsigned)(c - c_begin + 1) * (unsigned)A.G + (unsigned)P.wait_test;
                bool ok = false;
                for (long long it = 0; it < P.grid_wait_limit; ++it) {
                    if (ld_acquire(A.arrive) >= target) {
                        ok = true;
                        break;
                    }
                    __nanosleep(32);
                }
                if (!ok && lane == 0) {
                    atomicOr(C.err, 4u);
                    *io.status = -4;  // ALADDIN_ERR_TIMEOUT
                    sm.stop = 2;
                }
                bk = 0ull;
                bw = NONE;
                bf = 0;
                // up to 8 entries a lane loaded together, then any beyond 256 CTAs
                ulonglong2 xv[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int q = lane + 32 * k;
                    xv[k] = q < A.G ? __ldcg(&A.xrec[par * A.G + q]) : make_ulonglong2(0ull, NONE);
                }
                for (int q = lane + 256; q < A.G; q += 32) {
                    const ulonglong2 v = __ldcg(&A.xrec[par * A.G + q]);
                    const int iq = (int)v.y;
                    better_f(bk, bw, bf, v.x, iq == NONE ? NONE : (iq & 0x1fffffff),
                             iq == NONE ? 0 : (iq >> 29) & 3);
                }
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int iq = (int)xv[k].y;
                    better_f(bk, bw, bf, xv[k].x, iq == NONE ? NONE : (iq & 0x1fffffff),
                             iq == NONE ? 0 : (iq >> 29) & 3);
                }
                reduce_f(bk, bw, bf);
                if (lane == 0) sm.gwin[par] = bw == NONE ? NONE : (bw | (bf << 29));
            }
            __syncthreads();
            if (sm.stop) break;
            const int gw = sm.gwin[par];
            bw = gw == NONE ? NONE : (gw & 0x1fffffff);
            bf = gw == NONE ? 0 : (gw >> 29) & 3;
        }
        const int winner = !cr.valid ? -2 : (bw == NONE ? -1 : bw);
        if (winner >= 0 && (bf & 1)) {
            if (tid == 0 && g == 0) {
                *io.status = -2;  // ALADDIN_ERR_CAPACITY
                if (!io.sim)
                    for (int k = c; k < n_cand; ++k) io.placement[k] = -1;
            }
            pend_w = -1;
            break;
        }
        pend_w = (winner >= w_lo && winner < w_lo + nloc) ? winner : -1;
        pend_small = (bf & 2) != 0;  // the reduced winner's flags: the same in every thread
        pa = a;
        pr = r;
        prl = rl;
        pwd = wd;
        if (g == 0 && tid == 0) {
            if (io.sim && io.sim_pl) {
                io.sim_pl[c] = winner;
                io.sim_tix[c] = tix;
            }
            if (!io.sim) {
                io.placement[c] = winner;
            } else if (winner >= 0) {
                io.counters[1] += 1;
            } else {
                const double tau_alone = C.scaled[0] * (P.k1d * (double)a + P.c1d);
                // a decode instance has no TTFT budget to absorb a wait
                if (winner == -2 || P.decode || wd + io.H + tau_alone > P.T_pred)
                    io.counters[0] += 1;
                else io.wl[keep++] = tix;
            }
        }
    }
    if (pend_w >= 0) {
        const bool small = NW > 4 && pend_small;
        if (warp < (small ? 4 : NW)) rebuild(pend_w, small, nullptr);
    }
    if (g == 0 && tid == 0 && io.sim && !sm.stop && *io.status == 0) {
        if (io.sim_n) *io.sim_n = n_cand;
        *io.n_wait = keep;
        if (io.stop_at_fail && io.counters[0] > 0) {
            *io.status = 1;
            io.counters[2] = (unsigned long long)io.hb;
        }
    }
}

// Shared memory of k_round2 for a slice of `slice` workers holding rc rows.
template <int E>
static size_t r2_smem(int slice, int rc)
{
    return ((sizeof(R2Smem<E>) + 15) / 16) * 16 + (size_t)slice * (16 + 8 + 4 + 4) +
           (size_t)slice * (rc + R2_RHO_PAD) * 2;
}
constexpr int R2_MIN_RC = 64;  // fewer rows per worker in shared memory: use the plain round

// Grid of the sliced round for W workers of cap slots: G CTAs, each holding
// the first rc rows of its slice of workers in shared memory. max_ctas = 1
// asks for one CTA (then rc shrinks with W). false: no sliced round fits.
template <int E>
static bool r2_plan(int W, int cap, int K, int sms, int smem_max, int max_ctas, int* G_out,
                    int* rc_out)
{
    if (K > 65536) return false;  // breakpoints held as 16-bit rho - 1
    if (sms > ROUND_XBUF_SMS) return false;
    const size_t budget = (size_t)smem_max - 1024;
    const size_t base = r2_smem<E>(0, 0);
    if (budget <= base + 32 + 2 * (R2_MIN_RC + R2_RHO_PAD)) return false;
    // As few CTAs as hold every worker's rows; beyond the CTAs allowed, the
    // slices hold only the first rc rows of each worker.
    int rc = cap;
    const long long slice_max = (long long)((budget - base) / (32 + 2 * (size_t)(rc + R2_RHO_PAD)));
    int G = (int)((W + slice_max - 1) / slice_max);
    const int gmax = max_ctas < sms ? max_ctas : sms;
    if (G > gmax) {
        G = gmax;
        const long long sl = (W + G - 1) / G;
        rc = ((int)((((budget - base) / (size_t)sl) - 32) / 2) - R2_RHO_PAD) & ~7;
        if (rc < R2_MIN_RC) return false;
    }
    *G_out = G;
    *rc_out = rc;
    return true;
}

template <int E>
static cudaError_t round2_e(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                            cudaStream_t st, bool* used)
{
    *used = false;
    DevInfo d;
    cudaError_t e = device_info(&d);
    if (e != cudaSuccess) return e;
    int G = 0, rc = 0;
    // several CTAs need a cooperative launch
    const int max_ctas = (io.single_cta || !d.coop) ? 1 : d.sms;
    if (!r2_plan<E>(C.W, C.cap, P.K, d.sms, d.smem_optin, max_ctas, &G, &rc)) return cudaSuccess;
    const int slice = (C.W + G - 1) / G;
    const size_t smem = r2_smem<E>(slice, rc);
    if ((e = allow_max_smem<k_round2<E>>()) != cudaSuccess) return e;
    R2Args A;
    A.P = P;
    A.C = C;
    A.io = io;
    A.G = G;
    A.slice = slice;
    A.rc = rc;
    A.xrec = reinterpret_cast<ulonglong2*>(io.xbuf);
    A.arrive = reinterpret_cast<unsigned int*>(A.xrec + 2 * ROUND_XBUF_SMS);
    if (G > 1) {
        e = cudaMemsetAsync(A.arrive, 0, sizeof(unsigned int), st);
        if (e != cudaSuccess) return e;
        void* args[] = {&A};
        e = cudaLaunchCooperativeKernel((const void*)k_round2<E>, dim3(G), dim3(R2_THREADS), args,
                                        smem, st);
    } else {
        k_round2<E><<<1, R2_THREADS, smem, st>>>(A);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) *used = true;
    return e;
}

template <int E>
static cudaError_t round_e(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                           cudaStream_t st)
{
    const size_t smem = sizeof(RoundSmem<E>);
    if (smem > 48 * 1024) {
        const cudaError_t e = allow_max_smem<k_round<E>>();
        if (e != cudaSuccess) return e;
    }
    k_round<E><<<1, ROUND_THREADS, smem, st>>>(P, C, io);
    return cudaGetLastError();
}

int round_ctas(int W, int cap, int K, bool single_cta)
{
    DevInfo d;
    if (device_info(&d) != cudaSuccess) {
        cudaGetLastError();
        return -1;
    }
    const int sms = d.sms, smem_max = d.smem_optin;
    const int max_ctas = (single_cta || !d.coop) ? 1 : sms;
    int G = 0, rc = 0;
    bool ok = false;
    switch (lanes_per_worker(cap)) {
    case 1: ok = r2_plan<1>(W, cap, K, sms, smem_max, max_ctas, &G, &rc); break;
    case 2: ok = r2_plan<2>(W, cap, K, sms, smem_max, max_ctas, &G, &rc); break;
    case 4: ok = r2_plan<4>(W, cap, K, sms, smem_max, max_ctas, &G, &rc); break;
    case 8: ok = r2_plan<8>(W, cap, K, sms, smem_max, max_ctas, &G, &rc); break;
    case 16: ok = r2_plan<16>(W, cap, K, sms, smem_max, max_ctas, &G, &rc); break;
    case 32: ok = r2_plan<32>(W, cap, K, sms, smem_max, max_ctas, &G, &rc); break;
    default: return -1;
    }
    if (ok) return G;
    return lanes_per_worker(cap) <= 16 ? 0 : -1;  // the plain round holds up to 512 slots
}

cudaError_t launch_round(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                         cudaStream_t st)
{
    if (io.xbuf) {
        bool used = false;
        cudaError_t e = cudaSuccess;
        switch (lanes_per_worker(C.cap)) {
        case 1: e = round2_e<1>(P, C, io, st, &used); break;
        case 2: e = round2_e<2>(P, C, io, st, &used); break;
        case 4: e = round2_e<4>(P, C, io, st, &used); break;
        case 8: e = round2_e<8>(P, C, io, st, &used); break;
        case 16: e = round2_e<16>(P, C, io, st, &used); break;
        case 32: e = round2_e<32>(P, C, io, st, &used); break;
        default: return cudaErrorInvalidValue;
        }
        if (e != cudaSuccess || used) return e;
    }
    switch (lanes_per_worker(C.cap)) {
    case 1: return round_e<1>(P, C, io, st);
    case 2: return round_e<2>(P, C, io, st);
    case 4: return round_e<4>(P, C, io, st);
    case 8: return round_e<8>(P, C, io, st);
    case 16: return round_e<16>(P, C, io, st);
    default: return cudaErrorNotSupported;  // 1,024 slots need the sliced round
    }
}

}  // namespace aladdin
