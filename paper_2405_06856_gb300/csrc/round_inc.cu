// K4, incremental: one greedy best-fit placement round (Algorithm 1) that
// re-scores only the workers the round has modified.
//
// Committing a candidate to worker i only adds a request to i: every other
// worker keeps its state, its table and its capacity_norm. So once every
// candidate of the round has been scored against the round-start state (the
// K3 scoring kernel, flags written in capacity_norm rank order), candidate c's
// choice is the better of
//   * the first feasible worker, in the round-start rank order, that the round
//     has not modified yet (its round-start flag is still exact), and
//   * the feasible worker of largest key among the modified ones, evaluated
//     afresh against their rebuilt tables (adding requests only raises a
//     worker's key, so a modified worker may overtake unmodified ones).
// One CTA runs the chain. The modified workers (usually a few dozen to a few
// hundred a round, against thousands of workers) keep their breakpoints,
// counts, records and keys in shared memory, and a bit set marks their rank
// positions. Per candidate the threads scan its flag row for the first
// unmodified feasible position (32 positions per word) and evaluate the
// modified workers; one block reduction picks the winner. The winner is
// committed lazily: at the next step a group of warps appends the request
// and rebuilds the winner's table, evaluating the next candidate against it
// in the same pass, while the other warps do the scan and the evaluations.
// No grid-wide exchange is needed. When the modified workers outgrow the
// shared-memory slots the kernel stops at that candidate and the sliced
// round (k_round2) finishes the rest from the current state.
#include <algorithm>

#include "round_common.cuh"

namespace aladdin {

constexpr int RI_THREADS = 512;
constexpr int RI_WARPS = RI_THREADS / 32;
constexpr int RI_WIN = 1024;       // rank positions whose entries stay in shared memory
constexpr int RI_MAX_SLOTS = 2048; // modified workers held in shared memory, at most
constexpr int RI_RC_MAX = 256;     // breakpoint rows a modified worker keeps in shared memory
constexpr size_t RI_FLAGS_MAX = (size_t)512 << 20;  // bytes of rank-order flags a chunk holds

// The rebuild group of the winner's table: tables of up to 256 slots, one
// warp per 32 slots; larger tables, RI_NW_BIG warps with the build sized to
// the worker's count (EW elements a lane cover the capacity).
#ifndef ALADDIN_RI_NW_BIG
#define ALADDIN_RI_NW_BIG 12
#endif
template <int E>
struct RISplit {
    static constexpr int NW = E <= 8 ? E : ALADDIN_RI_NW_BIG;
    static constexpr int EW = E <= 8 ? 1 : (E + NW - 1) / NW <= 2 ? 2 : 4;
};

// Round-start entry of a rank position: the worker there, its key and count.
struct __align__(16) RankEnt {
    unsigned long long key;
    int w;
    int n;
};

struct RIArgs {
    DevParams P;
    ClusterDev C;
    RoundIO io;                // direct mode; in/pred/wait/placement of this chunk
    const uint8_t* F;          // [n_cand][ldf] flags of the round-start state, rank order
    int ldf;                   // row stride of F (a multiple of 32)
    RankEnt* rank_ent;         // [W] scratch, written at kernel start
    int* c_stop;               // out: first candidate left to the sliced round
    int mmax;                  // modified-worker slots
    int rc;                    // breakpoint rows a slot holds
    int nwin;                  // rank positions held in shared memory
};

template <int E>
struct RISmem {
    BuildSmem<RISplit<E>::EW, RISplit<E>::NW> build;
    unsigned long long bk[2][RI_WARPS];
    int bw[2][RI_WARPS];
    int bf[2][RI_WARPS];
    CandRec cand[2];           // candidate records (parity of the step)
    int craw[2][4];            // prompt, predicted, real output length
    double cwd[2];             // wait (ms)
};

// Winner flags carried through the reductions: bit 29 the worker is full,
// bit 28 it is unmodified (then bits 0..26 hold its rank position, else its
// slot), bit 27 its count after the append fits the 4-warp rebuild.
constexpr int RI_FULL = 1 << 29;
constexpr int RI_UNMOD = 1 << 28;
constexpr int RI_SMALL = 1 << 27;
constexpr int RI_IDX = (1 << 27) - 1;

__device__ __forceinline__ int ri_flags(int idx, int n, int cap)
{
    return idx | (n >= cap ? RI_FULL : 0) | (n + 1 <= 128 ? RI_SMALL : 0);
}

// Bit b of the result: column 32 k + b of the flag row is 15 (feasible).
__device__ __forceinline__ unsigned feasible_bits(const uint8_t* row, int k)
{
    const uint4* p = reinterpret_cast<const uint4*>(row + 32 * (size_t)k);
    const uint4 u0 = __ldg(p), u1 = __ldg(p + 1);
    const unsigned w[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
    unsigned bits = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        // bytes equal to 15 -> 0xff, else 0; their low bits gathered into a
        // nibble by a multiply (no two partial products overlap)
        const unsigned eq = __vcmpeq4(w[i], 0x0f0f0f0fu) & 0x01010101u;
        bits |= ((eq * 0x10204080u) >> 28) << (4 * i);
    }
    return bits;
}

template <int E>
__global__ void __launch_bounds__(RI_THREADS, 1) k_round_inc(RIArgs A)
{
    constexpr int NW = RISplit<E>::NW, EW = RISplit<E>::EW;
    static_assert(NW * EW * 32 >= E * 32 && NW <= 12, "the rebuild group covers the capacity");
    constexpr bool NW_INSERT = NW > 1;
    extern __shared__ __align__(16) unsigned char smraw[];
    RISmem<E>& sm = *reinterpret_cast<RISmem<E>*>(smraw);
    const int mmax = A.mmax, rc = A.rc, nwin = A.nwin;
    const int rs = rc + R2_RHO_PAD;  // an odd number of words a slot
    unsigned char* tail = smraw + ((sizeof(RISmem<E>) + 15) / 16) * 16;
    RankEnt* win = reinterpret_cast<RankEnt*>(tail);
    float4* mwrec = reinterpret_cast<float4*>(win + nwin);
    unsigned long long* mkey = reinterpret_cast<unsigned long long*>(mwrec + mmax);
    int* mw = reinterpret_cast<int*>(mkey + mmax);
    int* mR = mw + mmax;
    int* mn = mR + mmax;
    const DevParams& P = A.P;
    const ClusterDev& C = A.C;
    const RoundIO& io = A.io;
    const int W = C.W, cap = C.cap;
    const int nwords = (W + 31) >> 5;
    unsigned* modbits = reinterpret_cast<unsigned*>(mn + mmax);
    unsigned short* rho = reinterpret_cast<unsigned short*>(modbits + ((nwords + 3) & ~3));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_cand = io.n_cand;

    // round-start rank entries: global scratch, the first nwin in shared memory
    for (int p = tid; p < W; p += RI_THREADS) {
        const int w = C.order[p];
        RankEnt e;
        e.key = C.key[w];
        e.w = w;
        e.n = C.n[w];
        A.rank_ent[p] = e;
        if (p < nwin) win[p] = e;
    }
    for (int k = tid; k < nwords; k += RI_THREADS) modbits[k] = 0u;
    // the prefetching thread (in the last warp, never part of a rebuild)
    const bool pf = tid == RI_THREADS - 1;
    auto fetch = [&](int c, int par) {
        const int32_t a = io.in[c], r = io.pred[c];
        const float wf = io.wait ? io.wait[c] : 0.0f;
        sm.cand[par] = make_cand(P, a, r, wf, c);
        sm.craw[par][0] = a;
        sm.craw[par][1] = r;
        sm.craw[par][2] = r;
        sm.cwd[par] = (double)wf;
    };
    if (pf && n_cand > 0) fetch(0, 0);
    __syncthreads();

    int mcount = 0;           // slots in use (every thread tracks the same value)
    int last_pos = -1;        // rank position marked modified at the previous step
    int pend_w = -1, pend_s = -1;  // the previous step's winner, not yet appended
    bool pend_small = false;  // its new count fits the 4-warp rebuild
    int32_t pa = 0, pr = 0, prl = 0;
    double pwd = 0.0;
    int stop_at = n_cand;     // first candidate left to the sliced round

    auto append = [&](int w, int s) {  // the rebuild group commits the owed request
        if (tid == 0) {
            const int nw = mn[s] >= 0 ? mn[s] : C.n[w];
            const long long slot = (long long)w * C.cap + nw;
            C.in[slot] = pa;
            C.gen[slot] = 0;
            C.pred[slot] = pr;
            C.real[slot] = prl;
            C.tdec[slot] = 0.0;
            C.pend[slot] = 1;
            C.wait[slot] = pwd;
            C.n[w] = nw + 1;
            mn[s] = nw + 1;
        }
    };
    auto rebuild = [&](int w, int s, bool small, const CandRec* cand) -> unsigned {
        SliceCache sc{rho + (long long)s * rs, rc, &mR[s], &mwrec[s], &mkey[s]};
        append(w, s);
        if constexpr (NW > 4) {
            if (small) {
                group_sync<4>();
                return build_table_fit<1, 4, true>(P, C, w, mn[s],
                                                   reinterpret_cast<unsigned char*>(&sm.build),
                                                   &sc, cand);
            }
        }
        group_sync<NW>();
        return build_table_fit<EW, NW, NW_INSERT>(P, C, w, mn[s],
                                                  reinterpret_cast<unsigned char*>(&sm.build), &sc,
                                                  cand);
    };

    int c = 0;
    for (; c < n_cand; ++c) {
        const int par = c & 1;
        const CandRec cr = sm.cand[par];
        const int32_t a = sm.craw[par][0], r = sm.craw[par][1], rl = sm.craw[par][2];
        const double wd = sm.cwd[par];
        unsigned long long bk = 0ull;
        int bw = NONE, bf = 0;
        const bool rebuilding = pend_w >= 0;
        const int nwr = !rebuilding ? 0 : (NW > 4 && pend_small ? 4 : NW);  // rebuild warps
        if (warp < nwr) {
            const unsigned f = rebuild(pend_w, pend_s, nwr == 4 && NW > 4, cr.valid ? &cr : nullptr);
            if (tid == 0 && cr.valid && f == 15u)
                bk = mkey[pend_s], bw = pend_w, bf = ri_flags(pend_s, mn[pend_s], cap);
        } else {
            if (cr.valid) {
                const int first = tid - 32 * nwr, stride = RI_THREADS - 32 * nwr;
                // the modified workers, against their current tables
                for (int i = first; i < mcount; i += stride) {
                    if (i == pend_s) continue;
                    const int w = mw[i];
                    const long long rb = (long long)w * C.rows;
                    const int p = r2_find(rho + (long long)i * rs, mR[i], rc, cr.ri, C.tab, rb);
                    const long long row = rb + p;
                    const float4* t = C.tab + row * ROW_F4;
                    float m;
                    const unsigned f =
                        eval_pair_mode(P.approx != 0, t[0], t[1], C.tab2[row], mwrec[i],
                                       P.approx ? C.wapx[w] : make_float2(0.0f, 0.0f), cr, m);
                    if (f == 15u) better_f(bk, bw, bf, mkey[i], w, ri_flags(i, mn[i], cap));
                }
                // the first unmodified feasible position of every word of the
                // candidate's round-start flag row
                const uint8_t* frow = A.F + (size_t)c * A.ldf;
                for (int k = first; k < nwords; k += stride) {
                    unsigned bits = feasible_bits(frow, k) & ~modbits[k];
                    if (k == (last_pos >> 5) && last_pos >= 0) bits &= ~(1u << (last_pos & 31));
                    const int left = W - 32 * k;
                    if (left < 32) bits &= (1u << left) - 1u;
                    if (bits) {
                        const int pos = 32 * k + __ffs(bits) - 1;
                        const RankEnt e = pos < nwin ? win[pos] : A.rank_ent[pos];
                        better_f(bk, bw, bf, e.key, e.w, ri_flags(pos, e.n, cap) | RI_UNMOD);
                    }
                }
            }
            if (pf && c + 1 < n_cand) fetch(c + 1, par ^ 1);
        }
        reduce_f(bk, bw, bf);
        if (lane == 0) {
            sm.bk[par][warp] = bk;
            sm.bw[par][warp] = bw;
            sm.bf[par][warp] = bf;
        }
        __syncthreads();
        bk = lane < RI_WARPS ? sm.bk[par][lane] : 0ull;
        bw = lane < RI_WARPS ? sm.bw[par][lane] : NONE;
        bf = lane < RI_WARPS ? sm.bf[par][lane] : 0;
        reduce_f(bk, bw, bf);  // every thread ends with the winner
        const int winner = !cr.valid ? -2 : (bw == NONE ? -1 : bw);
        if (winner >= 0 && (bf & RI_FULL)) {
            if (tid == 0) {
                *io.status = -2;  // ALADDIN_ERR_CAPACITY
                for (int k = c; k < n_cand; ++k) io.placement[k] = -1;
            }
            pend_w = -1;
            break;
        }
        int s = -1;
        last_pos = -1;
        if (winner >= 0) {
            if (bf & RI_UNMOD) {
                if (mcount == mmax) {  // no slot left: the sliced round takes over here
                    stop_at = c;
                    pend_w = -1;  // the previous winner was appended at this step's start
                    break;
                }
                s = mcount++;
                last_pos = bf & RI_IDX;
                if (tid == 0) {
                    mw[s] = winner;
                    mn[s] = -1;  // the append reads the round-start count
                    modbits[last_pos >> 5] |= 1u << (last_pos & 31);
                }
            } else {
                s = bf & RI_IDX;
            }
        }
        pend_w = winner >= 0 ? winner : -1;
        pend_s = s;
        pend_small = winner >= 0 && (bf & RI_SMALL) != 0;  // the same in every thread
        pa = a;
        pr = r;
        prl = rl;
        pwd = wd;
        if (tid == 0) io.placement[c] = winner;
    }
    if (pend_w >= 0) {
        const int nwr = NW > 4 && pend_small ? 4 : NW;
        if (warp < nwr) rebuild(pend_w, pend_s, nwr == 4 && NW > 4, nullptr);
    }
    if (tid == 0) *A.c_stop = stop_at;
}

// Shared memory of k_round_inc: the fixed part, nwin rank entries, mmax slots
// of rc rows, and the modified-position bit set of W workers.
template <int E>
static size_t ri_smem(int W, int nwin, int mmax, int rc)
{
    const int nwords = (W + 31) >> 5;
    return ((sizeof(RISmem<E>) + 15) / 16) * 16 + (size_t)nwin * sizeof(RankEnt) +
           (size_t)mmax * (16 + 8 + 4 * 3) + (size_t)((nwords + 3) & ~3) * 4 +
           (size_t)mmax * (rc + R2_RHO_PAD) * 2;
}

template <int E>
static bool ri_plan(int W, int cap, int K, int smem_max, int* nwin, int* mmax, int* rc)
{
    if (K > 65536) return false;  // breakpoints held as 16-bit rho - 1
    const size_t budget = (size_t)smem_max - 1024;
    const int nw = W < RI_WIN ? W : RI_WIN;
    int r = cap < RI_RC_MAX ? cap : RI_RC_MAX;
    const size_t base = ri_smem<E>(W, nw, 0, r);
    const size_t per = 16 + 8 + 4 * 3 + (size_t)(r + R2_RHO_PAD) * 2;
    if (budget <= base + 64 * per) return false;  // too few slots to be worth it
    size_t m = (budget - base) / per;
    if (m > RI_MAX_SLOTS) m = RI_MAX_SLOTS;
    if (m > (size_t)W) m = W;
    *nwin = nw;
    *mmax = (int)m;
    *rc = r;
    return true;
}

template <int E>
static cudaError_t round_inc_e(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                               const RoundIncBuffers& B, cudaStream_t st, bool* used)
{
    *used = false;
    DevInfo d;
    cudaError_t e = device_info(&d);
    if (e != cudaSuccess) return e;
    int nwin = 0, mmax = 0, rc = 0;
    if (!ri_plan<E>(C.W, C.cap, P.K, d.smem_optin, &nwin, &mmax, &rc)) return cudaSuccess;
    if (P.round_slots_max > 0 && mmax > P.round_slots_max) mmax = P.round_slots_max;
    const size_t smem = ri_smem<E>(C.W, nwin, mmax, rc);
    if ((e = allow_max_smem<k_round_inc<E>>()) != cudaSuccess) return e;
    const int ldf = (C.W + 31) & ~31;
    const size_t per_row = (size_t)ldf;
    int chunk = (int)std::min<size_t>((size_t)io.n_cand, std::max<size_t>(1, RI_FLAGS_MAX / per_row));
    if (P.round_chunk > 0 && chunk > P.round_chunk) chunk = P.round_chunk;
    for (int c0 = 0; c0 < io.n_cand; c0 += chunk) {
        const int n = std::min(chunk, io.n_cand - c0);
        if (c0 > 0 && (e = launch_rank(C, st)) != cudaSuccess) return e;  // the chunk's start state
        // every candidate of the chunk against the current state, rank order
        e = launch_score(P, C, n, io.in + c0, io.pred + c0, io.wait ? io.wait + c0 : nullptr, B.flags,
                         nullptr, nullptr, nullptr, nullptr, B.score, io.round_open || c0 > 0, st,
                         nullptr, nullptr, false, C.order, ldf);
        if (e != cudaSuccess) return e;
        RIArgs A;
        A.P = P;
        A.C = C;
        A.io = io;
        A.io.in = io.in + c0;
        A.io.pred = io.pred + c0;
        A.io.wait = io.wait ? io.wait + c0 : nullptr;
        A.io.placement = io.placement + c0;
        A.io.n_cand = n;
        A.F = B.flags;
        A.ldf = ldf;
        A.rank_ent = reinterpret_cast<RankEnt*>(B.rank);
        A.c_stop = B.c_stop;
        A.mmax = mmax;
        A.rc = rc;
        A.nwin = nwin;
        k_round_inc<E><<<1, RI_THREADS, smem, st>>>(A);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        // the sliced round places what the incremental round left (nothing
        // when every candidate was placed: it returns at once)
        RoundIO rest = A.io;
        rest.c_first = B.c_stop;
        if ((e = launch_round(P, C, rest, st)) != cudaSuccess) return e;
    }
    *used = true;
    return cudaSuccess;
}

template <int E>
static size_t flag_bytes_e(const DevParams& P, const ClusterDev& C, const RoundIO& io)
{
    DevInfo d;
    if (device_info(&d) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    int nwin = 0, mmax = 0, rc = 0;
    if (!ri_plan<E>(C.W, C.cap, P.K, d.smem_optin, &nwin, &mmax, &rc)) return 0;
    const size_t ldf = (size_t)((C.W + 31) & ~31);
    const size_t chunk = std::min<size_t>((size_t)io.n_cand, std::max<size_t>(1, RI_FLAGS_MAX / ldf));
    return chunk * ldf;
}

size_t round_inc_flag_bytes(const DevParams& P, const ClusterDev& C, const RoundIO& io)
{
    if (io.sim || P.groups > 1 || P.wait_test || io.n_cand <= 0) return 0;
    switch (lanes_per_worker(C.cap)) {
    case 1: return flag_bytes_e<1>(P, C, io);
    case 2: return flag_bytes_e<2>(P, C, io);
    case 4: return flag_bytes_e<4>(P, C, io);
    case 8: return flag_bytes_e<8>(P, C, io);
    case 16: return flag_bytes_e<16>(P, C, io);
    case 32: return flag_bytes_e<32>(P, C, io);
    default: return 0;
    }
}

cudaError_t launch_round_inc(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                             const RoundIncBuffers& B, cudaStream_t st, bool* used)
{
    *used = false;
    if (io.sim || P.groups > 1 || P.wait_test || io.n_cand <= 0) return cudaSuccess;
    switch (lanes_per_worker(C.cap)) {
    case 1: return round_inc_e<1>(P, C, io, B, st, used);
    case 2: return round_inc_e<2>(P, C, io, B, st, used);
    case 4: return round_inc_e<4>(P, C, io, B, st, used);
    case 8: return round_inc_e<8>(P, C, io, B, st, used);
    case 16: return round_inc_e<16>(P, C, io, B, st, used);
    case 32: return round_inc_e<32>(P, C, io, B, st, used);
    default: return cudaSuccess;
    }
}

}  // namespace aladdin
