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
// modified workers; one block reduction picks the winner. The winner's
// request is appended at the decision; at the next step a group of warps
// rebuilds its table (inserting the appended keys into its sorted order),
// evaluating the next candidate against it in the same pass, while the other
// warps do the scan and the evaluations (and, on tables of up to 128 slots,
// a second group looks one candidate ahead: see below). No grid-wide exchange
// is needed. When the modified workers outgrow the
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

// Look-ahead (tables of up to 128 slots, rebuilt by at most 4 warps): while
// one group rebuilds the pending worker's table and evaluates candidate c on
// it, RI_LA - 1 more groups build that worker's state with c (and c + 1)
// appended as well (evaluation only, nothing committed) and evaluate c + 1
// (and c + 2) on it, and the remaining warps scan and evaluate for every one
// of those candidates. When c goes to the pending worker, c + 1 is decided in
// the same step, and so on: a step places up to RI_LA candidates. Most
// candidates of a best-fit round go to the worker that took the previous one.
#ifndef ALADDIN_RI_LA
#define ALADDIN_RI_LA 2
#endif
constexpr int RI_LA = ALADDIN_RI_LA;  // candidates a look-ahead step may place

template <int E>
constexpr bool ri_lookahead()
{
    return RISplit<E>::NW <= 4;
}

template <int E>
struct RISmem {
    BuildSmem<RISplit<E>::EW, RISplit<E>::NW> build;
    // the look-ahead groups' scratch
    BuildSmem<1, ri_lookahead<E>() ? RISplit<E>::NW : 1> bla[ri_lookahead<E>() ? RI_LA - 1 : 1];
    unsigned long long bk[2][RI_LA][RI_WARPS];  // [step parity][candidate c + j][warp]
    int bw[2][RI_LA][RI_WARPS];
    int bf[2][RI_LA][RI_WARPS];
    CandRec cand[8];           // candidate records, by candidate index mod 8
    int craw[8][4];            // prompt, predicted, real output length
    double cwd[8];             // wait (ms)
    unsigned long long la_key[RI_LA]; // the look-ahead states' capacity_norm keys
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
    auto fetch = [&](int k) {
        const int b = k & 7;
        const int32_t a = io.in[k], r = io.pred[k];
        const float wf = io.wait ? io.wait[k] : 0.0f;
        sm.cand[b] = make_cand(P, a, r, wf, k);
        sm.craw[b][0] = a;
        sm.craw[b][1] = r;
        sm.craw[b][2] = r;
        sm.cwd[b] = (double)wf;
    };
    int fetched = 0;  // candidates fetched (meaningful in the prefetching thread)
    if (pf)
        while (fetched < n_cand && fetched < 2) fetch(fetched++);

    constexpr bool LA = ri_lookahead<E>();
    int mcount = 0;           // slots in use (every thread tracks the same value)
    int last_pos = -1;        // rank position marked modified at the previous step
    int pend_w = -1, pend_s = -1;  // the worker whose table is owed a rebuild
    int pend_cnt = 0;         // requests appended to it since its table was built
    bool pend_small = false;  // its count fits the 4-warp rebuild
    int stop_at = n_cand;     // first candidate left to the sliced round
    int c_step = 0;           // the step's first candidate

    // tid 0: candidate k's request into worker w's next slot (slot s)
    auto append = [&](int w, int s, int k) {
        const int b = k & 7;
        const int nw = mn[s] >= 0 ? mn[s] : C.n[w];
        const long long slot = (long long)w * C.cap + nw;
        C.in[slot] = sm.craw[b][0];
        C.gen[slot] = 0;
        C.pred[slot] = sm.craw[b][1];
        C.real[slot] = sm.craw[b][2];
        C.tdec[slot] = 0.0;
        C.pend[slot] = 1;
        C.wait[slot] = sm.cwd[b];
        C.n[w] = nw + 1;
        mn[s] = nw + 1;
    };
    // the rebuild group commits the worker's table, inserting the `ins`
    // requests appended since its last build into that build's sorted keys.
    // With the look-ahead, the sorted keys are stored after the step's
    // barrier (skey_store): the look-ahead group reads the previous ones.
    auto rebuild = [&](int w, int s, bool small, int ins, const CandRec* cand) -> unsigned {
        SliceCache sc{rho + (long long)s * rs, rc, &mR[s], &mwrec[s], &mkey[s]};
        unsigned char* bs = reinterpret_cast<unsigned char*>(&sm.build);
        if constexpr (NW > 4) {
            if (small) return build_table_fit<1, 4, true>(P, C, w, mn[s], bs, &sc, cand);
        }
        return build_table_fit<EW, NW, NW_INSERT, 1, 0, false, !LA>(P, C, w, mn[s], bs, &sc, cand,
                                                                    nullptr, ins);
    };
    auto skey_store = [&](int w, int s) {  // the rebuild group, after its build
        if constexpr (LA && NW > 1) {
            const int n = mn[s];
            for (int x = tid; x < n; x += 32 * NW) C.skey[(long long)w * C.cap + x] = sm.build.sorted[x];
        }
    };
    // candidate cq (index k): the modified workers other than the pending
    // one, against their current tables, and the first unmodified feasible
    // position of every word of its round-start flag row
    auto scan_eval = [&](const CandRec& cq, int k, int first, int stride, unsigned long long& bk,
                         int& bw, int& bf) {
        if (!cq.valid) return;
        for (int i = first; i < mcount; i += stride) {
            if (i == pend_s) continue;
            const int w = mw[i];
            const long long rb = (long long)w * C.rows;
            const int p = r2_find(rho + (long long)i * rs, mR[i], rc, cq.ri, C.tab, rb);
            const long long row = rb + p;
            const float4* t = C.tab + row * ROW_F4;
            float m;
            const unsigned f =
                eval_pair_mode(P.approx != 0, t[0], t[1], C.tab2[row], mwrec[i],
                               P.approx ? C.wapx[w] : make_float2(0.0f, 0.0f), cq, m);
            if (f == 15u) better_f(bk, bw, bf, mkey[i], w, ri_flags(i, mn[i], cap));
        }
        const uint8_t* frow = A.F + (size_t)k * A.ldf;
        for (int kw = first; kw < nwords; kw += stride) {
            unsigned bits = feasible_bits(frow, kw) & ~modbits[kw];
            if (kw == (last_pos >> 5) && last_pos >= 0) bits &= ~(1u << (last_pos & 31));
            const int left = W - 32 * kw;
            if (left < 32) bits &= (1u << left) - 1u;
            if (bits) {
                const int pos = 32 * kw + __ffs(bits) - 1;
                const RankEnt e = pos < nwin ? win[pos] : A.rank_ent[pos];
                better_f(bk, bw, bf, e.key, e.w, ri_flags(pos, e.n, cap) | RI_UNMOD);
            }
        }
    };

    // look-ahead group g (1 .. RI_LA - 1, warps g NW .. g NW + NW - 1): the
    // pending worker with candidates c .. c + g - 1 appended as well,
    // evaluated for c + g. The group's first thread writes their requests
    // into the slots past the worker's count: the append writes the same
    // values there when a candidate is placed on the worker, and otherwise
    // they lie past the count, where no build or evaluation reads.
    auto la_eval = [&](int g, int nw, int ins, const CandRec* cq) -> unsigned {
        if (tid == 32 * NW * g) {
            for (int j = 0; j < g; ++j) {
                const int b = (c_step + j) & 7;
                const long long slot = (long long)pend_w * C.cap + nw + j;
                C.in[slot] = sm.craw[b][0];
                C.gen[slot] = 0;
                C.pred[slot] = sm.craw[b][1];
                C.real[slot] = sm.craw[b][2];
                C.tdec[slot] = 0.0;
                C.pend[slot] = 1;
                C.wait[slot] = sm.cwd[b];
            }
        }
        unsigned char* bs = reinterpret_cast<unsigned char*>(&sm.bla[g - 1]);
        if (g == 1) {
            group_sync<NW, 2>();
            return build_table_fit<1, NW, NW_INSERT, 2, NW, true>(P, C, pend_w, nw + 1, bs, nullptr,
                                                                  cq, &sm.la_key[1], ins);
        }
        group_sync<NW, 3>();
        return build_table_fit<1, NW, NW_INSERT, 3, 2 * NW, true>(P, C, pend_w, nw + 2, bs, nullptr,
                                                                  cq, &sm.la_key[2], ins);
    };

    int c = 0;
    for (int stp = 0; c < n_cand; ++stp) {
        __syncthreads();  // the last step's appends, slots and fetched records are visible
        c_step = c;
        const int par = stp & 1;
        const CandRec cr = sm.cand[c & 7];
        const bool rebuilding = pend_w >= 0;
        // candidates looked at this step: c, and while valid and room is left
        // on the pending worker, c + 1 .. c + RI_LA - 1
        int la = 1;
        if constexpr (LA) {
            if (rebuilding && cr.valid) {
                while (la < RI_LA && c + la < n_cand && sm.cand[(c + la) & 7].valid &&
                       mn[pend_s] + la + 1 <= cap)
                    ++la;
            }
        }
        const int nwr = !rebuilding ? 0 : (NW > 4 && pend_small ? 4 : NW);  // rebuild warps
        const int scan0 = la > 1 ? la * NW : nwr;  // first scanning warp
        unsigned long long bk[RI_LA];
        int bw[RI_LA], bf[RI_LA];
#pragma unroll
        for (int j = 0; j < RI_LA; ++j) bk[j] = 0ull, bw[j] = NONE, bf[j] = 0;
        if (warp < nwr) {
            const unsigned f = rebuild(pend_w, pend_s, nwr == 4 && NW > 4, pend_cnt,
                                       cr.valid ? &cr : nullptr);
            if (tid == 0 && cr.valid && f == 15u)
                bk[0] = mkey[pend_s], bw[0] = pend_w, bf[0] = ri_flags(pend_s, mn[pend_s], cap);
        } else if (warp < scan0) {
            if constexpr (LA) {
                const int g = warp / NW;  // 1 .. la - 1
                const int nw = mn[pend_s];
                const CandRec cq = sm.cand[(c + g) & 7];
                const unsigned f = la_eval(g, nw, pend_cnt + g, &cq);
                if (tid == 32 * NW * g && f == 15u) {
#pragma unroll
                    for (int j = 1; j < RI_LA; ++j)
                        if (j == g)
                            bk[j] = sm.la_key[j], bw[j] = pend_w,
                            bf[j] = ri_flags(pend_s, nw + j, cap);
                }
            }
        } else {
            const int first = tid - 32 * scan0, stride = RI_THREADS - 32 * scan0;
#pragma unroll
            for (int j = 0; j < RI_LA; ++j)
                if (j < la) scan_eval(sm.cand[(c + j) & 7], c + j, first, stride, bk[j], bw[j], bf[j]);
            if (pf)
                while (fetched < n_cand && fetched < c + 2 * RI_LA) fetch(fetched++);
        }
#pragma unroll
        for (int j = 0; j < RI_LA; ++j)
            if (j < la) reduce_f(bk[j], bw[j], bf[j]);
        if (lane == 0) {
#pragma unroll
            for (int j = 0; j < RI_LA; ++j) {
                sm.bk[par][j][warp] = bk[j];
                sm.bw[par][j][warp] = bw[j];
                sm.bf[par][j][warp] = bf[j];
            }
        }
        __syncthreads();
        if (warp < nwr) skey_store(pend_w, pend_s);
        unsigned long long kk = lane < RI_WARPS ? sm.bk[par][0][lane] : 0ull;
        int ww = lane < RI_WARPS ? sm.bw[par][0][lane] : NONE;
        int ff = lane < RI_WARPS ? sm.bf[par][0][lane] : 0;
        reduce_f(kk, ww, ff);  // every thread ends with the winner
        const int winner = !cr.valid ? -2 : (ww == NONE ? -1 : ww);
        if (winner >= 0 && (ff & RI_FULL)) {
            if (tid == 0) {
                *io.status = -2;  // ALADDIN_ERR_CAPACITY
                for (int k = c; k < n_cand; ++k) io.placement[k] = -1;
            }
            pend_w = -1;
            break;
        }
        // c + 1, c + 2 are decided now while their predecessors went to the
        // pending worker: every other worker's state is the one their
        // evaluations saw
        int placed = 1;
        if (la > 1 && winner == pend_w) {
            for (int j = 1; j < la; ++j) {
                unsigned long long k2 = lane < RI_WARPS ? sm.bk[par][j][lane] : 0ull;
                int w2 = lane < RI_WARPS ? sm.bw[par][j][lane] : NONE;
                int f2 = lane < RI_WARPS ? sm.bf[par][j][lane] : 0;
                reduce_f(k2, w2, f2);
                if (w2 != pend_w) break;
                ++placed;
            }
        }
        int s = -1;
        last_pos = -1;
        if (winner >= 0) {
            if (ff & RI_UNMOD) {
                if (mcount == mmax) {  // no slot left: the sliced round takes over here
                    stop_at = c;
                    pend_w = -1;  // the pending worker's table was rebuilt at this step
                    break;
                }
                s = mcount++;
                last_pos = ff & RI_IDX;
                if (tid == 0) {
                    mw[s] = winner;
                    mn[s] = -1;  // the append reads the round-start count
                    modbits[last_pos >> 5] |= 1u << (last_pos & 31);
                }
            } else {
                s = ff & RI_IDX;
            }
        }
        if (tid == 0) {
            io.placement[c] = winner;
            if (winner >= 0) append(winner, s, c);
            for (int j = 1; j < placed; ++j) {
                io.placement[c + j] = winner;
                append(winner, s, c + j);
            }
        }
        pend_w = winner >= 0 ? winner : -1;
        pend_s = s;
        pend_cnt = placed;
        pend_small = winner >= 0 && (ff & RI_SMALL) != 0;  // the same in every thread
        c += placed;
    }
    __syncthreads();  // the last appends are visible to the rebuild group
    if (pend_w >= 0) {
        const int nwr = NW > 4 && pend_small ? 4 : NW;
        if (warp < nwr) {
            rebuild(pend_w, pend_s, nwr == 4 && NW > 4, pend_cnt, nullptr);
            skey_store(pend_w, pend_s);
        }
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
