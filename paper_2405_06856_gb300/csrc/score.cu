// K3: batched candidate x worker scoring.
//
// Candidates are validated, turned into per-candidate constants and
// counting-sorted by predicted output length. A CTA owns a tile of
// SCORE_WARPS x 32 x SLOTS consecutive workers and a contiguous range of the
// sorted candidates; the grid is one wave of CTAs with equal shares. Candidate
// records are staged into shared memory in chunks by TMA bulk copies (double
// buffered, mbarrier completion). Each lane keeps, per worker, the table row of
// the segment containing the current candidate length and the next row, so a
// breakpoint crossing is a register move while the row after it is fetched in
// the background; a pair costs the O(1) bound arithmetic only. Flags and
// margins of one candidate are one coalesced row segment per warp (streaming
// stores); argbest is the smallest capacity_norm rank among feasible workers,
// reduced per warp, merged across the CTA's warps in shared memory and
// committed with one atomic per CTA and candidate.
#include "aladdin_host.h"

namespace aladdin {

constexpr int SCORE_WARPS = 4;
constexpr int SCORE_CHUNK = 256;

__global__ void k_cand_count(DevParams P, int n, const int32_t* __restrict__ in,
                             const int32_t* __restrict__ pred, const float* __restrict__ wait,
                             int32_t* hist, unsigned int* best)
{
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= n) return;
    const int32_t a = in[c], r = pred[c];
    const float w = wait ? wait[c] : 0.0f;
    const bool ok = a >= 0 && r >= 1 && (long long)a + r <= (long long)P.K && w >= 0.0f &&
                    w <= 3.0e38f;
    atomicAdd(&hist[ok ? r : 0], 1);
    best[c] = 0xffffffffu;
}

// Exclusive scan of hist[0..K] in place (one CTA).
constexpr int SCAN_THREADS = 1024;

__global__ void __launch_bounds__(SCAN_THREADS) k_scan_hist(int32_t* hist, int len)
{
    __shared__ int32_t wsum[SCAN_THREADS / 32];
    const int per = (len + SCAN_THREADS - 1) / SCAN_THREADS;
    const int b0 = threadIdx.x * per;
    const int b1 = min(b0 + per, len);
    int32_t sum = 0;
    for (int i = b0; i < b1; ++i) sum += hist[i];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t incl = sum;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int32_t u = __shfl_up_sync(FULL, incl, d);
        if (lane >= d) incl += u;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int32_t v = wsum[lane];
        int32_t vi = v;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int32_t u = __shfl_up_sync(FULL, vi, d);
            if (lane >= d) vi += u;
        }
        wsum[lane] = vi - v;
    }
    __syncthreads();
    int32_t run = wsum[warp] + incl - sum;
    for (int i = b0; i < b1; ++i) {
        const int32_t h = hist[i];
        hist[i] = run;
        run += h;
    }
}

// Sorted record (3 x float4): {a, r, 1/r, Ua}, {inv_d1, nXd1, inv_d2, Zc},
// {valid ? r : 0, original index, low and high words of index * W (the start
// of the candidate's output row)}.
constexpr int REC_F4 = 3;

struct ScoreArgs {
    ClusterDev C;
    const float4* __restrict__ cand;
    int n_cand;
    uint8_t* flags;
    float* margin;
    unsigned int* best;
    int tiles, chunks;
    int approx;  // approximate-mode constraints (b) and (d)
    long long wait_limit;  // mbarrier polls before a wait gives up
    int withhold;          // test hook: the first candidate copy is not issued
    const int32_t* order;  // nullptr, or rank order: output column k is worker order[k]
    int ld;                // output row stride (elements)
};

__global__ void k_cand_scatter(DevParams P, int n, int W, const int32_t* __restrict__ in,
                               const int32_t* __restrict__ pred, const float* __restrict__ wait,
                               int32_t* cursor, float4* sorted)
{
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= n) return;
    const CandRec rec = make_cand(P, in[c], pred[c], wait ? wait[c] : 0.0f, c);
    const int pos = atomicAdd(&cursor[rec.valid ? rec.ri : 0], 1);
    const unsigned long long rowoff = (unsigned long long)c * (unsigned long long)W;
    float4* o = sorted + (size_t)pos * REC_F4;
    o[0] = make_float4(rec.a, rec.r, rec.inv_r, rec.Ua);
    o[1] = make_float4(rec.inv_d1, rec.nXd1, rec.inv_d2, rec.Zc);
    o[2] = make_float4(__int_as_float(rec.valid ? rec.ri : 0), __int_as_float(c),
                       __uint_as_float((unsigned)(rowoff & 0xffffffffull)),
                       __uint_as_float((unsigned)(rowoff >> 32)));
}

struct Row {
    float4 v0, v1;
};

__device__ __forceinline__ Row load_row(const float4* __restrict__ tab, long long row)
{
    const float4* t = tab + row * ROW_F4;
    Row r;
    r.v0 = __ldg(t);
    r.v1 = __ldg(t + 1);
    return r;
}

__device__ __forceinline__ unsigned prmt(unsigned a, unsigned b, unsigned sel)
{
    unsigned d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// Flag bytes of SLOTS pairs from the sign bits of their group headrooms
// d[g][k] (bit g of byte k set iff d[g][k] >= 0). prmt with the
// sign-replicate selector (bit 3 of a selector nibble) turns the top byte of
// each headroom into 0x00 / 0xff, one byte per slot.
template <int SLOTS>
__device__ __forceinline__ unsigned pack_flags(const float (&d)[4][SLOTS])
{
    unsigned acc = 0;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        unsigned S;
        if (SLOTS == 4) {
            const unsigned t1 = prmt(__float_as_uint(d[g][0]), __float_as_uint(d[g][1 % SLOTS]), 0x00fbu);
            const unsigned t2 = prmt(__float_as_uint(d[g][2 % SLOTS]), __float_as_uint(d[g][3 % SLOTS]), 0x00fbu);
            S = prmt(t1, t2, 0x5410u);
        } else {
            S = prmt(__float_as_uint(d[g][0]), __float_as_uint(d[g][1 % SLOTS]), 0x00fbu);
        }
        const unsigned mask = SLOTS == 4 ? 0x01010101u : 0x0101u;
        acc |= ~S & (mask << g);
    }
    return acc;
}

#ifndef ALADDIN_SCORE_SLOTS
#define ALADDIN_SCORE_SLOTS 4
#endif
#ifndef ALADDIN_SCORE_MINB
#define ALADDIN_SCORE_MINB 5
#endif
constexpr int CHUNK = 256;                   // candidates per staged chunk
constexpr unsigned ERR_TIMEOUT_BIT = 4u;

__device__ __forceinline__ unsigned smem_addr(const void* p)
{
    return (unsigned)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(unsigned long long* bar, unsigned count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// One elected thread: expect `bytes` and start the bulk copy of `bytes`
// (multiple of 16, both addresses 16-byte aligned) from global to shared.
__device__ __forceinline__ void tma_load(void* dst, const void* src, unsigned bytes,
                                         unsigned long long* bar)
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// Bounded wait for the phase with the given parity; false if `limit` polls
// ran out.
__device__ __forceinline__ bool mbar_wait(unsigned long long* bar, unsigned parity, long long limit)
{
    for (long long it = 0; it < limit; ++it) {
        unsigned done;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
            : "=r"(done)
            : "r"(smem_addr(bar)), "r"(parity)
            : "memory");
        if (done) return true;
    }
    return false;
}

struct VecArgs {
    ClusterDev C;
    const float4* __restrict__ cand;   // sorted records, REC_F4 float4 each
    int n_cand;
    uint8_t* flags;
    float* margin;
    unsigned int* best;
    int tiles;       // worker tiles of SCORE_WARPS * 32 * SLOTS
    int per_tile;    // CTAs per tile
    long long wait_limit;  // mbarrier polls before a wait gives up
    int withhold;    // test hook, 1: the first chunk's copy is not issued (its wait runs out)
    const int32_t* order;  // nullptr, or rank order: output column k is worker order[k]
};

struct __align__(16) ScoreSmem {
    float4 cs[2][CHUNK * REC_F4];
    unsigned kmin[SCORE_WARPS][CHUNK];
    unsigned long long bar[2];
    int stop;
};

// Worker state of one lane slot: the fields of the current table row that a
// pair reads, the next row (raw), and the worker's record.
#ifndef ALADDIN_SCORE_PF
#define ALADDIN_SCORE_PF 1
#endif

// Ask L1 to hold a row (32 bytes).
__device__ __forceinline__ void prefetch_row(const float4* tab, long long row)
{
    asm volatile("prefetch.global.L1 [%0];" ::"l"(tab + row * ROW_F4));
}

template <bool PEND>
struct Slot {
    float kvB1, kvE, np1n, b0n, b1, nh, pmA, Gt;
    float pmAp, Gpt;           // PEND only
    int rnext;                 // rho_{p+1} of the current row
#if !ALADDIN_SCORE_PF
    Row nxt;                   // row p + 1
    float2 nxt2;               // its side entry (PEND only)
#endif
};

template <bool PEND>
__device__ __forceinline__ void take_row(Slot<PEND>& q, const Row& r, const float2 e)
{
    q.rnext = __float_as_int(r.v0.x);
    q.kvB1 = r.v0.y;
    q.kvE = r.v0.z;
    q.b0n = r.v0.w;
    q.b1 = r.v1.x;
    q.nh = r.v1.y;
    q.np1n = fmaf(2.0f, r.v1.y, -1.0f);
    q.pmA = r.v1.z;
    q.Gt = r.v1.w;
    if (PEND) {
        q.pmAp = e.x;
        q.Gpt = e.y;
    }
}

// One CTA = SCORE_WARPS warps x 32 lanes x SLOTS consecutive workers and one
// contiguous range of sorted candidates (one wave of CTAs, equal shares).
// Requires W % 4 == 0 and 16-byte aligned outputs. PEND: some worker holds
// requests placed in an open round (pending prefill and its TTFT/ATGT bounds).
#ifndef ALADDIN_STORE_HINT
#define ALADDIN_STORE_HINT 1
#endif
template <typename T>
__device__ __forceinline__ void st_out(T* p, T v)
{
#if ALADDIN_STORE_HINT
    __stcs(p, v);
#else
    *p = v;
#endif
}

template <int SLOTS, bool SF, bool SMG, bool ARG, bool PEND, bool FULLT, bool APPROX>
__global__ void __launch_bounds__(SCORE_WARPS * 32, PEND ? 3 : ALADDIN_SCORE_MINB) k_score(VecArgs A)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    ScoreSmem& sm = *reinterpret_cast<ScoreSmem*>(smraw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int W = A.C.W;
    const int tile = blockIdx.x % A.tiles;
    const int part = blockIdx.x / A.tiles;
    const int cb = (int)(((long long)A.n_cand * part) / A.per_tile);
    const int ce = (int)(((long long)A.n_cand * (part + 1)) / A.per_tile);
    if (cb >= ce) return;  // CTA-uniform
    const int nchunks = (ce - cb + CHUNK - 1) / CHUNK;

    if (tid == 0) {
        mbar_init(&sm.bar[0], 1);
        mbar_init(&sm.bar[1], 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        sm.stop = 0;
    }
    __syncthreads();
    if (tid == 0 && !A.withhold) {
        const int n0 = min(CHUNK, ce - cb);
        tma_load(sm.cs[0], A.cand + (size_t)cb * REC_F4, (unsigned)n0 * (REC_F4 * 16u), &sm.bar[0]);
    }

    const int wbase = (tile * SCORE_WARPS + warp) * 32 * SLOTS;
    const int w0 = wbase + lane * SLOTS;
    const bool live = FULLT || w0 < W;
    const bool warp_live = FULLT || wbase < W;
    uint8_t* const fbase = SF ? A.flags + (live ? w0 : 0) : nullptr;
    float* const mbase = SMG ? A.margin + (live ? w0 : 0) : nullptr;
    const int last_row = A.C.rows - 1;

    Slot<PEND> ss[SLOTS];
    int p[SLOTS], wk[SLOTS];
    float inv_s[SLOTS], nZO[SLOTS], ZW[SLOTS];
    float bd[APPROX ? SLOTS : 1], bq[APPROX ? SLOTS : 1];  // approximate-mode bounds
    unsigned rank[SLOTS];
    int nb = 0;  // smallest next breakpoint over this lane's workers
    bool have_rows = false;
    // The KV and decode-time bounds of a pair depend on the worker's row and
    // the candidate's predicted length only (not on its prompt or wait):
    // computed once for a run of candidates of equal length on unchanged rows
    // (the candidates are sorted by length), minus each candidate's a after.
    float xkv[SLOTS], xdt[SLOTS];
    int x_ri = -1;  // the length they hold (warp-uniform); -1: none

    for (int k = 0; k < nchunks; ++k) {
        const int buf = k & 1;
        const int c0 = cb + k * CHUNK;
        const int nc = min(CHUNK, ce - c0);
        if (tid == 0 && k + 1 < nchunks) {
            const int c1 = c0 + CHUNK;
            const int n1 = min(CHUNK, ce - c1);
            tma_load(sm.cs[buf ^ 1], A.cand + (size_t)c1 * REC_F4, (unsigned)n1 * (REC_F4 * 16u),
                     &sm.bar[buf ^ 1]);
        }
        if (!mbar_wait(&sm.bar[buf], (unsigned)((k >> 1) & 1), A.wait_limit)) {
            if (lane == 0) atomicOr(A.C.err, ERR_TIMEOUT_BIT);
            sm.stop = 1;
        }
        __syncthreads();
        if (sm.stop) {
            // the copy into the other buffer is in flight: let it land first
            // (with the full limit whatever the cluster's test setting)
            if (tid == 0 && k + 1 < nchunks)
                mbar_wait(&sm.bar[buf ^ 1], (unsigned)(((k + 1) >> 1) & 1), MBAR_WAIT_POLLS);
            return;
        }
        const float4* cs = sm.cs[buf];
        if (warp_live) {
            if (!have_rows) {
                const int r_first = __float_as_int(cs[2].x);
#pragma unroll
                for (int s = 0; s < SLOTS; ++s) {
                    wk[s] = live ? (A.order ? __ldg(&A.order[w0 + s]) : w0 + s) : W - 1;
                    const long long rb = (long long)wk[s] * A.C.rows;
                    p[s] = find_row(A.C.tab, rb, __ldg(&A.C.R[wk[s]]), r_first);
                    const long long pn = rb + min(p[s] + 1, last_row);
                    take_row<PEND>(ss[s], load_row(A.C.tab, rb + p[s]),
                                   PEND ? __ldg(&A.C.tab2[rb + p[s]]) : make_float2(0.f, 0.f));
#if ALADDIN_SCORE_PF
                    prefetch_row(A.C.tab, pn);
#else
                    ss[s].nxt = load_row(A.C.tab, pn);
                    if (PEND) ss[s].nxt2 = __ldg(&A.C.tab2[pn]);
#endif
                    const float4 wr = __ldg(&A.C.wrec[wk[s]]);
                    inv_s[s] = wr.x;
                    nZO[s] = -wr.y;
                    ZW[s] = wr.z;
                    rank[s] = live ? (unsigned)__float_as_int(wr.w) : 0xffffffffu;
                    if constexpr (APPROX) {
                        const float2 wa = __ldg(&A.C.wapx[wk[s]]);
                        bd[s] = wa.x;
                        bq[s] = wa.y;
                    }
                }
                nb = ss[0].rnext;
#pragma unroll
                for (int s = 1; s < SLOTS; ++s) nb = min(nb, ss[s].rnext);
                have_rows = true;
            }
            unsigned* const kbase = &sm.kmin[warp][0];
            auto rec_off = [&](int i) {  // start of candidate i's output row
                const float4 q4 = cs[i * REC_F4 + 2];
                return ((unsigned long long)__float_as_uint(q4.w) << 32) | __float_as_uint(q4.z);
            };
            auto rec_ri = [&](int i) { return __float_as_int(cs[i * REC_F4 + 2].x); };
            // Step every slot to the row whose segment holds ri (when some lane
            // of the warp needs it); the next row is in L1 already, the one
            // after is fetched now and needed only at the next crossing.
            auto step_rows = [&](int ri) {
                if (__any_sync(FULL, ri >= nb)) {
                    x_ri = -1;
#pragma unroll
                    for (int s = 0; s < SLOTS; ++s) {
                        while (ri >= ss[s].rnext && p[s] < last_row) {
                            p[s] += 1;
                            const long long rb = (long long)wk[s] * A.C.rows;
                            const long long pn = rb + min(p[s] + 1, last_row);
#if ALADDIN_SCORE_PF
                            take_row<PEND>(ss[s], load_row(A.C.tab, rb + p[s]),
                                           PEND ? __ldg(&A.C.tab2[rb + p[s]]) : make_float2(0.f, 0.f));
                            prefetch_row(A.C.tab, pn);
#else
                            take_row<PEND>(ss[s], ss[s].nxt, ss[s].nxt2);
                            ss[s].nxt = load_row(A.C.tab, pn);
                            if (PEND) ss[s].nxt2 = __ldg(&A.C.tab2[pn]);
#endif
                        }
                    }
                    nb = ss[0].rnext;
#pragma unroll
                    for (int s = 1; s < SLOTS; ++s) nb = min(nb, ss[s].rnext);
                }
            };
            // The group headrooms and margins of candidate i on this lane's
            // workers (current rows), and its argbest key.
            auto eval = [&](int i, float (&d)[4][SLOTS], float (&m)[SLOTS], unsigned& kmin) {
                const float4 q0 = cs[i * REC_F4], q1 = cs[i * REC_F4 + 1];
                const float a = q0.x, r = q0.y, ir = q0.z, Ua = q0.w;
                const float id1 = q1.x, nX = q1.y, id2 = q1.z, Zc = q1.w;
                kmin = 0xffffffffu;
                if constexpr (!APPROX) {
                    const int ri = rec_ri(i);
                    if (ri != x_ri) {  // warp-uniform
#pragma unroll
                        for (int s = 0; s < SLOTS; ++s) {
                            xkv[s] = fminf(ss[s].kvB1, fmaf(r, ss[s].np1n, ss[s].kvE));
                            xdt[s] = fminf(ss[s].pmA, fmaf(ss[s].Gt, id1, nX));
                        }
                        x_ri = ri;
                    }
                }
#pragma unroll
                for (int s = 0; s < SLOTS; ++s) {
                    const Slot<PEND>& t = ss[s];
                    d[0][s] = (APPROX ? fminf(t.kvB1, fmaf(r, t.np1n, t.kvE)) : xkv[s]) - a;
                    const float tt = fmaf(Zc, inv_s[s], nZO[s]);
                    if constexpr (APPROX) {
                        // (d) and (b) of the placement MIP; Ua holds a + gamma r
                        d[2][s] = bd[s % (APPROX ? SLOTS : 1)] - a;
                        d[3][s] = bq[s % (APPROX ? SLOTS : 1)] - Ua;
                        d[1][s] = (PEND ? fminf(tt, ZW[s]) : tt) - a;
                    } else {
                        d[2][s] = xdt[s] - a;
                        const float ca = fmaf(t.b0n, ir, fmaf(t.nh, r, Ua - t.b1));
                        if (PEND) {
                            d[1][s] = fminf(tt, ZW[s]) - a;
                            d[3][s] = fmin3(t.pmAp - a, fmaf(t.Gpt, id2, Ua), ca);
                        } else {
                            d[1][s] = tt - a;
                            d[3][s] = ca;
                        }
                    }
                    m[s] = fmin3(fminf(d[0][s], d[1][s]), d[2][s], d[3][s]);
                    if (ARG) kmin = min(kmin, (__float_as_uint(m[s]) & 0x80000000u) | rank[s]);
                }
            };
            auto store = [&](int i, const float (&d)[4][SLOTS], const float (&m)[SLOTS]) {
                if (!live) return;
                const unsigned long long off = rec_off(i);
                if (SF) {
                    const unsigned f = pack_flags<SLOTS>(d);
                    if (SLOTS == 4) st_out(reinterpret_cast<unsigned int*>(fbase + off), f);
                    else st_out(reinterpret_cast<unsigned short*>(fbase + off), (unsigned short)f);
                }
                if (SMG) {
                    if (SLOTS == 4)
                        st_out(reinterpret_cast<float4*>(mbase + off),
                               make_float4(m[0], m[1], m[2 % SLOTS], m[3 % SLOTS]));
                    else
                        st_out(reinterpret_cast<float2*>(mbase + off), make_float2(m[0], m[1]));
                }
            };
            auto score_one = [&](int i) {
                float d[4][SLOTS], m[SLOTS];
                unsigned kmin;
                eval(i, d, m, kmin);
                store(i, d, m);
                if (ARG) kbase[i] = __reduce_min_sync(FULL, kmin);  // same value from every lane
            };

            // invalid candidates sort first (bucket 0): a prefix of the chunk
            int i = 0;
            for (; i < nc && rec_ri(i) == 0; ++i) {  // warp-uniform
                if (live) {
                    const unsigned long long off = rec_off(i);
#pragma unroll
                    for (int s = 0; s < SLOTS; ++s) {
                        if (SF) fbase[off + s] = 0x80;
                        if (SMG) mbase[off + s] = __int_as_float(0x7fc00000);
                    }
                }
                if (ARG) kbase[i] = 0xffffffffu;
            }
            // two candidates at a time on the same rows (independent chains the
            // scheduler interleaves); one at a time where a breakpoint lies
            // between them
            for (; i + 1 < nc; i += 2) {
                step_rows(rec_ri(i));
                if (__any_sync(FULL, rec_ri(i + 1) >= nb)) {
                    score_one(i);
                    step_rows(rec_ri(i + 1));
                    score_one(i + 1);
                } else {
                    float d0[4][SLOTS], m0[SLOTS], d1[4][SLOTS], m1[SLOTS];
                    unsigned k0, k1;
                    eval(i, d0, m0, k0);
                    eval(i + 1, d1, m1, k1);
                    store(i, d0, m0);
                    store(i + 1, d1, m1);
                    if (ARG) {
                        kbase[i] = __reduce_min_sync(FULL, k0);
                        kbase[i + 1] = __reduce_min_sync(FULL, k1);
                    }
                }
            }
            if (i < nc) {
                step_rows(rec_ri(i));
                score_one(i);
            }
        } else if (ARG) {
            for (int i = lane; i < nc; i += 32) sm.kmin[warp][i] = 0xffffffffu;
        }
        __syncthreads();
        if (ARG) {
            for (int i = tid; i < nc; i += SCORE_WARPS * 32) {
                unsigned v = sm.kmin[0][i];
#pragma unroll
                for (int w = 1; w < SCORE_WARPS; ++w) v = min(v, sm.kmin[w][i]);
                if (v < 0x80000000u) atomicMin(A.best + __float_as_int(cs[REC_F4 * i + 2].y), v);
            }
        }
        __syncthreads();  // buffer `buf` and kmin are reused two chunks later
    }
}

// Fallback for W % 4 != 0 or unaligned outputs: one worker per lane, scalar
// stores, candidate records read from global memory.
template <bool SF, bool SMG, bool ARG>
__global__ void __launch_bounds__(SCORE_WARPS * 32) k_score_scalar(ScoreArgs A)
{
    const int lane = threadIdx.x & 31;
    const int unit = blockIdx.x * SCORE_WARPS + (threadIdx.x >> 5);
    if (unit >= A.tiles * A.chunks) return;
    const int tile = unit % A.tiles, chunk = unit / A.tiles;
    const int W = A.C.W;
    const int w = tile * 32 + lane;  // output column
    const bool live = w < W;
    const int wc = live ? (A.order ? __ldg(&A.order[w]) : w) : W - 1;  // its worker
    const int c0 = chunk * SCORE_CHUNK;
    const int c1 = min(c0 + SCORE_CHUNK, A.n_cand);
    const long long rb = (long long)wc * A.C.rows;
    const int last_row = A.C.rows - 1;
    const float4* recs = reinterpret_cast<const float4*>(A.cand);
    int p = find_row(A.C.tab, rb, A.C.R[wc], __float_as_int(__ldg(&recs[(size_t)c0 * REC_F4 + 2].x)));
    Row cur = load_row(A.C.tab, rb + p);
    float2 ext = __ldg(&A.C.tab2[rb + p]);
    const float4 wr = __ldg(&A.C.wrec[wc]);
    const float2 wa = A.approx ? __ldg(&A.C.wapx[wc]) : make_float2(0.0f, 0.0f);
    const unsigned rank = live ? (unsigned)__float_as_int(wr.w) : 0xffffffffu;
    for (int c = c0; c < c1; ++c) {
        const float4* cp = recs + (size_t)c * REC_F4;
        const float4 q0 = __ldg(cp), q1 = __ldg(cp + 1), q2 = __ldg(cp + 2);
        CandRec cr;
        cr.a = q0.x; cr.r = q0.y; cr.inv_r = q0.z; cr.Ua = q0.w;
        cr.inv_d1 = q1.x; cr.nXd1 = q1.y; cr.inv_d2 = q1.z; cr.Zc = q1.w;
        cr.ri = __float_as_int(q2.x);
        cr.orig = __float_as_int(q2.y);
        const size_t off = (size_t)cr.orig * (size_t)A.ld + (size_t)w;
        if (cr.ri == 0) {
            if (live) {
                if (SF) A.flags[off] = 0x80;
                if (SMG) A.margin[off] = __int_as_float(0x7fc00000);
            }
            continue;
        }
        while (cr.ri >= __float_as_int(cur.v0.x) && p < last_row) {
            p += 1;
            cur = load_row(A.C.tab, rb + p);
            ext = __ldg(&A.C.tab2[rb + p]);
        }
        float m;
        const unsigned f = eval_pair_mode(A.approx != 0, cur.v0, cur.v1, ext, wr, wa, cr, m);
        if (live) {
            if (SF) A.flags[off] = (uint8_t)f;
            if (SMG) __stcs(A.margin + off, m);
        }
        if (ARG) {
            unsigned kmin = (f == 15u) ? rank : 0xffffffffu;
            kmin = __reduce_min_sync(FULL, kmin);
            if (lane == 0 && kmin != 0xffffffffu) atomicMin(A.best + cr.orig, kmin);
        }
    }
}

template <int SLOTS, bool SF, bool SMG, bool ARG, bool PEND, bool FULLT, bool APPROX>
static cudaError_t launch_vec(const ScoreArgs& A0, cudaStream_t st)
{
    VecArgs A;
    A.C = A0.C;
    A.cand = reinterpret_cast<const float4*>(A0.cand);
    A.n_cand = A0.n_cand;
    A.flags = A0.flags;
    A.margin = A0.margin;
    A.best = A0.best;
    A.tiles = (A.C.W + SCORE_WARPS * 32 * SLOTS - 1) / (SCORE_WARPS * 32 * SLOTS);
    A.wait_limit = A0.wait_limit;
    A.withhold = A0.withhold;
    A.order = A0.order;
    const size_t smem = sizeof(ScoreSmem);
    DevInfo d;
    cudaError_t e = device_info(&d);
    if (e != cudaSuccess) return e;
    int per_sm = 0;  // occupancy of this instantiation on this device (cached)
    e = kernel_occupancy<k_score<SLOTS, SF, SMG, ARG, PEND, FULLT, APPROX>>(SCORE_WARPS * 32, smem,
                                                                          &per_sm);
    if (e != cudaSuccess) return e;
    // one wave: per_tile CTAs share each worker tile's candidates equally
    const int wave = per_sm * d.sms;
    int per_tile = wave / A.tiles;
    if (per_tile < 1) per_tile = 1;
    const int max_parts = (A.n_cand + 63) / 64;  // at least 64 candidates per CTA
    if (per_tile > max_parts) per_tile = max_parts;
    A.per_tile = per_tile;
    k_score<SLOTS, SF, SMG, ARG, PEND, FULLT, APPROX><<<A.tiles * per_tile, SCORE_WARPS * 32, smem, st>>>(A);
    return cudaGetLastError();
}

template <bool PEND, bool FULLT, bool APPROX>
static cudaError_t dispatch_vec3(bool sf, bool smg, bool arg, const ScoreArgs& A, cudaStream_t st)
{
    constexpr int S = ALADDIN_SCORE_SLOTS;
    if (sf && smg && arg) return launch_vec<S, true, true, true, PEND, FULLT, APPROX>(A, st);
    if (sf && smg) return launch_vec<S, true, true, false, PEND, FULLT, APPROX>(A, st);
    if (sf && arg) return launch_vec<S, true, false, true, PEND, FULLT, APPROX>(A, st);
    if (smg && arg) return launch_vec<S, false, true, true, PEND, FULLT, APPROX>(A, st);
    if (sf) return launch_vec<S, true, false, false, PEND, FULLT, APPROX>(A, st);
    if (smg) return launch_vec<S, false, true, false, PEND, FULLT, APPROX>(A, st);
    return launch_vec<S, false, false, true, PEND, FULLT, APPROX>(A, st);
}

template <bool PEND, bool FULLT>
static cudaError_t dispatch_vec2(bool approx, bool sf, bool smg, bool arg, const ScoreArgs& A,
                                 cudaStream_t st)
{
    return approx ? dispatch_vec3<PEND, FULLT, true>(sf, smg, arg, A, st)
                  : dispatch_vec3<PEND, FULLT, false>(sf, smg, arg, A, st);
}

template <bool PEND>
static cudaError_t dispatch_vec(bool approx, bool sf, bool smg, bool arg, const ScoreArgs& A,
                                cudaStream_t st)
{
    // every lane of every CTA tile holds a worker: no per-lane predicate
    const bool full = A.C.W % (SCORE_WARPS * 32 * ALADDIN_SCORE_SLOTS) == 0;
    return full ? dispatch_vec2<PEND, true>(approx, sf, smg, arg, A, st)
                : dispatch_vec2<PEND, false>(approx, sf, smg, arg, A, st);
}

// prepare_score_kernels: every k_score instantiation dispatch_vec can reach
// (seven output combinations x pending x full tile x approximate), the scalar
// variants and the candidate preparation, finalize and detail kernels.
template <bool PEND, bool FULLT, bool APPROX>
static cudaError_t prepare_vec3()
{
    constexpr int S = ALADDIN_SCORE_SLOTS;
    constexpr int T = SCORE_WARPS * 32;
    constexpr size_t M = sizeof(ScoreSmem);
    int ps = 0;
    cudaError_t e;
    if ((e = kernel_occupancy<k_score<S, true, true, true, PEND, FULLT, APPROX>>(T, M, &ps)) ||
        (e = kernel_occupancy<k_score<S, true, true, false, PEND, FULLT, APPROX>>(T, M, &ps)) ||
        (e = kernel_occupancy<k_score<S, true, false, true, PEND, FULLT, APPROX>>(T, M, &ps)) ||
        (e = kernel_occupancy<k_score<S, false, true, true, PEND, FULLT, APPROX>>(T, M, &ps)) ||
        (e = kernel_occupancy<k_score<S, true, false, false, PEND, FULLT, APPROX>>(T, M, &ps)) ||
        (e = kernel_occupancy<k_score<S, false, true, false, PEND, FULLT, APPROX>>(T, M, &ps)) ||
        (e = kernel_occupancy<k_score<S, false, false, true, PEND, FULLT, APPROX>>(T, M, &ps)))
        return e;
    return cudaSuccess;
}

template <bool SF, bool SMG, bool ARG>
static void launch_scalar(const ScoreArgs& A0, cudaStream_t st)
{
    ScoreArgs A = A0;
    A.tiles = (A.C.W + 31) / 32;
    const int units = A.tiles * A.chunks;
    k_score_scalar<SF, SMG, ARG><<<(units + SCORE_WARPS - 1) / SCORE_WARPS, SCORE_WARPS * 32, 0, st>>>(A);
}

__global__ void k_finalize(DevParams P, int n, const int32_t* __restrict__ in,
                           const int32_t* __restrict__ pred, const float* __restrict__ wait,
                           const unsigned int* __restrict__ best, const int32_t* __restrict__ order,
                           int32_t* argbest)
{
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= n) return;
    const int32_t a = in[c], r = pred[c];
    const float w = wait ? wait[c] : 0.0f;
    const bool ok = a >= 0 && r >= 1 && (long long)a + r <= (long long)P.K && w >= 0.0f &&
                    w <= 3.0e38f;
    const unsigned b = best[c];
    argbest[c] = !ok ? -2 : (b == 0xffffffffu ? -1 : order[b]);
}

// Verification outputs: exact KV peak and the candidate's projected decode
// time, from the exact integer aggregates of the row (one thread per pair).
__global__ void k_detail(DevParams P, ClusterDev C, int n, const int32_t* __restrict__ in,
                         const int32_t* __restrict__ pred, const float* __restrict__ wait,
                         int64_t* kv_peak, float* t_cand)
{
    const long long total = (long long)n * C.W;
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(idx / C.W);
        const int w = (int)(idx % C.W);
        const int32_t a = in[c], r = pred[c];
        const float wt = wait ? wait[c] : 0.0f;
        const bool ok = a >= 0 && r >= 1 && (long long)a + r <= (long long)P.K && wt >= 0.0f &&
                        wt <= 3.0e38f;
        if (!ok) {
            if (kv_peak) kv_peak[idx] = -1;
            if (t_cand) t_cand[idx] = __int_as_float(0x7fc00000);
            continue;
        }
        const long long rb = (long long)w * C.rows;
        const int p = find_row(C.tab, rb, C.R[w], r);
        const AuxRow x = C.aux[rb + p];
        const long long h = P.h, jj = P.j, rr = r, aa = a, np = x.n;
        long long pk = h * (x.A + rr * np) + jj * np + h * (aa + rr) + jj;
        if (x.PM != LL_NONE) pk = max(pk, x.PM + h * aa + jj);
        pk = max(pk, x.SM);
        if (kv_peak) kv_peak[idx] = pk;
        if (t_cand) {
            const double X1 = (double)(x.PR + rr * (np + 1));
            const double X2 = (double)(x.PRA + rr * (x.A + aa) + (np + 1) * (rr * (rr + 1) / 2));
            const double sc = (double)C.scale[w];
            t_cand[idx] = (float)(sc * (P.c3d * (double)rr + P.c2d * X1 + P.k2d * X2));
        }
    }
}

cudaError_t prepare_score_kernels()
{
    cudaError_t e;
    if ((e = prepare_vec3<false, false, false>()) || (e = prepare_vec3<false, false, true>()) ||
        (e = prepare_vec3<false, true, false>()) || (e = prepare_vec3<false, true, true>()) ||
        (e = prepare_vec3<true, false, false>()) || (e = prepare_vec3<true, false, true>()) ||
        (e = prepare_vec3<true, true, false>()) || (e = prepare_vec3<true, true, true>()))
        return e;
    cudaFuncAttributes fa;
    const void* kerns[] = {
        (const void*)k_score_scalar<true, true, true>, (const void*)k_score_scalar<true, true, false>,
        (const void*)k_score_scalar<true, false, true>, (const void*)k_score_scalar<false, true, true>,
        (const void*)k_score_scalar<true, false, false>, (const void*)k_score_scalar<false, true, false>,
        (const void*)k_score_scalar<false, false, true>, (const void*)k_cand_count,
        (const void*)k_scan_hist, (const void*)k_cand_scatter, (const void*)k_finalize,
        (const void*)k_detail};
    for (const void* k : kerns)
        if ((e = cudaFuncGetAttributes(&fa, k)) != cudaSuccess) return e;
    return cudaSuccess;
}

cudaError_t launch_cand_prep(const DevParams& P, int W, int n, const int32_t* in,
                             const int32_t* pred, const float* wait, const ScoreBuffers& B,
                             cudaStream_t st)
{
    if (n <= 0) return cudaSuccess;
    const int tb = 256, nb = (n + tb - 1) / tb;
    cudaError_t e = cudaMemsetAsync(B.hist, 0, sizeof(int32_t) * (size_t)(P.K + 1), st);
    if (e != cudaSuccess) return e;
    k_cand_count<<<nb, tb, 0, st>>>(P, n, in, pred, wait, B.hist, B.best);
    k_scan_hist<<<1, SCAN_THREADS, 0, st>>>(B.hist, P.K + 1);
    k_cand_scatter<<<nb, tb, 0, st>>>(P, n, W, in, pred, wait, B.hist, B.sorted);
    return cudaGetLastError();
}

cudaError_t launch_score(const DevParams& P, const ClusterDev& C, int n, const int32_t* in,
                         const int32_t* pred, const float* wait, uint8_t* flags, float* margin,
                         int32_t* argbest, int64_t* kv_peak, float* t_cand, const ScoreBuffers& B,
                         bool pend, cudaStream_t st, cudaEvent_t ev0, cudaEvent_t ev1,
                         bool prepared, const int32_t* ranked, int ld)
{
    if (n <= 0) return cudaSuccess;
    cudaError_t e;
    const int tb = 256, nb = (n + tb - 1) / tb;
    const bool need_score = flags || margin || argbest;
    const int row = ld > 0 ? ld : C.W;  // output row stride
    if (need_score) {
        if (!prepared && (e = launch_cand_prep(P, row, n, in, pred, wait, B, st)) != cudaSuccess)
            return e;

        ScoreArgs A;
        A.C = C;
        A.cand = B.sorted;
        A.n_cand = n;
        A.flags = flags;
        A.margin = margin;
        A.best = argbest ? B.best : nullptr;
        A.chunks = (n + SCORE_CHUNK - 1) / SCORE_CHUNK;
        A.tiles = 0;
        A.approx = P.approx;
        A.wait_limit = P.mbar_wait_limit;
        A.withhold = P.wait_test;
        A.order = ranked;
        A.ld = row;
        if (ev0) cudaEventRecord(ev0, st);
        const bool vec = (C.W % 4 == 0) && (row % 4 == 0) && (((uintptr_t)flags & 3) == 0) &&
                         (((uintptr_t)margin & 15) == 0);
        const bool sf = flags != nullptr, smg = margin != nullptr, arg = argbest != nullptr;
        if (vec) {
            const bool ap = P.approx != 0;
            e = pend ? dispatch_vec<true>(ap, sf, smg, arg, A, st)
                     : dispatch_vec<false>(ap, sf, smg, arg, A, st);
            if (e != cudaSuccess) return e;
        } else {
            if (sf && smg && arg) launch_scalar<true, true, true>(A, st);
            else if (sf && smg) launch_scalar<true, true, false>(A, st);
            else if (sf && arg) launch_scalar<true, false, true>(A, st);
            else if (smg && arg) launch_scalar<false, true, true>(A, st);
            else if (sf) launch_scalar<true, false, false>(A, st);
            else if (smg) launch_scalar<false, true, false>(A, st);
            else launch_scalar<false, false, true>(A, st);
        }
        if (ev1) cudaEventRecord(ev1, st);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        if (argbest) {
            k_finalize<<<nb, tb, 0, st>>>(P, n, in, pred, wait, B.best, C.order, argbest);
            e = cudaGetLastError();
            if (e != cudaSuccess) return e;
        }
    }
    if (kv_peak || t_cand) {
        const long long total = (long long)n * C.W;
        const long long nblk = (total + 255) / 256;
        const int blocks = (int)(nblk < 65536 ? nblk : 65536);
        k_detail<<<blocks, 256, 0, st>>>(P, C, n, in, pred, wait, kv_peak, t_cand);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace aladdin
