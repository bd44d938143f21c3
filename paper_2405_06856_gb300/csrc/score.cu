// K3: batched candidate x worker scoring.
//
// Candidates are validated, turned into per-candidate constants and
// counting-sorted by predicted output length. A warp owns a tile of
// 32 x SLOTS consecutive workers (SLOTS per lane) and sweeps a chunk of the
// sorted candidates: each lane keeps the table row of each of its workers in
// registers and only steps to the next row when the candidate's length
// crosses that worker's next breakpoint, so a pair costs one row compare and
// the O(1) bound arithmetic of eval_pair. Flags and margins of one candidate
// are written as one coalesced row segment per warp (streaming stores); the
// per-candidate argbest is the smallest capacity_norm rank among feasible
// workers (warp min-reduction, one atomic per warp and candidate).
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

__global__ void k_cand_scatter(DevParams P, int n, const int32_t* __restrict__ in,
                               const int32_t* __restrict__ pred, const float* __restrict__ wait,
                               int32_t* cursor, CandRec* sorted)
{
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= n) return;
    const CandRec rec = make_cand(P, in[c], pred[c], wait ? wait[c] : 0.0f, c);
    const int pos = atomicAdd(&cursor[rec.valid ? rec.ri : 0], 1);
    sorted[pos] = rec;
}

struct ScoreArgs {
    ClusterDev C;
    const CandRec* __restrict__ cand;
    int n_cand;
    uint8_t* flags;
    float* margin;
    unsigned int* best;
    int tiles, chunks;
};

__device__ __forceinline__ void load_row(const float4* __restrict__ tab, long long row, float4& v0,
                                         float4& v1, float4& v2)
{
    const float4* t = tab + row * ROW_F4;
    v0 = __ldg(t);
    v1 = __ldg(t + 1);
    v2 = __ldg(t + 2);
}

template <int SLOTS, bool STORE, bool VEC>
__global__ void __launch_bounds__(SCORE_WARPS * 32) k_score(ScoreArgs A)
{
    const int lane = threadIdx.x & 31;
    const int unit = blockIdx.x * SCORE_WARPS + (threadIdx.x >> 5);
    if (unit >= A.tiles * A.chunks) return;  // warp-uniform
    const int tile = unit % A.tiles;
    const int chunk = unit / A.tiles;
    const int W = A.C.W;
    const int w0 = tile * 32 * SLOTS + lane * SLOTS;
    const int c0 = chunk * SCORE_CHUNK;
    const int c1 = min(c0 + SCORE_CHUNK, A.n_cand);

    float4 v0[SLOTS], v1[SLOTS], v2[SLOTS], wr[SLOTS];
    int p[SLOTS], Rk[SLOTS];
    long long rb[SLOTS];
    unsigned rk[SLOTS];
    bool live[SLOTS];
    const int r_first = __ldg(&A.cand[c0].ri);
#pragma unroll
    for (int k = 0; k < SLOTS; ++k) {
        const int w = w0 + k;
        live[k] = w < W;
        const int wc = live[k] ? w : 0;
        rb[k] = (long long)wc * A.C.rows;
        const int R = live[k] ? A.C.R[wc] : 0;
        Rk[k] = R;
        p[k] = live[k] ? find_row(A.C.tab, rb[k], R, r_first) : 0;
        load_row(A.C.tab, rb[k] + p[k], v0[k], v1[k], v2[k]);
        wr[k] = __ldg(&A.C.wrec[wc]);
        rk[k] = (unsigned)__float_as_int(wr[k].w);
    }

    for (int c = c0; c < c1; ++c) {
        const float4* cp = reinterpret_cast<const float4*>(A.cand + c);
        const float4 q0 = __ldg(cp), q1 = __ldg(cp + 1), q2 = __ldg(cp + 2);
        CandRec cr;
        cr.a = q0.x; cr.r = q0.y; cr.inv_r = q0.z; cr.U = q0.w;
        cr.inv_d1 = q1.x; cr.nXd1 = q1.y; cr.inv_d2 = q1.z; cr.Zc = q1.w;
        cr.ri = __float_as_int(q2.x);
        cr.orig = __float_as_int(q2.y);
        cr.valid = __float_as_int(q2.z);
        const size_t rowoff = (size_t)cr.orig * (size_t)W;
        if (!cr.valid) {
            if (STORE) {
#pragma unroll
                for (int k = 0; k < SLOTS; ++k)
                    if (live[k]) {
                        if (A.flags) A.flags[rowoff + w0 + k] = 0x80;
                        if (A.margin) A.margin[rowoff + w0 + k] = __int_as_float(0x7fc00000);
                    }
            }
            continue;
        }
        unsigned bestv = 0xffffffffu;
        unsigned fpack = 0;
        float mg[SLOTS];
#pragma unroll
        for (int k = 0; k < SLOTS; ++k) {
            mg[k] = 0.0f;
            if (live[k]) {
                while (cr.ri >= __float_as_int(v0[k].x) && p[k] < Rk[k]) {
                    p[k] += 1;
                    load_row(A.C.tab, rb[k] + p[k], v0[k], v1[k], v2[k]);
                }
                float m;
                const unsigned f = eval_pair(v0[k], v1[k], v2[k], wr[k], cr, m);
                mg[k] = m;
                fpack |= f << (8 * k);
                if (f == 15u) bestv = min(bestv, rk[k]);
            }
        }
        if (STORE) {
            if (VEC) {
                if (live[0]) {
                    if (A.flags)
                        __stcs(reinterpret_cast<unsigned int*>(A.flags + rowoff + w0), fpack);
                    if (A.margin)
                        __stcs(reinterpret_cast<float4*>(A.margin + rowoff + w0),
                               make_float4(mg[0], mg[SLOTS > 1 ? 1 : 0], mg[SLOTS > 2 ? 2 : 0],
                                           mg[SLOTS > 3 ? 3 : 0]));
                }
            } else {
#pragma unroll
                for (int k = 0; k < SLOTS; ++k)
                    if (live[k]) {
                        if (A.flags) A.flags[rowoff + w0 + k] = (uint8_t)((fpack >> (8 * k)) & 0xffu);
                        if (A.margin) __stcs(A.margin + rowoff + w0 + k, mg[k]);
                    }
            }
        }
        if (A.best) {
            bestv = __reduce_min_sync(FULL, bestv);
            if (lane == 0 && bestv != 0xffffffffu) atomicMin(A.best + cr.orig, bestv);
        }
    }
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

cudaError_t launch_score(const DevParams& P, const ClusterDev& C, int n, const int32_t* in,
                         const int32_t* pred, const float* wait, uint8_t* flags, float* margin,
                         int32_t* argbest, int64_t* kv_peak, float* t_cand, const ScoreBuffers& B,
                         cudaStream_t st, cudaEvent_t ev0, cudaEvent_t ev1)
{
    if (n <= 0) return cudaSuccess;
    cudaError_t e;
    const int tb = 256, nb = (n + tb - 1) / tb;
    const bool need_score = flags || margin || argbest;
    if (need_score) {
        e = cudaMemsetAsync(B.hist, 0, sizeof(int32_t) * (size_t)(P.K + 1), st);
        if (e != cudaSuccess) return e;
        k_cand_count<<<nb, tb, 0, st>>>(P, n, in, pred, wait, B.hist, B.best);
        k_scan_hist<<<1, SCAN_THREADS, 0, st>>>(B.hist, P.K + 1);
        k_cand_scatter<<<nb, tb, 0, st>>>(P, n, in, pred, wait, B.hist, B.sorted);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;

        ScoreArgs A;
        A.C = C;
        A.cand = B.sorted;
        A.n_cand = n;
        A.flags = flags;
        A.margin = margin;
        A.best = argbest ? B.best : nullptr;
        A.chunks = (n + SCORE_CHUNK - 1) / SCORE_CHUNK;
        const bool store = flags || margin;
        if (ev0) cudaEventRecord(ev0, st);
        const bool vec = (C.W % 4 == 0) && (((uintptr_t)flags & 3) == 0) &&
                         (((uintptr_t)margin & 15) == 0);
        if (store && vec) {
            A.tiles = (C.W + 127) / 128;
            const int units = A.tiles * A.chunks;
            k_score<4, true, true><<<(units + SCORE_WARPS - 1) / SCORE_WARPS, SCORE_WARPS * 32, 0, st>>>(A);
        } else if (store) {
            A.tiles = (C.W + 31) / 32;
            const int units = A.tiles * A.chunks;
            k_score<1, true, false><<<(units + SCORE_WARPS - 1) / SCORE_WARPS, SCORE_WARPS * 32, 0, st>>>(A);
        } else {
            A.tiles = (C.W + 127) / 128;
            const int units = A.tiles * A.chunks;
            k_score<4, false, false><<<(units + SCORE_WARPS - 1) / SCORE_WARPS, SCORE_WARPS * 32, 0, st>>>(A);
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
