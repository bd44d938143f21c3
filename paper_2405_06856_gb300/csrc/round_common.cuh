// Device helpers of the two best-fit round kernels (the sliced round k_round2
// and the incremental round k_round_inc): the rebuild group's split, the
// shared-memory breakpoint search and the (key, lowest index) reductions.
#pragma once

#include "aladdin_host.h"

namespace aladdin {

template <int E>
struct R2Split {
    // up to 256 slots: NW warps cover the capacity with one element a lane;
    // larger tables: 12 warps (4 left for evaluation) with up to E/8
    // elements a lane, the build sized to the worker's count
    static constexpr int NW = E <= 8 ? E : 12;
    static constexpr int EW = E <= 8 ? 1 : E / 8;
};
// Breakpoint rows of a worker in shared memory are 16-bit; rc (a multiple of
// 8) plus this pad makes the per-worker stride an odd number of 32-bit words,
// so that lanes searching neighbouring workers start on different banks.
constexpr int R2_RHO_PAD = 2;
constexpr int NONE = 0x7fffffff;

// Row of remaining length r: the first row q whose rho_{q+1} exceeds r (row R
// is unbounded). Shared memory holds rho_{q+1} - 1 for the first rc rows; a
// worker with more rows continues in the table's global rows.
__device__ __forceinline__ int r2_find(const unsigned short* rho, int R, int rc, int r,
                                       const float4* tab, long long rowbase)
{
    const int Rs = R < rc ? R : rc;
    int lo = 0, hi = Rs;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if ((int)rho[mid] >= r) hi = mid;
        else lo = mid + 1;
    }
    if (lo == Rs && R > Rs) {
        hi = R;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (__float_as_int(tab[(rowbase + mid) * ROW_F4].x) > r) hi = mid;
            else lo = mid + 1;
        }
    }
    return lo;
}

// better() carrying the winner's "worker full" flag along.
__device__ __forceinline__ void better_f(unsigned long long& bk, int& bw, int& bf,
                                         unsigned long long ok, int ow, int of)
{
    if (ow != NONE && (bw == NONE || ok > bk || (ok == bk && ow < bw))) {
        bk = ok;
        bw = ow;
        bf = of;
    }
}

// Warp-wide best_f: the largest key, then the lowest worker index among equal
// keys (warp max/min reductions on the key's halves); every lane ends with it.
__device__ __forceinline__ void reduce_f(unsigned long long& bk, int& bw, int& bf)
{
    const bool has = bw != NONE;
    const unsigned hi = has ? (unsigned)(bk >> 32) : 0u;
    const unsigned lo = has ? (unsigned)bk : 0u;
    const unsigned mhi = __reduce_max_sync(FULL, hi);
    const unsigned mlo = __reduce_max_sync(FULL, hi == mhi ? lo : 0u);
    const bool top = has && hi == mhi && lo == mlo;
    const unsigned widx = __reduce_min_sync(FULL, top ? (unsigned)bw : 0xffffffffu);
    const unsigned who = __ballot_sync(FULL, top && (unsigned)bw == widx);
    const int of = __shfl_sync(FULL, bf, who ? __ffs(who) - 1 : 0);
    if (who) {
        bk = ((unsigned long long)mhi << 32) | mlo;
        bw = (int)widx;
        bf = of;
    } else {
        bk = 0ull;
        bw = NONE;
        bf = 0;
    }
}

}  // namespace aladdin
