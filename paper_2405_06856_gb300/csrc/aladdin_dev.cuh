// Device-side data layout and the two primitives every kernel of the library
// shares: building one worker's projection table (one warp per worker) and
// evaluating one (candidate, worker) pair against a table row in O(1).
//
// Method (Sec. 3 and Sec. 4.2 of arxiv 2405.06856). For worker i with requests
// j (context a_j = l_in + l_out, remaining decode iterations r_j) the future
// iteration s has b(s) = #{r_j >= s} active requests holding
// K(s) = sum_{r_j >= s} (a_j + s) context tokens; its KV usage is
// h K(s) + j b(s) (Eq. kv cache) and it lasts t(s) = c3 + c2 b(s) + k2 K(s)
// (Eq. iter time). Sorting the distinct remaining lengths rho_1 < ... < rho_R
// turns both curves into segments on which b is constant: with
// n_p = #{r_j > rho_p}, A_p = sum_{r_j > rho_p} a_j,
//   K(s) = A_p + s n_p                      for rho_p < s <= rho_{p+1},
//   T(x) = sum_{s<=x} t(s) = c2 PR_p + k2 PRA_p + x (c3 + c2 n_p + k2 A_p)
//          + k2 n_p x (x + 1) / 2           for rho_p <= x <= rho_{p+1},
// where PR_p = sum_{r_j <= rho_p} r_j and
// PRA_p = sum_{r_j <= rho_p} (r_j a_j + r_j (r_j + 1) / 2) are exact integer
// prefix sums. KV grows inside a segment, so its maximum sits at a breakpoint
// (the paper's observation that a request's KV peaks just before it finishes).
//
// A candidate (prompt a, predicted output r, wait w) inserts one breakpoint.
// Every constraint of the placement test is monotone and affine in a, so each
// becomes "a <= bound" with a bound that is O(1) to evaluate from the row p of
// the segment containing r (rho_p <= r < rho_{p+1}):
//   KV (e):  a <= floor((M - j - PM_p)/h) and
//            a <= floor((M - j(n_p+1))/h) - A_p - r (n_p + 1), and no KV peak
//            after the candidate exceeds M (SM_p <= M);
//   TTFT (c): a <= (T_pre - w - off)/(s k1) - c1/k1 - P, and the same for the
//            largest wait among this round's placements;
//   ongoing (d), requests finishing with or before the candidate:
//            a <= min_{r_j <= r} (u_j - s(k1 P + c1)) / (s (k2 r_j + k1)),
//            u_j = sigma_j - s (c2 r_j + k2 r_j (r_j + 1)/2), a prefix minimum;
//            requests finishing after it:
//            a <= (min_{r_j > r} sigma_j / s - s(k1 P + c1)/s - X(r)) / (k2 r + k1),
//            X(r) = c2 r + k2 r (r + 1) / 2, a suffix minimum;
//   new requests (no stall): the same with k1 = 0 and P = 0;
//   candidate: a <= theta T_dec/(s k2) - X(r)/(k2 r) - T_u(r)/(k2 r).
// Here sigma_j = theta T_dec r_j + bank_j - T(r_j) is request j's slack before
// the candidate, s the worker's latency scale and P its pending prefill tokens.
// The pair's margin is the smallest bound minus a.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace aladdin {

constexpr unsigned FULL = 0xffffffffu;
constexpr int ROW_F4 = 2;               // float4 per table row
constexpr long long LL_NONE = (-0x7fffffffffffffffLL - 1);

struct DevParams {
    float k1, c1, k2, c2, c3;
    int32_t h, j;
    float T_pre, T_dec, gamma, theta;
    int32_t K, cap;
    int32_t approx;  // 1: the MIP's constraints (b) and (d) replace the projection
    // derived in double on the host, rounded once
    float c2_over_k2, c3_over_k2, c1_over_k1, inv_k1, theta_Tdec, thTdec_over_k2;
    // double copies for execution (advance) and exact capacity_norm keys
    double k1d, c1d, k2d, c2d, c3d, T_pred, T_decd, gammad, thetad;
    // realized latencies above these count as SLO violations (execution)
    double T_pre_viol, T_dec_viol;
    int32_t want_aux;        // 1: table builds also write the exact aggregates (AuxRow)
                             // that only the verification outputs read
    int32_t decode;          // 1: decode instance of split-phase inference (no prefill)
    int32_t policy;          // ALADDIN_POLICY_* of placement rounds
    int32_t groups;          // G > 1: request q is placed only on workers w = q (mod G)
    unsigned long long seed; // SplitMix64 seed of the power-of-two draws
    // Bounded device waits: polls before a wait gives up, sets the sticky
    // timeout bit and leaves the kernel (ALADDIN_ERR_TIMEOUT).
    long long grid_wait_limit;  // the placement round's grid exchange
    long long mbar_wait_limit;  // the scoring kernel's candidate-copy barriers
    int32_t wait_test;          // test hook, 1: the next waits run out by design (the
                                // round's exchange waits for one arrival more than its
                                // CTAs make; the scoring kernel withholds its first copy)
    int32_t round_slots_max;    // test hook (0: off): at most this many modified-worker
                                // slots in the incremental round
    int32_t round_chunk;        // test hook (0: off): at most this many candidates per
                                // chunk of the incremental round
};

// Relative slack of a realized latency over its SLO before the execution step
// counts it as a violation: the rounding of the fp32 placement test.
constexpr double SLO_TOL = 1e-5;

// Exact integer aggregates of one table row (verification outputs only).
struct __align__(16) AuxRow {
    long long PM;   // max_{m <= p} KV(rho_m) + h rho_m, LL_NONE for p = 0
    long long SM;   // max_{m > p} KV(rho_m), 0 if none
    long long A;    // sum_{r_j > rho_p} a_j
    long long PR;   // sum_{r_j <= rho_p} r_j
    long long PRA;  // sum_{r_j <= rho_p} (r_j a_j + r_j (r_j + 1) / 2)
    int32_t n;      // #{r_j > rho_p}
    int32_t rho;    // rho_p
};

struct ClusterDev {
    int32_t W, cap, rows;      // rows per worker = cap + 1
    const float* scale;        // [W] latency coefficient multiplier
    const double* scaled;      // [W] the same in double (execution)
    const int32_t* M;          // [W] KV capacity (slots)
    float* off;                // [W] ms from the round's time to the next iteration start
    double* clock;             // [W] absolute ms of the next iteration start
    int32_t* n;                // [W] requests
    int32_t* in;               // [W*cap]
    int32_t* gen;              // [W*cap]
    int32_t* pred;             // [W*cap]
    double* tdec;              // [W*cap] decode time so far (ms)
    float* bank;               // [W*cap] banked decode slack of an ongoing request,
                               // (float)(theta T_dec l_out - t^dec) in double, written
                               // wherever l_out or t^dec change (unused while pending)
    uint8_t* pend;             // [W*cap] 1: placed this round, prefill pending
    double* wait;              // [W*cap] pending: wait since arrival at placement
    float4* tab;               // [W*rows*ROW_F4] scoring rows
    float2* tab2;              // [W*rows] bounds of requests placed in an open round
    AuxRow* aux;               // [W*rows]
    int32_t* R;                // [W] breakpoints
    float4* wrec;              // [W] {1/s, ZO, ZW, rank bits}
    unsigned long long* key;   // [W] order-preserving code of capacity_norm^2 (0: unusable)
    int32_t* order;            // [W] worker at rank
    unsigned long long* rk;    // [ceil(W / 1024) * 1024] ranking scratch: keys sorted per chunk
    int32_t* ri;               // [same] their workers
    unsigned int* err;         // sticky error bits (1: invalid request)
    int32_t* ovf;              // [W] workers left to the full-capacity table build
    int* novf;                 // their count
    uint32_t* skey;            // [W*cap] (r << 10 | slot) of the requests in sorted order,
                               // written by every table build
    float2* wapx;              // [W] approximate mode: prompt bounds of (d) and of (b)
                               // before the candidate's gamma * l_pred
    int32_t* real;             // [W*cap] real output length (= pred unless a trace
                               // carries prediction errors)
    long long* le;             // [W] Algorithm 2's output-length error l^e
    int32_t* be;               // [W] Algorithm 2's batch-size error b^e
    double* err_e;             // [W] Algorithm 2's scratch: k2 l^e + c2 b^e
    const int32_t* repred;     // [K+1] re-prediction table, or nullptr (x + 1)
};

// Table row p of a worker (2 x float4, 32 bytes) and its side entry:
//  v0 = {rho_{p+1} (int bits; INT_MAX for the last row), kvB1, kvE, beta0n}
//  v1 = {beta1s, nh, pmA, Gt}
//  tab2 = {pmAp, Gpt}: only requests placed in an open round use these
// kvB1 = floor((M - j - PM_p)/h) (+inf for p = 0, -inf if SM_p > M)
// kvE  = floor((M - j (n_p + 1))/h) - A_p
// beta0n = -(c2/k2 PR_p + PRA_p); beta1s = (c3 + c2 n_p)/k2 + A_p + n_p/2 - theta T_dec/(s k2)
// nh = -n_p/2 (so -(n_p + 1) = 2 nh - 1); pmA / pmAp prefix-minimum bounds of
// ongoing / new requests with r_j <= rho_p; Gt / Gpt = suffix-minimum slack of
// ongoing / new requests with r_j > rho_p, over s, ongoing ones less the
// stall's constant part.

// Derived per-candidate values (3 x float4), identical for every worker.
// Bounds are compared with the prompt length a as headrooms bound - a; the
// candidate's decode bound carries a in Ua = U - a with U = -c2/k2 - (r + 1)/2.
struct __align__(16) CandRec {
    float a, r, inv_r, Ua;             // prompt, output, 1/r, U - a
    float inv_d1, nXd1, inv_d2, Zc;    // 1/(k2 r + k1), -X(r)/(k2 r + k1), 1/(k2 r), (T_pre - w)/k1
    int32_t ri, orig, valid, pad;
};

__device__ __forceinline__ float f_inf() { return __int_as_float(0x7f800000); }

// Banked decode slack of a request that has generated g tokens in td ms
// (Table 1's t^dec): theta T_dec g - td in double, rounded once to float.
__device__ __forceinline__ float banked_slack(const DevParams& P, int g, double td)
{
    return (float)(P.thetad * P.T_decd * (double)g - td);
}

// min(a, b, c): the three-operand form of min.f32 (sm_100 and later), the
// same value as fminf(fminf(a, b), c) in one instruction.
__device__ __forceinline__ float fmin3(float a, float b, float c)
{
    float d;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ long long floor_div_ll(long long x, long long d)
{
    if (d == 1) return x;
    long long q = x / d;
    if ((x % d != 0) && (x < 0)) q -= 1;
    return q;
}

__device__ __forceinline__ CandRec make_cand(const DevParams& P, int32_t in, int32_t pred, float w,
                                             int32_t orig)
{
    CandRec c;
    const bool ok = in >= 0 && pred >= 1 && (long long)in + pred <= (long long)P.K &&
                    w >= 0.0f && w <= 3.0e38f;
    const int32_t r = ok ? pred : 1;
    const float rf = (float)r;
    const float a = ok ? (float)in : 0.0f;
    c.a = a;
    c.r = rf;
    c.inv_r = 1.0f / rf;
    // approximate mode: a + gamma * l_pred, the candidate's share of (b)
    c.Ua = P.approx ? fmaf(P.gamma, rf, a) : (-P.c2_over_k2 - 0.5f * (rf + 1.0f)) - a;
    const float d1 = P.k2 * rf + P.k1;
    c.inv_d1 = 1.0f / d1;
    const float X = P.c2 * rf + P.k2 * (0.5f * rf * (rf + 1.0f));
    c.nXd1 = -X * c.inv_d1;
    c.inv_d2 = 1.0f / (P.k2 * rf);
    // decode instance: no TTFT test (the bound is +inf for every worker)
    c.Zc = P.decode ? f_inf() : (P.T_pre - (ok ? w : 0.0f)) * P.inv_k1;
    c.ri = ok ? r : 0;
    c.orig = orig;
    c.valid = ok ? 1 : 0;
    c.pad = 0;
    return c;
}

// Headroom of one pair per constraint group (bound - a): d[0] KV, d[1] TTFT,
// d[2] ongoing ATGT, d[3] new ATGT. The flags are the groups with d >= 0 and
// the margin is min(d).
__device__ __forceinline__ void pair_headroom(const float4 v0, const float4 v1, const float2 ext,
                                              const float4 wr, const CandRec& c, float (&d)[4])
{
    const float np1n = fmaf(2.0f, v1.y, -1.0f);
    d[0] = fminf(v0.y, fmaf(c.r, np1n, v0.z)) - c.a;
    d[1] = fminf(fmaf(c.Zc, wr.x, -wr.y), wr.z) - c.a;
    d[2] = fminf(v1.z, fmaf(v1.w, c.inv_d1, c.nXd1)) - c.a;
    d[3] = fmin3(ext.x - c.a, fmaf(ext.y, c.inv_d2, c.Ua),
                 fmaf(v0.w, c.inv_r, fmaf(v1.y, c.r, c.Ua - v1.x)));
}

// Bounds of one pair; returns the four flag bits, writes the margin.
__device__ __forceinline__ unsigned eval_pair(const float4 v0, const float4 v1, const float2 ext,
                                              const float4 wr, const CandRec& c, float& margin)
{
    float d[4];
    pair_headroom(v0, v1, ext, wr, c, d);
    margin = fmin3(fminf(d[0], d[1]), d[2], d[3]);
    return (d[0] >= 0.0f ? 1u : 0u) | (d[1] >= 0.0f ? 2u : 0u) | (d[2] >= 0.0f ? 4u : 0u) |
           (d[3] >= 0.0f ? 8u : 0u);
}

// eval_pair in either mode; wa = the worker's approximate-mode bounds.
__device__ __forceinline__ unsigned eval_pair_mode(bool approx, const float4 v0, const float4 v1,
                                                   const float2 ext, const float4 wr,
                                                   const float2 wa, const CandRec& c,
                                                   float& margin)
{
    if (!approx) return eval_pair(v0, v1, ext, wr, c, margin);
    float d[4];
    const float np1n = fmaf(2.0f, v1.y, -1.0f);
    d[0] = fminf(v0.y, fmaf(c.r, np1n, v0.z)) - c.a;
    d[1] = fminf(fmaf(c.Zc, wr.x, -wr.y), wr.z) - c.a;
    d[2] = wa.x - c.a;
    d[3] = wa.y - c.Ua;
    margin = fmin3(fminf(d[0], d[1]), d[2], d[3]);
    return (d[0] >= 0.0f ? 1u : 0u) | (d[1] >= 0.0f ? 2u : 0u) | (d[2] >= 0.0f ? 4u : 0u) |
           (d[3] >= 0.0f ? 8u : 0u);
}

// Row index p of worker w containing remaining length r: the first row whose
// rho_{p+1} exceeds r (row R has rho_{R+1} = INT_MAX).
// NC: read through the read-only path (only for tables not written by the
// running kernel).
template <bool NC = true>
__device__ __forceinline__ int find_row(const float4* tab, long long rowbase, int R, int r)
{
    int lo = 0, hi = R;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        const float* px = &tab[(rowbase + mid) * ROW_F4].x;
        const int nxt = __float_as_int(NC ? __ldg(px) : *px);
        if (nxt > r) hi = mid;
        else lo = mid + 1;
    }
    return lo;
}

// ---------------------------------------------------------------------------
// Warp-level scans over the E x 32 element layout (element x = e * 32 + lane).

template <typename T>
struct OpMin {
    __device__ __forceinline__ T operator()(T a, T b) const { return a < b ? a : b; }
};
template <typename T>
struct OpMax {
    __device__ __forceinline__ T operator()(T a, T b) const { return a > b ? a : b; }
};
template <typename T>
struct OpAdd {
    __device__ __forceinline__ T operator()(T a, T b) const { return a + b; }
};

// One value set of a fused scan: v[E] scanned over x with operator op.
// Several independent sets advance level by level together (scan_*_fused),
// so that their shuffles issue back to back instead of one latency chain per
// set; only the E row totals chain through a carry.
template <int E, typename T, typename Op>
struct ScanSet {
    static constexpr int kE = E;
    using value_type = T;
    T (&v)[E];
    Op op;
    T ident;
    T u[E], tot[E];
    T total;
    __device__ __forceinline__ ScanSet(T (&x)[E], Op o, T id) : v(x), op(o), ident(id) {}
    __device__ __forceinline__ void fetch_up(int d)
    {
#pragma unroll
        for (int e = 0; e < E; ++e) u[e] = __shfl_up_sync(FULL, v[e], d);
    }
    __device__ __forceinline__ void apply_up(int d, int lane)
    {
#pragma unroll
        for (int e = 0; e < E; ++e)
            if (lane >= d) v[e] = op(v[e], u[e]);
    }
    __device__ __forceinline__ void fetch_down(int d)
    {
#pragma unroll
        for (int e = 0; e < E; ++e) u[e] = __shfl_down_sync(FULL, v[e], d);
    }
    __device__ __forceinline__ void apply_down(int d, int lane)
    {
#pragma unroll
        for (int e = 0; e < E; ++e)
            if (lane + d < 32) v[e] = op(v[e], u[e]);
    }
    __device__ __forceinline__ void fetch_tot_prefix()
    {
#pragma unroll
        for (int e = 0; e < E; ++e) tot[e] = __shfl_sync(FULL, v[e], 31);
    }
    __device__ __forceinline__ void carry_prefix()
    {
        T carry = ident;
#pragma unroll
        for (int e = 0; e < E; ++e) {
            v[e] = op(carry, v[e]);
            carry = op(carry, tot[e]);
        }
        total = carry;
    }
    __device__ __forceinline__ void fetch_tot_suffix()
    {
#pragma unroll
        for (int e = 0; e < E; ++e) {
            tot[e] = __shfl_sync(FULL, v[e], 0);
            u[e] = __shfl_down_sync(FULL, v[e], 1);
        }
    }
    __device__ __forceinline__ void carry_suffix(int lane)
    {
        T carry = ident;
#pragma unroll
        for (int e = E - 1; e >= 0; --e) {
            const T nx = lane == 31 ? ident : u[e];
            v[e] = op(nx, carry);
            carry = op(carry, tot[e]);
        }
        total = carry;
    }
};

template <int E, typename T, typename Op>
__device__ __forceinline__ ScanSet<E, T, Op> scan_set(T (&v)[E], Op op, T ident)
{
    return ScanSet<E, T, Op>(v, op, ident);
}

// Sets are fused while the values in flight fit in registers (E <= 4);
// with more elements per lane the E chains of each set already overlap.
constexpr int FUSE_MAX_E = 4;

template <typename... S>
__device__ __forceinline__ void scan_prefix_sets(S&... s)
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        (s.fetch_up(d), ...);
        (s.apply_up(d, lane), ...);
    }
    (s.fetch_tot_prefix(), ...);
    (s.carry_prefix(), ...);
}

template <typename... S>
__device__ __forceinline__ void scan_suffix_excl_sets(S&... s)
{
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        (s.fetch_down(d), ...);
        (s.apply_down(d, lane), ...);
    }
    (s.fetch_tot_suffix(), ...);
    (s.carry_suffix(lane), ...);
}

// Inclusive prefix scans over x of every set; each set's total in .total.
template <typename S0, typename... S>
__device__ __forceinline__ void scan_prefix_fused(S0& s0, S&... s)
{
    if constexpr (S0::kE <= FUSE_MAX_E) {
        scan_prefix_sets(s0, s...);
    } else {
        scan_prefix_sets(s0);
        (scan_prefix_sets(s), ...);
    }
}

// Exclusive suffix scans over x (elements y > x) of every set; totals in .total.
template <typename S0, typename... S>
__device__ __forceinline__ void scan_suffix_excl_fused(S0& s0, S&... s)
{
    if constexpr (S0::kE <= FUSE_MAX_E) {
        scan_suffix_excl_sets(s0, s...);
    } else {
        scan_suffix_excl_sets(s0);
        (scan_suffix_excl_sets(s), ...);
    }
}

template <typename T, typename Op>
__device__ __forceinline__ T warp_reduce(T v, Op op)
{
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) v = op(v, __shfl_xor_sync(FULL, v, d));
    return v;
}

// Scratch of one table build: EW element rows per lane, NW warps per worker.
template <int EW, int NW = 1>
struct BuildSmem {
    static constexpr int N = 32 * EW * NW;
    long long kvrho[N + 1];
    int32_t a[N];
    float bank[N];
    float Tp[N + 1];
    unsigned sorted[NW > 1 ? N : 1];  // cooperative builds: merged keys
    alignas(16) unsigned runs[NW > 1 ? N : 1];  // each warp's keys (read as uint4)
    long long pll[6][NW];             // per-warp partials
    double pdm[NW];
    float pf[7][NW];
    int pi[5][NW];
    unsigned cflag;
    unsigned newk[8];                 // insertion: the appended keys
    uint8_t pend[N];
};

// Barrier of the NW warps building one table (NW consecutive warps of the
// CTA when NW > 1; a named barrier, 1 unless the caller runs two builds side
// by side, so that the other warps may run on).
template <int NW, int BAR = 1>
__device__ __forceinline__ void group_sync()
{
    if constexpr (NW == 1) {
        __syncwarp();
    } else {
        asm volatile("bar.sync %0, %1;" ::"n"(BAR), "r"(NW * 32) : "memory");
    }
}

// Lanes of the smallest power of two >= NW.
template <int NW>
constexpr int lanes_p2()
{
    return NW <= 1 ? 1 : NW <= 2 ? 2 : NW <= 4 ? 4 : NW <= 8 ? 8 : NW <= 16 ? 16 : 32;
}

// Cross-warp combination of per-warp scan totals: the carry into warp q
// (op over warps before q for a prefix, after q for a suffix) and the total.
// Lane k < NW of every warp reads warp k's partial; a shuffle scan over those
// lanes gives every lane the carries and the total (log2 NW steps, the same
// exact min / max / integer results as a sequential fold).
template <int NW, typename T, typename Op>
__device__ __forceinline__ T carry_in(const T* part, int q, bool suffix, Op op, T ident, T& all)
{
    const int lane = threadIdx.x & 31;
    T incl = lane < NW ? part[lane] : ident;
#pragma unroll
    for (int d = 1; d < lanes_p2<NW>(); d <<= 1) {
        if (!suffix) {
            const T u = __shfl_up_sync(FULL, incl, d);
            if (lane >= d) incl = op(u, incl);
        } else {
            const T u = __shfl_down_sync(FULL, incl, d);
            if (lane + d < 32) incl = op(incl, u);
        }
    }
    all = __shfl_sync(FULL, incl, suffix ? 0 : NW - 1);
    const int src = suffix ? q + 1 : q - 1;  // inclusive value of the neighbour
    const T c = __shfl_sync(FULL, incl, src >= 0 && src < NW ? src : 0);
    return src >= 0 && src < NW ? c : ident;
}

// Combination over the NW warps of a value every warp holds (lane k reads
// warp k's entry; xor reduction over the lanes).
template <int NW, typename T, typename Op>
__device__ __forceinline__ T combine_warps(const T* part, Op op, T ident)
{
    const int lane = threadIdx.x & 31;
    T v = lane < NW ? part[lane] : ident;
#pragma unroll
    for (int d = lanes_p2<NW>() / 2; d > 0; d >>= 1) v = op(v, __shfl_xor_sync(FULL, v, d));
    return __shfl_sync(FULL, v, 0);  // lanes past the reduced ones get it too
}

template <int NW, typename Set>
__device__ __forceinline__ void add_carry_prefix(Set& st, typename Set::value_type* part, int q)
{
    if constexpr (NW > 1) {
        typename Set::value_type all;
        const auto c = carry_in<NW>(part, q, false, st.op, st.ident, all);
#pragma unroll
        for (int e = 0; e < Set::kE; ++e) st.v[e] = st.op(c, st.v[e]);
        st.total = all;
    }
}

template <int NW, typename Set>
__device__ __forceinline__ void add_carry_suffix(Set& st, typename Set::value_type* part, int q)
{
    if constexpr (NW > 1) {
        typename Set::value_type all;
        const auto c = carry_in<NW>(part, q, true, st.op, st.ident, all);
#pragma unroll
        for (int e = 0; e < Set::kE; ++e) st.v[e] = st.op(st.v[e], c);
        st.total = all;
    }
}

// One table row in its stored form (see the layout above) and its exact
// integer aggregates.
struct RowVals {
    float4 v0, v1;
    float2 ext;
    AuxRow aux;
};

__device__ __forceinline__ RowVals make_row(const DevParams& P, float inv_s, int M, long long P_pend,
                                            int rho, int rho_next, int n_p, long long A,
                                            long long PR, long long PRA, long long PM, long long SM,
                                            float pmA, float pmAp, float smS, float smSp)
{
    float kvB1;
    if (SM > (long long)M) kvB1 = -f_inf();
    else if (PM == LL_NONE) kvB1 = f_inf();
    else kvB1 = (float)floor_div_ll((long long)M - P.j - PM, P.h);
    const float kvE = (float)(floor_div_ll((long long)M - (long long)P.j * (n_p + 1), P.h) - A);
    const float nf = (float)n_p;
    RowVals o;
    o.v0.x = __int_as_float(rho_next);
    o.v0.y = kvB1;
    o.v0.z = kvE;
    o.v0.w = -(P.c2_over_k2 * (float)PR + (float)PRA);
    o.v1.x = P.c3_over_k2 + P.c2_over_k2 * nf + (float)A + 0.5f * nf - P.thTdec_over_k2 * inv_s;
    o.v1.y = -0.5f * nf;
    o.v1.z = pmA;
    o.v1.w = smS * inv_s - (P.k1 * (float)P_pend + P.c1);
    o.ext = make_float2(pmAp, smSp * inv_s);
    o.aux.PM = PM;
    o.aux.SM = SM;
    o.aux.A = A;
    o.aux.PR = PR;
    o.aux.PRA = PRA;
    o.aux.n = n_p;
    o.aux.rho = rho;
    return o;
}

__device__ __forceinline__ void store_row(const ClusterDev& C, long long rowid, const RowVals& o,
                                          bool aux)
{
    float4* t = C.tab + rowid * ROW_F4;
    t[0] = o.v0;
    t[1] = o.v1;
    C.tab2[rowid] = o.ext;
    if (aux) C.aux[rowid] = o.aux;
}

// Shared-memory copies of one worker's breakpoints, record and key, kept by
// the sliced placement round (pointers to this worker's entries).
struct SliceCache {
    unsigned short* rho;  // rho_{q+1} - 1 of rows q = 0..min(R, rc)-1
    int rc;               // rows held
    int* R;
    float4* wrec;
    unsigned long long* key;
};

// Build worker w's table (rows 0..R), its record and its capacity_norm key.
// Called by all lanes of NW warps (warps W0..W0+NW-1 of the CTA when NW > 1,
// synchronised by named barrier BAR); element x = (q EW + e) 32 + lane of
// the group's warp q, so 32 EW NW slots are covered. Requests are loaded from
// the slot arrays, the first n_in of them (the worker's count when n_in < 0);
// an invalid request (in < 0, gen outside [0, pred), in + pred > K) makes the
// worker infeasible for every candidate and sets err bit 1. With `cache`, the
// worker's shared-memory copies are refreshed as well. With a valid `cand`,
// the candidate is evaluated against the new table by the lane that holds
// its row, and every lane returns its flags (else 0). EVAL: the evaluation
// only (a state that is not committed): nothing is written outside `sm`
// except the state's capacity_norm key into *key_out. INSERT: the last `ins`
// slots (1 to 3) were appended since the build that left its sorted keys in
// skey, and are inserted into that order instead of sorting afresh (ins up
// to INS_MAX). !SKEY:
// the sorted keys are left in sm.sorted for the caller to store (a caller
// that runs an evaluation of the same worker beside this build).
constexpr int INS_MAX = 5;  // appended keys an insertion build takes

template <int EW, int NW = 1, bool INSERT = false, int BAR = 1, int W0 = 0, bool EVAL = false,
          bool SKEY = true>
__device__ unsigned build_table(const DevParams& P, const ClusterDev& C, int w,
                                BuildSmem<EW, NW>& sm, const SliceCache* cache = nullptr,
                                const CandRec* cand = nullptr, int n_in = -1,
                                unsigned long long* key_out = nullptr, int ins = 1)
{
    static_assert(!INSERT || NW > 1, "the insertion path is for cooperative builds");
    constexpr int E = EW;
    constexpr int RUN = 32 * EW;  // elements per warp
    const int lane = threadIdx.x & 31;
    const int q = NW > 1 ? (int)(threadIdx.x >> 5) - W0 : 0;
    const int x0 = q * RUN;
    const long long base = (long long)w * C.cap;
    const long long rowbase = (long long)w * C.rows;
    // Independent loads first: the slot loads do not wait for n (slots below
    // the capacity lie inside the worker's slot range; those past n are
    // masked). A build may cover more elements than the capacity (padding).
    const int n = n_in >= 0 ? n_in : C.n[w];
    const float s = C.scale[w];
    const int M = C.M[w];
    const float off = C.off[w];
    const float rank_bits = C.wrec[w].w;
    constexpr bool PRELOAD = E <= FUSE_MAX_E;  // registers allow it
    constexpr int EL = PRELOAD ? E : 1;
    int l_pd[EL], l_g[EL], l_pr[EL], l_in[EL];
    float l_bk[EL];
    double l_wt[EL];
    unsigned l_sk[INSERT ? E : 1];
    if constexpr (INSERT) {
        // The previous build's sorted keys (all requests but the last `ins`,
        // which were appended since).
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int x = x0 + e * 32 + lane;
            l_sk[e] = x < C.cap ? C.skey[base + x] : 0xffffffffu;
        }
    }
    if constexpr (PRELOAD) {
#pragma unroll
        for (int e = 0; e < EL; ++e) {
            const int x = x0 + e * 32 + lane;
            const long long slot = base + x;
            l_pd[e] = 0;
            l_g[e] = l_pr[e] = l_in[e] = 0;
            l_bk[e] = 0.0f;
            l_wt[e] = 0.0;
            if (x < C.cap) {
                l_pd[e] = C.pend[slot];
                l_g[e] = C.gen[slot];
                l_pr[e] = C.pred[slot];
                l_in[e] = C.in[slot];
                l_bk[e] = C.bank[slot];
                l_wt[e] = C.wait[slot];
            }
        }
    }
    const float inv_s = 1.0f / s;

    unsigned key[E];
    long long sumP = 0, sumIn = 0, sumPred = 0;
    float wpmax = -f_inf();
    int npend = 0;
    int bad = 0;
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int i = x0 + e * 32 + lane;
        if (i < n) {
            const long long slot = base + i;
            const int pd = PRELOAD ? l_pd[e % EL] : C.pend[slot];
            const int g = pd ? 0 : (PRELOAD ? l_g[e % EL] : C.gen[slot]);
            const int pr = PRELOAD ? l_pr[e % EL] : C.pred[slot];
            const int in = PRELOAD ? l_in[e % EL] : C.in[slot];
            if (in < 0 || g < 0 || g >= pr || (long long)in + pr > (long long)P.K) bad = 1;
            int r = pr - g;
            r = r < 1 ? 1 : (r > P.K ? P.K : r);
            int a = in + g;
            a = a < 0 ? 0 : (a > P.K ? P.K : a);
            key[e] = ((unsigned)r << 10) | (unsigned)i;
            sm.a[i] = a;
            sm.pend[i] = (uint8_t)pd;
            sm.bank[i] = pd ? 0.0f : (PRELOAD ? l_bk[e % EL] : C.bank[slot]);
            sumIn += in;
            sumPred += pr;
            if (pd) {
                sumP += in;
                wpmax = fmaxf(wpmax, (float)(PRELOAD ? l_wt[e % EL] : C.wait[slot]));
                npend += 1;
            }
        } else {
            key[e] = 0xffffffffu;
        }
    }
    // Sums over the worker's requests (warp shuffles interleaved, then the
    // NW warp partials in warp order).
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
        const long long o0 = __shfl_xor_sync(FULL, sumP, d);
        const long long o1 = __shfl_xor_sync(FULL, sumIn, d);
        const long long o2 = __shfl_xor_sync(FULL, sumPred, d);
        const float o3 = __shfl_xor_sync(FULL, wpmax, d);
        const int o4 = __shfl_xor_sync(FULL, npend, d);
        sumP += o0;
        sumIn += o1;
        sumPred += o2;
        wpmax = wpmax > o3 ? wpmax : o3;
        npend += o4;
    }
    bad = __any_sync(FULL, bad);
    if constexpr (NW > 1) {
        if (lane == 0) {
            sm.pll[0][q] = sumP;
            sm.pll[1][q] = sumIn;
            sm.pll[2][q] = sumPred;
            sm.pf[0][q] = wpmax;
            sm.pi[0][q] = npend;
            sm.pi[1][q] = bad;
        }
    }
    group_sync<NW, BAR>();
    if constexpr (NW > 1) {
        sumP = combine_warps<NW>(sm.pll[0], OpAdd<long long>(), 0LL);
        sumIn = combine_warps<NW>(sm.pll[1], OpAdd<long long>(), 0LL);
        sumPred = combine_warps<NW>(sm.pll[2], OpAdd<long long>(), 0LL);
        wpmax = combine_warps<NW>(sm.pf[0], OpMax<float>(), -f_inf());
        npend = combine_warps<NW>(sm.pi[0], OpAdd<int>(), 0);
        bad = combine_warps<NW>(sm.pi[1], OpMax<int>(), 0);
    }
    // Approximate mode: prompt bounds of (d) (stall within the smallest
    // theta-scaled saved decode time) and of (b) (weighted context within
    // theta * l_d(n + 1), Eq. input limit), in fp64, rounded once.
    float2 wa = make_float2(0.0f, 0.0f);
    if (P.approx) {
        double dmin = __longlong_as_double(0x7ff0000000000000ll);  // +inf: nothing decoding
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int i = x0 + e * 32 + lane;
            if (i < n) {  // reloaded: the preloaded registers stay short-lived
                const long long slot = base + i;
                if (!C.pend[slot])  // decode time saved so far, theta-scaled
                    dmin = fmin(dmin, P.thetad * (P.T_decd * (double)C.gen[slot] - C.tdec[slot]));
            }
        }
#pragma unroll
        for (int d = 16; d > 0; d >>= 1) dmin = fmin(dmin, __shfl_xor_sync(FULL, dmin, d));
        if constexpr (NW > 1) {
            if (lane == 0) sm.pdm[q] = dmin;
            group_sync<NW, BAR>();
            dmin = combine_warps<NW>(sm.pdm, OpMin<double>(), dmin);
        }
        const double s_d = C.scaled[w];
        if (P.decode) {
            wa.x = f_inf();  // no prefill, no stall: (d) is vacuous
        } else {
            const double tau0 = s_d * (P.k1d * (double)sumP + P.c1d);
            wa.x = (float)((dmin - tau0) / (s_d * P.k1d));
        }
        const double ld = (P.T_decd / s_d - P.c3d - P.c2d * (double)(n + 1)) / P.k2d;
        wa.y = (float)(P.thetad * ld - ((double)sumIn + P.gammad * (double)sumPred));
    }

    // capacity_norm key (one lane; code 0 is kept for a worker holding an
    // invalid request): capacity_norm^2 is exact (integer and half-integer
    // terms below 2^53) and non-negative doubles order like their bit
    // patterns; with gamma = 1/2 the same order comes from integers.
    // Row 0, the record and the key are written by the last lane of the last
    // warp, which holds the highest elements (often padding) and so has the
    // fewest rows of its own to write.
    const bool row0_lane = q == NW - 1 && lane == 31;
    unsigned long long kq = 0ull;
    if (row0_lane && !bad) {
        if (P.gammad == 0.5) {
            // 4 capacity_norm^2 = (2B)^2 + (2 sum in + sum pred)^2 in integers
            // (the same order and ties as the exact double value)
            const unsigned long long b2 = 2ull * (unsigned long long)n;
            const unsigned long long s2 = 2ull * (unsigned long long)sumIn + (unsigned long long)sumPred;
            kq = b2 * b2 + s2 * s2 + 1ull;
        } else {
            const double kB = (double)n;
            const double kL = __dadd_rn((double)sumIn, __dmul_rn(P.gammad, (double)sumPred));
            const double kQ = __dadd_rn(__dmul_rn(kB, kB), __dmul_rn(kL, kL));
            kq = (unsigned long long)__double_as_longlong(kQ) + 1ull;
        }
    }

    constexpr int N = BuildSmem<EW, NW>::N;
    // Cooperative builds of up to 256 slots rank every key by counting the
    // keys below it (keys of valid requests are distinct); larger ones sort
    // each warp's run and merge the runs.
    constexpr bool COUNT_RANK = NW > 1 && N <= 256 && !INSERT;
    if constexpr (INSERT) {
        // Insert the appended requests' keys into the previous sorted order
        // (keys are distinct): a new key lands after the old and new keys
        // below it, an old key moves up by the new keys below it.
        const int n0 = n - ins;  // keys of the previous order
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int x = x0 + e * 32 + lane;
            if (x < n0) sm.runs[x] = l_sk[e];
            if (x >= n0 && x < n) sm.newk[x - n0] = key[e];
        }
        group_sync<NW, BAR>();
        unsigned nk[INS_MAX];
        int pos[INS_MAX];
#pragma unroll
        for (int j = 0; j < INS_MAX; ++j) {
            nk[j] = j < ins ? sm.newk[j] : 0xffffffffu;
            pos[j] = 0;
        }
#pragma unroll
        for (int j = 0; j < INS_MAX; ++j) {
            if (j >= ins) break;  // uniform
            int lo;  // old keys below nk[j]
            if constexpr (E == 1) {
                // one key a thread: a barrier reduction over the group
                const unsigned below = (x0 + lane < n0 && l_sk[0] < nk[j]) ? 1u : 0u;
                unsigned cnt;
                asm volatile("{\n .reg .pred p;\n setp.ne.u32 p, %2, 0;\n"
                             " bar.red.popc.u32 %0, %3, %1, p;\n}"
                             : "=r"(cnt)
                             : "r"(NW * 32), "r"(below), "n"(BAR)
                             : "memory");
                lo = (int)cnt;
            } else {
                int hi = n0;
                lo = 0;
                while (lo < hi) {
                    const int mid = (lo + hi) >> 1;
                    if (sm.runs[mid] < nk[j]) lo = mid + 1;
                    else hi = mid;
                }
            }
            pos[j] = lo;
#pragma unroll
            for (int j2 = 0; j2 < INS_MAX; ++j2) pos[j] += (j2 < ins && nk[j2] < nk[j]) ? 1 : 0;
        }
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int x = x0 + e * 32 + lane;
            if (x < n0) {
                const unsigned k = l_sk[e];
                int sh = 0;
#pragma unroll
                for (int j = 0; j < INS_MAX; ++j) sh += (j < ins && nk[j] < k) ? 1 : 0;
                sm.sorted[x + sh] = k;
            }
        }
        if (q == 0 && lane < ins) {
#pragma unroll
            for (int j = 0; j < INS_MAX; ++j)
                if (j == lane) sm.sorted[pos[j]] = nk[j];
        }
        group_sync<NW, BAR>();
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int x = x0 + e * 32 + lane;
            key[e] = x < n ? sm.sorted[x] : 0xffffffffu;
        }
    }
    if constexpr (COUNT_RANK) {
#pragma unroll
        for (int e = 0; e < E; ++e) sm.runs[x0 + e * 32 + lane] = key[e];
        group_sync<NW, BAR>();
        int rank[E];
#pragma unroll
        for (int e = 0; e < E; ++e) rank[e] = 0;
        const uint4* run4 = reinterpret_cast<const uint4*>(sm.runs);
#pragma unroll 8
        for (int k = 0; k < N / 4; ++k) {
            const uint4 v = run4[k];
#pragma unroll
            for (int e = 0; e < E; ++e)
                rank[e] += (v.x < key[e]) + (v.y < key[e]) + (v.z < key[e]) + (v.w < key[e]);
        }
#pragma unroll
        for (int e = 0; e < E; ++e)
            if (x0 + e * 32 + lane < n) sm.sorted[rank[e]] = key[e];
        group_sync<NW, BAR>();
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int x = x0 + e * 32 + lane;
            key[e] = x < n ? sm.sorted[x] : 0xffffffffu;
        }
    }
    // Bitonic sort of (r, slot) keys, ascending, within each warp's run.
#pragma unroll
    for (int k = 2; k <= (COUNT_RANK || INSERT ? 1 : RUN); k <<= 1) {
#pragma unroll
        for (int jj = k >> 1; jj > 0; jj >>= 1) {
            if (jj >= 32) {
                const int je = jj >> 5;
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    if ((e & je) == 0) {
                        const int e2 = e | je;
                        const bool asc = ((e * 32 + lane) & k) == 0;
                        const unsigned lo = min(key[e], key[e2]);
                        const unsigned hi = max(key[e], key[e2]);
                        key[e] = asc ? lo : hi;
                        key[e2] = asc ? hi : lo;
                    }
                }
            } else {
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    const bool asc = ((e * 32 + lane) & k) == 0;
                    const unsigned v = __shfl_xor_sync(FULL, key[e], jj);
                    const bool lower = (lane & jj) == 0;
                    key[e] = (asc == lower) ? min(key[e], v) : max(key[e], v);
                }
            }
        }
    }
    if constexpr (NW > 1 && !COUNT_RANK && !INSERT) {
        // Merge the NW sorted runs: a key's rank is its position in its run
        // plus the keys of the other runs before it (equal padding keys of
        // earlier runs first).
#pragma unroll
        for (int e = 0; e < E; ++e) sm.runs[x0 + e * 32 + lane] = key[e];
        group_sync<NW, BAR>();
#pragma unroll
        for (int e = 0; e < E; ++e) {
            // In every other run, the count of keys before this one: a
            // fixed-step search, the NW searches advancing together.
            int cnt[NW];
#pragma unroll
            for (int q2 = 0; q2 < NW; ++q2) cnt[q2] = 0;
#pragma unroll
            for (int st = RUN; st >= 1; st >>= 1) {
#pragma unroll
                for (int q2 = 0; q2 < NW; ++q2) {
                    const int probe = cnt[q2] + st;
                    if (probe <= RUN) {
                        const unsigned v = sm.runs[q2 * RUN + probe - 1];
                        if (q2 < q ? v <= key[e] : v < key[e]) cnt[q2] = probe;
                    }
                }
            }
            int rank = e * 32 + lane;
#pragma unroll
            for (int q2 = 0; q2 < NW; ++q2)
                if (q2 != q) rank += cnt[q2];
            sm.sorted[rank] = key[e];
        }
        group_sync<NW, BAR>();
#pragma unroll
        for (int e = 0; e < E; ++e) key[e] = sm.sorted[x0 + e * 32 + lane];
    }

    int r[E], a[E], pd[E];
    float bank[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int x = x0 + e * 32 + lane;
        if (x < n) {
            r[e] = (int)(key[e] >> 10);
            const int i = (int)(key[e] & 1023u);
            a[e] = sm.a[i];
            pd[e] = sm.pend[i];
            bank[e] = sm.bank[i];
        } else {
            r[e] = 0x7fffffff;
            a[e] = 0;
            pd[e] = 0;
            bank[e] = 0.0f;
        }
    }
    // The sorted order, kept for the next build's insertion.
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int x = x0 + e * 32 + lane;
        if (!EVAL && SKEY && x < n) C.skey[base + x] = key[e];
    }
    // Neighbours in sorted order.
    int rnext[E], first[E], last[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int x = x0 + e * 32 + lane;
        int nx, pv;
        if constexpr (NW > 1) {
            nx = x + 1 < n ? (int)(sm.sorted[x + 1] >> 10) : -1;
            pv = x > 0 && x - 1 < n ? (int)(sm.sorted[x - 1] >> 10) : -1;
        } else {
            const int dn = __shfl_down_sync(FULL, r[e], 1);
            const int up = __shfl_up_sync(FULL, r[e], 1);
            int wrap_n = -1, wrap_p = -1;
            if (e + 1 < E) wrap_n = __shfl_sync(FULL, r[e + 1 < E ? e + 1 : e], 0);
            if (e > 0) wrap_p = __shfl_sync(FULL, r[e > 0 ? e - 1 : e], 31);
            nx = lane < 31 ? dn : wrap_n;
            pv = lane > 0 ? up : wrap_p;
        }
        const bool valid = x < n;
        rnext[e] = nx;
        first[e] = valid && (x == 0 || pv != r[e]);
        last[e] = valid && (x == n - 1 || nx != r[e]);
    }
    int r0;
    if constexpr (NW > 1) r0 = n > 0 ? (int)(sm.sorted[0] >> 10) : 0x7fffffff;
    else r0 = __shfl_sync(FULL, r[0], 0);
    // Prefix sums over the sorted order.
    // (r and a are at most K <= 65536 and a table holds at most 1,024
    // requests, so their sums fit 32 bits; the r a sums need 64)
    int rowid[E];
    int pre_r[E], pre_a[E];
    long long pre_ra[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const bool valid = x0 + e * 32 + lane < n;
        rowid[e] = first[e];
        const long long rr = valid ? (long long)r[e] : 0;
        const long long aa = valid ? (long long)a[e] : 0;
        pre_r[e] = (int)rr;
        pre_ra[e] = rr * aa + rr * (rr + 1) / 2;
        pre_a[e] = (int)aa;
    }
    auto s_row = scan_set(rowid, OpAdd<int>(), 0);
    auto s_r = scan_set(pre_r, OpAdd<int>(), 0);
    auto s_ra = scan_set(pre_ra, OpAdd<long long>(), 0LL);
    auto s_a = scan_set(pre_a, OpAdd<int>(), 0);
    scan_prefix_fused(s_row, s_r, s_ra, s_a);
    if constexpr (NW > 1) {
        if (lane == 0) {
            sm.pi[2][q] = s_row.total;
            sm.pi[3][q] = s_r.total;
            sm.pll[4][q] = s_ra.total;
            sm.pi[4][q] = s_a.total;
        }
        group_sync<NW, BAR>();
        add_carry_prefix<NW>(s_row, sm.pi[2], q);
        add_carry_prefix<NW>(s_r, sm.pi[3], q);
        add_carry_prefix<NW>(s_ra, sm.pll[4], q);
        add_carry_prefix<NW>(s_a, sm.pi[4], q);
    }
    const int R = s_row.total;
    const long long tot_a = s_a.total;

    // Per-breakpoint KV and cumulative decode time.
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int x = x0 + e * 32 + lane;
        if (first[e]) {
            const long long b_at = n - x;
            const long long Kat = tot_a - (pre_a[e] - a[e]) + (long long)r[e] * b_at;
            sm.kvrho[rowid[e]] = (long long)P.h * Kat + (long long)P.j * b_at;
        }
        if (last[e]) {
            const long long np = n - (x + 1);
            const long long rr = r[e];
            const long long A = tot_a - pre_a[e];
            const long long Sb = pre_r[e] + rr * np;
            const long long SK = pre_ra[e] + np * (rr * (rr + 1) / 2) + rr * A;
            sm.Tp[rowid[e]] = s * (P.c3 * (float)rr + P.c2 * (float)Sb + P.k2 * (float)SK);
        }
    }
    group_sync<NW, BAR>();

    // Per-request bounds and slacks.
    const float stall0 = s * (P.k1 * (float)sumP + P.c1);
    float pmA[E], pmAp[E], smS[E], smSp[E];
    long long PMx[E], SMx[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int x = x0 + e * 32 + lane;
        const bool valid = x < n;
        pmA[e] = f_inf();
        pmAp[e] = f_inf();
        smS[e] = f_inf();
        smSp[e] = f_inf();
        PMx[e] = LL_NONE;
        SMx[e] = LL_NONE;
        if (valid) {
            const float rf = (float)r[e];
            const float Tj = sm.Tp[rowid[e]];
            const float sigma = P.theta_Tdec * rf + bank[e] - Tj;
            const float u = sigma - s * (P.c2 * rf + P.k2 * (0.5f * rf * (rf + 1.0f)));
            if (pd[e]) {
                pmAp[e] = u / (s * P.k2 * rf);
                smSp[e] = sigma;
            } else {
                pmA[e] = (u - stall0) / (s * (P.k2 * rf + P.k1));
                smS[e] = sigma;
            }
        }
        if (last[e]) {
            const long long kv = sm.kvrho[rowid[e]];
            PMx[e] = kv + (long long)P.h * r[e];
            SMx[e] = kv;
        }
    }
    auto s_pmA = scan_set(pmA, OpMin<float>(), f_inf());
    auto s_pmAp = scan_set(pmAp, OpMin<float>(), f_inf());
    auto s_PM = scan_set(PMx, OpMax<long long>(), LL_NONE);
    auto s_smS = scan_set(smS, OpMin<float>(), f_inf());
    auto s_smSp = scan_set(smSp, OpMin<float>(), f_inf());
    auto s_SM = scan_set(SMx, OpMax<long long>(), LL_NONE);
    scan_prefix_fused(s_pmA, s_pmAp, s_PM);
    scan_suffix_excl_fused(s_smS, s_smSp, s_SM);
    if constexpr (NW > 1) {
        if (lane == 0) {
            sm.pf[1][q] = s_pmA.total;
            sm.pf[2][q] = s_pmAp.total;
            sm.pll[0][q] = s_PM.total;  // the request sums were consumed above
            sm.pf[3][q] = s_smS.total;
            sm.pf[4][q] = s_smSp.total;
            sm.pll[1][q] = s_SM.total;
        }
        group_sync<NW, BAR>();
        add_carry_prefix<NW>(s_pmA, sm.pf[1], q);
        add_carry_prefix<NW>(s_pmAp, sm.pf[2], q);
        add_carry_prefix<NW>(s_PM, sm.pll[0], q);
        add_carry_suffix<NW>(s_smS, sm.pf[3], q);
        add_carry_suffix<NW>(s_smSp, sm.pf[4], q);
        add_carry_suffix<NW>(s_SM, sm.pll[1], q);
    }
    const float smS0 = s_smS.total;
    const float smSp0 = s_smSp.total;
    const long long SM0 = s_SM.total;

    // Worker record (every lane; the first lane stores it).
    float4 wr;
    wr.x = inv_s;
    // TTFT bounds (the candidate's Zc is +inf on a decode instance, and so is
    // its bound Zc / s - wr.y)
    wr.y = P.decode ? 0.0f : off * inv_s * P.inv_k1 + P.c1_over_k1 + (float)sumP;
    wr.z = (npend > 0 && !P.decode)
               ? (P.T_pre - wpmax - off) * inv_s * P.inv_k1 - P.c1_over_k1 - (float)sumP
               : f_inf();
    wr.w = rank_bits;
    const bool want = cand != nullptr && cand->valid;
    const int rc = want ? cand->ri : 0;
    unsigned cf = 0;
    bool mine = false;

    if (!bad) {
#pragma unroll
        for (int e = 0; e < E; ++e) {
            const int xe = x0 + e * 32 + lane;
            const int nxe = (xe == n - 1) ? 0x7fffffff : rnext[e];
            // an evaluation build forms only the candidate's row
            if (last[e] && (!EVAL || (want && r[e] <= rc && rc < nxe))) {
                const int x = xe;
                const int np = n - (x + 1);
                const long long A = tot_a - pre_a[e];
                const int nxt = nxe;
                const long long SM = SMx[e] == LL_NONE ? 0 : SMx[e];
                const RowVals o = make_row(P, inv_s, M, sumP, r[e], nxt, np, A, pre_r[e], pre_ra[e],
                                           PMx[e], SM, pmA[e], pmAp[e], smS[e], smSp[e]);
                if constexpr (!EVAL) store_row(C, rowbase + rowid[e], o, P.want_aux != 0);
                if (cache && rowid[e] < R && rowid[e] < cache->rc)
                    cache->rho[rowid[e]] = (unsigned short)(nxt - 1);
                if (want && r[e] <= rc && rc < nxt) {
                    float m;
                    cf = eval_pair_mode(P.approx, o.v0, o.v1, o.ext, wr, wa, *cand, m);
                    mine = true;
                }
            }
        }
    }
    if (row0_lane && (!EVAL || (want && (bad || n == 0 || rc < r0)))) {
        RowVals o;
        if (!bad) {
            o = make_row(P, inv_s, M, sumP, 0, n > 0 ? r0 : 0x7fffffff, n, tot_a, 0, 0, LL_NONE,
                         SM0 == LL_NONE ? 0 : SM0, f_inf(), f_inf(), smS0, smSp0);
            if constexpr (!EVAL) C.R[w] = R;
        } else {
            // An invalid request: no candidate fits this worker.
            o = make_row(P, inv_s, M, 0, 0, 0x7fffffff, 0, 0, 0, 0, LL_NONE, (long long)M + 1,
                         f_inf(), f_inf(), f_inf(), f_inf());
            if constexpr (!EVAL) {
                C.R[w] = 0;
                atomicOr(C.err, 1u);
            }
        }
        if constexpr (!EVAL) store_row(C, rowbase, o, P.want_aux != 0);
        if (want && (bad || n == 0 || rc < r0)) {
            float m;
            cf = eval_pair_mode(P.approx, o.v0, o.v1, o.ext, wr, wa, *cand, m);
            mine = true;
        }
        if constexpr (!EVAL) {
            C.wrec[w] = wr;
            if (P.approx) C.wapx[w] = wa;
            C.key[w] = kq;
        }
        if (cache) {
            if (!bad && n > 0 && R > 0) cache->rho[0] = (unsigned short)(r0 - 1);
            *cache->R = bad ? 0 : R;
            *cache->wrec = wr;
            *cache->key = kq;
        }
    }
    if constexpr (EVAL) {
        if (row0_lane && key_out) *key_out = kq;
    }
    if constexpr (NW > 1) {
        if (mine) sm.cflag = cf;  // exactly one lane of the group holds the row
        group_sync<NW, BAR>();
        return want ? sm.cflag : 0u;
    } else {
        __syncwarp();
        if (!want) return 0u;
        const unsigned who = __ballot_sync(FULL, mine);
        return __shfl_sync(FULL, cf, who ? __ffs(who) - 1 : 0);
    }
}

// build_table with the fewest elements per lane that cover the worker's n
// requests (a table of 1,024 slots holding 300 requests sorts and scans 512
// elements, not 1,024). smem holds a BuildSmem<EWMAX, NW>; the smaller
// variants use a prefix of it. n is the worker's current count (uniform over
// the NW warps).
template <int EWMAX, int NW, bool INSERT = false, int BAR = 1, int W0 = 0, bool EVAL = false,
          bool SKEY = true>
__device__ __forceinline__ unsigned build_table_fit(const DevParams& P, const ClusterDev& C, int w,
                                                    int n, unsigned char* smem,
                                                    const SliceCache* cache = nullptr,
                                                    const CandRec* cand = nullptr,
                                                    unsigned long long* key_out = nullptr,
                                                    int ins = 1)
{
    // an evaluation build is given its count (beyond the worker's own)
    const int n_in = EVAL ? n : -1;
    if constexpr (EWMAX >= 4) {
        if (n > 64 * NW)  // more than the EW = 2 variant covers
            return build_table<4, NW, INSERT, BAR, W0, EVAL, SKEY>(
                P, C, w, *reinterpret_cast<BuildSmem<4, NW>*>(smem), cache, cand, n_in, key_out,
                ins);
    }
    if constexpr (EWMAX >= 2) {
        if (n > 32 * NW)
            return build_table<2, NW, INSERT, BAR, W0, EVAL, SKEY>(
                P, C, w, *reinterpret_cast<BuildSmem<2, NW>*>(smem), cache, cand, n_in, key_out,
                ins);
    }
    return build_table<1, NW, INSERT, BAR, W0, EVAL, SKEY>(
        P, C, w, *reinterpret_cast<BuildSmem<1, NW>*>(smem), cache, cand, n_in, key_out, ins);
}

}  // namespace aladdin
