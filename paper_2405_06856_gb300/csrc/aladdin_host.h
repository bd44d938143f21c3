// Host-side internals shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>

#include <atomic>

#include "aladdin_dev.cuh"

namespace aladdin {

// Default poll limits of the bounded device waits (about a second each).
constexpr long long GRID_WAIT_POLLS = 1ll << 22;  // the round's grid exchange
constexpr long long MBAR_WAIT_POLLS = 1ll << 26;  // the scoring kernel's copy barriers

// Elements per lane of the per-warp table builder for a slot capacity.
inline int lanes_per_worker(int cap) { return cap / 32; }

// Requests in CSR form on the device (worker w holds [off[w], off[w+1]) of
// the arrays; tdec nullable), packed into the cluster's slots.
struct PackSrc {
    const int32_t* off;
    const int32_t* in;
    const int32_t* gen;
    const int32_t* pred;
    const float* tdec;
};
// K2: rebuild the tables of `count` workers (all workers when list == nullptr).
// With src (list == nullptr), every worker's requests are first packed from
// src into its slots by the warp that builds its table, in the same kernel.
cudaError_t launch_build(const DevParams& P, const ClusterDev& C, const int32_t* list, int count,
                         cudaStream_t st, const PackSrc* src = nullptr);
// The banked decode slack (ClusterDev::bank) of every slot from its l_out and
// t^dec, after the host wrote the slot arrays.
cudaError_t launch_bank(const DevParams& P, const ClusterDev& C, cudaStream_t st);
// capacity_norm ranks (descending key, lowest index on ties) and rank -> worker.
cudaError_t launch_rank(const ClusterDev& C, cudaStream_t st);

// float4 words of one sorted candidate record, the scoring kernels' input
// (layout and writer: k_cand_scatter in score.cu)
constexpr int CAND_REC_F4 = 3;

struct ScoreBuffers {
    float4* sorted;        // [n_cand * CAND_REC_F4] sorted candidate records
    int32_t* hist;         // [K + 2]
    unsigned int* best;    // [n_cand]
};

// K3 pipeline: validate + derive + counting-sort candidates by predicted
// output, score every pair, finalize argbest. Device pointers only. With
// prepared, the candidates were sorted into B by launch_cand_prep already
// (its stream ordered before st by the caller). With ranked (C.order), the
// flags and margins are written in rank order: column k of a row is worker
// ranked[k] (argbest unaffected).
cudaError_t launch_score(const DevParams& P, const ClusterDev& C, int n_cand, const int32_t* in,
                         const int32_t* pred, const float* wait, uint8_t* flags, float* margin,
                         int32_t* argbest, int64_t* kv_peak, float* t_cand, const ScoreBuffers& B,
                         bool pend, cudaStream_t st, cudaEvent_t ev0 = nullptr,
                         cudaEvent_t ev1 = nullptr, bool prepared = false,
                         const int32_t* ranked = nullptr, int ld = 0);
// The candidate preparation of launch_score alone (it reads no table): the
// validated per-candidate records sorted by predicted output, and the
// argbest keys reset. W is the cluster's worker count (output row stride).
cudaError_t launch_cand_prep(const DevParams& P, int W, int n_cand, const int32_t* in,
                             const int32_t* pred, const float* wait, const ScoreBuffers& B,
                             cudaStream_t st);

// K4: one greedy round over candidates in index order.
struct RoundIO {
    // direct mode
    const int32_t* in;
    const int32_t* pred;
    const float* wait;
    int n_cand;
    int32_t* placement;
    // trace mode (fleet simulation): candidates = waiting list then arrivals
    int sim;
    const double* t_arr;
    const int32_t* tin;
    const int32_t* tpred;
    long long* wl;           // waiting list (trace indices), rewritten in place
    int* n_wait;             // device
    long long arr_begin, arr_end;
    double t_now, H;
    unsigned long long* counters;  // [0] failed, [1] placed, [2] heartbeat of the halt
    int* status;             // device: 0 ok, 1 halted at the first failure, -2 capacity
    int stop_at_fail;
    long long hb;
    // exchange buffer of the sliced round (ROUND_XBUF_BYTES), or nullptr to
    // use the single-CTA round
    void* xbuf;
    // power-of-two draws: request id of direct-mode candidate c is rid0 + c
    long long rid0;
    // trace mode: real output lengths (nullable: exact predictions), and, when
    // sim_pl is set, every candidate's placement (-1 none, -2 invalid), trace
    // index and the candidate count, for Algorithm 2 after the round
    const int32_t* treal;
    int32_t* sim_pl;
    long long* sim_tix;
    int* sim_n;
    // host routing only: never the multi-CTA (cooperative) sliced round, for
    // simulations that run side by side with others
    int single_cta;
    // direct mode: device pointer to the first candidate still to place (the
    // ones before it were placed by the incremental round), or nullptr (0)
    const int* c_first;
    // direct mode: some worker holds requests placed earlier in the open round
    int round_open;
};
constexpr int ROUND_XBUF_SMS = 1024;  // largest SM count the exchange buffer serves
constexpr size_t ROUND_XBUF_BYTES = 32 * (size_t)ROUND_XBUF_SMS + 16;
cudaError_t launch_round(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                         cudaStream_t st);
// CTAs of the best-fit round launch_round runs for W workers of cap slots
// (K the length limit): > 1 cooperative, 1 the sliced round on one CTA, 0 the
// plain single-CTA round, -1 none (a single-CTA request beyond what one CTA
// holds at 1,024 slots, or a failed device query).
int round_ctas(int W, int cap, int K, bool single_cta);

// Scratch of the incremental round (grow-only, owned by the cluster).
struct RoundIncBuffers {
    uint8_t* flags;        // [chunk][(W + 31) & ~31] rank-order flags of the round-start state
    void* rank;            // [W] 16-byte rank entries
    int* c_stop;           // one int
    ScoreBuffers score;    // candidate preparation of the pre-scoring (chunk candidates)
};
// Bytes of the incremental round's flag buffer for n_cand candidates (0: the
// incremental round does not apply and needs nothing).
size_t round_inc_flag_bytes(const DevParams& P, const ClusterDev& C, const RoundIO& io);
// K4, incremental (direct-mode best-fit rounds of one scheduling group): every
// candidate scored against the round-start state, then a single-CTA chain
// that re-scores only the workers it modified; the sliced round finishes any
// candidates left when the modified workers outgrow shared memory. *used =
// false: not applicable (trace mode, several groups, the wait test hook),
// nothing launched.
cudaError_t launch_round_inc(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                             const RoundIncBuffers& B, cudaStream_t st, bool* used);

// Attributes of the current device that launches size themselves by, read
// once per device and cached (thread-safe).
struct DevInfo {
    int device, sms, smem_optin, coop;
};
cudaError_t device_info(DevInfo* out);

// Raises Kern's dynamic shared-memory limit to the device maximum, once per
// device. The limit is a process-wide property of the kernel; at the maximum,
// launches of every size are allowed, so threads launching the kernel with
// different sizes cannot undercut one another, and later launches skip the
// driver call.
template <auto Kern>
cudaError_t allow_max_smem()
{
    static std::atomic<unsigned long long> done{0};  // one bit per device ordinal < 64
    DevInfo d;
    cudaError_t e = device_info(&d);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = d.device < 64 ? 1ull << d.device : 0ull;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(Kern, cudaFuncAttributeMaxDynamicSharedMemorySize, d.smem_optin);
    if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_acq_rel);
    return e;
}

// Resident CTAs per SM of Kern at `threads` threads and `smem` bytes of
// dynamic shared memory (whose limit is raised to `smem` for the kernel), queried
// once per device ordinal < 64 and cached (thread-safe; concurrent first
// queries compute and store the same value).
template <auto Kern>
cudaError_t kernel_occupancy(int threads, size_t smem, int* per_sm)
{
    static std::atomic<int> cache[64];  // 0: not queried on that device yet
    DevInfo d;
    cudaError_t e = device_info(&d);
    if (e != cudaSuccess) return e;
    const bool slot = d.device >= 0 && d.device < 64;
    int v = slot ? cache[d.device].load(std::memory_order_acquire) : 0;
    if (v == 0) {
        if ((e = cudaFuncSetAttribute(Kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)smem)) != cudaSuccess)
            return e;
        int ps = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&ps, Kern, threads, smem);
        if (e != cudaSuccess) return e;
        v = ps < 1 ? 1 : ps;
        if (slot) cache[d.device].store(v, std::memory_order_release);
    }
    *per_sm = v;
    return cudaSuccess;
}

// Loads every kernel the scoring path (launch_score) may launch on the
// current device and caches its launch configuration, so that later scoring
// calls on that device reach neither the module loader (which places kernel
// code in device memory on a kernel's first use) nor a device query.
cudaError_t prepare_score_kernels();

// Execution of every worker for dt ms from t_now.
// stats: device [0] prefills run, [1] finished, [2] max TTFT bits, [3] max
// ATGT bits (non-negative doubles compare like their bit patterns), realized
// violations [4] TTFT, [5] ATGT, [6] KV-overflow iterations, prediction-error
// events [7] re-predictions, [8] early finishes. halt (device, nullable):
// nothing runs when *halt != 0. fail (device, nullable): every violation is
// also added to it (the simulation's failure counter). Each worker's error
// events are added to C.le / C.be.
constexpr int STATS_N = 9;
cudaError_t launch_advance(const DevParams& P, const ClusterDev& C, double t_now, double dt,
                           unsigned long long* stats, const int* halt, cudaStream_t st,
                           unsigned long long* fail = nullptr);

// A best-fit round of a placement call under grouped scheduling (P.groups >
// 1, direct mode): one CTA per group, the groups in parallel. A group whose
// chosen worker is full stops (status -2); placements -1 / -2 as launch_round.
cudaError_t launch_round_groups(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                                cudaStream_t st);

// One round of a load-balancing policy (JSQ or power of two choices; the
// RoundIO of launch_round): each candidate goes to the policy's worker
// without a feasibility test. Tables are not rebuilt.
cudaError_t launch_round_queue(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                               cudaStream_t st);

// Algorithm 2 over one round's placements. Direct mode (io.sim == 0): the
// candidates io.in / io.pred / io.wait (io.n_cand) and io.placement (updated);
// trace mode: io.sim_pl / io.sim_tix / *io.sim_n with the trace arrays and
// io.t_now. Errors from C.le / C.be; moves (device, nullable) receives the
// number of moves and obj (device, nullable, 2 doubles) the summed distance
// before and after. Tables of the two workers of every move are rebuilt.
cudaError_t launch_rebalance(const DevParams& P, const ClusterDev& C, const RoundIO& io,
                             int* moves, double* obj, cudaStream_t st);

// Exact integer sums over a trace for the worker-configuration model:
// sums[0] = sum of predicted outputs (decode iterations), sums[1] = sum over
// requests and their iterations of the context l_in + s. Device pointers.
cudaError_t launch_trace_demand(const int32_t* in, const int32_t* pred, long long n,
                                unsigned long long* sums, cudaStream_t st);

// What another translation unit may read of a cluster (see cluster_view).
struct ClusterView {
    int device;
    cudaStream_t stream;
    DevParams dp;
    ClusterDev dev;
    bool round_open;
};

}  // namespace aladdin

struct aladdin_cluster;
namespace aladdin {
int cluster_view(aladdin_cluster* cl, ClusterView* v);
}  // namespace aladdin
