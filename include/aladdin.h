/*
 * aladdin.h - C ABI of the GB300 scheduler hot path of Aladdin
 * ("Aladdin: Joint Placement and Scaling for SLO-Aware LLM Serving",
 * arxiv 2405.06856).
 *
 * The library scores candidate queries against serving workers (Sec. 4.2:
 * constraints (c), (d), (e) with the paper's KV, prefill and decode models of
 * Sec. 3), places them greedily with the best-fit heuristic (Algorithm 1) and
 * searches the minimum number of workers per worker configuration (Sec. 4.1,
 * Sec. 6.4). Every computation runs in CUDA kernels on the current GPU; there
 * is no CPU fallback.
 *
 * Conventions
 *  - Lengths are int32 token counts, times are milliseconds.
 *  - Pointer arguments may point to host memory or to device memory of the
 *    cluster's GPU; the library inspects each pointer. Page-locked host memory
 *    that the GPU can address (cudaHostAlloc, cudaHostRegister, torch
 *    pin_memory) is read and written in place by the kernels, like device
 *    memory; pageable host memory is staged through device buffers. With
 *    device pointers only, a call is asynchronous on the cluster's stream;
 *    when any argument is in host memory the call returns after the stream
 *    has completed.
 *  - The caller owns every buffer it passes; the library never frees caller
 *    memory and keeps no pointer to it after the call returns.
 *  - Pair outputs are row-major [candidate][worker].
 *  - Every function returns ALADDIN_OK (0) or a negative error code; nothing
 *    else crosses the ABI. Results are deterministic: the same inputs give the
 *    same bytes.
 */
#ifndef ALADDIN_H
#define ALADDIN_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ALADDIN_OK 0
#define ALADDIN_ERR_ARG (-1)      /* null pointer, bad size, length or coefficient */
#define ALADDIN_ERR_CAPACITY (-2) /* a worker would exceed its request slots b_cap */
#define ALADDIN_ERR_CUDA (-3)     /* a CUDA runtime call failed */
#define ALADDIN_ERR_TIMEOUT (-4)  /* a bounded device-side wait expired */
#define ALADDIN_ERR_NOMEM (-5)    /* device or host allocation failed */
#define ALADDIN_ERR_STATE (-6)    /* the cluster holds an invalid request (see
                                     aladdin_cluster_load) */
#define ALADDIN_ERR_SCRATCH (-7)  /* more candidates than aladdin_score_noalloc's
                                     fixed scratch holds */

/* Pair flags (one byte per (candidate, worker)). */
#define ALADDIN_FLAG_KV 1u        /* (e): KV usage stays within capacity every iteration */
#define ALADDIN_FLAG_TTFT 2u      /* (c): candidate and this round's placements meet T_pre */
#define ALADDIN_FLAG_ONGOING 4u   /* (d): requests decoding at round start absorb the stall */
#define ALADDIN_FLAG_NEW 8u       /* candidate and this round's placements meet T_dec */
#define ALADDIN_FEASIBLE 15u      /* all four */
#define ALADDIN_FLAG_INVALID 128u /* the candidate itself is invalid (see aladdin_score) */

#define ALADDIN_NONE (-1)         /* argbest / placement: no feasible worker */
#define ALADDIN_INVALID (-2)      /* argbest / placement: the candidate is invalid */

/* Decode-SLO constraints of a placement (the flag bits 4 and 8):
 *   EXACT   every request's remaining decode projected iteration by iteration
 *           with the candidate added (the stall of this round's prefill
 *           charged to the requests decoding at round start);
 *   APPROX  the placement MIP's own constraints (Sec. 4.2): bit 4 is (d), the
 *           stall within theta * min_j (T_dec * l_out_j - t_dec_j) over the
 *           requests decoding at round start; bit 8 is (b), sum over the
 *           worker's requests and the candidate of (l_in + gamma * l_pred)
 *           within theta * l_d(B) with Eq. input limit l_d(b) = (T_dec /
 *           lat_scale - c3 - c2 b) / k2 and B the requests with the candidate.
 * KV (bit 1) and TTFT (bit 2) are the same in both modes. */
#define ALADDIN_MODE_EXACT 0
#define ALADDIN_MODE_APPROX 1

/* Serving setting of the workers (Sec. 5.1):
 *   MIXED   default continuous batching: prefill and decode on the same
 *           worker; a round's prefill stalls the worker's decoding requests.
 *   DECODE  split-phase inference: the workers are decode instances and a
 *           request arrives with its prompt processed by a prefill instance
 *           (its prompt's KV cache comes with it). No prefill runs on the
 *           worker, so nothing is stalled (tau = 0 in (d) and in the exact
 *           projection) and TTFT (c) is not tested: flag bit 2 is always set
 *           and (d) of the approximate mode is vacuous (bit 4 set). In the
 *           simulation a request that no worker takes at the first heartbeat
 *           after its arrival fails (nothing absorbs a wait). */
#define ALADDIN_PHASE_MIXED 0
#define ALADDIN_PHASE_DECODE 1

/* Placement policy of aladdin_place_round, aladdin_simulate and
 * aladdin_min_workers (Sec. 6.1 baselines, Sec. 6.4); scoring is the same
 * under every policy.
 *   BESTFIT  Algorithm 1: the feasible worker of largest capacity_norm.
 *   JSQ      join the shortest queue: the worker holding the fewest requests,
 *            lowest index on ties, without a feasibility test.
 *   PO2      power of two choices: two workers drawn uniformly at random, the
 *            one holding fewer requests (the first drawn on ties), without a
 *            feasibility test. Draw k (0, 1) of request id q is output
 *            2 q + k + 1 of the SplitMix64 stream seeded with params.seed
 *            (Steele, Lea, Flood, OOPSLA 2014), mapped to a worker as
 *            (upper 32 bits x W) >> 32. Request ids are trace indices in the
 *            simulation and, in aladdin_place_round, the count of candidates
 *            the cluster was given in earlier rounds plus the index in the
 *            call. */
#define ALADDIN_POLICY_BESTFIT 0
#define ALADDIN_POLICY_JSQ 1
#define ALADDIN_POLICY_PO2 2

/* Performance models and SLOs (Sec. 3, Sec. 4.2).
 *   prefill iteration (Eq. prefill iter time): t_pre = k1 * sum(l_in) + c1
 *   decode iteration  (Eq. iter time):         t_d = k2 * sum(context) + c2 * b + c3
 *   KV usage          (Eq. kv cache):          kv = h * (l_in + l_out) + j
 * Requirements: k1, k2 > 0; c1, c2, c3 >= 0; h >= 1; j >= 0; T_pre > 0;
 * T_dec > c3 (Eq. input limit); 0 < theta <= 1; gamma >= 0; 2 <= K <= 65536;
 * b_cap a power of two in [32, 1024]; mode, phase and policy one of the
 * values above; rebalance 0 or 1; 0 <= groups <= 65536. Request ids (for the
 * power-of-two draws and the groups) are trace indices in the simulation and
 * the running candidate count in aladdin_place_round; aladdin_rebalance uses
 * the ids of the latest aladdin_place_round. */
typedef struct aladdin_params {
    double k1, c1;       /* prefill: ms per input token, ms */
    double k2, c2, c3;   /* decode: ms per context token, ms per request, ms */
    int32_t h, j;        /* KV slots per context token, per request */
    double T_pre;        /* TTFT SLO (ms) */
    double T_dec;        /* average token generation time SLO (ms per token) */
    double gamma;        /* capacity_norm weight of predicted output (Sec. 4.2) */
    double theta;        /* SLO scaling knob of (b), (d) */
    int32_t K;           /* sequence limit: l_in + l_pred <= K for every request */
    int32_t b_cap;       /* request slots per worker (ongoing + this round's) */
    int32_t mode;        /* ALADDIN_MODE_EXACT or ALADDIN_MODE_APPROX */
    int32_t phase;       /* ALADDIN_PHASE_MIXED or ALADDIN_PHASE_DECODE */
    int32_t policy;      /* ALADDIN_POLICY_BESTFIT, _JSQ or _PO2 */
    uint64_t seed;       /* SplitMix64 seed of the power-of-two draws */
    int32_t rebalance;   /* 1: Algorithm 2 after every best-fit round of a simulation
                            (see aladdin_rebalance); 0: off */
    int32_t groups;      /* distributed grouped scheduling (Appendix A): G > 1 groups,
                            request id q in group q mod G placed only on workers
                            w = g (mod G); 0 or 1: one central scheduler */
} aladdin_params;

/* One worker configuration (Sec. 4.1): GPUs per worker, KV capacity in KV
 * slots (< 2^24), and a multiplier applied to every latency coefficient. */
typedef struct aladdin_worker_cfg {
    int32_t gpus;
    int64_t kv_capacity;
    double lat_scale;
} aladdin_worker_cfg;

typedef struct aladdin_cluster aladdin_cluster;

/* Create a cluster of n_workers workers on the current CUDA device, bound to
 * cuda_stream (a cudaStream_t; NULL = the legacy default stream).
 * Worker w's ongoing requests (Table 1: l_in, l_out generated so far, l_pred)
 * are [req_off[w], req_off[w+1]) of in / gen / pred; req_off has
 * n_workers + 1 entries. tdec_ms (nullable) gives each request's decode time
 * so far (Table 1: t^dec); when NULL every request is taken to have used
 * exactly its theta-scaled budget so far. Each request needs in >= 0,
 * 0 <= gen < pred and in + pred <= K; each worker at most b_cap requests.
 * Errors: ALADDIN_ERR_ARG, ALADDIN_ERR_CAPACITY, ALADDIN_ERR_NOMEM,
 * ALADDIN_ERR_CUDA. On error *out is NULL. */
int aladdin_cluster_create(const aladdin_params* params, int32_t n_workers,
                           const aladdin_worker_cfg* cfg, const int32_t* req_off,
                           const int32_t* in, const int32_t* gen, const int32_t* pred,
                           const float* tdec_ms, void* cuda_stream, aladdin_cluster** out);

int aladdin_cluster_destroy(aladdin_cluster* cl);

/* Replace every worker's requests (same layout as aladdin_cluster_create) and
 * rebuild the per-worker projection tables: packing into device slots, sorting
 * of remaining lengths, breakpoints, prefix sums, KV and latency curves at the
 * breakpoints and the capacity_norm ranking (Sec. 4.2). Pageable host inputs
 * are validated on the host before upload (ALADDIN_ERR_ARG /
 * ALADDIN_ERR_CAPACITY). Device and page-locked host inputs are packed and
 * validated on the GPU: a worker holding an invalid request is made infeasible
 * for every candidate and the cluster records ALADDIN_ERR_STATE, which
 * aladdin_cluster_status returns. Any round in progress is discarded
 * and the cluster clock is kept. */
int aladdin_cluster_load(aladdin_cluster* cl, const int32_t* req_off, const int32_t* in,
                         const int32_t* gen, const int32_t* pred, const float* tdec_ms);

/* Score n_cand candidates (prompt length in[c], predicted output pred[c],
 * wait_ms[c] since arrival, nullable = 0) against every worker.
 *  flags  [n_cand*W] (nullable): ALADDIN_FLAG_* bits per pair.
 *  margin [n_cand*W] (nullable): the largest prompt length the worker could
 *         accept for this candidate (all constraints are monotone in it)
 *         minus in[c]; >= 0 exactly when the pair is feasible, -inf when no
 *         prompt length fits.
 *  argbest[n_cand] (nullable): Algorithm 1's choice: the feasible worker with
 *         the largest capacity_norm, lowest index on ties; ALADDIN_NONE if no
 *         worker is feasible.
 * A candidate with in < 0, pred < 1, in + pred > K or a negative or
 * non-finite wait is invalid: its flags are ALADDIN_FLAG_INVALID, its margins
 * NaN and its argbest ALADDIN_INVALID; the call still succeeds. Outputs of a
 * pending round (placements so far) are included in the state scored. */
int aladdin_score(aladdin_cluster* cl, int32_t n_cand, const int32_t* in, const int32_t* pred,
                  const float* wait_ms, uint8_t* flags, float* margin, int32_t* argbest);

/* aladdin_cluster_load followed by aladdin_score in one call (a scheduling
 * heartbeat: the workers' new state, then the waiting requests scored
 * against it), with the same arguments and results. When every array is
 * device memory (or mapped page-locked host memory) the candidates are
 * validated and sorted on a second stream while the cluster's stream packs
 * the state and builds the tables; the two join before the scoring kernel,
 * and the call stays ordered on the cluster's stream like the two calls.
 * Otherwise it runs the two calls in sequence. */
int aladdin_cluster_load_score(aladdin_cluster* cl, const int32_t* req_off, const int32_t* in,
                               const int32_t* gen, const int32_t* pred, const float* tdec_ms,
                               int32_t n_cand, const int32_t* cand_in, const int32_t* cand_pred,
                               const float* wait_ms, uint8_t* flags, float* margin,
                               int32_t* argbest);

/* As aladdin_score, plus two verification outputs per pair (each nullable):
 * kv_peak [n_cand*W]: the worker's peak KV usage over all future iterations
 * with the candidate added (exact integer), and t_cand_ms [n_cand*W]: the
 * candidate's projected total decode time on the worker. */
int aladdin_score_detail(aladdin_cluster* cl, int32_t n_cand, const int32_t* in,
                         const int32_t* pred, const float* wait_ms, uint8_t* flags,
                         float* margin, int32_t* argbest, int64_t* kv_peak, float* t_cand_ms);

/* Maximum candidates per call of aladdin_score_noalloc. */
#define ALADDIN_NOALLOC_MAX_CAND 32768

/* aladdin_score for callers that cannot allocate device memory during the
 * call: processes whose device memory is reserved up front by another
 * allocator (a serving engine owning the whole KV-cache pool leaves nothing
 * for a cudaMalloc to take), real-time scheduling loops that must not pay the
 * allocator's latency or its implicit synchronisation. The paper has no
 * counterpart; this is a property of the library.
 * Same inputs, outputs and results as aladdin_score, but every pointer must be
 * device memory of the cluster's GPU, or managed memory (ALADDIN_ERR_ARG
 * otherwise, before anything is launched), the call is asynchronous on the
 * cluster's stream, and it calls no allocator: its scratch is a fixed device
 * array (about 2 MB) built into the library, held by every GPU that loads it
 * until the process exits.
 * n_cand may be at most ALADDIN_NOALLOC_MAX_CAND (ALADDIN_ERR_SCRATCH
 * otherwise). The first call on a device sets up that device: it looks up the
 * array's device address and loads every scoring kernel with its launch
 * configuration; make that first call before any stream capture. All calls
 * share the array: calls that overlap on the GPU (several streams, or several
 * clusters on one device) race on it, and the caller must serialize them.
 * cudaDeviceReset while the library is in use is not supported. */
int aladdin_score_noalloc(aladdin_cluster* cl, int32_t n_cand, const int32_t* in,
                          const int32_t* pred, const float* wait_ms, uint8_t* flags,
                          float* margin, int32_t* argbest);

/* One placement round: candidates in index order, each placed in the state
 * left by the earlier placements, where it becomes a request of this round
 * (prefill pending, gen = 0). With ALADDIN_POLICY_BESTFIT (Algorithm 1) the
 * worker is the feasible one of largest capacity_norm; with JSQ or PO2 it is
 * the policy's choice, feasible or not. placement[c] = worker, ALADDIN_NONE
 * if no worker is feasible (best-fit; the cluster is fixed: no worker is
 * opened), ALADDIN_INVALID for an invalid candidate. Returns
 * ALADDIN_ERR_CAPACITY if a chosen worker has no free slot (placements up to
 * that candidate are kept, the later ones are ALADDIN_NONE). With grouped
 * scheduling (params.groups > 1) and best-fit the groups are independent
 * schedulers and run in parallel, one CTA each: a group whose chosen worker
 * is full stops there (its later candidates ALADDIN_NONE), the others go on,
 * and the call returns ALADDIN_ERR_CAPACITY. */
int aladdin_place_round(aladdin_cluster* cl, int32_t n_cand, const int32_t* in,
                        const int32_t* pred, const float* wait_ms, int32_t* placement);

/* Execute every worker for dt_ms from the cluster clock (continuous batching,
 * Sec. 2.1): at its next iteration boundary a worker runs the prefill of this
 * round's placements (stalling its decoding requests; on a decode instance
 * they join the batch without one), then decode iterations back to back
 * while they start before clock + dt_ms; finished requests leave. The clock
 * then advances by dt_ms and a new round begins.
 * stats (nullable, host, 7 doubles) accumulates since creation:
 * [0] requests whose prefill ran (joined the batch, on a decode instance),
 * [1] requests finished, [2] largest realized TTFT (ms; mixed setting only),
 * [3] largest realized ATGT (ms per token), and the realized violations:
 * [4] TTFTs above T_pre, [5] ATGTs above T_dec (each beyond a relative 1e-5,
 * the rounding of the fp32 placement test), [6] decode iterations whose KV
 * usage h * context + j * batch exceeded the worker's capacity. stats has 9
 * doubles: [7] re-predictions and [8] early finishes (both zero here: a
 * cluster built by this API holds exact predictions; the simulation follows
 * a trace's real lengths). */
int aladdin_cluster_advance(aladdin_cluster* cl, double dt_ms, double* stats);

/* Copy the cluster state to host arrays (each nullable): n[W] requests per
 * worker, and per slot [W*b_cap] in, gen, pred, pending (1 = placed this
 * round). Synchronous. */
int aladdin_cluster_state(aladdin_cluster* cl, int32_t* n, int32_t* in, int32_t* gen,
                          int32_t* pred, uint8_t* pending);

/* Algorithm 2 (Sec. 4.3, re-balancing with prediction error) over a round
 * that aladdin_place_round placed (n_cand candidates in, pred, wait_ms, and
 * their placement[], updated in place), before the round executes. le[w] and
 * be[w] (W entries each) are worker w's output-length and batch-size errors
 * (l^e, b^e): the tokens and requests its running requests deviate from
 * their predictions (+ for a request that outgrew its prediction, by the
 * added length; - for one that finished early, by the unused length). Its
 * error e_w = k2 l^e + c2 b^e places it relative to Eq. input limit; the
 * distance |e_w| / sqrt(k2^2 + c2^2) of that error line to the origin is
 * what the moves reduce, summed over workers. In index order, a placement on
 * a worker with e > 0 moves to the worker with e < 0 that is feasible for it
 * in the current state (all four flags, a free slot) and lowers the sum the
 * most: gain (e_x - e_y) - |e_x - d| - |e_y + d| > 0 with d = k2 pred + c2;
 * equal gains go to the larger capacity_norm, then the lower index. Moved
 * requests stay pending (prefill at the new worker's next boundary).
 * *moves (nullable) receives the number of moves, obj (nullable, host, 2
 * doubles) the summed distance before and after. Errors as
 * aladdin_place_round. */
int aladdin_rebalance(aladdin_cluster* cl, int32_t n_cand, const int32_t* in,
                      const int32_t* pred, const float* wait_ms, int32_t* placement,
                      const int64_t* le, const int32_t* be, int32_t* moves, double* obj);

/* Checkpoint and resume of a cluster's state (no counterpart in the paper):
 * the requests of every slot (l_in, l_out, l_pred, real length, decode time
 * so far, pending flag, wait), every worker's count, clock, offset and
 * Algorithm 2 errors, and the cluster's clock, open-round flag and request
 * ids. aladdin_cluster_save with buf NULL stores the size in *bytes;
 * otherwise it writes that many bytes to buf (host memory, *bytes at least
 * the size; synchronous). aladdin_cluster_restore loads such a buffer into
 * a cluster of the same worker count and request slots (its own parameters
 * and worker configurations stay) and rebuilds the tables and the
 * capacity_norm ranking, so that the cluster continues exactly as the saved
 * one would. ALADDIN_ERR_ARG for a buffer that is too short, not a
 * checkpoint, or of another shape. */
int aladdin_cluster_save(aladdin_cluster* cl, void* buf, int64_t* bytes);
int aladdin_cluster_restore(aladdin_cluster* cl, const void* buf, int64_t bytes);

/* Kernel timing (tracing): while enabled, CUDA events on the cluster's stream
 * bracket every launch of the candidate x worker scoring kernel. Each call
 * waits for the stream, returns in *kernel_ms (nullable) the summed event time
 * of the launches bracketed since the previous call and in *launches
 * (nullable) their number, forgets them, and turns the timing on (enable != 0)
 * or off. */
int aladdin_cluster_timing(aladdin_cluster* cl, int32_t enable, double* kernel_ms,
                           int64_t* launches);

/* ALADDIN_OK; ALADDIN_ERR_TIMEOUT if a kernel gave up a bounded wait (its
 * outputs for that call are incomplete); ALADDIN_ERR_STATE if an invalid
 * request was loaded from device or page-locked host memory; or
 * ALADDIN_ERR_CUDA. Errors are sticky. Synchronous. */
int aladdin_cluster_status(aladdin_cluster* cl);

/* Test hook of the failure handling of bounded device waits; the paper has
 * no counterpart. Every spin-wait of the library's kernels is bounded: the
 * placement round's grid exchange polls an arrival counter at most
 * grid_polls times (default 2^22, about a second) and the scoring kernel
 * polls each candidate-copy mbarrier at most mbar_polls times (default
 * 2^26); a wait that runs out sets the cluster's sticky timeout bit and its
 * kernel returns (aladdin_place_round returns ALADDIN_ERR_TIMEOUT, scoring
 * calls leave it to aladdin_cluster_status). 0 keeps a default. run_out = 1
 * makes the next waits run out by design, without any fault: the round's
 * exchange waits for one arrival more than its CTAs make, and the scoring
 * kernel does not issue its first candidate copy. For tests only: a cluster
 * whose wait ran out keeps an incomplete round or incomplete outputs.
 * ALADDIN_ERR_ARG for negative limits or run_out outside {0, 1}. */
int aladdin_cluster_test_waits(aladdin_cluster* cl, int64_t grid_polls, int64_t mbar_polls,
                               int32_t run_out);

/* Test hook of the incremental placement round; the paper has no
 * counterpart. A best-fit round first scores every candidate against the
 * round-start state, then re-evaluates only the workers it modifies, holding
 * them in a bounded number of shared-memory slots; when they run out, the
 * round continues with the sliced round from the current state, and very
 * large rounds are split into chunks of candidates, each a fresh incremental
 * round. max_slots > 0 caps the slots and chunk > 0 the candidates per chunk,
 * so that tests reach both paths on small clusters (0: the defaults). The
 * placements do not depend on either. ALADDIN_ERR_ARG for negative values. */
int aladdin_cluster_test_round(aladdin_cluster* cl, int32_t max_slots, int32_t chunk);

/* A request trace: arrival times (ms, non-decreasing), prompt and predicted
 * output lengths, and optionally prediction errors (Sec. 4.3): real[q] is the
 * output length request q really generates (the scheduler sees only
 * pred[q]); when a request has generated x tokens, reached its prediction
 * and not finished, it is re-predicted to repred[x] (at least x + 1, at most
 * K - in), the output length a predictor expects of a request known to
 * exceed x (repred has K + 1 entries; NULL: x + 1). real NULL: predictions
 * are exact. Host arrays. */
typedef struct aladdin_trace {
    int64_t n;
    const double* t_arr_ms;
    const int32_t* in;
    const int32_t* pred;
    const int32_t* real;     /* nullable, 1 <= real[q], in[q] + real[q] <= K */
    const int32_t* repred;   /* nullable, K + 1 entries */
} aladdin_trace;

/* Minimum-worker search (Sec. 4.1, Sec. 6.4): for every worker configuration
 * options[o], the smallest number of identical workers in [1, n_max] that
 * serves the whole trace with no failed request under params.policy and
 * params.phase (see aladdin_simulate; heartbeat every heartbeat_ms). Found by
 * doubling then bisection; each simulation runs on the GPU. JSQ and PO2
 * admit without a test, so their simulations drain the workers after the
 * last arrival to realize every request's latencies; best-fit's admissions
 * meet them by construction. n_workers[o] = -1 if n_max workers fail.
 * best_option (nullable) receives the option with the fewest total GPUs
 * (gpus * n_workers; first on ties), total_gpus (nullable) that total. Trace
 * arrays are host memory.
 * Execution: cuda_stream carries the trace upload (synchronised before any
 * simulation starts). The simulations run side by side on host threads of
 * the library, each on a non-blocking stream of its own on the current
 * device, with device memory from a private stream-ordered pool that is
 * trimmed on return: the options' searches at once, and per search the next
 * doubling steps or the next levels of bisection at once. The result equals
 * that of the sequential doubling-and-bisection search. Returns when every
 * simulation has finished. */
int aladdin_min_workers(const aladdin_params* params, int32_t n_options,
                        const aladdin_worker_cfg* options, const aladdin_trace* trace,
                        double heartbeat_ms, int32_t n_max, void* cuda_stream,
                        int32_t* n_workers, int32_t* best_option, int64_t* total_gpus);

/* Simulate the trace on n identical workers of configuration cfg (the check
 * inside aladdin_min_workers). At every heartbeat the arrivals so far that
 * are not placed form one placement round (params.policy), then the workers
 * execute until the next heartbeat. A request fails when it can no longer be
 * placed in time: best-fit in the mixed setting keeps an unplaced request
 * waiting while its wait at the next heartbeat plus its prefill alone stay
 * within T_pre; on a decode instance it fails at its first heartbeat; JSQ and
 * PO2 place every request at once and one whose worker has no free slot
 * fails. Every realized violation (aladdin_cluster_advance stats [4]-[6])
 * counts as a failure too. With prediction errors in the trace requests run
 * to their real lengths (re-predicted as they outgrow predictions), and with
 * params.rebalance (best-fit only) Algorithm 2 (aladdin_rebalance) runs after
 * every round on the errors the workers recorded since the previous
 * heartbeat, which then restart from zero. out (host, 9 doubles):
 * [0] failures, [1] placed requests, [2] heartbeats run, [3] largest realized
 * TTFT, [4] largest realized ATGT, [5] realized violations (included in
 * [0]), [6] re-predictions, [7] early finishes, [8] requests moved by
 * Algorithm 2. With stop_at_fail the simulation ends at the heartbeat after
 * the first failure; with drain it continues after the last arrival until
 * every worker is idle. */
int aladdin_simulate(const aladdin_params* params, const aladdin_worker_cfg* cfg, int32_t n,
                     const aladdin_trace* trace, double heartbeat_ms, int32_t stop_at_fail,
                     int32_t drain, void* cuda_stream, double* out);

/* ------------------------------------------------------------------------
 * Worker configuration (Sec. 4.1) and the worker-count model (Sec. 5.2).
 */

/* Tensor-parallel model of a worker of N_g GPUs (Sec. 4.1): compute time
 * k4 / N_g + c4 (Eq. TP compute), all-reduce time kc (N_g - 1) / N_g, KV
 * capacity N_g m_gpu - m_model (KV slots). */
typedef struct aladdin_tp_model {
    double k4, c4;     /* compute: ms, split across GPUs / not split */
    double kc;         /* all-reduce overhead scale (ms) */
    double m_gpu;      /* KV slots one GPU's memory holds */
    double m_model;    /* KV slots the model's weights take from a worker */
} aladdin_tp_model;

/* Worker configurations for gpus[o] GPUs per worker (o < n): kv_capacity =
 * floor(N_g m_gpu - m_model) and lat_scale = (k4 / N_g + c4 + kc (N_g - 1) /
 * N_g) / (k4 + c4), the iteration time relative to one GPU, which multiplies
 * every latency coefficient of aladdin_params (written to out[o]).
 * ALADDIN_ERR_ARG if a coefficient is negative or not finite, k4 + c4 <= 0, a
 * GPU count is below 1, or a capacity falls outside [1, 2^24). Host arrays;
 * no GPU work. */
int aladdin_tp_configs(const aladdin_tp_model* tp, int32_t n, const int32_t* gpus,
                       aladdin_worker_cfg* out);

/* Demand of a trace (Sec. 4.1, "learned from the historical data"): over
 * every decode iteration s = 1..l_pred of every request, the KV the request
 * holds, h (l_in + s) + j (the footprint vector w of (e)), averaged into
 * *m_r, and its context l_in + s averaged into *l_ave (each nullable). The
 * sums are exact integers reduced on the GPU; each average is one division.
 * Trace arrays are host memory; synchronous on cuda_stream. */
int aladdin_trace_demand(const aladdin_params* params, const aladdin_trace* trace,
                         void* cuda_stream, double* m_r, double* l_ave);

/* Eq. max throughput of each worker configuration options[o]: decode tokens
 * per ms per GPU, T_max = min(b_kv / (g t(b_kv)), B / (g T_dec)), with the KV
 * batch b_kv = kv_capacity / m_r, its iteration time t(b) = lat_scale (c3 +
 * c2 b + k2 b l_ave) (Eq. iter time) and the SLO batch B = (T_dec /
 * lat_scale - c3) / (c2 + k2 l_ave) (Eq. input limit); m_r and l_ave are the
 * trace's demand (aladdin_trace_demand). Both batches stay fractional, as in
 * the equation. t_max[o] (nullable) receives T_max, *best_option the option
 * of largest T_max (the optimal worker configuration; first on ties).
 * Trace arrays are host memory; synchronous. */
int aladdin_pick_config(const aladdin_params* params, int32_t n_options,
                        const aladdin_worker_cfg* options, const aladdin_trace* trace,
                        void* cuda_stream, double* t_max, int32_t* best_option);

/* Eq. total_worker_pre, N_w = ceil(k5 r_a + c5) for arrival rates r_a > R:
 * for each trace k (requests arriving at rate rates[k], requests per second)
 * the minimum number of workers of configuration cfg that serves it
 * (aladdin_min_workers: params.policy and params.phase, heartbeat_ms, at
 * most n_max workers) into n_workers[k], then k5 and c5 by ordinary least
 * squares over the traces whose rate exceeds R and whose search succeeded.
 * Returns ALADDIN_ERR_ARG (after filling n_workers, with k5 = c5 = 0) when
 * fewer than two such traces, or only one distinct rate, remain. Trace arrays
 * are host memory; every simulation runs on the GPU, the traces' searches
 * side by side (as in aladdin_min_workers). */
int aladdin_fit_workers(const aladdin_params* params, const aladdin_worker_cfg* cfg,
                        int32_t n_traces, const aladdin_trace* traces, const double* rates,
                        double R, double heartbeat_ms, int32_t n_max, void* cuda_stream,
                        int32_t* n_workers, double* k5, double* c5);

/* Eq. total_worker_pre: *n_workers = ceil(k5 rate + c5). ALADDIN_ERR_ARG if
 * the value is not finite or outside the int64 range. */
int aladdin_predict_workers(double k5, double c5, double rate, int64_t* n_workers);

/* Number of scheduling groups of distributed scheduling (Appendix A,
 * Eq. group_arrival_limit). Requests arriving at rate_a (requests per second)
 * are dealt round-robin to G groups (params.groups), so group i gets the rate
 * r_i = rate_a / G and n_workers / G workers (n_workers e.g. from
 * aladdin_predict_workers). G must satisfy
 *   r_i <= rate_max      rate_max = r(T_s), the arrival rate one scheduler
 *                        places within the scheduling latency limit T_s
 *                        (measured by the caller);
 *   n_workers / G >= 1 / (2 e)   if about half of the groups need one extra
 *                        worker, the extra workers stay within a fraction e
 *                        of the central scheduler's (the printed bound stands
 *                        on r_i; it is read as the workers per group that the
 *                        text derives, e = 10% giving five workers a group).
 * *groups receives the fewest such G (the least extra workers): the smallest
 * G >= 1 with G rate_max >= rate_a, if G <= 2 e n_workers and G <= n_workers.
 * ALADDIN_ERR_ARG if no G meets both, or for rate_a < 0, rate_max <= 0,
 * e <= 0 (or any of them not finite), n_workers < 1 or a null groups. */
int aladdin_pick_groups(double rate_a, double rate_max, double e, int64_t n_workers,
                        int64_t* groups);

#ifdef __cplusplus
}
#endif

#endif /* ALADDIN_H */
