// Execution step of the fleet simulation (continuous batching, Sec. 2.1): one
// warp per worker runs, from the worker's next iteration boundary, the prefill
// of this round's placements (Eq. prefill iter time; it stalls the decoding
// requests), then decode iterations back to back (Eq. iter time) while they
// start before t_now + dt. Each iteration adds one token to every active
// request; requests that reach their predicted length leave and their
// realized ATGT (decode time over decode tokens, Sec. 2.2) is recorded. On a
// decode instance (split-phase inference) the round's placements join the
// batch at the boundary with no prefill and no TTFT. Realized violations are
// counted: TTFT above T_pre, ATGT above T_dec (each beyond SLO_TOL) and
// decode iterations whose KV usage h * context + j * batch exceeds the
// worker's capacity M (what a placement without a feasibility test, JSQ or
// power of two, can cause). With prediction errors (Sec. 4.3) a request runs
// to its real length: one that reaches its prediction first is re-predicted
// from the re-prediction table, one that finishes before its prediction
// finishes early; both are Algorithm 2's error events (C.le, C.be). A lane
// keeps each request's next event point min(real, pred) in registers and
// reads the slot arrays only at events.
// Times accumulate in fp64 with explicitly rounded operations, in the same
// order as the CPU reference, so both sides produce the same schedule.
#include "aladdin_host.h"

namespace aladdin {

constexpr int ADV_WARPS = 4;

__device__ __forceinline__ void atomic_max_nonneg(unsigned long long* addr, double v)
{
    atomicMax(addr, (unsigned long long)__double_as_longlong(v));
}

template <int E>
__global__ void __launch_bounds__(ADV_WARPS * 32)
k_advance(DevParams P, ClusterDev C, double t_now, double dt, unsigned long long* stats,
          const int* halt, unsigned long long* fail)
{
    if (halt && *halt != 0) return;
    const int lane = threadIdx.x & 31;
    const int w = blockIdx.x * ADV_WARPS + (threadIdx.x >> 5);
    if (w >= C.W) return;  // warp-uniform
    const int n = C.n[w];
    const long long base = (long long)w * C.cap;
    const double s = C.scaled[w];
    const double t_end = __dadd_rn(t_now, dt);

    int in[E], gen[E], evt[E];  // evt: min(real, pred), the next event point
    double tdec[E];
    unsigned alive = 0;  // bit e: element e holds a request
    // events of one step: |le_acc| <= slots x iterations x K < 2^31
    int le_acc = 0, be_acc = 0, nrep = 0, nearly = 0;
    long long Pint = 0;
    int npend = 0;
    double maxttft = 0.0, maxatgt = 0.0;
    unsigned long long nfin = 0, vttft = 0, vatgt = 0, vkv = 0;
    const long long Mw = C.M[w];
    double start = C.clock[w] > t_now ? C.clock[w] : t_now;
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int x = e * 32 + lane;
        if (x < n) alive |= 1u << e;
        in[e] = gen[e] = 0;
        evt[e] = 1;
        tdec[e] = 0.0;
        if (x < n) {
            const long long slot = base + x;
            in[e] = C.in[slot];
            gen[e] = C.gen[slot];
            evt[e] = min(C.pred[slot], C.real[slot]);
            tdec[e] = C.tdec[slot];
            if (C.pend[slot]) {
                Pint += in[e];
                npend += 1;
            }
        }
    }
    Pint = warp_reduce(Pint, OpAdd<long long>());
    npend = warp_reduce(npend, OpAdd<int>());
    if (npend > 0 && P.decode) {
        // decode instance: the placements join the batch, nothing is stalled
#pragma unroll
        for (int e = 0; e < E; ++e) {
            if (!((alive >> e) & 1u)) continue;
            if (C.pend[base + e * 32 + lane]) {
                gen[e] = 0;
                tdec[e] = 0.0;
            }
        }
    } else if (npend > 0) {
        const double tau = __dmul_rn(s, __dadd_rn(__dmul_rn(P.k1d, (double)Pint), P.c1d));
        const double lead = __dsub_rn(start, t_now);
#pragma unroll
        for (int e = 0; e < E; ++e) {
            if (!((alive >> e) & 1u)) continue;
            const long long slot = base + e * 32 + lane;
            if (C.pend[slot]) {
                const double ttft = __dadd_rn(__dadd_rn(C.wait[slot], lead), tau);
                maxttft = fmax(maxttft, ttft);
                vttft += ttft > P.T_pre_viol ? 1 : 0;
                gen[e] = 0;
                tdec[e] = 0.0;
            } else {
                tdec[e] = __dadd_rn(tdec[e], tau);
            }
        }
        start = __dadd_rn(start, tau);
    }
    // Decode iterations (bounded: every iteration adds a token to every active
    // request, so at most max(real) iterations run).
    for (;;) {
        int b = 0;
        long long K = 0;
#pragma unroll
        for (int e = 0; e < E; ++e)
            if ((alive >> e) & 1u) {
                b += 1;
                K += (long long)in[e] + gen[e] + 1;
            }
        b = warp_reduce(b, OpAdd<int>());
        K = warp_reduce(K, OpAdd<long long>());
        if (b == 0 || !(start < t_end)) break;
        vkv += (long long)P.h * K + (long long)P.j * b > Mw ? 1 : 0;
        const double t = __dmul_rn(
            s, __dadd_rn(__dadd_rn(P.c3d, __dmul_rn(P.c2d, (double)b)), __dmul_rn(P.k2d, (double)K)));
#pragma unroll
        for (int e = 0; e < E; ++e)
            if ((alive >> e) & 1u) {
                gen[e] += 1;
                tdec[e] = __dadd_rn(tdec[e], t);
                if (gen[e] >= evt[e]) {
                    const long long slot = base + e * 32 + lane;
                    const int pr = C.pred[slot], rl = C.real[slot];
                    if (gen[e] >= rl) {
                        if (rl < pr) {  // finished before its prediction
                            le_acc += rl - pr;
                            be_acc -= 1;
                            nearly += 1;
                        }
                        const double atgt = __ddiv_rn(tdec[e], (double)gen[e]);
                        maxatgt = fmax(maxatgt, atgt);
                        vatgt += atgt > P.T_dec_viol ? 1 : 0;
                        nfin += 1;
                        alive &= ~(1u << e);
                    } else {  // reached its prediction unfinished: re-predict
                        int np = C.repred ? C.repred[gen[e]] : gen[e] + 1;
                        np = max(np, gen[e] + 1);
                        if ((long long)in[e] + np > (long long)P.K) np = P.K - in[e];
                        le_acc += np - pr;
                        be_acc += 1;
                        nrep += 1;
                        C.pred[slot] = np;
                        evt[e] = min(np, rl);
                    }
                }
            }
        start = __dadd_rn(start, t);
    }
    // Write the surviving requests back in their order, densely.
    int pos = 0;
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const unsigned bal = __ballot_sync(FULL, (alive >> e) & 1u);
        const int before = __popc(bal & ((1u << lane) - 1u));
        const long long src = base + e * 32 + lane;
        // read the fields that are not kept in registers before any write
        double wt = 0.0;
        int pr = 1, rl = 1;
        if ((alive >> e) & 1u) {
            wt = C.wait[src];
            pr = C.pred[src];
            rl = C.real[src];
        }
        __syncwarp();
        if ((alive >> e) & 1u) {
            const long long dst = base + pos + before;
            C.in[dst] = in[e];
            C.gen[dst] = gen[e];
            C.pred[dst] = pr;
            C.real[dst] = rl;
            C.tdec[dst] = tdec[e];
            C.bank[dst] = banked_slack(P, gen[e], tdec[e]);
            C.pend[dst] = 0;
            C.wait[dst] = wt;
        }
        __syncwarp();
        pos += __popc(bal);
    }
    maxttft = warp_reduce(maxttft, OpMax<double>());
    maxatgt = warp_reduce(maxatgt, OpMax<double>());
    nfin = warp_reduce(nfin, OpAdd<unsigned long long>());
    vttft = warp_reduce(vttft, OpAdd<unsigned long long>());
    vatgt = warp_reduce(vatgt, OpAdd<unsigned long long>());
    le_acc = warp_reduce(le_acc, OpAdd<int>());
    be_acc = warp_reduce(be_acc, OpAdd<int>());
    nrep = warp_reduce(nrep, OpAdd<int>());
    nearly = warp_reduce(nearly, OpAdd<int>());
    if (lane == 0) {
        C.n[w] = pos;
        if (le_acc || be_acc) {  // one warp per worker: no other writer
            C.le[w] += (long long)le_acc;
            C.be[w] += be_acc;
        }
        C.clock[w] = start;
        C.off[w] = start > t_end ? (float)__dsub_rn(start, t_end) : 0.0f;
        if (stats) {
            if (npend) atomicAdd(&stats[0], (unsigned long long)npend);
            if (nfin) atomicAdd(&stats[1], nfin);
            if (npend && !P.decode) atomic_max_nonneg(&stats[2], maxttft);
            if (nfin) atomic_max_nonneg(&stats[3], maxatgt);
            if (vttft) atomicAdd(&stats[4], vttft);
            if (vatgt) atomicAdd(&stats[5], vatgt);
            if (vkv) atomicAdd(&stats[6], vkv);
            if (nrep) atomicAdd(&stats[7], (unsigned long long)nrep);
            if (nearly) atomicAdd(&stats[8], (unsigned long long)nearly);
        }
        const unsigned long long v = vttft + vatgt + vkv;
        if (fail && v) atomicAdd(fail, v);
    }
}

template <int E>
static cudaError_t advance_e(const DevParams& P, const ClusterDev& C, double t_now, double dt,
                             unsigned long long* stats, const int* halt, unsigned long long* fail,
                             cudaStream_t st)
{
    const int blocks = (C.W + ADV_WARPS - 1) / ADV_WARPS;
    k_advance<E><<<blocks, ADV_WARPS * 32, 0, st>>>(P, C, t_now, dt, stats, halt, fail);
    return cudaGetLastError();
}

cudaError_t launch_advance(const DevParams& P, const ClusterDev& C, double t_now, double dt,
                           unsigned long long* stats, const int* halt, cudaStream_t st,
                           unsigned long long* fail)
{
    switch (lanes_per_worker(C.cap)) {
    case 1: return advance_e<1>(P, C, t_now, dt, stats, halt, fail, st);
    case 2: return advance_e<2>(P, C, t_now, dt, stats, halt, fail, st);
    case 4: return advance_e<4>(P, C, t_now, dt, stats, halt, fail, st);
    case 8: return advance_e<8>(P, C, t_now, dt, stats, halt, fail, st);
    case 16: return advance_e<16>(P, C, t_now, dt, stats, halt, fail, st);
    case 32: return advance_e<32>(P, C, t_now, dt, stats, halt, fail, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace aladdin
