/*
 * Aladdin scheduler oracle: a plain, slow CPU restatement of the scheduling
 * rules of "Aladdin: Joint Placement and Scaling for SLO-Aware LLM Serving"
 * (arxiv 2405.06856), in fp64, stepping every worker's future one decode
 * iteration at a time.
 *
 * TEST INFRASTRUCTURE ONLY. Only the tests, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py may load or call this library. It shares no
 * code, header, table or constant with the CUDA library, and the product
 * path never reaches it.
 *
 * Models (Sec. 3). Where the paper is garbled or silent these readings are
 * taken: Eq. kv cache's r is l_out, the tokens generated so far; Eq. iter
 * time holds for every batch size b >= 1; ATGT is enforced over the
 * remaining iterations plus the banked slack of Table 1's t^dec; the stall
 * of a round's prefill hits only the requests decoding at round start.
 *   KV usage      Eq. kv cache: a request with c context tokens holds h*c + j
 *                 KV slots. In its s-th remaining decode iteration a request
 *                 with l_in input and l_out generated tokens holds
 *                 l_in + l_out + s tokens (footprint vector w of constraint (e),
 *                 Sec. 4.2), and nothing after its last iteration.
 *   Prefill       Eq. prefill iter time: t_pre = k1 * sum(l_in) + c1.
 *   Decode        Eq. iter time: t_d = (k2 * l_ave + c2) * b + c3
 *                 = k2 * (context tokens of the batch) + c2 * b + c3, used for
 *                 every batch size b >= 1.
 *   Worker scale  every latency coefficient of worker i is multiplied by
 *                 scale[i] (1/sqrt(GPUs) in the mixed-config workload).
 *
 * Placement test of a candidate c (prompt l_in = a_c, predicted output r_c,
 * waiting w_c ms) on worker i (Sec. 4.2, constraints (c), (d), (e); the exact
 * per-request decode projection replaces the approximate constraint (b)):
 *   tau      = t_pre(P_i + a_c): the prefill of every request placed on i in
 *              this round (P_i input tokens) plus the candidate; it stalls the
 *              requests that were decoding at round start.
 *   KV       for every future iteration s: KV(s) <= M_i            (e)
 *   TTFT     w + off_i + tau <= T_pre for the candidate and for every request
 *              already placed on i in this round                  (c)
 *   ongoing  tau + D_j <= theta * T_dec * r_j + bank_j              (d)
 *   new      D_q <= theta * T_dec * r_q for the candidate and the requests
 *              placed on i in this round (no stall: they decode after it)
 *   where D_j is the projected time of request j's r_j remaining decode
 *   iterations with the candidate added, off_i the time until worker i's next
 *   iteration boundary, and bank_j = theta * T_dec * l_out_j - t_dec_j the
 *   decode time request j saved so far (Table 1: t^dec_j; 0 when no history
 *   is given).
 *
 * Every quantity above is affine in the candidate's prompt length l (KV
 * tokens and tau grow by one token per unit of l; D_j by k2 for every
 * iteration the candidate shares with j). The oracle carries each quantity
 * as (value at l = 0, coefficient of l) while stepping, which gives for every
 * constraint the largest admissible l. The pair's margin is the smallest of
 * these bounds minus a_c: the number of extra prompt tokens the worker could
 * still absorb for this candidate (negative: infeasible).
 *
 * Approximate mode (mode 1): the MIP's own decode constraints replace the
 * projection of groups 2 and 3, as the paper states them (Sec. 4.2):
 *   (d) ongoing  tau <= theta * min_j (T_dec * l_out_j - t_dec_j) over the
 *                requests decoding at round start (t_dec_j = theta * T_dec *
 *                l_out_j when no history is given)
 *   (b) new      sum over the worker's requests and the candidate of
 *                (l_in + gamma * l_pred) <= theta * l_d(B), B = requests with
 *                the candidate, l_d(b) = (T_dec / scale_i - c3 - c2 b) / k2
 *                (Eq. input limit).
 * KV (e) and TTFT (c) are as in the exact mode.
 *
 * Serving setting (phase):
 *   0 mixed     continuous batching with prefill and decode on the same
 *               worker (Sec. 5.1, default continuous batching).
 *   1 decode    split-phase inference (Sec. 5.1): the worker is a decode
 *               instance; requests arrive with their prompt processed
 *               elsewhere, so no prefill runs on it. Nothing stalls its
 *               decoding requests (tau = 0), TTFT (c) is the prefill
 *               instance's concern and is not tested, and in the approximate
 *               mode (d) is vacuous. A request arrives holding its prompt's
 *               KV, as in the mixed setting.
 * Placement policy (Sec. 6.1 baselines, Sec. 6.4):
 *   0 best-fit  Algorithm 1 (the feasibility test above, capacity_norm order).
 *   1 JSQ       join the shortest queue: the worker holding the fewest
 *               requests, lowest index on ties; no feasibility test.
 *   2 Po2       power of two choices: two workers drawn uniformly at random
 *               (SplitMix64, below), the one holding fewer requests, the
 *               first drawn on ties; no feasibility test.
 * Grouped scheduling (Appendix A, distributed scheduling): with G > 1 groups
 * the requests are dealt to groups round-robin (request id q to group
 * q mod G) and each group's scheduler places only on its own workers
 * (worker w belongs to group w mod G), under the same policy; Algorithm 2
 * moves requests within their group.
 * In the simulation a placement that breaks an SLO shows up when the
 * workers execute: a realized TTFT above T_pre, a realized ATGT above T_dec
 * (each beyond a relative 1e-5) or an iteration whose KV exceeds M counts as
 * a violation and fails the run like an unplaced request.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    double k1, c1;        /* prefill: ms per input token, ms */
    double k2, c2, c3;    /* decode: ms per context token, ms per request, ms */
    int64_t h, j;         /* KV slots per context token, per request */
    double T_pre, T_dec;  /* TTFT SLO, per-token decode SLO (ms) */
    double gamma, theta;  /* capacity_norm weight, SLO scaling knob */
    int64_t K;            /* sequence limit (input + output tokens) */
    int64_t mode;         /* 0: exact decode projection; 1: approximate
                             constraints (b) and (d) of the MIP (Sec. 4.2) */
    int64_t phase;        /* 0: mixed prefill + decode; 1: decode instance */
    int64_t policy;       /* 0: best-fit; 1: JSQ; 2: power of two choices */
    uint64_t seed;        /* SplitMix64 seed of the power-of-two draws */
    int64_t rebalance;    /* 1: Algorithm 2 after every placement round (simulation) */
    int64_t groups;       /* G > 1: distributed grouped scheduling (Appendix A) */
} orc_params;

/* Relative slack of a realized latency over its SLO before it counts as a
 * violation (the rounding of the fp32 placement test). */
#define ORC_SLO_TOL 1e-5

/* Cluster state in fixed-stride slots: worker w owns slots
 * [w*cap, w*cap + n[w]). */
typedef struct {
    int32_t W, cap;
    const int64_t* M;     /* [W] KV capacity (slots) */
    const double* scale;  /* [W] latency coefficient multiplier */
    double* off;          /* [W] ms from now to the worker's next iteration start */
    double* clock;        /* [W] absolute ms at which the worker's next iteration
                             starts (simulation only; may be NULL for scoring) */
    int32_t* n;           /* [W] requests on the worker */
    int32_t* in;          /* [W*cap] input length */
    int32_t* gen;         /* [W*cap] output tokens generated so far */
    int32_t* pred;        /* [W*cap] predicted output length */
    double* tdec;         /* [W*cap] decode time so far (ms), or NULL */
    uint8_t* pend;        /* [W*cap] 1: placed in the current round, prefill pending */
    double* wait;         /* [W*cap] pending requests: wait since arrival (ms) */
    int64_t* rid;         /* [W*cap] request id (simulation only), or NULL */
    int32_t* real;        /* [W*cap] real output length (unknown to the scheduler), or
                             NULL: every prediction is exact */
    int64_t* le;          /* [W] Algorithm 2's output-length error l^e, or NULL */
    int32_t* be;          /* [W] Algorithm 2's batch-size error b^e, or NULL */
    const int32_t* repred;/* [K+1] re-prediction: the output length predicted for a
                             request that has generated x tokens without finishing,
                             or NULL (x + 1) */
} orc_cluster;

typedef struct {
    uint8_t flags;        /* bit0 KV, bit1 TTFT, bit2 ongoing ATGT, bit3 new ATGT */
    double margin;        /* largest admissible prompt length minus a_c (tokens) */
    double mscale;        /* token scale of the binding latency bound; 0 if KV binds */
    int64_t kv_peak;      /* peak KV over all future iterations with the candidate */
    double t_cand;        /* candidate's projected decode time, all iterations (ms) */
    double near;          /* over the latency groups, the smallest |min slack / scale|
                             at a_c: how close the closest flag bit is to flipping */
} orc_pair;

enum { ORC_OK = 0, ORC_ERR_ARG = -1, ORC_ERR_CAPACITY = -2, ORC_ERR_MEM = -3 };

/* ---------------------------------------------------------------------- */
/* A worker's own future, stepped one decode iteration at a time:
 *   b[s] = number of its requests still decoding in iteration s,
 *   Kt[s] = context tokens they hold in iteration s,   s = 1..S.         */
typedef struct {
    int32_t S;
    int64_t* b;
    int64_t* Kt;
} orc_future;

static int32_t remaining(const orc_cluster* cl, int64_t slot)
{
    return cl->pred[slot] - (cl->pend[slot] ? 0 : cl->gen[slot]);
}

static int64_t context(const orc_cluster* cl, int64_t slot)
{
    return (int64_t)cl->in[slot] + (cl->pend[slot] ? 0 : cl->gen[slot]);
}

static int future_build(const orc_cluster* cl, int w, orc_future* f)
{
    int64_t base = (int64_t)w * cl->cap;
    int32_t S = 0;
    for (int q = 0; q < cl->n[w]; ++q) {
        int32_t r = remaining(cl, base + q);
        if (r > S) S = r;
    }
    f->S = S;
    f->b = (int64_t*)calloc((size_t)S + 2, sizeof(int64_t));
    f->Kt = (int64_t*)calloc((size_t)S + 2, sizeof(int64_t));
    if (!f->b || !f->Kt) return ORC_ERR_MEM;
    for (int32_t s = 1; s <= S; ++s) {
        int64_t b = 0, K = 0;
        for (int q = 0; q < cl->n[w]; ++q) {
            int64_t slot = base + q;
            if (remaining(cl, slot) >= s) {
                b += 1;
                K += context(cl, slot) + s;
            }
        }
        f->b[s] = b;
        f->Kt[s] = K;
    }
    return ORC_OK;
}

static void future_free(orc_future* f)
{
    free(f->b);
    free(f->Kt);
    f->b = f->Kt = NULL;
    f->S = 0;
}

static int64_t floor_div(int64_t x, int64_t d) /* d > 0 */
{
    int64_t q = x / d;
    if ((x % d != 0) && (x < 0)) q -= 1;
    return q;
}

/* Running minimum of the constraint bounds; gmin[g] is the smallest relative
 * slack (slack / scale, signed) among group g's constraints at a_c. */
typedef struct {
    double bound, bscale;
    double gmin[4];
    int ok[4];
} orc_acc;

/* A latency constraint slack(l) = slack0 - slope * l >= 0; scale_a is the sum
 * of the magnitudes of its terms at l = a (the size rounding acts on). */
static void lat_constraint(orc_acc* A, int group, double slack0, double slope,
                           double scale_a, double a)
{
    double slack_a = slack0 - slope * a;
    if (!(slack_a >= 0.0)) A->ok[group] = 0;
    double b;
    if (slope > 0.0) b = slack0 / slope;
    else b = slack0 >= 0.0 ? INFINITY : -INFINITY;
    if (b < A->bound) {
        A->bound = b;
        A->bscale = slope > 0.0 ? scale_a / slope : 0.0;
    }
    double rel = slack_a / (scale_a > 0.0 ? scale_a : 1.0);
    if (rel < A->gmin[group]) A->gmin[group] = rel;
}

/* Evaluate candidate (a_c, r_c, w_c) on worker w. T0, T1 are scratch arrays of
 * at least max(S, r_c) + 1 doubles. */
static void eval_pair(const orc_params* p, const orc_cluster* cl, int w, const orc_future* f,
                      double* T0, double* T1, int32_t a_c, int32_t r_c, double w_c, orc_pair* out)
{
    const double sc = cl->scale[w];
    const int64_t M = cl->M[w];
    const int64_t base = (int64_t)w * cl->cap;
    const int32_t S = f->S > r_c ? f->S : r_c;

    /* Step every future iteration with the candidate added. The candidate holds
     * l + s tokens in its s-th iteration (it has generated nothing yet). */
    int64_t kv_hi0 = INT64_MIN; /* max KV at l = 0 over iterations shared with the candidate */
    int64_t kv_lo = 0;          /* max KV over iterations after the candidate finished */
    int64_t kv_peak = 0;
    T0[0] = 0.0;
    T1[0] = 0.0;
    for (int32_t s = 1; s <= S; ++s) {
        int64_t bw = s <= f->S ? f->b[s] : 0;
        int64_t Kw = s <= f->S ? f->Kt[s] : 0;
        int with_c = s <= r_c;
        int64_t b = bw + (with_c ? 1 : 0);
        int64_t K0 = Kw + (with_c ? s : 0); /* context tokens at l = 0 */
        int64_t kv0 = p->h * K0 + p->j * b;
        int64_t kv_a = kv0 + (with_c ? p->h * (int64_t)a_c : 0);
        if (kv_a > kv_peak) kv_peak = kv_a;
        if (with_c) {
            if (kv0 > kv_hi0) kv_hi0 = kv0;
        } else if (kv0 > kv_lo) {
            kv_lo = kv0;
        }
        double t0 = sc * (p->c3 + p->c2 * (double)b + p->k2 * (double)K0);
        double t1 = with_c ? sc * p->k2 : 0.0;
        T0[s] = T0[s - 1] + t0;
        T1[s] = T1[s - 1] + t1;
    }

    orc_acc A;
    A.bound = INFINITY;
    A.bscale = 0.0;
    for (int g = 0; g < 4; ++g) A.gmin[g] = INFINITY;
    for (int g = 0; g < 4; ++g) A.ok[g] = 1;
    const double a = (double)a_c;

    /* (e) KV capacity. */
    double bkv;
    if (kv_lo > M) {
        bkv = -INFINITY;
        A.ok[0] = 0;
    } else {
        bkv = (double)floor_div(M - kv_hi0, p->h);
        if (kv_hi0 + p->h * (int64_t)a_c > M) A.ok[0] = 0;
    }

    /* Prefill of this round's placements plus the candidate (Eq. prefill). */
    double P = 0.0;
    for (int q = 0; q < cl->n[w]; ++q)
        if (cl->pend[base + q]) P += (double)cl->in[base + q];
    /* A decode instance runs no prefill: no stall and no TTFT test. */
    const int decode = p->phase == 1;
    const double tau0 = decode ? 0.0 : sc * (p->k1 * P + p->c1);
    const double tau1 = decode ? 0.0 : sc * p->k1;
    const double tau_a = tau0 + tau1 * a;
    const double off = cl->off ? cl->off[w] : 0.0;

    /* (c) TTFT of the candidate and of this round's earlier placements. */
    if (!decode) {
        lat_constraint(&A, 1, p->T_pre - w_c - off - tau0, tau1, p->T_pre + w_c + off + tau_a, a);
        for (int q = 0; q < cl->n[w]; ++q) {
            int64_t slot = base + q;
            if (!cl->pend[slot]) continue;
            double wq = cl->wait[slot];
            lat_constraint(&A, 1, p->T_pre - wq - off - tau0, tau1, p->T_pre + wq + off + tau_a,
                           a);
        }
    }

    if (p->mode == 1) {
        /* (d) as stated: the stall within theta times the smallest decode time
         * an ongoing request has saved so far (vacuous without a prefill). */
        for (int q = 0; q < cl->n[w] && !decode; ++q) {
            int64_t slot = base + q;
            if (cl->pend[slot]) continue;
            double g = (double)cl->gen[slot];
            double td = cl->tdec ? cl->tdec[slot] : p->theta * p->T_dec * g;
            double saved = p->theta * (p->T_dec * g - td);
            lat_constraint(&A, 2, saved - tau0, tau1, fabs(saved) + tau_a, a);
        }
        /* (b) with Eq. input limit: weighted context of the batch with the
         * candidate within theta * l_d(B). */
        double L = 0.0;
        for (int q = 0; q < cl->n[w]; ++q)
            L += (double)cl->in[base + q] + p->gamma * (double)cl->pred[base + q];
        double B = (double)cl->n[w] + 1.0;
        double ld = (p->T_dec / sc - p->c3 - p->c2 * B) / p->k2;
        double cap_b = p->theta * ld - L - p->gamma * (double)r_c;
        lat_constraint(&A, 3, cap_b, 1.0, fabs(p->theta * ld) + L + p->gamma * (double)r_c + a, a);
        {
            double D0 = T0[r_c], D1 = T1[r_c];
            out->t_cand = D0 + D1 * a;
        }
    } else {
    /* (d) ongoing requests: stall plus remaining decode within their budget. */
    for (int q = 0; q < cl->n[w]; ++q) {
        int64_t slot = base + q;
        int32_t r = remaining(cl, slot);
        double D0 = T0[r], D1 = T1[r];
        if (cl->pend[slot]) {
            double budget = p->theta * p->T_dec * (double)r;
            lat_constraint(&A, 3, budget - D0, D1, budget + D0 + D1 * a, a);
        } else {
            double bank = 0.0;
            if (cl->tdec) bank = p->theta * p->T_dec * (double)cl->gen[slot] - cl->tdec[slot];
            double budget = p->theta * p->T_dec * (double)r + bank;
            lat_constraint(&A, 2, budget - tau0 - D0, tau1 + D1,
                           p->theta * p->T_dec * (double)r + fabs(bank) + tau_a + D0 + D1 * a, a);
        }
    }
    /* The candidate's own decode. */
    {
        double budget = p->theta * p->T_dec * (double)r_c;
        double D0 = T0[r_c], D1 = T1[r_c];
        lat_constraint(&A, 3, budget - D0, D1, budget + D0 + D1 * a, a);
        out->t_cand = D0 + D1 * a;
    }
    }

    double bound = A.bound, bscale = A.bscale;
    if (bkv <= bound) {
        bound = bkv;
        bscale = 0.0;
    }
    out->flags = (uint8_t)((A.ok[0] ? 1 : 0) | (A.ok[1] ? 2 : 0) | (A.ok[2] ? 4 : 0) | (A.ok[3] ? 8 : 0));
    out->margin = bound - a;
    out->mscale = bscale;
    out->kv_peak = kv_peak;
    /* A group's flag is the sign of its smallest slack; arithmetic with a
     * relative error below e per constraint can flip it only when that
     * smallest relative slack lies within e of zero. */
    double near = INFINITY;
    for (int g = 0; g < 4; ++g)
        if (fabs(A.gmin[g]) < near) near = fabs(A.gmin[g]);
    out->near = near;
}

/* ---------------------------------------------------------------------- */
/* Algorithm 1 ordering: workers sorted on capacity_norm from large to small;
 * capacity_norm = L2 norm of (batch size B, sum over requests of
 * l_in + gamma * l_pred) (Sec. 4.2, Scheduling heuristic). Equal norms keep
 * index order. */
typedef struct {
    double norm;
    int32_t w;
} orc_key;

static int key_cmp(const void* x, const void* y)
{
    const orc_key* a = (const orc_key*)x;
    const orc_key* b = (const orc_key*)y;
    if (a->norm > b->norm) return -1;
    if (a->norm < b->norm) return 1;
    return a->w < b->w ? -1 : (a->w > b->w ? 1 : 0);
}

double orc_capacity_norm(const orc_params* p, const orc_cluster* cl, int w)
{
    int64_t base = (int64_t)w * cl->cap;
    double B = (double)cl->n[w];
    double L = 0.0;
    for (int q = 0; q < cl->n[w]; ++q)
        L += (double)cl->in[base + q] + p->gamma * (double)cl->pred[base + q];
    return sqrt(B * B + L * L);
}

static int capacity_order(const orc_params* p, const orc_cluster* cl, int32_t* order)
{
    orc_key* keys = (orc_key*)malloc(sizeof(orc_key) * (size_t)cl->W);
    if (!keys) return ORC_ERR_MEM;
    for (int w = 0; w < cl->W; ++w) {
        keys[w].norm = orc_capacity_norm(p, cl, w);
        keys[w].w = w;
    }
    qsort(keys, (size_t)cl->W, sizeof(orc_key), key_cmp);
    for (int i = 0; i < cl->W; ++i) order[i] = keys[i].w;
    free(keys);
    return ORC_OK;
}

int orc_order(const orc_params* p, const orc_cluster* cl, int32_t* order)
{
    return capacity_order(p, cl, order);
}

static int32_t max_remaining(const orc_cluster* cl)
{
    int32_t S = 0;
    for (int w = 0; w < cl->W; ++w)
        for (int q = 0; q < cl->n[w]; ++q) {
            int32_t r = remaining(cl, (int64_t)w * cl->cap + q);
            if (r > S) S = r;
        }
    return S;
}

static int32_t max_of(const int32_t* x, int64_t n)
{
    int32_t m = 0;
    for (int64_t i = 0; i < n; ++i)
        if (x[i] > m) m = x[i];
    return m;
}

static void store_pair(const orc_pair* r, int64_t k, uint8_t* flags, double* margin, double* mscale,
                       int64_t* kvpeak, double* tcand, double* near)
{
    if (flags) flags[k] = r->flags;
    if (margin) margin[k] = r->margin;
    if (mscale) mscale[k] = r->mscale;
    if (kvpeak) kvpeak[k] = r->kv_peak;
    if (tcand) tcand[k] = r->t_cand;
    if (near) near[k] = r->near;
}

/* Score every (candidate, worker) pair; outputs are row-major [c][w]; every
 * output pointer may be NULL. argbest[c] is the first feasible worker in
 * capacity_norm order, -1 if none. */
int orc_score(const orc_params* p, const orc_cluster* cl, int32_t C, const int32_t* cin,
              const int32_t* cpred, const double* cwait, uint8_t* flags, double* margin,
              double* mscale, int64_t* kvpeak, double* tcand, double* near, int32_t* argbest)
{
    const int W = cl->W;
    int32_t S = max_remaining(cl);
    int32_t Sc = max_of(cpred, C);
    if (Sc > S) S = Sc;
    double* T0 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    double* T1 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    uint8_t* feas = (uint8_t*)calloc((size_t)C * (size_t)W, 1);
    int32_t* order = (int32_t*)malloc(sizeof(int32_t) * (size_t)W);
    if (!T0 || !T1 || !feas || !order) return ORC_ERR_MEM;
    for (int w = 0; w < W; ++w) {
        orc_future f;
        if (future_build(cl, w, &f) != ORC_OK) return ORC_ERR_MEM;
        for (int32_t c = 0; c < C; ++c) {
            orc_pair r;
            eval_pair(p, cl, w, &f, T0, T1, cin[c], cpred[c], cwait ? cwait[c] : 0.0, &r);
            int64_t k = (int64_t)c * W + w;
            store_pair(&r, k, flags, margin, mscale, kvpeak, tcand, near);
            feas[k] = r.flags == 15;
        }
        future_free(&f);
    }
    if (argbest) {
        if (capacity_order(p, cl, order) != ORC_OK) return ORC_ERR_MEM;
        for (int32_t c = 0; c < C; ++c) {
            argbest[c] = -1;
            for (int i = 0; i < W; ++i)
                if (feas[(int64_t)c * W + order[i]]) {
                    argbest[c] = order[i];
                    break;
                }
        }
    }
    free(T0);
    free(T1);
    free(feas);
    free(order);
    return ORC_OK;
}

/* Score a list of (candidate, worker) pairs; outputs are per pair. */
int orc_score_pairs(const orc_params* p, const orc_cluster* cl, int64_t npairs,
                    const int32_t* pc, const int32_t* pw, const int32_t* cin,
                    const int32_t* cpred, const double* cwait, uint8_t* flags, double* margin,
                    double* mscale, int64_t* kvpeak, double* tcand, double* near)
{
    int32_t S = max_remaining(cl);
    for (int64_t k = 0; k < npairs; ++k)
        if (cpred[pc[k]] > S) S = cpred[pc[k]];
    double* T0 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    double* T1 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    if (!T0 || !T1) return ORC_ERR_MEM;
    for (int64_t k = 0; k < npairs; ++k) {
        orc_future f;
        if (future_build(cl, pw[k], &f) != ORC_OK) return ORC_ERR_MEM;
        orc_pair r;
        int32_t c = pc[k];
        eval_pair(p, cl, pw[k], &f, T0, T1, cin[c], cpred[c], cwait ? cwait[c] : 0.0, &r);
        store_pair(&r, k, flags, margin, mscale, kvpeak, tcand, near);
        future_free(&f);
    }
    free(T0);
    free(T1);
    return ORC_OK;
}

/* KV curve of worker w with candidate (a_c, r_c): kv[s-1] = KV(s), s = 1..S,
 * S = max(worker's longest remaining, r_c). Returns S (or < 0 on error); kv
 * must hold at least K entries. */
int32_t orc_kv_curve(const orc_params* p, const orc_cluster* cl, int w, int32_t a_c, int32_t r_c,
                     int64_t* kv)
{
    orc_future f;
    if (future_build(cl, w, &f) != ORC_OK) return ORC_ERR_MEM;
    int32_t S = f.S > r_c ? f.S : r_c;
    for (int32_t s = 1; s <= S; ++s) {
        int64_t b = (s <= f.S ? f.b[s] : 0) + (s <= r_c ? 1 : 0);
        int64_t K = (s <= f.S ? f.Kt[s] : 0) + (s <= r_c ? (int64_t)a_c + s : 0);
        kv[s - 1] = p->h * K + p->j * b;
    }
    future_free(&f);
    return S;
}

/* ---------------------------------------------------------------------- */
/* SplitMix64 (G. Steele, D. Lea, C. Flood, "Fast splittable pseudorandom
 * number generators", OOPSLA 2014): the n-th output (n = 1, 2, ...) of the
 * stream seeded with s is mix(s + n * 0x9E3779B97F4A7C15), all mod 2^64. */
uint64_t orc_splitmix64(uint64_t s, uint64_t n)
{
    uint64_t z = s + n * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* Draw k (0 or 1) of the power-of-two choice for request id rid: output
 * 2 rid + k + 1 of the seeded stream, mapped to [0, W) by its upper 32 bits
 * times W over 2^32. */
int32_t orc_po2_draw(uint64_t seed, int64_t rid, int k, int32_t W)
{
    uint64_t x = orc_splitmix64(seed, 2ull * (uint64_t)rid + (uint64_t)k + 1ull);
    return (int32_t)(((x >> 32) * (uint64_t)W) >> 32);
}

/* Grouped scheduling: may request rid be placed on worker w? */
static int same_group(const orc_params* p, int w, int64_t rid)
{
    return p->groups <= 1 || (int64_t)w % p->groups == rid % p->groups;
}

/* The worker a load-balancing policy picks (JSQ or power of two choices)
 * among the workers of the request's group; -1 if the group has none. */
static int pick_by_queue(const orc_params* p, const orc_cluster* cl, int64_t rid)
{
    const int G = p->groups > 1 ? (int)p->groups : 1;
    const int g = (int)(rid % G);
    const int Wg = cl->W > g ? (cl->W - g + G - 1) / G : 0; /* workers g, g + G, ... */
    if (Wg == 0) return -1;
    if (p->policy == 1) {
        int best = g;
        for (int w = g + G; w < cl->W; w += G)
            if (cl->n[w] < cl->n[best]) best = w;
        return best;
    }
    int w1 = g + G * orc_po2_draw(p->seed, rid, 0, Wg);
    int w2 = g + G * orc_po2_draw(p->seed, rid, 1, Wg);
    return cl->n[w2] < cl->n[w1] ? w2 : w1;
}

/* ---------------------------------------------------------------------- */
/* One placement round, candidates in index (arrival) order. Best-fit
 * (Algorithm 1): each goes to the first feasible worker in capacity_norm
 * order of the current state. JSQ / power of two: each goes to the worker the
 * policy picks, feasible or not. The request becomes a pending request there
 * (gen = 0, prefill at the worker's next iteration). placement[c] = worker,
 * or -1 if no worker is feasible (best-fit; the cluster is fixed, nothing is
 * opened). A chosen worker without a free slot is ORC_ERR_CAPACITY, or, with
 * refuse_full (simulation of JSQ / power of two), placement -3 and the round
 * goes on. The power-of-two draws use crid[c] (c if crid is NULL). */
static int place_round_impl(const orc_params* p, orc_cluster* cl, int32_t C, const int32_t* cin,
                            const int32_t* cpred, const int32_t* creal, const double* cwait,
                            const int64_t* crid, int32_t* placement, int refuse_full);

int orc_place_round(const orc_params* p, orc_cluster* cl, int32_t C, const int32_t* cin,
                    const int32_t* cpred, const double* cwait, const int64_t* crid,
                    int32_t* placement)
{
    return place_round_impl(p, cl, C, cin, cpred, NULL, cwait, crid, placement, 0);
}

/* Append a request of the open round to worker w (gen 0, prefill pending). */
static void append_request(orc_cluster* cl, int w, int32_t a, int32_t r, int32_t real,
                           double wait, int64_t rid)
{
    int64_t slot = (int64_t)w * cl->cap + cl->n[w];
    cl->in[slot] = a;
    cl->gen[slot] = 0;
    cl->pred[slot] = r;
    if (cl->tdec) cl->tdec[slot] = 0.0;
    cl->pend[slot] = 1;
    cl->wait[slot] = wait;
    if (cl->rid) cl->rid[slot] = rid;
    if (cl->real) cl->real[slot] = real;
    cl->n[w] += 1;
}

/* Remove slot q of worker w: the worker's last slot moves into it. */
static void remove_slot(orc_cluster* cl, int w, int q)
{
    int64_t slot = (int64_t)w * cl->cap + q;
    int64_t last = (int64_t)w * cl->cap + cl->n[w] - 1;
    cl->in[slot] = cl->in[last];
    cl->gen[slot] = cl->gen[last];
    cl->pred[slot] = cl->pred[last];
    if (cl->tdec) cl->tdec[slot] = cl->tdec[last];
    cl->pend[slot] = cl->pend[last];
    cl->wait[slot] = cl->wait[last];
    if (cl->rid) cl->rid[slot] = cl->rid[last];
    if (cl->real) cl->real[slot] = cl->real[last];
    cl->n[w] -= 1;
}

static int place_round_impl(const orc_params* p, orc_cluster* cl, int32_t C, const int32_t* cin,
                            const int32_t* cpred, const int32_t* creal, const double* cwait,
                            const int64_t* crid, int32_t* placement, int refuse_full)
{
    const int W = cl->W;
    if (p->policy != 0) {
        for (int32_t c = 0; c < C; ++c) {
            int64_t rid = crid ? crid[c] : c;
            int w = pick_by_queue(p, cl, rid);
            if (w < 0 || cl->n[w] >= cl->cap) {
                if (!refuse_full) {
                    for (int32_t k = c; k < C; ++k) placement[k] = -1;
                    return ORC_ERR_CAPACITY;
                }
                placement[c] = -3;
                continue;
            }
            append_request(cl, w, cin[c], cpred[c], creal ? creal[c] : cpred[c],
                           cwait ? cwait[c] : 0.0, rid);
            placement[c] = w;
        }
        return ORC_OK;
    }
    int32_t S = (int32_t)p->K + 2;
    double* T0 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    double* T1 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    int32_t* order = (int32_t*)malloc(sizeof(int32_t) * (size_t)W);
    orc_future* fut = (orc_future*)calloc((size_t)W, sizeof(orc_future));
    uint8_t* have = (uint8_t*)calloc((size_t)W, 1);
    if (!T0 || !T1 || !order || !fut || !have) return ORC_ERR_MEM;
    int rc = ORC_OK;
    /* With groups each group is its own scheduler: a group whose chosen worker
     * has no free slot stops there (that candidate and its later ones stay
     * unplaced) while the other groups go on; the round then reports
     * ORC_ERR_CAPACITY. */
    const int64_t G = p->groups > 1 ? p->groups : 1;
    uint8_t* stopped = G > 1 ? (uint8_t*)calloc((size_t)G, 1) : NULL;
    int cap_hit = 0;
    if (G > 1 && !stopped) return ORC_ERR_MEM;
    for (int32_t c = 0; c < C && rc == ORC_OK; ++c) {
        placement[c] = -1;
        const int64_t rid = crid ? crid[c] : c;
        if (stopped && stopped[rid % G]) continue;
        if (capacity_order(p, cl, order) != ORC_OK) { rc = ORC_ERR_MEM; break; }
        for (int i = 0; i < W; ++i) {
            int w = order[i];
            if (!same_group(p, w, rid)) continue;
            if (!have[w]) {
                if (future_build(cl, w, &fut[w]) != ORC_OK) { rc = ORC_ERR_MEM; break; }
                have[w] = 1;
            }
            orc_pair r;
            eval_pair(p, cl, w, &fut[w], T0, T1, cin[c], cpred[c], cwait ? cwait[c] : 0.0, &r);
            if (r.flags != 15) continue;
            if (cl->n[w] >= cl->cap) {
                if (stopped) {
                    stopped[rid % G] = 1;
                    cap_hit = 1;
                } else {
                    rc = ORC_ERR_CAPACITY;
                }
                break;
            }
            append_request(cl, w, cin[c], cpred[c], creal ? creal[c] : cpred[c],
                           cwait ? cwait[c] : 0.0, crid ? crid[c] : c);
            future_free(&fut[w]);
            have[w] = 0;
            placement[c] = w;
            break;
        }
    }
    for (int w = 0; w < W; ++w)
        if (have[w]) future_free(&fut[w]);
    free(T0);
    free(T1);
    free(order);
    free(fut);
    free(have);
    free(stopped);
    if (rc == ORC_OK && cap_hit) rc = ORC_ERR_CAPACITY;
    return rc;
}

/* ---------------------------------------------------------------------- */
/* Execute every worker from heartbeat time t_now for dt ms (continuous
 * batching, Sec. 2.1): at its next iteration boundary (max(clock, t_now)) a
 * worker first runs the prefill of this round's placements (stalling its
 * decoding requests), then decode iterations back to back while they start
 * before t_now + dt. Finished requests leave; their realized TTFT and ATGT
 * (decode time / decode tokens, Sec. 2.2) are appended to the record arrays
 * (rec_* may be NULL; *nrec counts). On a decode instance (phase 1) the
 * round's placements join the batch at the boundary without a prefill and
 * record no TTFT. viol (nullable, 3 counters) accumulates the realized
 * violations: [0] TTFT above T_pre, [1] ATGT above T_dec (each beyond the
 * relative ORC_SLO_TOL), [2] decode iterations whose KV usage
 * h * context + j * batch exceeds M. With real lengths (cl->real) a request
 * finishes when it has generated its real length; a request that reaches its
 * prediction first is re-predicted (cl->repred) and counted in ev[0] (nullable),
 * an early finish in ev[1]; both update Algorithm 2's per-worker errors
 * (cl->le, cl->be). The realized ATGT divides by the tokens generated.
 * Afterwards off[w] is the time from t_now + dt to the worker's next iteration
 * start. */
int orc_advance(const orc_params* p, orc_cluster* cl, double t_now, double dt,
                int64_t* rec_rid, double* rec_val, uint8_t* rec_kind, int64_t* nrec,
                int64_t rec_cap, int64_t* viol, int64_t* ev)
{
    const double t_end = t_now + dt;
    const int decode = p->phase == 1;
    for (int w = 0; w < cl->W; ++w) {
        const double sc = cl->scale[w];
        const int64_t base = (int64_t)w * cl->cap;
        double start = cl->clock[w] > t_now ? cl->clock[w] : t_now;
        double P = 0.0;
        int any = 0;
        for (int q = 0; q < cl->n[w]; ++q)
            if (cl->pend[base + q]) { P += (double)cl->in[base + q]; any = 1; }
        if (any && decode) {
            for (int q = 0; q < cl->n[w]; ++q) {
                int64_t slot = base + q;
                if (!cl->pend[slot]) continue;
                cl->pend[slot] = 0;
                cl->gen[slot] = 0;
                cl->tdec[slot] = 0.0;
            }
        } else if (any) {
            double tau = sc * (p->k1 * P + p->c1);
            for (int q = 0; q < cl->n[w]; ++q) {
                int64_t slot = base + q;
                if (cl->pend[slot]) {
                    double ttft = cl->wait[slot] + (start - t_now) + tau;
                    if (rec_rid && *nrec < rec_cap) {
                        rec_rid[*nrec] = cl->rid ? cl->rid[slot] : slot;
                        rec_val[*nrec] = ttft;
                        rec_kind[*nrec] = 0;
                    }
                    *nrec += 1;
                    if (viol && ttft > p->T_pre * (1.0 + ORC_SLO_TOL)) viol[0] += 1;
                    cl->pend[slot] = 0;
                    cl->gen[slot] = 0;
                    cl->tdec[slot] = 0.0;
                } else {
                    cl->tdec[slot] += tau;
                }
            }
            start += tau;
        }
        while (cl->n[w] > 0 && start < t_end) {
            int64_t b = cl->n[w], K = 0;
            for (int q = 0; q < cl->n[w]; ++q) K += context(cl, base + q) + 1;
            if (viol && p->h * K + p->j * b > cl->M[w]) viol[2] += 1;
            double t = sc * (p->c3 + p->c2 * (double)b + p->k2 * (double)K);
            for (int q = 0; q < cl->n[w]; ++q) {
                cl->gen[base + q] += 1;
                cl->tdec[base + q] += t;
            }
            start += t;
            /* Prediction errors (Sec. 4.3, Algorithm 2's indicators): a request
             * that reaches its predicted length without finishing is
             * re-predicted (l^e grows by the added length, b^e by one); one
             * that finishes before its prediction lowers l^e by the unused
             * length and b^e by one. */
            for (int q = 0; q < cl->n[w]; ++q) {
                int64_t slot = base + q;
                int32_t real = cl->real ? cl->real[slot] : cl->pred[slot];
                int32_t g = cl->gen[slot];
                if (g >= real) {
                    if (real < cl->pred[slot]) {
                        if (cl->le) cl->le[w] += (int64_t)real - cl->pred[slot];
                        if (cl->be) cl->be[w] -= 1;
                        if (ev) ev[1] += 1;
                    }
                } else if (g >= cl->pred[slot]) {
                    int32_t np = cl->repred ? cl->repred[g] : g + 1;
                    if (np < g + 1) np = g + 1;
                    if ((int64_t)cl->in[slot] + np > p->K) np = (int32_t)(p->K - cl->in[slot]);
                    if (cl->le) cl->le[w] += (int64_t)np - cl->pred[slot];
                    if (cl->be) cl->be[w] += 1;
                    if (ev) ev[0] += 1;
                    cl->pred[slot] = np;
                }
            }
            /* Retire finished requests; the last slot moves into the hole. */
            for (int q = 0; q < cl->n[w];) {
                int64_t slot = base + q;
                int32_t real = cl->real ? cl->real[slot] : cl->pred[slot];
                if (cl->gen[slot] >= real) {
                    double atgt = cl->tdec[slot] / (double)cl->gen[slot];
                    if (rec_rid && *nrec < rec_cap) {
                        rec_rid[*nrec] = cl->rid ? cl->rid[slot] : slot;
                        rec_val[*nrec] = atgt;
                        rec_kind[*nrec] = 1;
                    }
                    *nrec += 1;
                    if (viol && atgt > p->T_dec * (1.0 + ORC_SLO_TOL)) viol[1] += 1;
                    remove_slot(cl, w, q);
                } else {
                    ++q;
                }
            }
        }
        cl->clock[w] = start;
        cl->off[w] = start > t_end ? start - t_end : 0.0;
    }
    return ORC_OK;
}

/* ---------------------------------------------------------------------- */
/* Algorithm 2 (Sec. 4.3, re-balancing with prediction error), run after a
 * placement round and before the round's requests execute. Worker i's errors
 * (l^e_i, b^e_i) define, through Eq. input limit (k2 l + c2 b = T_dec - c3),
 * the line k2 l + c2 b - (k2 l^e_i + c2 b^e_i) = 0 through its error point,
 * parallel to the SLO boundary; its distance to the origin is
 * |e_i| / sqrt(k2^2 + c2^2) with e_i = k2 l^e_i + c2 b^e_i. Moving a new
 * request j (predicted output l_j) from worker x to worker y moves l_j and one
 * request of error from x to y: e_x -= d_j, e_y += d_j with d_j = k2 l_j + c2.
 * The sum of distances is reduced greedily: the round's placements in index
 * order; one on an over-utilized worker (e_x > 0) moves to the under-utilized
 * worker (e_y < 0) that is feasible for it in the current state (all four
 * flags, a free slot) and lowers the sum the most, gain
 * (e_x - e_y) - |e_x - d_j| - |e_y + d_j| > 0; equal gains go to the larger
 * capacity_norm, then the lower index (with grouped scheduling, among the
 * workers of the request's group; its id is crid[c], c if NULL). A moved
 * request leaves its pending
 * slot on x and becomes a pending request of y. placement[] is updated;
 * *moves (nullable) counts the moves, obj (nullable, 2 doubles) receives the
 * sum of distances before and after. */
int orc_rebalance(const orc_params* p, orc_cluster* cl, int32_t C, const int32_t* cin,
                  const int32_t* cpred, const double* cwait, const int64_t* crid,
                  int32_t* placement, const int64_t* le, const int32_t* be, int32_t* moves,
                  double* obj)
{
    const int W = cl->W;
    double* e = (double*)malloc(sizeof(double) * (size_t)W);
    int32_t S = (int32_t)p->K + 2;
    double* T0 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    double* T1 = (double*)malloc(sizeof(double) * ((size_t)S + 2));
    if (!e || !T0 || !T1) return ORC_ERR_MEM;
    const double norm = sqrt(p->k2 * p->k2 + p->c2 * p->c2);
    double before = 0.0;
    for (int i = 0; i < W; ++i) {
        e[i] = p->k2 * (double)le[i] + p->c2 * (double)be[i];
        before += fabs(e[i]) / norm;
    }
    int32_t nmov = 0;
    for (int32_t c = 0; c < C; ++c) {
        int x = placement[c];
        if (x < 0 || !(e[x] > 0.0)) continue;
        double d = p->k2 * (double)cpred[c] + p->c2;
        double wc = cwait ? cwait[c] : 0.0;
        int best = -1;
        double bgain = 0.0, bnorm = 0.0;
        for (int y = 0; y < W; ++y) {
            if (y == x || !(e[y] < 0.0) || cl->n[y] >= cl->cap) continue;
            if (!same_group(p, y, crid ? crid[c] : c)) continue;
            double gain = ((e[x] - e[y]) - fabs(e[x] - d)) - fabs(e[y] + d);
            if (!(gain > 0.0)) continue;
            orc_future f;
            if (future_build(cl, y, &f) != ORC_OK) return ORC_ERR_MEM;
            orc_pair r;
            eval_pair(p, cl, y, &f, T0, T1, cin[c], cpred[c], wc, &r);
            future_free(&f);
            if (r.flags != 15) continue;
            double ny = orc_capacity_norm(p, cl, y);
            if (best < 0 || gain > bgain || (gain == bgain && ny > bnorm)) {
                best = y;
                bgain = gain;
                bnorm = ny;
            }
        }
        if (best < 0) continue;
        /* the request's pending slot on x: the last one with its values */
        int q = -1;
        for (int k = cl->n[x] - 1; k >= 0 && q < 0; --k) {
            int64_t slot = (int64_t)x * cl->cap + k;
            if (cl->pend[slot] && cl->in[slot] == cin[c] && cl->pred[slot] == cpred[c] &&
                cl->wait[slot] == wc)
                q = k;
        }
        if (q < 0) continue;
        int64_t slot = (int64_t)x * cl->cap + q;
        int32_t real = cl->real ? cl->real[slot] : cpred[c];
        int64_t rid = cl->rid ? cl->rid[slot] : c;
        remove_slot(cl, x, q);
        append_request(cl, best, cin[c], cpred[c], real, wc, rid);
        e[x] -= d;
        e[best] += d;
        placement[c] = best;
        nmov += 1;
    }
    double after = 0.0;
    for (int i = 0; i < W; ++i) after += fabs(e[i]) / norm;
    if (moves) *moves = nmov;
    if (obj) {
        obj[0] = before;
        obj[1] = after;
    }
    free(e);
    free(T0);
    free(T1);
    return ORC_OK;
}

/* ---------------------------------------------------------------------- */
/* Serve a request trace with N identical workers (large-scale simulation,
 * Sec. 6.4): heartbeats every H ms; at each, the arrivals so far that are not
 * yet placed form one placement round in arrival order, then every worker
 * executes until the next heartbeat. A request still unplaced whose wait at
 * the next heartbeat plus its prefill alone would exceed T_pre can no longer
 * meet its TTFT: it is counted as failed and dropped. On a decode instance
 * (phase 1) nothing absorbs a wait, so a request not placed at the first
 * heartbeat after its arrival fails (Algorithm 1 would have opened a worker
 * for it). JSQ and power of two place every request at once; one whose
 * worker has no free slot fails. Every realized violation (see orc_advance)
 * also counts as a failure. If drain is set the simulation continues without
 * arrivals until every worker is empty, so that every admitted request's
 * realized TTFT and ATGT are recorded. With real output lengths (rreal,
 * nullable: exact predictions) requests run to their real length and are
 * re-predicted with repred (nullable) when they outgrow a prediction; with
 * p->rebalance, Algorithm 2 (orc_rebalance) runs after every placement round
 * on the errors the execution recorded since the previous heartbeat, which
 * then restart from zero.
 * out[0] failed, out[1] placed, out[2] heartbeats, out[3] max realized TTFT,
 * out[4] max realized ATGT, out[5] realized records, out[6] realized
 * violations (included in out[0]), out[7] re-predictions, out[8] early
 * finishes, out[9] requests moved by Algorithm 2. */
int orc_simulate(const orc_params* p, int32_t N, int32_t cap, int64_t M, double scale,
                 int64_t R, const double* t_arr, const int32_t* rin, const int32_t* rpred,
                 const int32_t* rreal, const int32_t* repred, double H, int32_t stop_at_fail,
                 int32_t drain, double* out)
{
    orc_cluster cl;
    memset(&cl, 0, sizeof(cl));
    cl.W = N;
    cl.cap = cap;
    int64_t* Mv = (int64_t*)malloc(sizeof(int64_t) * (size_t)N);
    double* sv = (double*)malloc(sizeof(double) * (size_t)N);
    cl.off = (double*)calloc((size_t)N, sizeof(double));
    cl.clock = (double*)calloc((size_t)N, sizeof(double));
    cl.n = (int32_t*)calloc((size_t)N, sizeof(int32_t));
    size_t slots = (size_t)N * (size_t)cap;
    cl.in = (int32_t*)calloc(slots, sizeof(int32_t));
    cl.gen = (int32_t*)calloc(slots, sizeof(int32_t));
    cl.pred = (int32_t*)calloc(slots, sizeof(int32_t));
    cl.tdec = (double*)calloc(slots, sizeof(double));
    cl.pend = (uint8_t*)calloc(slots, 1);
    cl.wait = (double*)calloc(slots, sizeof(double));
    cl.rid = (int64_t*)calloc(slots, sizeof(int64_t));
    cl.real = (int32_t*)calloc(slots, sizeof(int32_t));
    cl.le = (int64_t*)calloc((size_t)N, sizeof(int64_t));
    cl.be = (int32_t*)calloc((size_t)N, sizeof(int32_t));
    cl.repred = repred;
    int32_t* creal = (int32_t*)malloc(sizeof(int32_t) * (size_t)(R > 0 ? R : 1));
    int64_t* wl = (int64_t*)malloc(sizeof(int64_t) * (size_t)(R > 0 ? R : 1));
    int32_t* cin = (int32_t*)malloc(sizeof(int32_t) * (size_t)(R > 0 ? R : 1));
    int32_t* cpr = (int32_t*)malloc(sizeof(int32_t) * (size_t)(R > 0 ? R : 1));
    double* cw = (double*)malloc(sizeof(double) * (size_t)(R > 0 ? R : 1));
    int32_t* pl = (int32_t*)malloc(sizeof(int32_t) * (size_t)(R > 0 ? R : 1));
    int64_t rec_cap = 4 * (R > 0 ? R : 1);
    int64_t* rr = (int64_t*)malloc(sizeof(int64_t) * (size_t)rec_cap);
    double* rv = (double*)malloc(sizeof(double) * (size_t)rec_cap);
    uint8_t* rk = (uint8_t*)malloc((size_t)rec_cap);
    if (!Mv || !sv || !cl.off || !cl.clock || !cl.n || !cl.in || !cl.gen || !cl.pred || !cl.tdec ||
        !cl.pend || !cl.wait || !cl.rid || !wl || !cin || !cpr || !cw || !pl || !rr || !rv || !rk ||
        !cl.real || !cl.le || !cl.be || !creal)
        return ORC_ERR_MEM;
    for (int w = 0; w < N; ++w) { Mv[w] = M; sv[w] = scale; }
    cl.M = Mv;
    cl.scale = sv;

    int64_t next = 0, nwait = 0, failed = 0, placed = 0, hb = 0, nrec = 0, violations = 0;
    int64_t events[2] = {0, 0}, moved = 0;
    double max_ttft = 0.0, max_atgt = 0.0;
    int rc = ORC_OK;
    for (;;) {
        double t = (double)hb * H;
        while (next < R && t_arr[next] <= t) wl[nwait++] = next++;
        if (nwait > 0) {
            for (int64_t i = 0; i < nwait; ++i) {
                cin[i] = rin[wl[i]];
                cpr[i] = rpred[wl[i]];
                creal[i] = rreal ? rreal[wl[i]] : rpred[wl[i]];
                cw[i] = t - t_arr[wl[i]];
            }
            rc = place_round_impl(p, &cl, (int32_t)nwait, cin, cpr, creal, cw, wl, pl, 1);
            if (rc != ORC_OK) break;
            if (p->rebalance && p->policy == 0) {
                int32_t mv = 0;
                rc = orc_rebalance(p, &cl, (int32_t)nwait, cin, cpr, cw, wl, pl, cl.le, cl.be,
                                   &mv, NULL);
                if (rc != ORC_OK) break;
                moved += mv;
            }
            int64_t keep = 0;
            for (int64_t i = 0; i < nwait; ++i) {
                if (pl[i] >= 0) { placed++; continue; }
                double tau_alone = scale * (p->k1 * (double)cin[i] + p->c1);
                if (pl[i] == -3 || p->phase == 1 || cw[i] + H + tau_alone > p->T_pre) failed++;
                else wl[keep++] = wl[i];
            }
            nwait = keep;
        }
        if (failed > 0 && stop_at_fail) break;
        int64_t nr0 = nrec;
        int64_t vv[3] = {0, 0, 0};
        for (int w = 0; w < N; ++w) {  /* Algorithm 2's errors restart every heartbeat */
            cl.le[w] = 0;
            cl.be[w] = 0;
        }
        orc_advance(p, &cl, t, H, rr, rv, rk, &nrec, rec_cap, vv, events);
        violations += vv[0] + vv[1] + vv[2];
        failed += vv[0] + vv[1] + vv[2];
        for (int64_t i = nr0; i < nrec && i < rec_cap; ++i) {
            if (rk[i] == 0 && rv[i] > max_ttft) max_ttft = rv[i];
            if (rk[i] == 1 && rv[i] > max_atgt) max_atgt = rv[i];
        }
        if (nrec > rec_cap / 2) nrec = 0; /* records are only used for the maxima */
        hb++;
        if (next >= R && nwait == 0) {
            if (!drain) break;
            int busy = 0;
            for (int w = 0; w < N; ++w) busy |= cl.n[w] > 0;
            if (!busy) break;
        }
    }
    out[0] = (double)failed;
    out[1] = (double)placed;
    out[2] = (double)hb;
    out[3] = max_ttft;
    out[4] = max_atgt;
    out[5] = (double)nrec;
    out[6] = (double)violations;
    out[7] = (double)events[0];
    out[8] = (double)events[1];
    out[9] = (double)moved;
    free(cl.real); free(cl.le); free(cl.be); free(creal);
    free(Mv); free(sv); free(cl.off); free(cl.clock); free(cl.n); free(cl.in); free(cl.gen);
    free(cl.pred); free(cl.tdec); free(cl.pend); free(cl.wait); free(cl.rid);
    free(wl); free(cin); free(cpr); free(cw); free(pl); free(rr); free(rv); free(rk);
    return rc;
}

/* Minimum-worker search (Sec. 4.1, Sec. 6.4): for each worker configuration
 * (GPUs per worker, KV capacity, latency scale) the smallest worker count N in
 * [1, n_max] that serves the whole trace with no failed request, found by
 * doubling then bisection. n_out[o] = -1 if even n_max fails. JSQ and power
 * of two admit without a test, so their runs drain the workers to see every
 * request's realized latencies; best-fit's admitted requests meet them by
 * construction. */
int orc_min_workers(const orc_params* p, int32_t n_opt, const int32_t* gpus, const int64_t* M,
                    const double* scale, int32_t cap, int64_t R, const double* t_arr,
                    const int32_t* rin, const int32_t* rpred, const int32_t* rreal,
                    const int32_t* repred, double H, int32_t n_max, int32_t* n_out)
{
    double out[10];
    const int32_t drain = p->policy != 0;
    for (int o = 0; o < n_opt; ++o) {
        int32_t lo = 0, hi = 1; /* lo fails (or is 0), hi to be tested */
        int found = 0;
        while (hi <= n_max) {
            int rc = orc_simulate(p, hi, cap, M[o], scale[o], R, t_arr, rin, rpred, rreal, repred,
                                  H, 1, drain, out);
            if (rc != ORC_OK) return rc;
            if (out[0] == 0.0) { found = 1; break; }
            lo = hi;
            hi = hi * 2 > n_max && hi < n_max ? n_max : hi * 2;
        }
        if (!found) { n_out[o] = -1; continue; }
        while (hi - lo > 1) {
            int32_t mid = lo + (hi - lo) / 2;
            int rc = orc_simulate(p, mid, cap, M[o], scale[o], R, t_arr, rin, rpred, rreal,
                                  repred, H, 1, drain, out);
            if (rc != ORC_OK) return rc;
            if (out[0] == 0.0) hi = mid;
            else lo = mid;
        }
        n_out[o] = hi;
        (void)gpus;
    }
    return ORC_OK;
}

/* ---------------------------------------------------------------------- */
/* Worker configuration (Sec. 4.1) and the worker-count model (Sec. 5.2).  */

/* Worker configurations from the tensor-parallel model of Sec. 4.1 for
 * N_g GPUs per worker: KV capacity M = N_g m_gpu - m_model, and the latency
 * multiplier of the decode model, the iteration time t_compute + t_comm with
 * t_compute = k4 / N_g + c4 (Eq. TP compute) and t_comm = kc (N_g - 1) / N_g
 * (the all-reduce overhead), relative to one GPU (k4 + c4). */
void orc_tp_config(double k4, double c4, double kc, double m_gpu, double m_model, int32_t g,
                   double* M, double* scale)
{
    double ng = (double)g;
    *M = ng * m_gpu - m_model;
    *scale = (k4 / ng + c4 + kc * (ng - 1.0) / ng) / (k4 + c4);
}

/* Mean KV demand of a running request, "learned from the historical data"
 * (Sec. 4.1, Eq. max throughput): over every decode iteration s = 1..l_pred
 * of every request of a trace, the KV the request holds, h (l_in + s) + j
 * (the footprint vector w of (e)), averaged; l_ave likewise for its context
 * l_in + s. A request counts once per iteration it runs (a time average). */
void orc_trace_demand(const orc_params* p, int64_t R, const int32_t* rin, const int32_t* rpred,
                      double* m_r, double* l_ave)
{
    double kv = 0.0, ctx = 0.0, it = 0.0;
    for (int64_t q = 0; q < R; ++q)
        for (int32_t s = 1; s <= rpred[q]; ++s) {
            kv += (double)(p->h * ((int64_t)rin[q] + s) + p->j);
            ctx += (double)((int64_t)rin[q] + s);
            it += 1.0;
        }
    *m_r = it > 0.0 ? kv / it : 0.0;
    *l_ave = it > 0.0 ? ctx / it : 0.0;
}

/* Eq. max throughput: decode tokens per ms per GPU of a worker of g GPUs,
 * KV capacity M and latency multiplier scale. The batch is bounded by the KV
 * cache, b_kv = M / m_r, and by the ATGT SLO: B, the batch whose iteration
 * scale (c3 + c2 B + k2 B l_ave) equals T_dec (Eq. iter time with the batch's
 * context B l_ave; Eq. input limit). T_max = min(b_kv / (g t(b_kv)),
 * B / (g T_dec)); both batches are kept fractional, as in the equation. */
double orc_max_throughput(const orc_params* p, int32_t g, double M, double scale, double m_r,
                          double l_ave)
{
    double b_kv = M / m_r;
    double t_kv = scale * (p->c3 + p->c2 * b_kv + p->k2 * (b_kv * l_ave));
    double B = (p->T_dec / scale - p->c3) / (p->c2 + p->k2 * l_ave);
    double by_kv = b_kv / ((double)g * t_kv);
    double by_slo = B / ((double)g * p->T_dec);
    return by_kv < by_slo ? by_kv : by_slo;
}

/* The worker configuration of largest T_max (first on ties); T_max of each
 * into tmax (nullable). */
int32_t orc_pick_config(const orc_params* p, int32_t n, const int32_t* gpus, const double* M,
                        const double* scale, double m_r, double l_ave, double* tmax)
{
    int32_t best = -1;
    double bv = 0.0;
    for (int32_t o = 0; o < n; ++o) {
        double v = orc_max_throughput(p, gpus[o], M[o], scale[o], m_r, l_ave);
        if (tmax) tmax[o] = v;
        if (best < 0 || v > bv) {
            best = o;
            bv = v;
        }
    }
    return best;
}

/* Eq. total_worker_pre: N_w = ceil(k5 r_a + c5) for arrival rates above R.
 * k5, c5 by ordinary least squares over the (rate, minimum workers) points
 * whose rate exceeds R. Returns the number of points used (< 2, or all rates
 * equal: no fit, k5 = c5 = 0). */
int32_t orc_fit_workers(int32_t n, const double* rate, const int32_t* nw, double R, double* k5,
                        double* c5)
{
    double m = 0.0, sx = 0.0, sy = 0.0, sxx = 0.0, sxy = 0.0;
    for (int32_t k = 0; k < n; ++k) {
        if (!(rate[k] > R)) continue;
        m += 1.0;
        sx += rate[k];
        sy += (double)nw[k];
        sxx += rate[k] * rate[k];
        sxy += rate[k] * (double)nw[k];
    }
    double den = m * sxx - sx * sx;
    if (m < 2.0 || !(den > 0.0)) {
        *k5 = 0.0;
        *c5 = 0.0;
        return (int32_t)m;
    }
    *k5 = (m * sxy - sx * sy) / den;
    *c5 = (sy - *k5 * sx) / m;
    return (int32_t)m;
}

int64_t orc_predict_workers(double k5, double c5, double rate)
{
    return (int64_t)ceil(k5 * rate + c5);
}

/* Appendix A, Eq. group_arrival_limit: the number G of scheduling groups of
 * distributed scheduling. Round-robin dealing gives group i the rate
 * r_i = rate_a / G and n_workers / G workers. Its scheduler must place
 * r_i within the latency limit T_s (r_i <= r(T_s) = rate_max), and the
 * group must keep at least 1 / (2e) workers, so that about half of the groups
 * needing one extra worker costs at most a fraction e of extra workers (the
 * printed lower bound stands on r_i; it is read as the workers per group the
 * text derives). Both conditions multiplied out: rate_a <= G rate_max and
 * 2 e n_workers >= G. The fewest such groups (the least extra workers), by
 * enumeration over G = 1 .. n_workers; 0 if none. */
int64_t orc_pick_groups(double rate_a, double rate_max, double e, int64_t n_workers)
{
    for (int64_t G = 1; G <= n_workers; ++G) {
        const int fast_enough = rate_a <= (double)G * rate_max;
        const int enough_workers = 2.0 * e * (double)n_workers >= (double)G;
        if (fast_enough && enough_workers) return G;
    }
    return 0;
}
