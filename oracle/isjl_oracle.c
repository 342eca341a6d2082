/*
 * isjl_oracle.c -- CPU oracle for the batched FCFS / LJF / ISJL simulator.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, step-by-step
 * statement of what the scheduling model of "Efficiency and Cost Alignment in
 * Batched LLM Serving via Resource-Fair Scheduling" computes.  Only the tests,
 * the package's smoke check and the benchmark's CPU-baseline leg may load it.
 * It shares no code, header, table or helper with the CUDA path.
 *
 * Model (Section 2, "Model"): request i needs o_i = prompt_i + output_i
 * tokens, processed one token per step; at most B requests run in a step;
 * progress a_i is the KV footprint; the fairness constraint (Eq. 1) bounds
 * max a - min a over the running set by the budget alpha (called delta here).
 * Service is contiguous: a started request runs every step until done
 * (integer program of Appendix A, constraint (2)).
 *
 * Cost (Section 5, Eq. batch-cost-progress): a nonempty step costs
 * c + tau*|S|*max r with r_i = a_i + 1.  Decomposition (Theorem "Profit
 * decomposition"): total = tau*Q + c*T + tau*E with Q = sum o(o+1)/2 and
 * E = sum over steps of sum_{i in S}(max r - r_i).
 *
 * Readings where the paper is silent:
 *   - KV cap: a running request reserves its peak footprint o_i; a start needs
 *     sum_{S} o_j + o_i <= kv_cap.  kv_cap = INT32_MAX is the paper's model.
 *   - In every policy the first KV failure ends all starts of that step.
 *   - "Longest" = (o descending, index ascending); arrival order = index order.
 *   - A request started in step k runs in step k; completion c_i = (last step
 *     it ran) + 1; T_busy counts nonempty steps, T_make = max c_i.
 *   - ISJL: see isjl_admit() below.
 *   - Robust-ISJL (Section 3.3): with an upper-bound slack e_i >= 0 the
 *     policies plan with u_i = o_i + e_i (sorting, M, cap_j, packs, Phase TWO
 *     order, KV reservation of u_i); requests still finish after o_i tokens
 *     and the gate uses their true progress.  e = 0 is the clairvoyant case.
 *
 * Parity unpinned (nothing the paper fixes decides these parts; the tests check
 * them only by invariants and hand-derived schedules):
 *   - the KV cap: beyond "sum of reservations <= kv_cap at every step" and the
 *     kv_cap = INT32_MAX reductions, the paper gives no value to compare with;
 *   - ISJL at 0 < alpha < infinity with B >= 3 when a pack holds a request
 *     longer than alpha, so that the gate can hold a plan entry back: pinned
 *     only by hand-derived worked examples, and it misses the 3/4 bound of the
 *     competitive-ratio theorem for Algorithm 2 on recorded tiny instances.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_FCFS 0
#define OR_LJF  1
#define OR_ISJL 2
#define OR_SJF  3   /* shortest first, continuous batching (Section 6 baseline) */
#define OR_ISJL_BETA 4   /* Algorithm "ISJL" with beta = (sqrt(17) - 1) / 4 * alpha */

#define OR_OK            0
#define OR_INVALID_ARG   1
#define OR_INFEASIBLE    2
#define OR_OOM           3
#define OR_STEP_LIMIT    5

#define ST_WAIT    0   /* not started, not in a plan (released or not) */
#define ST_PLANNED 1   /* placed in an ISJL Phase ONE plan, not started */
#define ST_RUN     2
#define ST_DONE    3

typedef struct {
    int64_t T_make, T_busy, O, Q, W, E, token_adv;
    int64_t sum_completion, sum_latency, sum_extent, max_extent;
    int64_t violations, kv_violations, peak_kv, peak_batch, status;
    double c_T, tau_Q, tau_E, cost, revenue, profit, throughput, ael;
} or_record;

typedef struct {
    int n, B, policy;
    int64_t alpha, beta, kv_cap;
    const int32_t *arr;
    int32_t *o;               /* planning length u_i (= o_i without predictions) */
    int32_t *ot;              /* true length o_i */
    int32_t *status, *a, *start, *compl;
    int32_t *by_len;          /* job ids sorted by (o desc, idx asc) */
    /* running set */
    int32_t *run;  int run_cnt;  int64_t kv_sum;
    /* FCFS */
    int next_fcfs;
    /* ISJL workers, 1-based: worker_job[j] running job or -1; plan FIFO */
    int32_t *worker_job, *plan_head, *plan_tail, *plan_next, *job_worker;
    int64_t plan_left;
    int64_t t0, d1;
    int32_t L1;               /* o_1 of the current stage (worker 1) */
    int32_t *long_of;         /* long_of[j]: o_j planned on worker j, 2..M */
    int flags;                /* ISJL reading variants (0 = the specified readings) */
    int broke;                /* the gate kept a free worker from a queued request */
} sim_t;

/* ---- sorting by (o desc, idx asc) --------------------------------------- */
static const int32_t *g_sort_o;
static int cmp_len(const void *x, const void *y) {
    int32_t i = *(const int32_t *)x, j = *(const int32_t *)y;
    if (g_sort_o[i] != g_sort_o[j]) return g_sort_o[i] > g_sort_o[j] ? -1 : 1;
    return i < j ? -1 : (i > j);
}

static int64_t min64(int64_t x, int64_t y) { return x < y ? x : y; }
static int64_t max64(int64_t x, int64_t y) { return x > y ? x : y; }

/* ---- common start / helpers ---------------------------------------------- */
static void start_job(sim_t *s, int32_t i, int64_t k, int worker) {
    s->status[i] = ST_RUN;
    s->a[i] = 0;
    s->start[i] = (int32_t)k;
    s->run[s->run_cnt++] = i;
    s->kv_sum += s->o[i];
    if (s->policy == OR_ISJL) { s->worker_job[worker] = i; s->job_worker[i] = worker; }
}

/* longest released request that is neither running, done nor planned */
static int32_t longest_waiting(const sim_t *s, int64_t k) {
    for (int p = 0; p < s->n; ++p) {
        int32_t i = s->by_len[p];
        if (s->status[i] == ST_WAIT && s->arr[i] <= k) return i;
    }
    return -1;
}

/* A_max(k): largest progress among running requests (0 when none run) */
static int64_t a_max(const sim_t *s) {
    int64_t m = 0;
    for (int q = 0; q < s->run_cnt; ++q) m = max64(m, s->a[s->run[q]]);
    return m;
}

/* beta = floor((sqrt(17) - 1) / 4 * alpha), exactly: the largest m >= 0 with
 * 4m + alpha <= alpha * sqrt(17), i.e. (4m + alpha)^2 <= 17 alpha^2.  Only
 * floor(beta) matters: o_1 - o_2 + beta is compared with integer sums. */
static int64_t beta_of(int64_t alpha) {
    if (alpha > 1000000) return alpha;           /* no plan can exist: o <= 65535 < alpha */
    int64_t m = (int64_t)(0.780776406404415 * (double)alpha);
    while (m > 0 && (4 * m + alpha) * (4 * m + alpha) > 17 * alpha * alpha) m--;
    while ((4 * (m + 1) + alpha) * (4 * (m + 1) + alpha) <= 17 * alpha * alpha) m++;
    return m;
}

/* shortest released request that is neither running, done nor planned */
static int32_t shortest_waiting(const sim_t *s, int64_t k) {
    for (int p = s->n - 1; p >= 0; --p) {
        int32_t i = s->by_len[p];
        if (s->status[i] == ST_WAIT && s->arr[i] <= k) {
            /* among equal lengths the lower index goes first */
            int32_t best = i;
            for (int q = p - 1; q >= 0 && s->o[s->by_len[q]] == s->o[i]; --q) {
                int32_t j = s->by_len[q];
                if (s->status[j] == ST_WAIT && s->arr[j] <= k) best = j;
            }
            return best;
        }
    }
    return -1;
}

/* ---- SJF (Section 2.1 example, continuous-batching remark; Section 6) ----- */
/* Each step admit released requests shortest first (ties: lower index) while
 * a slot is free and the KV reservation fits; the first that does not fit
 * ends admissions.  No fairness gate. */
static void sjf_admit(sim_t *s, int64_t k) {
    while (s->run_cnt < s->B) {
        int32_t i = shortest_waiting(s, k);
        if (i < 0) break;
        if (s->kv_sum + s->o[i] > s->kv_cap) break;
        start_job(s, i, k, 0);
    }
}

/* ---- FCFS (Section 2.1 example, continuous-batching remark) -------------- */
/* Each step admit released requests in arrival (= index) order while a slot
 * is free and the KV reservation fits; the first request that does not fit
 * ends admissions, so requests never overtake each other.  FCFS ignores the
 * fairness budget: it is the unconstrained baseline. */
static void fcfs_admit(sim_t *s, int64_t k) {
    while (s->run_cnt < s->B && s->next_fcfs < s->n && s->arr[s->next_fcfs] <= k) {
        int32_t i = s->next_fcfs;
        if (s->kv_sum + s->o[i] > s->kv_cap) break;
        start_job(s, i, k, 0);
        s->next_fcfs++;
    }
}

/* ---- LJF (Algorithm 1, static batching remark) -------------------------- */
/* When nothing runs, form a batch of the longest released requests (at most
 * B, stopping at the first KV failure) and hold it until every member is
 * done.  Offline with no KV cap this is exactly Algorithm 1's consecutive
 * groups o_1..o_B, o_{B+1}..o_{2B}, ... */
static void ljf_admit(sim_t *s, int64_t k) {
    if (s->run_cnt != 0) return;
    while (s->run_cnt < s->B) {
        int32_t i = longest_waiting(s, k);
        if (i < 0) break;
        if (s->kv_sum + s->o[i] > s->kv_cap) break;
        start_job(s, i, k, 0);
    }
}

/* ---- ISJL (Algorithm 2 with beta = alpha; online rolling form, Sec. 3.4) - */
/*
 * State: every worker is running a request, holds plan entries (reserved) or
 * is free.  A stage starts when nothing runs, no plan entry is left and the
 * released queue Q(k) is nonempty.  Phase ONE then fixes a plan: worker 1
 * gets the longest request o_1, to be started d1 steps after the stage start;
 * worker j in 2..M gets a pack of shorter requests followed by the j-th
 * longest request o_j; workers beyond M get a pack only.  Every start, planned
 * or not, needs the fairness gate A_max(k) <= alpha (Eq. 1: a request starts
 * at progress 0, so the gap it opens is the largest running progress) and the
 * KV reservation.  Phase TWO gives free workers the longest released request.
 *
 * The reading variants below exist only for the reading study (each is off by
 * default and none is part of the specified path):
 */
#define V_NO_WAIT_O1     1    /* o_j may start before o_1 has started */
#define V_D1_LAST        2    /* d1 from the pack of worker M alone */
#define V_P2_RESERVED    4    /* Phase TWO may use a worker whose plan entry waits */
#define V_REBUILD_REOPEN 8    /* new Phase ONE once the gate reopens after stopping Phase TWO */
#define V_LITERAL_LONG  16    /* o_2..o_M are not planned: packs scan every shorter request, Phase TWO starts the rest */
#define V_SHORT_PACKS   32    /* packs take only requests with o <= alpha */
#define V_CANCEL        64    /* a plan stopped by the gate goes back to the queue */
#define V_WAIVER       128    /* o_1's delay is skipped at a later step that finds nothing running */
#define V_UNGATED_PLAN 256    /* plan entries start without the gate (breaks Eq. 1; for contrast) */

static void plan_append(sim_t *s, int j, int32_t i) {
    s->status[i] = ST_PLANNED;
    s->plan_next[i] = -1;
    if (s->plan_head[j] < 0) s->plan_head[j] = i; else s->plan_next[s->plan_tail[j]] = i;
    s->plan_tail[j] = i;
    s->plan_left++;
}

/* Phase ONE over the workers wk[0..nw-1] (wk[0] plays worker 1, wk[j-1]
 * worker j).  Returns 1 if a plan was made, 0 if the stage goes straight to
 * Phase TWO (|Q| = 1, or the second longest request is no longer than alpha). */
static int isjl_phase_one(sim_t *s, int64_t k, const int32_t *wk, int nw, int32_t *Q, int64_t *packsum,
                          int64_t *budget, int32_t *visit) {
    const int64_t al = s->alpha;
    const int64_t be = s->beta;   /* beta = alpha (Algorithm 2), or Algorithm "ISJL"'s beta */
    int q = 0;
    for (int p = 0; p < s->n; ++p) {            /* Q(k) longest first, ties by index */
        int32_t i = s->by_len[p];
        if (s->status[i] == ST_WAIT && s->arr[i] <= k) Q[q++] = i;
    }
    s->t0 = k;
    s->d1 = 0;
    s->L1 = -1;
    if (q < 2 || (int64_t)s->o[Q[1]] <= al) return 0;

    /* M: how many of the B workers take a long request (o > alpha) */
    int n_long = 0;
    for (int p = 0; p < q && n_long < nw; ++p) if ((int64_t)s->o[Q[p]] > al) n_long++;
    const int64_t o1 = s->o[Q[0]];
    /* a pack member is at most theta = min{2 alpha, o_1 - o_M + beta} long
     * (for the short-packs variant also at most alpha) */
    int64_t theta = min64(2 * al, o1 - (int64_t)s->o[Q[n_long - 1]] + be);
    if (s->flags & V_SHORT_PACKS) theta = min64(theta, al);

    /* pack budgets: alpha on a worker without a long request; on worker j
     * (2 <= j <= M) the room that lets o_j still end within beta of o_1,
     * capped at 2 alpha.  Visiting order of the first fit: the workers without
     * a long request first, then the long ones from o_M back to o_2. */
    int nv = 0;
    for (int j = 1; j <= nw; ++j) { packsum[j] = 0; budget[j] = -1; }
    for (int j = n_long + 1; j <= nw; ++j) { budget[j] = al; visit[nv++] = j; }
    for (int j = n_long; j >= 2; --j) {
        budget[j] = min64(2 * al, o1 - (int64_t)s->o[Q[j - 1]] + be);
        visit[nv++] = j;
    }
    const int literal = (s->flags & V_LITERAL_LONG) != 0;
    s->status[Q[0]] = ST_PLANNED;
    if (!literal) for (int p = 1; p < n_long; ++p) s->status[Q[p]] = ST_PLANNED;

    /* first fit, longest candidate first; a candidate that fits nowhere stays queued */
    for (int p = literal ? 1 : n_long; p < q; ++p) {
        int32_t i = Q[p];
        int64_t oi = s->o[i];
        if (oi > theta) continue;
        for (int v = 0; v < nv; ++v) {
            int j = visit[v];
            if (packsum[j] + oi <= budget[j]) { plan_append(s, wk[j - 1], i); packsum[j] += oi; break; }
        }
    }
    /* worker 1 holds o_1; worker j (2..M) runs o_j after its pack */
    plan_append(s, wk[0], Q[0]);
    s->L1 = Q[0];
    for (int j = 0; j <= s->B; ++j) s->long_of[j] = -1;
    if (!literal)
        for (int j = 2; j <= n_long; ++j) { plan_append(s, wk[j - 1], Q[j - 1]); s->long_of[wk[j - 1]] = Q[j - 1]; }

    /* d1: the smallest delay after which o_1's progress is at most alpha when
     * the longest pack ends, min{max{max_j sum(w_j) - alpha, 0}, alpha} over
     * j = 2..M (the last-pack variant uses worker M's pack alone) */
    int64_t mx = 0;
    if (s->flags & V_D1_LAST) mx = n_long >= 2 ? packsum[n_long] : 0;
    else for (int j = 2; j <= n_long; ++j) mx = max64(mx, packsum[j]);
    s->d1 = min64(max64(mx - al, 0), al);
    return 1;
}

static int worker_free(const sim_t *s, int j) { return s->worker_job[j] < 0 && s->plan_head[j] < 0; }

/* ISJL admission for step k:
 *   1. a stage start runs Phase ONE;
 *   2. plan starts, workers 1..B in order: a worker that is not running starts
 *      its next plan entry if the gate and the KV reservation allow it; o_1
 *      also waits until k >= t0 + d1, and o_j (j >= 2) until o_1 has started
 *      (the pack runs alone, o_1 joins it, o_j follows the pack alongside
 *      o_1 -- Section 3.2's order, kept by Section 3.3's stages, which hold
 *      o_1 on worker 1 while the packs run).  An entry that cannot start
 *      waits on its worker;
 *   3. Phase TWO: while a worker is free, Q(k) is nonempty and the gate is
 *      open, the longest released request starts on the lowest free worker.
 * The first KV failure ends the step's starts.  Requests arriving during a
 * stage only join Q(k).  Starts have progress 0, so A_max(k) is the same for
 * every start of the step. */
static void isjl_admit(sim_t *s, int64_t k, int32_t *Q, int64_t *packsum, int64_t *budget, int32_t *wk) {
    const int nothing_runs = (s->run_cnt == 0);
    const int64_t amax = a_max(s);
    const int reopen = (s->flags & V_REBUILD_REOPEN) && s->broke && !nothing_runs && amax <= s->alpha;
    if (s->plan_left == 0 && (nothing_runs || reopen) && longest_waiting(s, k) >= 0) {
        int nw = 0;
        if (nothing_runs) {
            for (int j = 1; j <= s->B; ++j) wk[nw++] = j;
        } else {
            for (int j = 1; j <= s->B; ++j) if (worker_free(s, j)) wk[nw++] = j;
        }
        if (nw > 0) {
            isjl_phase_one(s, k, wk, nw, Q, packsum, budget, wk + s->B + 1);
            s->broke = 0;
        }
    }

    const int gate_ok = amax <= s->alpha;
    int stop = 0;
    for (int j = 1; j <= s->B && !stop; ++j) {
        int32_t e = s->plan_head[j];
        if (e < 0 || s->worker_job[j] >= 0) continue;
        if (!gate_ok && !(s->flags & V_UNGATED_PLAN)) {
            stop = 1;
            if (s->flags & V_CANCEL) {             /* the plan goes back to the queue */
                for (int w = 1; w <= s->B; ++w) {
                    for (int32_t x = s->plan_head[w]; x >= 0; x = s->plan_next[x]) s->status[x] = ST_WAIT;
                    s->plan_head[w] = s->plan_tail[w] = -1;
                    s->long_of[w] = -1;
                }
                s->plan_left = 0;
                s->L1 = -1;
            }
            break;
        }
        if (e == s->L1) {
            int over = k >= s->t0 + s->d1;
            if ((s->flags & V_WAIVER) && k > s->t0 && nothing_runs) over = 1;
            if (!over) continue;
        }
        if (e == s->long_of[j] && s->L1 >= 0 && s->status[s->L1] == ST_PLANNED && !(s->flags & V_NO_WAIT_O1))
            continue;
        if (s->kv_sum + s->o[e] > s->kv_cap) { stop = 1; break; }
        s->plan_head[j] = s->plan_next[e];
        if (s->plan_head[j] < 0) s->plan_tail[j] = -1;
        s->plan_left--;
        start_job(s, e, k, j);
    }
    if (stop || !gate_ok) {
        /* a free worker and a queued request that the closed gate keeps apart */
        if ((s->flags & V_REBUILD_REOPEN) && !gate_ok && longest_waiting(s, k) >= 0)
            for (int j = 1; j <= s->B; ++j) if (worker_free(s, j)) { s->broke = 1; break; }
        return;
    }

    for (;;) {
        int w = -1;
        for (int j = 1; j <= s->B && w < 0; ++j) if (worker_free(s, j)) w = j;
        if (w < 0 && (s->flags & V_P2_RESERVED))
            for (int j = 1; j <= s->B && w < 0; ++j) if (s->worker_job[j] < 0) w = j;
        if (w < 0) break;
        int32_t i = longest_waiting(s, k);
        if (i < 0) break;
        if (s->kv_sum + s->o[i] > s->kv_cap) break;
        start_job(s, i, k, w);
    }
}

/* ---- the run ------------------------------------------------------------- */
/* Simulate one instance under one policy.  delta is the fairness budget
 * (INT32_MAX = no constraint; ignored by FCFS and LJF except for counting
 * violations).  start_out/compl_out may be NULL.  Returns the status. */
int oracle_run_v(int policy, int B, int64_t delta, int64_t kv_cap, int n,
                 const int32_t *arrival, const int32_t *prompt, const int32_t *output, const int32_t *slack,
                 double c, double tau, double p0, int64_t max_steps, int flags,
                 int32_t *start_out, int32_t *compl_out, or_record *rec)
{
    memset(rec, 0, sizeof(*rec));
    if (n < 0 || B < 1 || delta < 0 || kv_cap < 1 || policy < 0 || policy > 4 || (n > 0 && (!arrival || !prompt || !output))) {
        rec->status = OR_INVALID_ARG; return OR_INVALID_ARG;
    }
    if (n == 0) return OR_OK;   /* an empty instance: nothing runs, every counter is 0 */
    for (int i = 0; i < n; ++i) {
        if (arrival[i] < 0 || prompt[i] < 0 || output[i] < 0 || (slack && slack[i] < 0) ||
            (i > 0 && arrival[i] < arrival[i - 1])) {
            rec->status = OR_INVALID_ARG; return OR_INVALID_ARG;
        }
    }
    sim_t S; memset(&S, 0, sizeof(S));
    sim_t *s = &S;
    s->n = n; s->B = B; s->policy = policy == OR_ISJL_BETA ? OR_ISJL : policy; s->alpha = delta;
    s->beta = policy == OR_ISJL_BETA ? beta_of(delta) : delta;
    s->kv_cap = kv_cap; s->arr = arrival; s->flags = flags;
    policy = s->policy;
    s->o = malloc(sizeof(int32_t) * n);
    s->ot = malloc(sizeof(int32_t) * n);
    s->status = malloc(sizeof(int32_t) * n);
    s->a = malloc(sizeof(int32_t) * n);
    s->start = malloc(sizeof(int32_t) * n);
    s->compl = malloc(sizeof(int32_t) * n);
    s->by_len = malloc(sizeof(int32_t) * n);
    s->run = malloc(sizeof(int32_t) * (size_t)(B < n ? B : n) + sizeof(int32_t));
    int32_t *Q = malloc(sizeof(int32_t) * n);
    int64_t *packsum = malloc(sizeof(int64_t) * (size_t)(B + 1));
    int64_t *budget = malloc(sizeof(int64_t) * (size_t)(B + 1));
    int32_t *wk = malloc(sizeof(int32_t) * (size_t)(2 * B + 2));   /* stage workers, then the first-fit order */
    s->worker_job = malloc(sizeof(int32_t) * (size_t)(B + 1));
    s->plan_head = malloc(sizeof(int32_t) * (size_t)(B + 1));
    s->plan_tail = malloc(sizeof(int32_t) * (size_t)(B + 1));
    s->plan_next = malloc(sizeof(int32_t) * n);
    s->job_worker = malloc(sizeof(int32_t) * n);
    s->long_of = malloc(sizeof(int32_t) * (size_t)(B + 1));
    int status = OR_OK;
    if (!s->o || !s->ot || !s->status || !s->a || !s->start || !s->compl || !s->by_len || !s->run || !Q ||
        !packsum || !budget || !wk || !s->worker_job || !s->plan_head || !s->plan_tail || !s->plan_next || !s->job_worker || !s->long_of) {
        status = OR_OOM; goto done;
    }

    /* o_i = prompt + output (Section 2: prompt and output tokens, one per step) */
    int64_t O = 0, Qsum = 0, sumA = 0, maxA = 0;
    for (int i = 0; i < n; ++i) {
        int64_t oi = (int64_t)prompt[i] + output[i];
        int64_t ui = oi + (slack ? slack[i] : 0);           /* planning length u_i >= o_i */
        if (oi < 1 || ui > kv_cap || ui > INT32_MAX / 2) { status = OR_INFEASIBLE; goto done; }
        s->o[i] = (int32_t)ui;
        s->ot[i] = (int32_t)oi;
        O += oi;
        Qsum += oi * (oi + 1) / 2;          /* Eq. intrinsic-resource-cost */
        sumA += arrival[i];
        if (arrival[i] > maxA) maxA = arrival[i];
        s->status[i] = ST_WAIT; s->a[i] = 0; s->start[i] = -1; s->compl[i] = -1;
        s->by_len[i] = i; s->plan_next[i] = -1; s->job_worker[i] = -1;
    }
    g_sort_o = s->o;
    qsort(s->by_len, (size_t)n, sizeof(int32_t), cmp_len);
    for (int j = 0; j <= B; ++j) {
        s->worker_job[j] = -1; s->plan_head[j] = -1; s->plan_tail[j] = -1; s->long_of[j] = -1;
    }
    if (max_steps <= 0) max_steps = O + maxA + 1;

    int done_cnt = 0;
    int64_t W = 0, E = 0, T_busy = 0, tok = 0, sum_ext = 0, max_ext = 0, viol = 0, kv_viol = 0;
    int64_t peak_kv = 0, peak_b = 0, T_make = 0, sum_c = 0;
    for (int64_t k = 0;; ++k) {
        if (k > max_steps) { status = OR_STEP_LIMIT; break; }
        /* retire: requests whose progress reached o_i in step k-1 */
        int w = 0;
        for (int q = 0; q < s->run_cnt; ++q) {
            int32_t i = s->run[q];
            if (s->a[i] == s->ot[i]) {
                s->status[i] = ST_DONE;
                s->compl[i] = (int32_t)k;
                s->kv_sum -= s->o[i];
                done_cnt++;
                sum_c += k;
                if (k > T_make) T_make = k;
                if (policy == OR_ISJL) s->worker_job[s->job_worker[i]] = -1;
            } else {
                s->run[w++] = i;
            }
        }
        s->run_cnt = w;
        if (done_cnt == n) break;

        /* admission */
        if (policy == OR_FCFS) fcfs_admit(s, k);
        else if (policy == OR_LJF) ljf_admit(s, k);
        else if (policy == OR_SJF) sjf_admit(s, k);
        else isjl_admit(s, k, Q, packsum, budget, wk);

        /* serve step k: every running request processes token r_i = a_i + 1 */
        if (s->run_cnt > 0) {
            int64_t m = 0, mn = INT64_MAX, kvs = 0;
            for (int q = 0; q < s->run_cnt; ++q) {
                int64_t r = (int64_t)s->a[s->run[q]] + 1;
                if (r > m) m = r;
                if (r < mn) mn = r;
                kvs += s->o[s->run[q]];
            }
            int64_t cnt = s->run_cnt;
            W += cnt * m;                                   /* |S| * max r   */
            for (int q = 0; q < s->run_cnt; ++q)            /* sum (max r - r_i) */
                E += m - ((int64_t)s->a[s->run[q]] + 1);
            int64_t ext = m - mn;                           /* Eq. 1 left side */
            sum_ext += ext;
            if (ext > max_ext) max_ext = ext;
            if (ext > delta) viol++;
            if (kvs > kv_cap) kv_viol++;
            if (kvs > peak_kv) peak_kv = kvs;
            if (cnt > peak_b) peak_b = cnt;
            for (int q = 0; q < s->run_cnt; ++q) s->a[s->run[q]] += 1;
            T_busy++;
            tok += cnt;
        }
    }

    rec->T_make = T_make; rec->T_busy = T_busy; rec->O = O; rec->Q = Qsum; rec->W = W; rec->E = E;
    rec->token_adv = tok; rec->sum_completion = sum_c; rec->sum_latency = sum_c - sumA;
    rec->sum_extent = sum_ext; rec->max_extent = max_ext; rec->violations = viol;
    rec->kv_violations = kv_viol; rec->peak_kv = peak_kv; rec->peak_batch = peak_b;
    /* cost decomposition C = tau Q + c T + tau E, profit = p0 O - C (Theorem
     * "Profit decomposition"); evaluated in this order, without contraction */
    rec->c_T = c * (double)T_busy;
    rec->tau_Q = tau * (double)Qsum;
    rec->tau_E = tau * (double)E;
    rec->cost = (rec->c_T + rec->tau_Q) + rec->tau_E;
    rec->revenue = p0 * (double)O;
    rec->profit = rec->revenue - rec->cost;
    rec->throughput = T_make > 0 ? (double)O / (double)T_make : 0.0;
    rec->ael = (double)sum_c / (double)n;
    if (start_out) memcpy(start_out, s->start, sizeof(int32_t) * n);
    if (compl_out) memcpy(compl_out, s->compl, sizeof(int32_t) * n);
done:
    rec->status = status;
    free(s->o); free(s->ot); free(s->status); free(s->a); free(s->start); free(s->compl); free(s->by_len);
    free(s->run); free(Q); free(packsum); free(budget); free(wk); free(s->worker_job); free(s->plan_head);
    free(s->plan_tail); free(s->plan_next); free(s->job_worker); free(s->long_of);
    return status;
}

/* The run with the specified readings (no variant flags). */
int oracle_run(int policy, int B, int64_t delta, int64_t kv_cap, int n,
               const int32_t *arrival, const int32_t *prompt, const int32_t *output, const int32_t *slack,
               double c, double tau, double p0, int64_t max_steps,
               int32_t *start_out, int32_t *compl_out, or_record *rec)
{
    return oracle_run_v(policy, B, delta, kv_cap, n, arrival, prompt, output, slack, c, tau, p0, max_steps, 0,
                        start_out, compl_out, rec);
}

/* Run many instances (row-major, n per row) under one (policy, delta) and
 * the ISJL reading variants `flags` (0: the specified readings).
 * rec has n_inst entries; start_out/compl_out are n_inst*n or NULL.
 * Returns the first nonzero status, else 0. */
int oracle_run_batch_v(int policy, int B, int64_t delta, int64_t kv_cap, int n_inst, int n,
                       const int32_t *arrival, const int32_t *prompt, const int32_t *output, const int32_t *slack,
                       double c, double tau, double p0, int64_t max_steps, int flags,
                       int32_t *start_out, int32_t *compl_out, or_record *rec)
{
    int first = 0;
    for (int t = 0; t < n_inst; ++t) {
        size_t off = (size_t)t * (size_t)n;
        int st = oracle_run_v(policy, B, delta, kv_cap, n, arrival + off, prompt + off, output + off,
                              slack ? slack + off : NULL, c, tau, p0, max_steps, flags,
                              start_out ? start_out + off : NULL, compl_out ? compl_out + off : NULL, rec + t);
        if (st && !first) first = st;
    }
    return first;
}

/* Run many instances under one (policy, delta) with the specified readings. */
int oracle_run_batch(int policy, int B, int64_t delta, int64_t kv_cap, int n_inst, int n,
                     const int32_t *arrival, const int32_t *prompt, const int32_t *output, const int32_t *slack,
                     double c, double tau, double p0, int64_t max_steps,
                     int32_t *start_out, int32_t *compl_out, or_record *rec)
{
    return oracle_run_batch_v(policy, B, delta, kv_cap, n_inst, n, arrival, prompt, output, slack, c, tau, p0,
                              max_steps, 0, start_out, compl_out, rec);
}

int oracle_record_size(void) { return (int)sizeof(or_record); }
int64_t oracle_beta(int64_t alpha) { return beta_of(alpha); }
