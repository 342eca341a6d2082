/*
 * opt_dp.c -- exact offline optimum of the fair batch-scheduling problem.
 *
 * TEST INFRASTRUCTURE ONLY (see isjl_oracle.c).  It defines OPT for the tiny
 * competitive-ratio checks by searching the schedules that the integer
 * program of Appendix A admits:
 *   (1) every request starts exactly once (at or after its release time),
 *   (2) it then runs contiguously for o_i steps,
 *   (3) at most B requests run in a step,
 *   (6) any two requests that run in the same step have progress within alpha,
 * plus, as in the simulator's reading, the KV reservation: the o_i of the
 * requests running in a step sum to at most kv_cap.  Deliberate waiting is
 * allowed (any start time is a decision).  The objective is the makespan.
 *
 * Method: breadth-first search over time.  A state lists, per request, "not
 * started", its progress while running, or "done".  From each state every
 * subset X of released, unstarted requests may start, subject to (3), the
 * KV reservation and (6) (a starting request has progress 0, so (6) needs
 * max progress of the running requests <= alpha when X is nonempty; pairs of
 * running requests keep their gap because they advance in lockstep).  Then
 * every running request advances one token.  The first level that reaches
 * "all done" is the optimal makespan.  Exponential; for n <= 9 requests of
 * length <= 62 only.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define BITS 6
#define CODE_NEW 0u
#define CODE_DONE 63u

typedef struct { uint64_t *keys; size_t cap, cnt; } hset;

static uint64_t mix(uint64_t x) {
    x ^= x >> 33; x *= 0xff51afd7ed558ccdULL; x ^= x >> 33; x *= 0xc4ceb9fe1a85ec53ULL; x ^= x >> 33;
    return x;
}
static int hs_init(hset *h, size_t cap) {
    h->cap = cap; h->cnt = 0;
    h->keys = malloc(cap * sizeof(uint64_t));
    if (!h->keys) return -1;
    memset(h->keys, 0xff, cap * sizeof(uint64_t));   /* all-ones = empty slot */
    return 0;
}
static int hs_insert(hset *h, uint64_t key);
static int hs_grow(hset *h) {
    hset g;
    if (hs_init(&g, h->cap * 2)) return -1;
    for (size_t i = 0; i < h->cap; ++i) if (h->keys[i] != UINT64_MAX) hs_insert(&g, h->keys[i]);
    free(h->keys);
    *h = g;
    return 0;
}
/* returns 1 if inserted, 0 if present, -1 on allocation failure */
static int hs_insert(hset *h, uint64_t key) {
    if ((h->cnt + 1) * 2 > h->cap && hs_grow(h)) return -1;
    size_t i = mix(key) & (h->cap - 1);
    while (h->keys[i] != UINT64_MAX) {
        if (h->keys[i] == key) return 0;
        i = (i + 1) & (h->cap - 1);
    }
    h->keys[i] = key; h->cnt++;
    return 1;
}

typedef struct { uint64_t *v; size_t n, cap; } vec;
static int vec_push(vec *a, uint64_t x) {
    if (a->n == a->cap) {
        size_t nc = a->cap ? a->cap * 2 : 1024;
        uint64_t *p = realloc(a->v, nc * sizeof(uint64_t));
        if (!p) return -1;
        a->v = p; a->cap = nc;
    }
    a->v[a->n++] = x;
    return 0;
}

static unsigned code_of(uint64_t st, int i) { return (unsigned)((st >> (BITS * i)) & 63u); }
static uint64_t with_code(uint64_t st, int i, unsigned c) {
    st &= ~((uint64_t)63u << (BITS * i));
    return st | ((uint64_t)c << (BITS * i));
}

/* Returns the optimal makespan, -1 for invalid input, -2 when the search
 * exceeds max_T levels, -3 on allocation failure. */
int64_t oracle_opt_makespan(int n, const int32_t *arrival, const int32_t *o, int B,
                            int64_t alpha, int64_t kv_cap, int64_t max_T)
{
    if (n < 1 || n > 9 || B < 1 || alpha < 0 || kv_cap < 1) return -1;
    int64_t maxA = 0;
    for (int i = 0; i < n; ++i) {
        if (o[i] < 1 || o[i] > 62 || arrival[i] < 0 || arrival[i] > 1000 || o[i] > kv_cap) return -1;
        if (arrival[i] > maxA) maxA = arrival[i];
    }
    /* state: 6 bits per request (0 = not started, 1..o = running with
     * progress code-1, 63 = done); bits 54.. hold min(t, maxA+1) so that
     * states before the last release are told apart by time */
    vec cur = {0}, nxt = {0};
    hset seen;
    if (hs_init(&seen, 1 << 16)) return -3;
    int64_t result = -2;
    if (vec_push(&cur, 0)) { result = -3; goto out; }
    hs_insert(&seen, 0);
    for (int64_t t = 0; t < max_T; ++t) {
        nxt.n = 0;
        uint64_t tnext = (uint64_t)((t + 1) < (maxA + 1) ? (t + 1) : (maxA + 1));
        for (size_t s = 0; s < cur.n; ++s) {
            uint64_t st = cur.v[s] & ((1ULL << (BITS * 9)) - 1);
            int nrun = 0, nnew = 0, cand[9];
            int64_t kv = 0, amax = 0;
            for (int i = 0; i < n; ++i) {
                unsigned cd = code_of(st, i);
                if (cd == CODE_NEW) { if (arrival[i] <= t) cand[nnew++] = i; }
                else if (cd != CODE_DONE) {
                    nrun++; kv += o[i];
                    if ((int64_t)(cd - 1) > amax) amax = cd - 1;
                }
            }
            for (uint32_t mask = 0; mask < (1u << nnew); ++mask) {
                int add = 0; int64_t kv2 = kv;
                for (int b = 0; b < nnew; ++b) if (mask >> b & 1u) { add++; kv2 += o[cand[b]]; }
                if (nrun + add > B || kv2 > kv_cap) continue;
                if (add > 0 && nrun > 0 && amax > alpha) continue;
                uint64_t ns = st;
                for (int b = 0; b < nnew; ++b) if (mask >> b & 1u) ns = with_code(ns, cand[b], 1u);
                int all_done = 1;
                for (int i = 0; i < n; ++i) {
                    unsigned cd = code_of(ns, i);
                    if (cd != CODE_NEW && cd != CODE_DONE) {
                        unsigned prog = cd;            /* progress after this step */
                        ns = with_code(ns, i, prog >= (unsigned)o[i] ? CODE_DONE : cd + 1);
                        cd = code_of(ns, i);
                    }
                    if (cd != CODE_DONE) all_done = 0;
                }
                if (all_done) { result = t + 1; goto out; }
                uint64_t key = ns | (tnext << (BITS * 9));
                int ins = hs_insert(&seen, key);
                if (ins < 0) { result = -3; goto out; }
                if (ins == 1 && vec_push(&nxt, key)) { result = -3; goto out; }
            }
        }
        vec tmp = cur; cur = nxt; nxt = tmp;
        if (cur.n == 0) break;
    }
out:
    free(cur.v); free(nxt.v); free(seen.keys);
    return result;
}
