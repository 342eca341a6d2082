// sim_kernel.cu -- the per-step simulation of FCFS, LJF and ISJL on sm_103a.
//
// One warp simulates one (instance, run) task; a persistent grid of warps
// pulls tasks from a global counter.  Within a task every step does, in the
// order of the paper's model (Section 2) and policies:
//   release   requests with A_i <= k join the pending queue Q(k)
//   retire    requests that finished in step k-1 leave the batch, c_i = k
//   admit     FCFS / LJF (Algorithm 1) / ISJL (Algorithm 2, Sec. 3.4 rolling)
//   advance   every running request processes token r_i = a_i + 1
//   cost      W += |S| max r, E += sum (max r - r_i), extent, T_busy
//             (Section 5, Eq. batch-cost-progress and the decomposition)
//
// Layout: worker (batch slot) w lives in lane w / SPL, register slot w % SPL,
// so a warp covers B <= 32 * SPL workers; the max / min / sum of the step are
// warp reductions (REDUX).  The pending queue is a bitset over the request
// positions of the instance sorted by (o desc, index asc): the longest pending
// request is the lowest set bit (two levels: 32-bit words plus a summary word
// per 32 words, in shared memory).  ISJL plans are per-worker FIFO lists
// linked through a global scratch array.
//
// Two variants share the admission code:
//   step kernel   advances every running request each step (the literal loop)
//   epoch kernel  jumps from event to event (arrival, completion, o_1's delay
//                 expiry) and adds the cost of the L steps in between in closed
//                 form; the running set is constant there and progress moves
//                 in lockstep, so every counter is identical.
// Admissions happen only at events: between events the running set, the KV
// reservation and the queue are unchanged and A_max only grows, so a step
// that could not start a request is followed by steps that cannot either.
#include <climits>
#include <cstdint>

#include "sim_internal.cuh"

namespace isjl {
namespace {

constexpr int32_t kNone = -1;

struct WarpSmem {
    int32_t *sjob;    // [B] request running on worker w
    int32_t *shead;   // [B] next ISJL plan entry of worker w (kNone = none)
    int32_t *stail;   // [B] last plan entry of worker w
    int32_t *slong;   // [B] long request o_j planned on worker j (1 <= j < n_long)
    uint32_t *pend0;  // [words0] bit p: sorted position p is pending
    uint32_t *pend1;  // [words1] bit w: pend0[w] != 0
};

__host__ __device__ inline int smem_words_per_warp(int B, int words0, int words1) {
    int w = 4 * B + words0 + words1;
    return (w + 3) & ~3;  // keep every warp's block 16-byte aligned
}

template <int SPL>
__device__ __forceinline__ int lowest_worker(uint32_t m) {
    const unsigned b = __ballot_sync(kFull, m != 0u);
    if (!b) return -1;
    const int l = __ffs(b) - 1;
    const uint32_t mm = __shfl_sync(kFull, m, l);
    return l * SPL + (__ffs(mm) - 1);
}

template <int SPL>
__device__ __forceinline__ int highest_worker(uint32_t m) {
    const unsigned b = __ballot_sync(kFull, m != 0u);
    if (!b) return -1;
    const int l = 31 - __clz(b);
    const uint32_t mm = __shfl_sync(kFull, m, l);
    return l * SPL + (31 - __clz(mm));
}

__device__ __forceinline__ int64_t warp_sum64(int64_t v) {
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(kFull, v, s);
    return v;
}

// first pending sorted position >= p, INT_MAX if none (uniform call)
__device__ __forceinline__ int bs_next(const WarpSmem &S, int words0, int words1, int p, int lane) {
    const int w0 = p >> 5;
    if (w0 >= words0) return INT_MAX;
    const uint32_t v = S.pend0[w0] & (~0u << (p & 31));
    if (v) return (w0 << 5) + __ffs(v) - 1;
    const int q = w0 + 1;
    if (q >= words0) return INT_MAX;
    const int w1 = q >> 5;
    const uint32_t u = S.pend1[w1] & (~0u << (q & 31));
    if (u) {
        const int ww = (w1 << 5) + __ffs(u) - 1;
        return (ww << 5) + __ffs(S.pend0[ww]) - 1;
    }
    for (int b1 = w1 + 1; b1 < words1; b1 += 32) {
        const int idx = b1 + lane;
        const uint32_t x = idx < words1 ? S.pend1[idx] : 0u;
        const unsigned b = __ballot_sync(kFull, x != 0u);
        if (b) {
            const int l = __ffs(b) - 1;
            const uint32_t xx = __shfl_sync(kFull, x, l);
            const int ww = ((b1 + l) << 5) + __ffs(xx) - 1;
            return (ww << 5) + __ffs(S.pend0[ww]) - 1;
        }
    }
    return INT_MAX;
}

__device__ __forceinline__ void bs_clear(const WarpSmem &S, int p, int lane) {
    if (lane == 0) {
        const int w = p >> 5;
        const uint32_t v = S.pend0[w] & ~(1u << (p & 31));
        S.pend0[w] = v;
        if (!v) S.pend1[w >> 5] &= ~(1u << (w & 31));
    }
    __syncwarp();
}

// number of pending positions < P (uniform call)
__device__ __forceinline__ int bs_count_below(const WarpSmem &S, int words0, int P, int lane) {
    const int full = P >> 5;
    int cnt = 0;
    for (int w = lane; w < full && w < words0; w += 32) cnt += __popc(S.pend0[w]);
    if (lane == 0 && (P & 31) && full < words0) cnt += __popc(S.pend0[full] & ((1u << (P & 31)) - 1u));
    return (int)__reduce_add_sync(kFull, (unsigned)cnt);
}

// first sorted position whose o is <= x (osorted is non-increasing); n if none
__device__ __forceinline__ int first_pos_le(const int32_t *os, int n, int64_t x) {
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if ((int64_t)__ldg(os + mid) <= x) hi = mid; else lo = mid + 1;
    }
    return lo;
}

template <int SPL, bool EPOCH>
__device__ __forceinline__ void run_task(const SimArgs &A, const WarpSmem &S, int lane, int64_t gwarp,
                                         int64_t task) {
    const int64_t inst = task / A.n_runs;
    const int run = (int)(task % A.n_runs);
    const int n = A.n, B = A.B;
    const int64_t base = inst * (int64_t)n;
    const int policy = A.runs.policy[run];
    const int64_t alpha = A.runs.delta[run];
    const int64_t kv_cap = A.kv_cap;
    const int32_t *__restrict__ arr = A.arrival + base;
    const int32_t *__restrict__ oarr = A.o + base;
    const int32_t *__restrict__ perm = A.perm + base;
    const int32_t *__restrict__ osrt = A.osorted + base;
    const int32_t *__restrict__ posof = A.posof + base;
    int32_t *__restrict__ pnext = A.plan_next + gwarp * (int64_t)n;
    const int64_t out_off = (int64_t)run * A.n_inst * n + base;
    int32_t *st_out = A.start_out ? A.start_out + out_off : nullptr;
    int32_t *co_out = A.compl_out ? A.compl_out + out_off : nullptr;
    const InstStats is = A.inst[inst];
    const int words0 = A.words0, words1 = A.words1;

    int64_t status = is.status;
    if (status == ISJL_OK && (int64_t)is.maxo > kv_cap) status = ISJL_ERR_INFEASIBLE;
    // step counters are int32: every schedule ends by sum o + max arrival
    if (status == ISJL_OK && is.O + (int64_t)is.maxA + 1 > (int64_t)INT_MAX) status = ISJL_ERR_INVALID_ARG;

    int64_t W = 0, E = 0, Tb = 0, tok = 0, sumc = 0, sumext = 0, maxext = 0, viol = 0, kvviol = 0;
    int64_t peakkv = 0, peakb = 0, Tmake = 0;

    if (status == ISJL_OK) {
        for (int w = lane; w < words0; w += 32) S.pend0[w] = 0u;
        for (int w = lane; w < words1; w += 32) S.pend1[w] = 0u;
        for (int w = lane; w < B; w += 32) { S.shead[w] = kNone; S.stail[w] = kNone; S.slong[w] = kNone; }
        __syncwarp();

        // per-lane worker slots: a_ = progress (step kernel) or start step (epoch kernel)
        int32_t a_[SPL], oo[SPL];
#pragma unroll
        for (int r = 0; r < SPL; ++r) { a_[r] = 0; oo[r] = 0; }
        uint32_t busy = 0u, resv = 0u;
        const int nv = B - lane * SPL;
        const uint32_t vmask = nv <= 0 ? 0u : (nv >= SPL ? (SPL == 32 ? ~0u : ((1u << SPL) - 1u)) : ((1u << nv) - 1u));

        int32_t k = 0, rel = 0, fcfs = 0, done = 0, run_cnt = 0, pend = 0;
        int64_t kv_sum = 0, sum_st = 0;
        int32_t plan_left = 0, t0 = 0, d1 = 0, L1 = kNone, nlong = 0;
        bool L1_started = true, adm_blocked = false;
        bool broken = false;   // an internal invariant failed: stop without touching memory
        const int64_t max_steps = A.max_steps > 0 ? A.max_steps : (is.O + (int64_t)is.maxA + 1);

        // start request e (length oe) on worker w at step k
        auto start = [&](int e, int oe, int w) {
            run_cnt++;
            kv_sum += oe;
            if (EPOCH) sum_st += k;
            const int l = w / SPL, rr = w - l * SPL;
            if (lane == l) {
#pragma unroll
                for (int r = 0; r < SPL; ++r)
                    if (r == rr) { a_[r] = EPOCH ? k : 0; oo[r] = oe; }
                busy |= 1u << rr;
                S.sjob[w] = e;
                if (st_out) st_out[e] = k;
            }
        };
        // requests of the workers in fin (per lane) complete at step c
        auto retire = [&](uint32_t fin, int32_t c) {
            if (!__ballot_sync(kFull, fin != 0u)) return;
            int nf = 0, of = 0;
            int64_t sf = 0;
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                if (fin >> r & 1u) {
                    nf++;
                    of += oo[r];
                    if (EPOCH) sf += a_[r];
                    if (co_out) co_out[S.sjob[lane * SPL + r]] = c;
                }
            }
            busy &= ~fin;
            nf = (int)__reduce_add_sync(kFull, (unsigned)nf);
            of = (int)__reduce_add_sync(kFull, (unsigned)of);
            if (EPOCH) sum_st -= warp_sum64(sf);
            done += nf;
            run_cnt -= nf;
            kv_sum -= of;
            sumc += (int64_t)nf * c;
            Tmake = c;
            adm_blocked = false;
        };
        // A_max(k): largest progress among running requests (0 if none)
        auto amax_now = [&]() -> int64_t {
            if (run_cnt == 0) return 0;
            if (EPOCH) {
                int m = INT_MAX;
#pragma unroll
                for (int r = 0; r < SPL; ++r) if (busy >> r & 1u) m = min(m, a_[r]);
                m = __reduce_min_sync(kFull, m);
                return (int64_t)k - m;
            } else {
                int m = 0;
#pragma unroll
                for (int r = 0; r < SPL; ++r) if (busy >> r & 1u) m = max(m, a_[r]);
                return (int64_t)__reduce_max_sync(kFull, m);
            }
        };

        // ISJL Phase ONE at a stage start (Algorithm 2 with beta = alpha)
        auto phase_one = [&]() {
            t0 = k; d1 = 0; L1 = kNone; L1_started = true; nlong = 0;
            if (pend < 2) return;                               // |Q| = 1: Phase TWO
            const int p1 = bs_next(S, words0, words1, 0, lane);
            if (p1 >= n) { broken = true; return; }
            const int64_t o1 = osrt[p1];
            const int p2 = bs_next(S, words0, words1, p1 + 1, lane);
            if (p2 >= n) { broken = true; return; }
            if ((int64_t)osrt[p2] <= alpha) return;             // o_2 <= alpha: Phase TWO
            // M = min{B, #{o > alpha}} over Q(k)
            const int cnt_long = bs_count_below(S, words0, first_pos_le(osrt, n, alpha), lane);
            const int nl = min(B, cnt_long);
            int32_t rem[SPL], psum[SPL];   // packing budget left / pack sum per worker
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                const int w = lane * SPL + r;
                rem[r] = (w >= nl && w < B) ? (int32_t)alpha : -1;   // workers M+1..B: alpha
                psum[r] = 0;
            }
            // the long requests o_1..o_M leave Q; worker j's budget cap_j
            int p = -1;
            int64_t o_last = o1;
            for (int j = 0; j < nl; ++j) {
                p = bs_next(S, words0, words1, p + 1, lane);
                if (p >= n) { broken = true; return; }
                const int e = perm[p];
                const int64_t oe = osrt[p];
                bs_clear(S, p, lane);
                if (j == 0) {
                    L1 = e;
                    if (lane == 0) { S.shead[0] = e; S.stail[0] = e; pnext[e] = kNone; }
                } else {
                    const int64_t cap = min(2 * alpha, o1 - oe + alpha);
                    if (lane == 0) S.slong[j] = e;
                    const int l = j / SPL, rr = j - l * SPL;
                    if (lane == l) {
#pragma unroll
                        for (int r = 0; r < SPL; ++r) if (r == rr) rem[r] = (int32_t)cap;
                    }
                }
                o_last = oe;
            }
            __syncwarp();
            pend -= nl;
            const int64_t theta = min(2 * alpha, o1 - o_last + alpha);
            // first fit of the shorter requests, in sorted order
            int maxrem = -1;
#pragma unroll
            for (int r = 0; r < SPL; ++r) maxrem = max(maxrem, rem[r]);
            maxrem = __reduce_max_sync(kFull, maxrem);
            int q = -1;
            for (;;) {
                const int64_t x = min(theta, (int64_t)maxrem);
                if (x < 1) break;
                // candidates with o > x fit nowhere now or later (budgets only shrink)
                q = bs_next(S, words0, words1, max(first_pos_le(osrt, n, x), q + 1), lane);
                if (q >= n) break;
                const int e = perm[q];
                const int oe = osrt[q];
                uint32_t mA = 0u, mB = 0u;
#pragma unroll
                for (int r = 0; r < SPL; ++r) {
                    const int w = lane * SPL + r;
                    const bool fits = rem[r] >= oe;
                    if (fits && w >= nl && w < B) mA |= 1u << r;
                    if (fits && w >= 1 && w < nl) mB |= 1u << r;
                }
                int w = lowest_worker<SPL>(mA);                 // workers M+1..B first
                if (w < 0) w = highest_worker<SPL>(mB);         // then M, M-1, ..., 2
                if (w < 0) { broken = true; return; }
                if (lane == 0) {
                    const int tl = S.stail[w];
                    if (tl < 0) S.shead[w] = e; else pnext[tl] = e;
                    S.stail[w] = e;
                    pnext[e] = kNone;
                }
                const int l = w / SPL, rr = w - l * SPL;
                if (lane == l) {
#pragma unroll
                    for (int r = 0; r < SPL; ++r) if (r == rr) { rem[r] -= oe; psum[r] += oe; }
                }
                bs_clear(S, q, lane);   // includes __syncwarp
                pend--;
                plan_left++;
                maxrem = -1;
#pragma unroll
                for (int r = 0; r < SPL; ++r) maxrem = max(maxrem, rem[r]);
                maxrem = __reduce_max_sync(kFull, maxrem);
            }
            // worker j (2..M) runs o_j after its pack
            for (int w = 1 + lane; w < nl; w += 32) {
                const int e = S.slong[w];
                const int tl = S.stail[w];
                if (tl < 0) S.shead[w] = e; else pnext[tl] = e;
                S.stail[w] = e;
                pnext[e] = kNone;
            }
            __syncwarp();
            plan_left += nl;
            // o_1 waits d1 = min{max{max_j sum(w_j) - alpha, 0}, alpha}, j = 2..M
            int mx = 0;
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                const int w = lane * SPL + r;
                if (w >= 1 && w < nl) mx = max(mx, psum[r]);
            }
            mx = __reduce_max_sync(kFull, mx);
            d1 = (int32_t)min(max((int64_t)mx - alpha, (int64_t)0), alpha);
            resv = 0u;
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                const int w = lane * SPL + r;
                if (w < B && S.shead[w] >= 0) resv |= 1u << r;
            }
            L1_started = false;
            nlong = nl;
        };

        auto admit = [&]() {
            if (policy == ISJL_POLICY_FCFS) {
                // arrival order; the first request that does not fit ends the step
                while (run_cnt < B && fcfs < rel) {
                    const int oe = oarr[fcfs];
                    if (kv_sum + oe > kv_cap) break;
                    const int w = lowest_worker<SPL>(vmask & ~busy);
                    if (w < 0) { broken = true; return; }
                    start(fcfs, oe, w);
                    fcfs++;
                }
            } else if (policy == ISJL_POLICY_LJF) {
                // static batch of the longest released requests when nothing runs
                if (run_cnt != 0) return;
                int p = -1;
                while (run_cnt < B && pend > 0) {
                    p = bs_next(S, words0, words1, p + 1, lane);
                    if (p >= n) { broken = true; return; }
                    const int oe = osrt[p];
                    if (kv_sum + oe > kv_cap) break;
                    const int e = perm[p];
                    const int w = lowest_worker<SPL>(vmask & ~busy);
                    if (w < 0) { broken = true; return; }
                    bs_clear(S, p, lane);
                    pend--;
                    start(e, oe, w);
                }
            } else {
                const bool nothing_runs = run_cnt == 0;
                if (nothing_runs && plan_left == 0 && pend > 0) phase_one();
                if (broken) return;
                bool stop = amax_now() > alpha;                  // the gate A_max(k) <= alpha
                if (!stop && plan_left > 0) {
                    // plan starts, workers in order
                    uint32_t cand = resv & ~busy;
                    for (;;) {
                        const unsigned b = __ballot_sync(kFull, cand != 0u);
                        if (!b) break;
                        const int l = __ffs(b) - 1;
                        const uint32_t m = __shfl_sync(kFull, cand, l);
                        const int rr = __ffs(m) - 1;
                        const int w = l * SPL + rr;
                        if (lane == l) cand &= ~(1u << rr);
                        const int e = S.shead[w];
                        if (w == 0 && e == L1) {
                            const bool over = ((int64_t)k >= (int64_t)t0 + d1) || (k > t0 && nothing_runs);
                            if (!over) continue;                 // o_1 still delayed
                        }
                        if (w >= 1 && w < nlong && e == S.slong[w] && !L1_started) continue;  // o_j after o_1
                        const int oe = oarr[e];
                        if (kv_sum + oe > kv_cap) { stop = true; break; }
                        const int nx = pnext[e];
                        __syncwarp();
                        if (lane == 0) { S.shead[w] = nx; if (nx < 0) S.stail[w] = kNone; }
                        __syncwarp();
                        if (nx < 0 && lane == l) resv &= ~(1u << rr);
                        plan_left--;
                        if (e == L1) L1_started = true;
                        start(e, oe, w);
                    }
                }
                if (!stop) {
                    // Phase TWO: longest released request onto a free worker
                    int p = -1;
                    while (pend > 0) {
                        const int w = lowest_worker<SPL>(vmask & ~busy & ~resv);
                        if (w < 0) break;
                        p = bs_next(S, words0, words1, p + 1, lane);
                        if (p >= n) { broken = true; return; }
                        const int oe = osrt[p];
                        if (kv_sum + oe > kv_cap) break;
                        const int e = perm[p];
                        bs_clear(S, p, lane);
                        pend--;
                        start(e, oe, w);
                    }
                }
            }
        };

        for (;;) {
            if ((int64_t)k > max_steps) { status = ISJL_ERR_STEP_LIMIT; break; }
            // release: arrivals are non-decreasing, so the released requests are a prefix
            if (rel < n && arr[rel] <= k) {
                adm_blocked = false;
                for (;;) {
                    const int i = rel + lane;
                    const bool ok = i < n && arr[i] <= k;
                    const unsigned b = __ballot_sync(kFull, ok);
                    if (ok && policy != ISJL_POLICY_FCFS) {
                        const int p = posof[i];
                        atomicOr(&S.pend0[p >> 5], 1u << (p & 31));
                        atomicOr(&S.pend1[p >> 10], 1u << ((p >> 5) & 31));
                    }
                    const int c = __popc(b);
                    rel += c;
                    pend += c;
                    if (c < 32) break;
                }
                __syncwarp();
            }
            if (EPOCH) {
                uint32_t fin = 0u;
#pragma unroll
                for (int r = 0; r < SPL; ++r)
                    if ((busy >> r & 1u) && a_[r] + oo[r] == k) fin |= 1u << r;
                retire(fin, k);
            }
            if (done == n) break;
            if (!EPOCH && policy == ISJL_POLICY_ISJL && !L1_started && k == t0 + d1) adm_blocked = false;
            if (EPOCH || !adm_blocked) {
                admit();
                adm_blocked = true;
                if (broken) { status = ISJL_ERR_STEP_LIMIT; break; }
            }

            if (!EPOCH) {
                if (run_cnt > 0) {
                    // advance every running request by one token
                    int rmax = 0, rmin = INT_MAX;
                    unsigned rsum = 0u;
                    uint32_t fin = 0u;
#pragma unroll
                    for (int r = 0; r < SPL; ++r) {
                        const bool bz = busy >> r & 1u;
                        const int rr = a_[r] + 1;          // token index processed now
                        if (bz) {
                            a_[r] = rr;
                            rmax = max(rmax, rr);
                            rmin = min(rmin, rr);
                            rsum += (unsigned)rr;
                            if (rr == oo[r]) fin |= 1u << r;
                        }
                    }
                    rmax = __reduce_max_sync(kFull, rmax);
                    rmin = __reduce_min_sync(kFull, rmin);
                    rsum = __reduce_add_sync(kFull, rsum);
                    const int64_t cnt = run_cnt;
                    W += cnt * rmax;
                    E += cnt * rmax - (int64_t)rsum;
                    const int64_t ext = rmax - rmin;
                    sumext += ext;
                    maxext = max(maxext, ext);
                    viol += ext > alpha;
                    kvviol += kv_sum > kv_cap;
                    peakkv = max(peakkv, kv_sum);
                    peakb = max(peakb, cnt);
                    Tb++;
                    tok += cnt;
                    retire(fin, k + 1);
                }
                k++;
            } else {
                // next event: arrival, completion or the end of o_1's delay
                int64_t nxt = rel < n ? (int64_t)arr[rel] : INT64_MAX;
                int mc = INT_MAX, mns = INT_MAX, mxs = INT_MIN;
#pragma unroll
                for (int r = 0; r < SPL; ++r) {
                    if (busy >> r & 1u) {
                        mc = min(mc, a_[r] + oo[r]);
                        mns = min(mns, a_[r]);
                        mxs = max(mxs, a_[r]);
                    }
                }
                mc = __reduce_min_sync(kFull, mc);
                mns = __reduce_min_sync(kFull, mns);
                mxs = __reduce_max_sync(kFull, mxs);
                if (run_cnt > 0) nxt = min(nxt, (int64_t)mc);
                if (policy == ISJL_POLICY_ISJL && !L1_started && (int64_t)t0 + d1 > k)
                    nxt = min(nxt, (int64_t)t0 + d1);
                if (nxt == INT64_MAX) { status = ISJL_ERR_STEP_LIMIT; break; }   // cannot progress
                if (run_cnt > 0) {
                    const int64_t L = nxt - k, s = run_cnt;
                    const int64_t m0 = (int64_t)k - mns + 1;       // max r at step k
                    const int64_t n0 = (int64_t)k - mxs + 1;       // min r at step k
                    const int64_t sr = s * ((int64_t)k + 1) - sum_st;   // sum r at step k
                    W += s * (L * m0 + L * (L - 1) / 2);
                    E += L * (s * m0 - sr);
                    const int64_t ext = m0 - n0;
                    sumext += L * ext;
                    maxext = max(maxext, ext);
                    viol += ext > alpha ? L : 0;
                    kvviol += kv_sum > kv_cap ? L : 0;
                    peakkv = max(peakkv, kv_sum);
                    peakb = max(peakb, s);
                    Tb += L;
                    tok += s * L;
                }
                if (nxt > INT_MAX) { status = ISJL_ERR_STEP_LIMIT; break; }
                k = (int32_t)nxt;
            }
        }
    }

    if (lane == 0) {
        isjl_record R;
        const bool bad_input = status == ISJL_ERR_INVALID_ARG || status == ISJL_ERR_INFEASIBLE;
        R.T_make = bad_input ? 0 : Tmake;
        R.T_busy = bad_input ? 0 : Tb;
        R.O = bad_input ? 0 : is.O;
        R.Q = bad_input ? 0 : is.Q;
        R.W = W;
        R.E = E;
        R.token_adv = tok;
        R.sum_completion = sumc;
        R.sum_latency = bad_input ? 0 : sumc - is.sumA;
        R.sum_extent = sumext;
        R.max_extent = maxext;
        R.violations = viol;
        R.kv_violations = kvviol;
        R.peak_kv = peakkv;
        R.peak_batch = peakb;
        R.status = status;
        if (bad_input) {
            R.c_T = R.tau_Q = R.tau_E = R.cost = R.revenue = R.profit = R.throughput = R.ael = 0.0;
        } else {
            // cost decomposition C = tau Q + c T + tau E, no contraction
            R.c_T = __dmul_rn(A.c, (double)Tb);
            R.tau_Q = __dmul_rn(A.tau, (double)is.Q);
            R.tau_E = __dmul_rn(A.tau, (double)E);
            R.cost = __dadd_rn(__dadd_rn(R.c_T, R.tau_Q), R.tau_E);
            R.revenue = __dmul_rn(A.p0, (double)is.O);
            R.profit = __dsub_rn(R.revenue, R.cost);
            R.throughput = Tmake > 0 ? __ddiv_rn((double)is.O, (double)Tmake) : 0.0;
            R.ael = __ddiv_rn((double)sumc, (double)n);
        }
        A.records[(int64_t)run * A.n_inst + inst] = R;
        if (status != ISJL_OK) atomicCAS(A.dev_status, 0, (int32_t)status);
    }
    __syncwarp();
}

template <int SPL, bool EPOCH>
__global__ void __launch_bounds__(kSimWarpsPerBlock * 32)
sim_kernel(SimArgs A, int64_t n_tasks) {
    extern __shared__ __align__(16) int32_t smem[];
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const int per = smem_words_per_warp(A.B, A.words0, A.words1);
    int32_t *b = smem + (size_t)wib * per;
    WarpSmem S;
    S.sjob = b;
    S.shead = b + A.B;
    S.stail = b + 2 * A.B;
    S.slong = b + 3 * A.B;
    S.pend0 = reinterpret_cast<uint32_t *>(b + 4 * A.B);
    S.pend1 = S.pend0 + A.words0;
    const int64_t gwarp = (int64_t)blockIdx.x * kSimWarpsPerBlock + wib;
    for (;;) {
        int t = 0;
        if (lane == 0) t = atomicAdd(A.task_counter, 1);
        t = __shfl_sync(kFull, t, 0);
        if ((int64_t)t >= n_tasks) break;
        run_task<SPL, EPOCH>(A, S, lane, gwarp, t);
    }
}

template <int SPL, bool EPOCH>
const void *kernel_ptr() { return reinterpret_cast<const void *>(&sim_kernel<SPL, EPOCH>); }

const void *pick_kernel(int spl, bool epoch) {
    switch (spl) {
        case 1:  return epoch ? kernel_ptr<1, true>() : kernel_ptr<1, false>();
        case 2:  return epoch ? kernel_ptr<2, true>() : kernel_ptr<2, false>();
        case 4:  return epoch ? kernel_ptr<4, true>() : kernel_ptr<4, false>();
        case 8:  return epoch ? kernel_ptr<8, true>() : kernel_ptr<8, false>();
        default: return epoch ? kernel_ptr<16, true>() : kernel_ptr<16, false>();
    }
}

}  // namespace

int slots_per_lane(int B) {
    int s = 1;
    while (32 * s < B) s <<= 1;
    return s;
}

size_t sim_smem_per_warp(int B, int n) {
    const int words0 = (n + 31) / 32, words1 = (words0 + 31) / 32;
    return (size_t)smem_words_per_warp(B, words0, words1) * 4;
}

static cudaError_t occupancy(int B, int n, bool epoch, int device, int *blocks_per_sm, int *sms, size_t *smem) {
    const void *k = pick_kernel(slots_per_lane(B), epoch);
    *smem = sim_smem_per_warp(B, n) * kSimWarpsPerBlock;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)*smem);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, k, kSimWarpsPerBlock * 32, *smem);
}

int sim_resident_warps(int B, int n, bool epoch, int device) {
    int bps = 0, sms = 0;
    size_t smem = 0;
    if (occupancy(B, n, epoch, device, &bps, &sms, &smem) != cudaSuccess || bps < 1) return 0;
    return bps * sms * kSimWarpsPerBlock;
}

cudaError_t launch_sim(const SimArgs &args, bool epoch, int total_warps, cudaStream_t s) {
    int bps = 0, sms = 0;
    size_t smem = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = occupancy(args.B, args.n, epoch, dev, &bps, &sms, &smem);
    if (e != cudaSuccess) return e;
    const int64_t n_tasks = args.n_inst * args.n_runs;
    int64_t blocks = total_warps / kSimWarpsPerBlock;
    const int64_t need = (n_tasks + kSimWarpsPerBlock - 1) / kSimWarpsPerBlock;
    if (blocks > need) blocks = need;
    if (blocks < 1) blocks = 1;
    const void *k = pick_kernel(slots_per_lane(args.B), epoch);
    SimArgs a = args;
    void *params[] = {&a, const_cast<int64_t *>(&n_tasks)};
    return cudaLaunchKernel(k, dim3((unsigned)blocks), dim3(kSimWarpsPerBlock * 32), params, smem, s);
}

}  // namespace isjl
