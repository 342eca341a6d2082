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
// Layout.  Worker (batch slot) w lives in lane w % 32, register row w / 32,
// so a warp holds B <= 32 * SPL workers.  The step kernel advances, each
// step, every slot of the rows that hold a running worker (a per-row-count
// instantiation of the step loop), straight-line: from 8 rows on, a slot's
// progress a is packed as (a << 16) | (65535 - a), so one add advances it and
// one per-half max collects both the step's max and (complemented) min, with
// idle slots set at the start of each stretch to values that lose both;
// below 8 rows an idle slot carries a progress below 0 as a signed value and
// at least 2^31 as an unsigned one (signed max, unsigned min).  The
// sum of progress over all steps is added per request, o (o + 1) / 2, when it
// starts (a run stopped early takes back the unserved part).  Values that
// change only at events (next
// arrival, earliest completion, start range, KV reservation) are kept as
// warp-uniform scalars, so the steps between two events run no branch and
// no warp reduction beyond the two of the step cost.  The pending
// queue is a bitset over the instance's request positions sorted by
// (o desc, index asc) -- the longest pending request is the lowest set bit --
// with a summary word per 32 words, in shared memory.  ISJL plans are
// per-worker FIFO lists linked through a global scratch array.
//
// Two variants share the admission code:
//   step kernel   advances every running request each step (the literal loop)
//   epoch kernel  jumps from event to event (arrival, completion, o_1's delay
//                 expiry) and adds the cost of the L steps in between in closed
//                 form; the running set is constant there and progress moves
//                 in lockstep, so every counter is identical.  While LJF has a
//                 batch running or ISJL's gate is shut, completions that do not
//                 change the running set's earliest or latest start are served
//                 in the same pass (a completion window).
// Admissions happen only at events: between events the running set, the KV
// reservation and the queue are unchanged and A_max only grows, so a step
// that could not start a request is followed by steps that cannot either.
// Arrivals that cannot start anything before the next completion are released
// at that completion, and an admission that starts several requests does so
// up to 32 (ISJL plan entries: all) at a time, with the same outcome as one
// start at a time.
#include <climits>
#include <cstdint>

#include "sim_internal.cuh"

namespace isjl {
namespace {

constexpr int32_t kNone = -1;
constexpr int32_t kIdle = -(1 << 30);   // idle-slot progress sentinel base (unpacked step kernel)
// step kernel with SPL >= 8: the progress a of a slot is packed as
// (a << 16) | (65535 - a)
constexpr uint32_t kPackedZero = 0xFFFFu;  // a = 0
constexpr uint32_t kPackedStep = 0xFFFFu;  // one step: a + 1 above, 65535 - (a + 1) below

struct WarpSmem {
    int32_t *sjob;    // [B] request running on worker w
    int32_t *shead;   // [B] next ISJL plan entry of worker w (kNone = none)
    int32_t *stail;   // [B] last plan entry of worker w
    int32_t *slong;   // [B] long request o_j planned on worker j (1 <= j < n_long)
    int32_t *srem;    // [B] ISJL packing budget of worker w at a stage start (Phase ONE only)
    int32_t *spsum;   // [B] ISJL pack sum on worker w in Phase ONE, then the o of its next plan entry
    int32_t *sres;    // [B] KV reserved by the request running on worker w (its planning length)
    uint32_t *pend0;  // [words0] bit p: sorted position p is pending
    uint32_t *pend1;  // [words1] bit w: pend0[w] != 0
};

__host__ __device__ inline int smem_words_per_warp(int B, int words0, int words1) {
    int w = 7 * B + words0 + words1;
    return (w + 3) & ~3;  // keep every warp's block 16-byte aligned
}

// lowest / highest worker whose row bit is set in the per-lane mask m
__device__ __forceinline__ int lowest_worker(uint32_t m, int lane) {
    const int v = m ? ((__ffs(m) - 1) << 5) + lane : INT_MAX;
    const int r = __reduce_min_sync(kFull, v);
    return r == INT_MAX ? -1 : r;
}
__device__ __forceinline__ int highest_worker(uint32_t m, int lane) {
    const int v = m ? ((31 - __clz(m)) << 5) + lane : -1;
    return __reduce_max_sync(kFull, v);
}

// a row count as a type, for the step loop's per-row-count instantiations
template <int N> struct RowCount { static constexpr int value = N; };

// Row counts the step loop is instantiated for, per SPL (ascending).  The
// loop advances the smallest of them covering every running worker; a few
// classes keep the kernel small (measured: 2 and 4 for SPL = 4; 2, 4 and 8
// for SPL = 8; 4, 8 and 16 for SPL = 16), and its steps are unrolled by two
// (four for SPL = 16).
template <int SPL> struct RowClasses;
template <> struct RowClasses<1> {
    static constexpr int n = 1;
    __host__ __device__ static constexpr int at(int i) { constexpr int v[1] = {1}; return v[i]; }
};
template <> struct RowClasses<2> {
    static constexpr int n = 2;
    __host__ __device__ static constexpr int at(int i) { constexpr int v[2] = {1, 2}; return v[i]; }
};
template <> struct RowClasses<4> {
    static constexpr int n = 2;
    __host__ __device__ static constexpr int at(int i) { constexpr int v[2] = {2, 4}; return v[i]; }
};
template <> struct RowClasses<8> {
    static constexpr int n = 3;
    __host__ __device__ static constexpr int at(int i) { constexpr int v[3] = {2, 4, 8}; return v[i]; }
};
template <> struct RowClasses<16> {
    static constexpr int n = 3;
    __host__ __device__ static constexpr int at(int i) { constexpr int v[3] = {4, 8, 16}; return v[i]; }
};

// rows advanced when the highest row holding a running worker is t - 1 (t = 0: none)
template <int SPL>
__device__ __forceinline__ int row_class(int t) {
    using C = RowClasses<SPL>;
    if (t <= 0) return 0;
    int r = SPL;
#pragma unroll
    for (int i = C::n - 1; i >= 0; --i) if (C::at(i) >= t) r = C::at(i);
    return r;
}
// call f(RowCount<rows>{}) for rows one of RowClasses<SPL> (indices LO..HI), by a tree of uniform branches
template <int SPL, int LO, int HI, class F>
__device__ __forceinline__ void dispatch_rows(int rows, F &f) {
    using C = RowClasses<SPL>;
    if constexpr (LO == HI) {
        f(RowCount<C::at(LO)>{});
    } else {
        constexpr int MID = (LO + HI) / 2;
        if (rows <= C::at(MID)) dispatch_rows<SPL, LO, MID>(rows, f);
        else dispatch_rows<SPL, MID + 1, HI>(rows, f);
    }
}

// per-16-bit-half unsigned maximum
__device__ __forceinline__ uint32_t vmax_u16x2(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("max.u16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// acc += a * b into a 64-bit accumulator with one wide multiply-add
__device__ __forceinline__ void mad_wide(int64_t &acc, uint32_t a, uint32_t b) {
    asm("mad.wide.u32 %0, %1, %2, %0;" : "+l"(acc) : "r"(a), "r"(b));
}

// warp sum of a 64-bit value (modulo 2^64) by three independent 32-bit warp
// reductions of its 22-, 22- and 20-bit pieces (each piece's sum is below 2^27)
__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v) {
    const uint32_t a = __reduce_add_sync(kFull, (uint32_t)v & 0x3FFFFFu);
    const uint32_t b = __reduce_add_sync(kFull, (uint32_t)(v >> 22) & 0x3FFFFFu);
    const uint32_t c = __reduce_add_sync(kFull, (uint32_t)(v >> 44));
    return (uint64_t)a + ((uint64_t)b << 22) + ((uint64_t)c << 44);
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

// highest pending sorted position, -1 if none (uniform call)
__device__ __forceinline__ int bs_last(const WarpSmem &S, int words1, int lane) {
    for (int b1 = (words1 - 1) & ~31; b1 >= 0; b1 -= 32) {
        const int idx = b1 + lane;
        const uint32_t x = idx < words1 ? S.pend1[idx] : 0u;
        const unsigned b = __ballot_sync(kFull, x != 0u);
        if (b) {
            const int l = 31 - __clz(b);
            const uint32_t xx = __shfl_sync(kFull, x, l);
            const int ww = ((b1 + l) << 5) + 31 - __clz(xx);
            return (ww << 5) + 31 - __clz(S.pend0[ww]);
        }
    }
    return -1;
}

// position of the k-th (0-based) set bit of x; k < popc(x)
__device__ __forceinline__ int nth_set_bit(uint32_t x, int k) {
    int pos = 0;
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) {
        const int c = __popc(x & ((1u << s) - 1u));
        if (k >= c) { k -= c; x >>= s; pos += s; }
    }
    return pos;
}

// number of pending positions < P (uniform call)
__device__ __forceinline__ int bs_count_below(const WarpSmem &S, int words0, int P, int lane) {
    const int full = P >> 5;
    int cnt = 0;
    for (int w = lane; w < full && w < words0; w += 32) cnt += __popc(S.pend0[w]);
    if (lane == 0 && (P & 31) && full < words0) cnt += __popc(S.pend0[full] & ((1u << (P & 31)) - 1u));
    return (int)__reduce_add_sync(kFull, (unsigned)cnt);
}

// first sorted position whose o is <= x (osorted is non-increasing); n if
// none (uniform call).  A 32-way search: each round the lanes sample 32
// evenly spaced positions of the bracket and a ballot keeps the sub-bracket
// holding the answer, so n = 1,000 takes two dependent loads and n = 10^5
// four, instead of a binary search's 10 and 17.
__device__ __forceinline__ int first_pos_le(const int32_t *os, int n, int64_t x, int lane) {
    int lo = 0, hi = n;                         // the answer lies in [lo, hi]
    while (hi - lo > 32) {
        const int step = (hi - lo + 31) >> 5;
        const int idx = lo + lane * step;
        const bool le = idx >= hi || (int64_t)__ldg(os + idx) <= x;
        const unsigned b = __ballot_sync(kFull, le);
        const int f = b ? __ffs(b) - 1 : 32;    // first sample at or after the answer
        if (f == 0) return lo;
        hi = min(hi, lo + f * step);
        lo = lo + (f - 1) * step + 1;
    }
    const int idx = lo + lane;
    const bool le = idx >= hi || (int64_t)__ldg(os + idx) <= x;
    const unsigned b = __ballot_sync(kFull, le);
    return b ? lo + __ffs(b) - 1 : lo + 32;
}

// One (instance, run) task under policy P, a compile-time constant (FCFS, LJF,
// SJF or ISJL; Algorithm "ISJL" runs the ISJL body with beta in the packing
// thresholds), so each policy's code holds only its own admission rule.
template <int SPL, bool EPOCH, int P>
__device__ __forceinline__ void run_task(const SimArgs &A, const WarpSmem &S, int lane, int64_t gwarp,
                                         int64_t inst, int run) {
    const int n_slots = A.n, B = A.B;
    const int64_t base = inst * (int64_t)n_slots;
    const InstStats is = A.inst[inst];
    const int n = is.n;                             // requests of this instance (<= n_slots)
    constexpr int policy = P;
    const int64_t alpha = A.runs.delta[run];
    const int64_t beta = A.runs.beta[run];
    const int64_t kv_cap = A.kv_cap;
    // reserved KV: at most B <= 512 running requests of length <= 65535, so
    // below 2^25; kept in 32 bits, against the cap clamped to INT_MAX (which
    // compares the same)
    const int32_t kv_lim = (int32_t)min(kv_cap, (int64_t)INT_MAX);
    const int32_t *__restrict__ arr = A.arrival + base;
    const int32_t *__restrict__ oarr = A.o + base;              // planning lengths (u_i)
    const int32_t *__restrict__ otru = A.otrue ? A.otrue + base : nullptr;   // true lengths
    const int32_t *__restrict__ perm = A.perm + base;
    const int32_t *__restrict__ osrt = A.osorted + base;
    const int32_t *__restrict__ posof = A.posof + base;
    int32_t *pnext = A.plan_next + gwarp * (int64_t)n_slots;
    const int64_t out_off = (int64_t)run * A.n_inst * n_slots + base;
    int32_t *st_out = A.start_out ? A.start_out + out_off : nullptr;
    int32_t *co_out = A.compl_out ? A.compl_out + out_off : nullptr;
    const int words0 = (n + 31) >> 5, words1 = (words0 + 31) >> 5;
    // packed progress in the step kernel's stretch pays off from 8 register
    // rows on (measured); fewer rows keep the signed / unsigned sentinel
    constexpr bool kPacked = !EPOCH && SPL >= 8;
    constexpr int32_t kStartA = EPOCH ? 0 : (kPacked ? (int32_t)kPackedZero : 0);

    int64_t status = is.status;
    if (status == ISJL_OK && (int64_t)is.maxo > kv_cap) status = ISJL_ERR_INFEASIBLE;
    // every schedule ends by sum o + max arrival; the idle sentinel needs steps < 2^30
    if (status == ISJL_OK && is.O + (int64_t)is.maxA + 1 >= (int64_t)(1 << 30)) status = ISJL_ERR_INVALID_ARG;
    // requests that never start / finish report -1: on an error status, in a
    // run the caller's max_steps may stop, and in the unused slots of a ragged
    // instance (a full run writes every other entry)
    if (status != ISJL_OK || A.max_steps > 0 || n < n_slots) {
        if (st_out) for (int i = lane; i < n_slots; i += 32) st_out[i] = -1;
        if (co_out) for (int i = lane; i < n_slots; i += 32) co_out[i] = -1;
    }

    // W = sum over steps of |S| max r; E = W - R, where R = sum over steps of
    // sum r equals the sum over served requests of a (a + 1) / 2 for the
    // tokens a each received (one per step from 1): the step kernel adds
    // o (o + 1) / 2 when a request starts and takes back the unserved part of
    // requests still running if a run stops early (the decomposition W = Q + E
    // of Section 5)
    int64_t W = 0, R = 0, E = 0, sumc = 0, sumext = 0;
    int32_t peakkv = 0;
    int32_t Tb = 0, tok = 0, maxext = 0, viol = 0, peakb = 0, Tmake = 0, kvviol = 0;

    if (status == ISJL_OK && n > 0) {
        for (int w = lane; w < words0; w += 32) S.pend0[w] = 0u;
        for (int w = lane; w < words1; w += 32) S.pend1[w] = 0u;
        for (int w = lane; w < B; w += 32) { S.shead[w] = kNone; S.stail[w] = kNone; S.slong[w] = kNone; }
        __syncwarp();

        // worker w = r * 32 + lane: sa = progress (step kernel) or start step
        // (epoch kernel), sc = completion step (INT_MAX when idle)
        int32_t sa[SPL], sc[SPL];
#pragma unroll
        for (int r = 0; r < SPL; ++r) { sa[r] = kIdle; sc[r] = INT_MAX; }
        uint32_t busy = 0u, resv = 0u;
        uint32_t lhead = 0u;    // worker's next plan entry is its long job o_j (waits for o_1)
        int32_t lane_cmin = INT_MAX;                 // earliest completion among this lane's workers
        int32_t lane_smin = INT_MAX, lane_smax = INT_MIN;   // start range (epoch kernel)
        const int nrow = (B - lane + 31) >> 5;       // rows holding a valid worker for this lane
        const uint32_t vmask = nrow >= 32 ? ~0u : ((1u << nrow) - 1u);
        const int32_t alpha32 = (int32_t)min(alpha, (int64_t)INT_MAX);

        int32_t k = 0, rel = 0, fcfs = 0, done = 0, run_cnt = 0, pend = 0;
        // step kernel: register rows [0, adv_rows) are advanced each step; every
        // running worker lies in them, and their idle slots hold the sentinel
        int adv_rows = 0;
        // step kernel: A_max at the current step, from the last step's max reduction
        int32_t amax_c = 0;
        bool amax_ok = false;
        int32_t kv_sum = 0;
        uint32_t sum_st = 0;   // epoch kernel: the running requests' start steps, summed modulo 2^32
        // the next 32 unreleased requests (from win_base): arrival and sorted position, per lane
        int32_t win_base = 0, win_a = INT_MAX, win_p = 0;
        auto load_window = [&]() {
            const int i = win_base + lane;
            win_a = i < n ? arr[i] : INT_MAX;
            win_p = (i < n && policy != ISJL_POLICY_FCFS) ? posof[i] : 0;
        };
        load_window();
        // uniform caches, changed only at events
        int32_t next_arr = __shfl_sync(kFull, win_a, 0);   // arrival of the next unreleased request
        int32_t hp = INT_MAX, ho = 0, he = 0, ho_pos = -1;   // longest pending position, its o and index
        bool hvalid = true;                            // hp is current (else recompute from the bitset)
        int32_t fo = -1;                               // o of the FCFS head (-1: not loaded)
        int32_t cmin = INT_MAX;                        // earliest completion step of the running set
        int32_t smin = INT_MAX, smax = INT_MIN;        // start range of the running set (epoch kernel)
        int32_t kv_over = 0;                           // reserved KV above the cap (never, by construction)
        int32_t plan_left = 0, t0 = 0, d1 = 0, L1 = kNone, nlong = 0;
        bool L1_started = true;
        bool broken = false;   // an internal invariant failed: stop without touching memory
        const int64_t max_steps = A.max_steps > 0 ? A.max_steps : (is.O + (int64_t)is.maxA + 1);
        const int32_t step_guard = (int32_t)min(max_steps + 1, (int64_t)INT_MAX);

        auto recompute_lane = [&]() {
            lane_cmin = INT_MAX;
            if (EPOCH) { lane_smin = INT_MAX; lane_smax = INT_MIN; }
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                lane_cmin = min(lane_cmin, sc[r]);               // idle slots hold INT_MAX
                if (EPOCH && (busy >> r & 1u)) { lane_smin = min(lane_smin, sa[r]); lane_smax = max(lane_smax, sa[r]); }
            }
        };
        // start request e (length oe) on worker w at step k
        auto start = [&](int e, int oe, int w) {
            const int oc = otru ? otru[e] : oe;          // it finishes after its true length
            run_cnt++;
            kv_sum += oe;                                // and reserves its planning length
            cmin = min(cmin, k + oc);
            peakkv = max(peakkv, kv_sum);
            peakb = max(peakb, run_cnt);
            kv_over = kv_sum > kv_lim;
            if (EPOCH) { sum_st += (uint32_t)k; smin = min(smin, k); smax = k; }
            if (!EPOCH) mad_wide(R, ((uint32_t)oc * (uint32_t)(oc + 1)) >> 1, 1u);   // oc (oc + 1) < 2^32
            const int owner = w & 31, row = w >> 5;
            if (!EPOCH && row >= adv_rows) adv_rows = row_class<SPL>(row + 1);
            if (!EPOCH && run_cnt == 1) { amax_c = 0; amax_ok = true; }   // the only request: progress 0
            if (lane == owner) {
#pragma unroll
                for (int r = 0; r < SPL; ++r)
                    if (r == row) { sa[r] = EPOCH ? k : kStartA; sc[r] = k + oc; }
                busy |= 1u << row;
                lane_cmin = min(lane_cmin, k + oc);
                S.sres[w] = oe;
                if (EPOCH) { lane_smin = min(lane_smin, k); lane_smax = max(lane_smax, k); }
                S.sjob[w] = e;
                if (st_out) st_out[e] = k;
            }
        };
        // warp-wide totals of c starts at step k made lane-parallel: kv_add their
        // reserved KV, my_cmin / rsum this lane's earliest completion and sum of
        // o (o + 1) / 2, top the highest row that received one, plus one
        auto commit_starts = [&](int c, int32_t kv_add, int32_t my_cmin, uint64_t rsum, int top) {
            __syncwarp();
            lane_cmin = min(lane_cmin, my_cmin);
            if (EPOCH && my_cmin != INT_MAX) { lane_smin = min(lane_smin, k); lane_smax = max(lane_smax, k); }
            const bool was_empty = run_cnt == 0;
            run_cnt += c;
            kv_sum += kv_add;
            cmin = min(cmin, (int32_t)__reduce_min_sync(kFull, (unsigned)my_cmin));
            peakkv = max(peakkv, kv_sum);
            peakb = max(peakb, run_cnt);
            kv_over = kv_sum > kv_lim;
            if (EPOCH) { sum_st += (uint32_t)c * (uint32_t)k; smin = min(smin, k); smax = k; }
            if (!EPOCH) {
                // rsum < 2^35 per lane: its low 24 bits and the rest summed by two reductions
                const unsigned lo = __reduce_add_sync(kFull, (unsigned)(rsum & 0xFFFFFFu));
                const unsigned hi = __reduce_add_sync(kFull, (unsigned)(rsum >> 24));
                R += ((int64_t)hi << 24) + (int64_t)lo;
                if (top > adv_rows) adv_rows = row_class<SPL>(top);
                if (was_empty) { amax_c = 0; amax_ok = true; }   // the new requests: progress 0
            }
        };
        // Start, at step k, the longest prefix of up to 32 candidates (lane l < m
        // holds request ce and its planning length co) whose KV reservations fit
        // and for which free workers remain, candidate i on the i-th lowest
        // worker of the free mask fm.  The same outcome as starting them one at
        // a time, each on the lowest free worker, until the first that does not
        // fit.  Returns how many started.
        auto bulk_start = [&](int m, int ce, int co, uint32_t fm) -> int {
            int pre = lane < m ? co : 0;                          // inclusive prefix of co
#pragma unroll
            for (int d = 1; d < 32; d <<= 1) {
                const int t = __shfl_up_sync(kFull, pre, d);
                if (lane >= d) pre += t;
            }
            const int nfree = (int)__reduce_add_sync(kFull, (unsigned)__popc(fm));
            const bool fit = lane < m && lane < nfree && kv_sum + pre <= kv_lim;
            const int c = __popc(__ballot_sync(kFull, fit));
            if (c == 0) return 0;
            const int oc_l = (otru && lane < c) ? otru[ce] : co;  // it finishes after its true length
            const uint32_t lt = (1u << lane) - 1u;
            int base = 0, top = 0;
            int32_t my_cmin = INT_MAX;
            uint64_t rsum = 0;
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                if (base < c) {
                    const bool f = fm >> r & 1u;
                    const unsigned rowf = __ballot_sync(kFull, f);
                    const int rank = base + __popc(rowf & lt);     // among the free workers, in w order
                    const int src = rank & 31;
                    const int e = __shfl_sync(kFull, ce, src);
                    const int oe = __shfl_sync(kFull, co, src);
                    const int oc = __shfl_sync(kFull, oc_l, src);
                    if (f && rank < c) {
                        const int w = (r << 5) + lane;
                        sa[r] = EPOCH ? k : kStartA;
                        sc[r] = k + oc;
                        busy |= 1u << r;
                        my_cmin = min(my_cmin, k + oc);
                        S.sres[w] = oe;
                        S.sjob[w] = e;
                        if (st_out) st_out[e] = k;
                        if (!EPOCH) rsum += ((uint32_t)oc * (uint32_t)(oc + 1)) >> 1;
                    }
                    if (rowf) top = r + 1;
                    base += __popc(rowf);
                }
            }
            commit_starts(c, __shfl_sync(kFull, pre, c - 1), my_cmin, rsum, top);
            return c;
        };
        // requests completing at step c leave their workers
        auto retire = [&](int32_t c) {
            uint32_t fm = 0u;
            unsigned sf = 0u;   // sum of (start - (c - 65536)) over finishing requests (epoch kernel)
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                const bool f = sc[r] == c;                   // idle slots hold INT_MAX
                fm |= (uint32_t)f << r;
                if (f) {
                    if (EPOCH) sf += (unsigned)(sa[r] - (c - 65536));
                    sc[r] = INT_MAX;
                    if (!EPOCH && !kPacked) sa[r] = kIdle;
                }
            }
            // per finishing request (usually one per warp): outputs and its KV release
            int nf = 0, of = 0;
            for (uint32_t m = fm; m; m &= m - 1u) {
                const int w = ((__ffs(m) - 1) << 5) + lane;
                nf++;
                of += S.sres[w];
                if (co_out) co_out[S.sjob[w]] = c;
            }
            busy &= ~fm;
            // unconditional where measured cheaper than the branch (not the epoch kernel's 16 rows)
            if (!EPOCH || SPL <= 8 || fm) recompute_lane();
            if (!EPOCH) adv_rows = row_class<SPL>((int)__reduce_max_sync(kFull, 32u - (unsigned)__clz((int)busy)));
            nf = (int)__reduce_add_sync(kFull, (unsigned)nf);
            of = (int)__reduce_add_sync(kFull, (unsigned)of);
            if (EPOCH)   // starts are within 65535 steps of c, so the offsets fit 32 bits
                sum_st -= __reduce_add_sync(kFull, sf) + (uint32_t)nf * (uint32_t)(c - 65536);
            done += nf;
            run_cnt -= nf;
            if (!EPOCH && nf > 0) amax_ok = false;
            kv_sum -= of;
            kv_over = kv_sum > kv_lim;
            sumc += (int64_t)nf * c;
            Tmake = c;
            cmin = __reduce_min_sync(kFull, lane_cmin);
            if (EPOCH) {
                smin = __reduce_min_sync(kFull, lane_smin);
                smax = __reduce_max_sync(kFull, lane_smax);
            }
        };
        // A_max(k): largest progress among running requests (0 if none)
        auto amax_now = [&]() -> int32_t {
            if (run_cnt == 0) return 0;
            if (EPOCH) return k - smin;
            if (!amax_ok) {
                if constexpr (kPacked) {
                    uint32_t m = 0u;    // packed progress: the larger value has the larger a
#pragma unroll
                    for (int r = 0; r < SPL; ++r) if (busy >> r & 1u) m = max(m, (uint32_t)sa[r]);
                    amax_c = (int32_t)(__reduce_max_sync(kFull, m) >> 16);
                } else {
                    int m = 0;
#pragma unroll
                    for (int r = 0; r < SPL; ++r) if (busy >> r & 1u) m = max(m, sa[r]);
                    amax_c = __reduce_max_sync(kFull, m);
                }
                amax_ok = true;
            }
            return amax_c;
        };

        auto release = [&]() {
            for (;;) {
                // released: window lanes at or after rel whose arrival is <= k (a prefix)
                const bool ok = win_base + lane >= rel && win_a <= k;
                const unsigned b = __ballot_sync(kFull, ok);
                if (policy != ISJL_POLICY_FCFS) {
                    if (ok) {
                        atomicOr(&S.pend0[win_p >> 5], 1u << (win_p & 31));
                        atomicOr(&S.pend1[win_p >> 10], 1u << ((win_p >> 5) & 31));
                    }
                    if (hvalid) hp = min(hp, __reduce_min_sync(kFull, ok ? win_p : INT_MAX));
                }
                const int c = __popc(b);
                rel += c;
                pend += c;
                if (rel < win_base + 32 || win_base + 32 >= n) break;
                win_base += 32;                           // window used up: load the next 32
                load_window();
            }
            __syncwarp();
            next_arr = rel < n ? __shfl_sync(kFull, win_a, (rel - win_base) & 31) : INT_MAX;
        };
        // longest pending position (INT_MAX if none), its o and request index
        auto head = [&]() -> int {
            if (!hvalid) { hp = bs_next(S, words0, words1, 0, lane); hvalid = true; }
            if (hp < n && ho_pos != hp) { ho = osrt[hp]; he = perm[hp]; ho_pos = hp; }
            return hp;
        };
        // remove the head position p (the longest pending request)
        auto pop_head = [&](int p) {
            bs_clear(S, p, lane);
            pend--;
            hp = bs_next(S, words0, words1, p + 1, lane);   // nothing pending below p
        };
        // sorted positions of the first m (1 <= m <= 32) pending requests at or
        // after position p0: lane l gets the l-th, lanes past the last one -1
        // (uniform call)
        auto first_pending_from = [&](int p0, int m) -> int {
            int mine = -1;
            for (int wb = (p0 >> 10) << 5, got = 0; got < m && wb < words0; wb += 32) {
                if (S.pend1[wb >> 5] == 0u) continue;           // no pending in these 32 words
                const int wi = wb + lane;
                uint32_t x = wi < words0 ? S.pend0[wi] : 0u;
                if (wi < (p0 >> 5)) x = 0u;                     // below p0
                else if (wi == (p0 >> 5)) x &= ~0u << (p0 & 31);
                const int c = __popc(x);
                int incl = c;
#pragma unroll
                for (int d = 1; d < 32; d <<= 1) {
                    const int t = __shfl_up_sync(kFull, incl, d);
                    if (lane >= d) incl += t;
                }
                const int excl = incl - c;
                const int jj = lane - got;                      // this lane's rank within the chunk
                int lo = 0;
#pragma unroll
                for (int sh = 16; sh > 0; sh >>= 1)
                    if (__shfl_sync(kFull, incl, lo + sh - 1) <= jj) lo += sh;
                const uint32_t xw = __shfl_sync(kFull, x, lo);
                const int ew = __shfl_sync(kFull, excl, lo);
                const int tot = __shfl_sync(kFull, incl, 31);
                if (lane < m && jj >= 0 && jj < tot) mine = ((wb + lo) << 5) + nth_set_bit(xw, jj - ew);
                got += tot;
            }
            return mine;
        };
        // the first m (1 <= m <= min(32, pend)) pending requests: the longest first
        auto first_pending = [&](int m) -> int {
            if (!hvalid) { hp = bs_next(S, words0, words1, 0, lane); hvalid = true; }
            return first_pending_from(hp, m);
        };
        // remove the lanes' positions p (where take) from the pending set
        auto clear_pending = [&](int p, bool take) {
            if (take) {
                const uint32_t bit = 1u << (p & 31);
                const uint32_t old = atomicAnd(&S.pend0[p >> 5], ~bit);
                if ((old & ~bit) == 0u) atomicAnd(&S.pend1[p >> 10], ~(1u << ((p >> 5) & 31)));
            }
            __syncwarp();
        };
        // start the longest pending requests (LJF's batch, ISJL's Phase TWO) on
        // the free workers of fm_base until one does not fit or the workers run out
        auto start_longest = [&](uint32_t fm_base) -> void {
            // one at a time for the first two starts (usually all there are),
            // then 32 at a time; every round first checks that the head fits
            for (int nseq = 0; pend > 0;) {
                const int w = lowest_worker(fm_base & ~busy, lane);
                if (w < 0) return;
                const int p = head();
                if (p >= n) { broken = true; return; }
                if (kv_sum + ho > kv_lim) return;
                if (nseq < 2) {
                    const int e = he, oe = ho;
                    pop_head(p);
                    start(e, oe, w);
                    nseq++;
                    continue;
                }
                const int m = min(32, pend);
                const int q = first_pending(m);
                if (__ballot_sync(kFull, lane < m && q < 0)) { broken = true; return; }
                const int ce = q >= 0 ? perm[q] : 0;
                const int co = q >= 0 ? osrt[q] : 0;
                const int c = bulk_start(m, ce, co, fm_base & ~busy);
                clear_pending(q, lane < c);
                pend -= c;
                if (c < m) { hp = __shfl_sync(kFull, q, c); return; }   // the first one left is the head
                hvalid = false;
            }
        };

        // ISJL plan starts of every candidate worker in cand (per-lane row
        // mask) at once, in worker order, until the first whose next entry does
        // not fit the KV cap (then true is returned: the gate of the step is
        // shut); entries that must wait (o_1 delayed unless over, an o_j before
        // o_1 has started) are skipped.  o_1 itself never comes here: worker 0
        // is always the first candidate and is started one at a time.
        auto plan_bulk = [&](uint32_t cand, bool over) -> bool {
            bool stopped = false;
            int c = 0, top = 0;
            int32_t kv_add = 0;
            int32_t my_cmin = INT_MAX;
            uint64_t rsum = 0;
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                if (!stopped) {
                    const int w = (r << 5) + lane;
                    bool el = cand >> r & 1u;
                    int e = 0, oe = 0;
                    if (el) {
                        e = S.shead[w];
                        if (w == 0 && e == L1 && !over) el = false;
                        if (w >= 1 && w < nlong && e == S.slong[w] && !L1_started) el = false;
                        if (el) oe = S.spsum[w];
                    }
                    int pre = el ? oe : 0;                      // prefix over this row, in lane order
#pragma unroll
                    for (int d = 1; d < 32; d <<= 1) {
                        const int t = __shfl_up_sync(kFull, pre, d);
                        if (lane >= d) pre += t;
                    }
                    const bool fits = el && kv_sum + kv_add + pre <= kv_lim;
                    const unsigned fb = __ballot_sync(kFull, fits);
                    if (fb != __ballot_sync(kFull, el)) stopped = true;   // the first one that does not fit
                    if (fits) {
                        const int nx = pnext[e];
                        const int onx = nx >= 0 ? oarr[nx] : 0;
                        S.shead[w] = nx;
                        const uint32_t bit = 1u << r;
                        if (nx < 0) { S.stail[w] = kNone; resv &= ~bit; } else S.spsum[w] = onx;
                        if (w >= 1 && w < nlong && nx >= 0 && nx == S.slong[w]) lhead |= bit;
                        else lhead &= ~bit;
                        const int oc = otru ? otru[e] : oe;     // it finishes after its true length
                        sa[r] = EPOCH ? k : kStartA;
                        sc[r] = k + oc;
                        busy |= bit;
                        my_cmin = min(my_cmin, k + oc);
                        S.sres[w] = oe;
                        S.sjob[w] = e;
                        if (st_out) st_out[e] = k;
                        if (!EPOCH) rsum += ((uint32_t)oc * (uint32_t)(oc + 1)) >> 1;
                    }
                    if (fb) top = r + 1;
                    c += __popc(fb);
                    kv_add += (int32_t)__reduce_add_sync(kFull, fits ? (unsigned)oe : 0u);
                }
            }
            if (c > 0) commit_starts(c, kv_add, my_cmin, rsum, top);
            plan_left -= c;
            return stopped;
        };

        // ISJL Phase ONE at a stage start (Algorithm 2 with beta = alpha)
        auto phase_one = [&]() {
            t0 = k; d1 = 0; L1 = kNone; L1_started = true; nlong = 0;
            if (pend < 2) return;                               // |Q| = 1: Phase TWO
            const int p1 = bs_next(S, words0, words1, 0, lane);
            if (p1 >= n) { broken = true; return; }
            const int64_t o1 = osrt[p1];
            const int p2 = bs_next(S, words0, words1, p1 + 1, lane);
            // cap_j = min{2 alpha, o_1 - o_j + beta}, theta likewise (beta = alpha in Algorithm 2)
            if (p2 >= n) { broken = true; return; }
            if ((int64_t)osrt[p2] <= alpha) return;             // o_2 <= alpha: Phase TWO
            // M = min{B, #{o > alpha}} over Q(k)
            const int cnt_long = bs_count_below(S, words0, first_pos_le(osrt, n, alpha, lane), lane);
            const int nl = min(B, cnt_long);
            // packing budget left / pack sum per worker, in shared memory
            for (int w = lane; w < B; w += 32) {
                S.srem[w] = w >= nl ? (int32_t)alpha : -1;   // workers M+1..B: alpha
                S.spsum[w] = 0;
            }
            __syncwarp();
            // the long requests o_1..o_M (the first M pending positions) leave Q;
            // worker j's budget cap_j.  Up to 32 at a time: a prefix sum of the
            // bitset words' popcounts gives each lane the word and bit of its rank
            int olast_l = 0;
            for (int wb = 0, taken = 0; taken < nl; wb += 32) {
                if (wb >= words0) { broken = true; return; }
                const int wi = wb + lane;
                const uint32_t x = wi < words0 ? S.pend0[wi] : 0u;
                const int c = __popc(x);
                int incl = c;                                   // inclusive count over lanes
#pragma unroll
                for (int d = 1; d < 32; d <<= 1) {
                    const int t = __shfl_up_sync(kFull, incl, d);
                    if (lane >= d) incl += t;
                }
                const int excl = incl - c;
                const int m = min(nl - taken, __shfl_sync(kFull, incl, 31));   // ranks from this chunk
                for (int r0 = 0; r0 < m; r0 += 32) {
                    const int jj = r0 + lane;                       // rank within the chunk
                    int lo = 0;                                     // lanes whose words end before it
#pragma unroll
                    for (int sh = 16; sh > 0; sh >>= 1)
                        if (__shfl_sync(kFull, incl, lo + sh - 1) <= jj) lo += sh;
                    const uint32_t xw = __shfl_sync(kFull, x, lo);
                    const int ew = __shfl_sync(kFull, excl, lo);
                    if (jj < m) {
                        const int p = ((wb + lo) << 5) + nth_set_bit(xw, jj - ew);
                        const int j = taken + jj;
                        const int e = perm[p];
                        const int oe = osrt[p];
                        if (j == 0) {
                            S.shead[0] = e; S.stail[0] = e; pnext[e] = kNone;
                        } else {
                            S.slong[j] = e;
                            S.srem[j] = (int32_t)min(2 * alpha, o1 - (int64_t)oe + beta);
                        }
                        if (j == nl - 1) olast_l = oe;
                    }
                }
                // the taken bits of this lane's word leave the bitset
                const int tk = min(max(m - excl, 0), c);
                if (tk > 0) {
                    const uint32_t y = tk == c ? 0u : x & (~0u << nth_set_bit(x, tk));
                    S.pend0[wi] = y;
                    if (y == 0u) atomicAnd(&S.pend1[wi >> 5], ~(1u << (wi & 31)));
                }
                taken += m;
            }
            __syncwarp();
            L1 = S.shead[0];
            const int64_t o_last = __reduce_max_sync(kFull, olast_l);
            pend -= nl;
            const int64_t theta = min(2 * alpha, o1 - o_last + beta);
            // first fit of the shorter requests, in sorted order.  Nothing runs
            // at a stage start, so the slot registers sa[] are free: they hold
            // the packing budgets left, worker r * 32 + lane in sa[r] (-1 for
            // worker 1 and past B: never chosen), and are reset to idle below.
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                const int w = (r << 5) + lane;
                sa[r] = w < B ? S.srem[w] : -1;
            }
            // maxrem bounds the largest budget from above; it is recomputed only
            // when a candidate no larger than it fits nowhere (budgets only shrink)
            int maxrem = -1;
#pragma unroll
            for (int r = 0; r < SPL; ++r) maxrem = max(maxrem, sa[r]);
            maxrem = __reduce_max_sync(kFull, maxrem);
            // this lane's rows whose worker takes no long request (M+1..B)
            uint32_t rows_short = 0u;
#pragma unroll
            for (int r = 0; r < SPL; ++r) rows_short |= (uint32_t)((r << 5) + lane >= nl) << r;
            int q = -1;
            int64_t x_prev = -1;
            int pos_x = 0;                                      // first sorted position with o <= x_prev
            for (;;) {
                const int64_t x = min(theta, (int64_t)maxrem);
                if (x < 1) break;
                // candidates with o > x fit nowhere now or later
                if (x != x_prev) { pos_x = first_pos_le(osrt, n, x, lane); x_prev = x; }
                q = bs_next(S, words0, words1, max(pos_x, q + 1), lane);
                if (q >= n) break;
                const int e = perm[q];
                const int oe = osrt[q];
                uint32_t fit = 0u;                              // rows whose budget takes it
#pragma unroll
                for (int r = 0; r < SPL; ++r) fit |= (uint32_t)(sa[r] >= oe) << r;
                int w = lowest_worker(fit & rows_short, lane);  // workers M+1..B first
                if (w < 0) w = highest_worker(fit & ~rows_short, lane);   // then M, M-1, ..., 2
                if (w < 0) {                                    // it stays queued; the bound was stale
                    int m = -1;
#pragma unroll
                    for (int r = 0; r < SPL; ++r) m = max(m, sa[r]);
                    maxrem = __reduce_max_sync(kFull, m);
                    continue;
                }
                {
                    const int dec = lane == (w & 31) ? oe : 0;   // the chosen worker's budget shrinks
#pragma unroll
                    for (int r = 0; r < SPL; ++r) sa[r] -= r == (w >> 5) ? dec : 0;
                }
                __syncwarp();
                if (lane == 0) {
                    const int tl = S.stail[w];
                    if (tl < 0) S.shead[w] = e; else pnext[tl] = e;
                    S.stail[w] = e;
                    pnext[e] = kNone;
                    S.spsum[w] += oe;
                }
                bs_clear(S, q, lane);   // includes __syncwarp
                pend--;
                plan_left++;
            }
#pragma unroll
            for (int r = 0; r < SPL; ++r) sa[r] = kIdle;
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
            for (int w = 1 + lane; w < nl; w += 32) mx = max(mx, S.spsum[w]);
            mx = __reduce_max_sync(kFull, mx);
            d1 = (int32_t)min(max((int64_t)mx - alpha, (int64_t)0), alpha);
            resv = 0u;
            lhead = 0u;
#pragma unroll
            for (int r = 0; r < SPL; ++r) {
                const int w = (r << 5) + lane;
                if (w < B && S.shead[w] >= 0) resv |= 1u << r;
                if (w >= 1 && w < nl && S.shead[w] == S.slong[w]) lhead |= 1u << r;
            }
            L1_started = false;
            nlong = nl;
            hvalid = false;                                // Phase ONE removed queued requests
            // spsum now caches the length of each worker's next plan entry
            for (int w = lane; w < B; w += 32) {
                const int e = S.shead[w];
                S.spsum[w] = e >= 0 ? oarr[e] : 0;
            }
            __syncwarp();
        };

        // After an admission, `blocked` says that no arrival alone can let a
        // request start before the next completion (or o_1's delay expiry):
        // FCFS with B full or its head not fitting the KV cap, LJF with a batch
        // running, SJF with B full, ISJL with its gate closed or its queue
        // stopped on the KV cap or on workers (an arrival never becomes a head
        // that fits better: it sorts after every pending request of its length).
        // Arrivals are then released at the next event instead of ending the
        // run of plain steps there.
        bool blocked = false;
        auto admit = [&]() {
            if (policy == ISJL_POLICY_FCFS) {
                // arrival order; the first request that does not fit ends the step
                blocked = false;
                // one at a time for the first two starts (usually all there are),
                // then 32 at a time; every round first checks that the head fits
                for (int nseq = 0;;) {
                    if (run_cnt >= B) { blocked = true; break; }
                    if (fcfs >= rel) break;
                    if (fo < 0) fo = oarr[fcfs];
                    if (kv_sum + fo > kv_lim) { blocked = true; break; }
                    if (nseq < 2) {
                        const int w = lowest_worker(vmask & ~busy, lane);
                        if (w < 0) { broken = true; return; }
                        start(fcfs, fo, w);
                        fcfs++;
                        fo = -1;
                        nseq++;
                        continue;
                    }
                    const int m = min(32, rel - fcfs);
                    const int i = fcfs + lane;
                    const int c = bulk_start(m, i, lane < m ? oarr[i] : 0, vmask & ~busy);
                    fcfs += c;
                    fo = -1;
                    if (c < m) { blocked = true; break; }        // the KV cap or B stopped it
                }
            } else if (policy == ISJL_POLICY_SJF) {
                // shortest released request first (ties: lower index), continuous
                // batching.  The pending requests of the smallest length omin are
                // the pending positions from the first with o <= omin upwards, in
                // start order; one at a time for the first two starts, then up to
                // 32 of them at a time
                for (int nseq = 0; run_cnt < B && pend > 0;) {
                    const int hi = bs_last(S, words1, lane);
                    if (hi < 0 || hi >= n) { broken = true; return; }
                    const int omin = osrt[hi];
                    if (kv_sum + omin > kv_lim) break;
                    const int g = first_pos_le(osrt, n, omin, lane);
                    if (nseq < 2) {
                        const int p = bs_next(S, words0, words1, g, lane);
                        if (p >= n) { broken = true; return; }
                        const int w = lowest_worker(vmask & ~busy, lane);
                        if (w < 0) { broken = true; return; }
                        const int e = perm[p];
                        bs_clear(S, p, lane);
                        pend--;
                        start(e, omin, w);
                        nseq++;
                        continue;
                    }
                    const int q = first_pending_from(g, min(32, pend));
                    const int mg = __popc(__ballot_sync(kFull, q >= 0));   // of this length, in order
                    if (mg == 0) { broken = true; return; }
                    const int c = bulk_start(mg, q >= 0 ? perm[q] : 0, omin, vmask & ~busy);
                    clear_pending(q, lane < c);
                    pend -= c;
                    hvalid = false;
                    if (c < mg) break;
                }
                blocked = run_cnt >= B;
            } else if (policy == ISJL_POLICY_LJF) {
                // static batch of the longest released requests when nothing runs
                blocked = run_cnt != 0;
                if (run_cnt != 0) return;
                start_longest(vmask);
                blocked = run_cnt != 0;
            } else {
                const bool nothing_runs = run_cnt == 0;
                if (nothing_runs && plan_left == 0 && pend > 0) phase_one();
                if (broken) return;
                // the gate A_max(k) <= alpha; progress stays below o <= 65535, so a
                // budget of at least 65535 never shuts it
                bool stop = alpha32 < 65535 && amax_now() > alpha32;
                if (!stop && plan_left > 0) {
                    // plan starts, workers in order; entries that must wait (o_1's
                    // delay, o_j before o_1) are filtered out up front
                    uint32_t cand = resv & ~busy;
                    if (!L1_started) {
                        cand &= ~lhead;
                        const bool over = k >= t0 + d1;
                        if (!over && lane == 0) cand &= ~1u;        // worker 0 holds o_1
                    }
                    for (int nseq = 0;;) {
                        if (nseq >= 2) {                            // the rest at once
                            if (__ballot_sync(kFull, cand != 0u)) {
                                const bool over = k >= t0 + d1;
                                stop = plan_bulk(cand, over);
                            }
                            break;
                        }
                        const int w = lowest_worker(cand, lane);
                        if (w < 0) break;
                        if (lane == (w & 31)) cand &= ~(1u << (w >> 5));
                        const int e = S.shead[w];
                        if (w == 0 && e == L1) {
                            const bool over = k >= t0 + d1;
                            if (!over) continue;                 // o_1 still delayed
                        }
                        if (w >= 1 && w < nlong && e == S.slong[w] && !L1_started) continue;  // o_j after o_1
                        const int oe = S.spsum[w];                 // o of the worker's next entry
                        if (kv_sum + oe > kv_lim) { stop = true; break; }
                        const int nx = pnext[e];
                        __syncwarp();
                        if (lane == 0) {
                            S.shead[w] = nx;
                            if (nx < 0) S.stail[w] = kNone; else S.spsum[w] = oarr[nx];
                        }
                        __syncwarp();
                        if (lane == (w & 31)) {
                            const uint32_t bit = 1u << (w >> 5);
                            if (nx < 0) resv &= ~bit;
                            if (w >= 1 && w < nlong && nx >= 0 && nx == S.slong[w]) lhead |= bit;
                            else lhead &= ~bit;
                        }
                        plan_left--;
                        if (e == L1) {
                            L1_started = true;
                            cand |= resv & ~busy & lhead;            // the o_j may start now
                        }
                        start(e, oe, w);
                        nseq++;
                    }
                }
                if (!stop) start_longest(vmask & ~resv);   // Phase TWO: longest released first
                blocked = stop || pend > 0;
            }
        };

        // steps k .. k + L - 1 with no event: advance rows [0, NR), which hold
        // every running worker, and add each step's cost.
        //   SPL >= 8: a slot's progress a is packed as (a << 16) | (65535 - a)
        //   (o <= 65535): one add of 0xFFFF advances both halves (no borrow: a < o
        //   while the request runs), and a per-half unsigned max over a lane's
        //   slots, then two warp max reductions, give max r (upper half) and
        //   65535 - min r (lower half).  Idle slots of these rows are first set
        //   to (0, L): after j steps they hold (j, L - j), at most the running
        //   slots' halves, since every running request has a >= j and none
        //   completes inside the stretch (min a + L <= its o <= 65535).
        //   SPL < 8: idle slots hold a value below 0 as a signed number and at
        //   least 2^31 as an unsigned one, so they lose the signed max and the
        //   unsigned min.
        auto plain_steps = [&](auto nr_tag, int L) {
            constexpr int NR = decltype(nr_tag)::value;
            const uint32_t cnt = (uint32_t)run_cnt;
            constexpr int kUnroll = SPL >= 16 ? 4 : 2;   // measured; more code costs instruction-cache misses
            if constexpr (kPacked) {
#pragma unroll
                for (int r = 0; r < NR; ++r)
                    if (!(busy >> r & 1u)) sa[r] = L;
                uint32_t last_mx = 0u, smx = 0u, sext = 0u;   // sums over the stretch: L, r < 2^16
#pragma unroll kUnroll
                for (int j = 0; j < L; ++j) {
                    uint32_t m = 0u;
#pragma unroll
                    for (int r = 0; r < NR; ++r) {
                        const uint32_t a = (uint32_t)sa[r] + kPackedStep;
                        sa[r] = (int32_t)a;
                        m = vmax_u16x2(m, a);
                    }
                    const uint32_t mx = __reduce_max_sync(kFull, m) >> 16;          // max r
                    const uint32_t lo = __reduce_max_sync(kFull, m & 0xFFFFu);      // 65535 - min r
                    const int ext = (int)(mx + lo) - 65535;
                    smx += mx;
                    sext += (uint32_t)ext;
                    maxext = max(maxext, ext);
                    viol += ext > alpha32;
                    last_mx = mx;
                }
                mad_wide(W, cnt, smx);                   // |S| max r, summed over the steps
                sumext += sext;
                amax_c = (int32_t)last_mx;               // max progress entering step k + L
            } else {
                int last_mx = 0;
                uint32_t smx = 0u, sext = 0u;            // sums over the stretch: L, r < 2^16
#pragma unroll kUnroll
                for (int j = 0; j < L; ++j) {
                    int mx = INT_MIN;
                    unsigned mn = 0xffffffffu;
#pragma unroll
                    for (int r = 0; r < NR; ++r) {
                        const int a = sa[r] + 1;
                        sa[r] = a;
                        mx = max(mx, a);
                        mn = min(mn, (unsigned)a);
                    }
                    mx = __reduce_max_sync(kFull, mx);
                    mn = __reduce_min_sync(kFull, mn);
                    const int ext = mx - (int)mn;
                    smx += (uint32_t)mx;
                    sext += (uint32_t)ext;
                    maxext = max(maxext, ext);
                    viol += ext > alpha32;
                    last_mx = mx;
                }
                mad_wide(W, cnt, smx);                   // |S| max r, summed over the steps
                sumext += sext;
                amax_c = last_mx;                        // max progress entering step k + L
            }
            amax_ok = true;
        };

        // epoch kernel: the step at which the running set's earliest or latest
        // start changes (the last completion among the requests that started at
        // smin, or at smax)
        auto window_end = [&]() -> int32_t {
            int32_t e_lo = INT_MIN, e_hi = INT_MIN;
#pragma unroll
            for (int r = 0; r < SPL; ++r)
                if (busy >> r & 1u) {
                    if (sa[r] == smin) e_lo = max(e_lo, sc[r]);
                    if (sa[r] == smax) e_hi = max(e_hi, sc[r]);
                }
            return min(__reduce_max_sync(kFull, e_lo), __reduce_max_sync(kFull, e_hi));
        };
        // epoch kernel: serve steps k .. K - 1 at once, K <= the step at which
        // the earliest or latest start changes.  Every running request i
        // (start s_i, completion c_i) runs L_i = min(c_i, K) - k of them, with
        // max r = t - smin + 1 at step t and r_i = t - s_i + 1:
        //   W += L_i (k - smin + 1) + L_i (L_i - 1) / 2,  E += L_i (s_i - smin),
        // and the extent smax - smin is constant.  Requests with c_i < K
        // complete inside the window and leave here.
        auto window = [&](int32_t K) {
            // twice the W term per slot: L_i (2 m0 - 1 + L_i), m0 = k - smin + 1;
            // all factors below 2^32
            const uint32_t m2 = 2u * (uint32_t)(k - smin) + 1u;
            uint64_t wl2 = 0, el = 0, cl = 0;
            uint32_t sl = 0;
            int32_t tl = 0, cmx = 0, nf = 0, of = 0;
            uint32_t fm = 0u;
#pragma unroll
            for (int r = 0; r < SPL; ++r)
                if (busy >> r & 1u) {
                    const int32_t c = sc[r];
                    const uint32_t Li = (uint32_t)(min(c, K) - k);
                    wl2 += (uint64_t)Li * (m2 + Li);
                    el += (uint64_t)Li * (uint32_t)(sa[r] - smin);
                    tl += (int32_t)Li;
                    if (c < K) {                                  // completes inside the window
                        const int w = (r << 5) + lane;
                        fm |= 1u << r;
                        cl += (uint32_t)c;
                        sl += (uint32_t)sa[r];
                        cmx = max(cmx, c);
                        nf++;
                        of += S.sres[w];
                        if (co_out) co_out[S.sjob[w]] = c;
                        sc[r] = INT_MAX;
                    }
                }
            busy &= ~fm;
            recompute_lane();
            W += (int64_t)(warp_sum_u64(wl2) >> 1);             // every slot's term is even
            E += (int64_t)warp_sum_u64(el);
            tok += (int32_t)__reduce_add_sync(kFull, (unsigned)tl);
            nf = (int32_t)__reduce_add_sync(kFull, (unsigned)nf);
            of = (int32_t)__reduce_add_sync(kFull, (unsigned)of);
            sumc += (int64_t)warp_sum_u64(cl);
            sum_st -= __reduce_add_sync(kFull, sl);
            const int32_t cm = (int32_t)__reduce_max_sync(kFull, (unsigned)cmx);
            if (nf > 0) Tmake = max(Tmake, cm);
            done += nf;
            run_cnt -= nf;
            kv_sum -= of;
            kv_over = kv_sum > kv_lim;
            cmin = __reduce_min_sync(kFull, lane_cmin);
            const int32_t ext = smax - smin;                  // unchanged inside the window
            const int32_t L = K - k;
            sumext += (int64_t)L * ext;
            maxext = max(maxext, ext);
            viol += ext > alpha32 ? L : 0;
            Tb += L;
        };

        // release every request with A_i <= k (a prefix: arrivals are non-decreasing)
        if (!EPOCH) {
            // ---------------------------------------------------- step kernel
            int32_t next_check = 0;   // the next step needing release / admission / the guard
            for (;;) {
                if (k >= next_check) {
                    if (k >= step_guard) { status = ISJL_ERR_STEP_LIMIT; break; }
                    if (done == n) break;
                    if (k >= next_arr) release();
                    admit();
                    if (broken) { status = ISJL_ERR_INTERNAL; break; }
                    next_check = blocked && run_cnt > 0 ? INT_MAX : next_arr;
                    if (policy == ISJL_POLICY_ISJL && !L1_started && t0 + d1 > k) next_check = min(next_check, t0 + d1);
                    next_check = min(next_check, step_guard);
                }
                if (run_cnt == 0) { k = next_check; continue; }   // idle steps: nothing to serve
                // no arrival, completion, delay expiry or guard before step e
                const int32_t e = min(next_check, cmin);
                const int L = e - k;
                {
                    auto f = [&](auto nr_tag) { plain_steps(nr_tag, L); };
                    if (adv_rows < 1) broken = true;
                    else dispatch_rows<SPL, 0, RowClasses<SPL>::n - 1>(adv_rows, f);
                }
                if (broken) { status = ISJL_ERR_INTERNAL; break; }
                Tb += L;
                tok += L * run_cnt;
                if (kv_over) kvviol += L;
                k = e;
                if (k == cmin && k < step_guard) {   // requests that finished in step k - 1 leave
                    retire(k);
                    next_check = k;
                }
            }
            // a request still running (a run stopped early) with progress a and
            // true length o = a + (completion - k) has served only a (a + 1) / 2
            int64_t unserved = 0;
#pragma unroll
            for (int r = 0; r < SPL; ++r)
                if (busy >> r & 1u) {
                    const uint32_t a = kPacked ? (uint32_t)sa[r] >> 16 : (uint32_t)sa[r];
                    const uint32_t o = a + (uint32_t)(sc[r] - k);
                    unserved += (int64_t)((o * (o + 1u)) >> 1) - (int64_t)((a * (a + 1u)) >> 1);
                }
            E = W - (R - warp_sum64(unserved));
        } else {
            // --------------------------------------------------- epoch kernel
            for (;;) {
                if (k >= step_guard) { status = ISJL_ERR_STEP_LIMIT; break; }   // k > max_steps
                if (k >= next_arr) release();
                if (k == cmin) retire(k);
                if (done == n) break;
                admit();
                if (broken) { status = ISJL_ERR_INTERNAL; break; }
                // next event: arrival, completion or the end of o_1's delay
                int32_t nxt = min(blocked && run_cnt > 0 ? INT_MAX : next_arr, cmin);
                if (policy == ISJL_POLICY_ISJL && !L1_started && t0 + d1 > k) nxt = min(nxt, t0 + d1);
                if (nxt == INT_MAX) { status = ISJL_ERR_STEP_LIMIT; break; }   // cannot progress
                nxt = min(nxt, step_guard);                          // serve no step past max_steps
                // LJF with a batch running, or ISJL with its gate shut (A_max only
                // grows while the earliest start stays): no request can start
                // before the running set's earliest or latest start changes, so
                // completions in between end no epoch of their own
                if (run_cnt > 0 && !kv_over && nxt == cmin &&
                    (policy == ISJL_POLICY_LJF || (policy == ISJL_POLICY_ISJL && k - smin > alpha32))) {
                    const int32_t K = min(window_end(), step_guard);
                    if (K > nxt) {
                        window(K);
                        k = K;
                        continue;
                    }
                }
                if (run_cnt > 0) {
                    // L steps, max r = m0 + t at step k + t, sum r = s m0 - sum (s_i - smin) + s t:
                    //   W += s (L m0 + L (L - 1) / 2),  E += L sum (s_i - smin)
                    // The epoch ends by the completion of the request that started at
                    // smin, so max r <= its o <= 65535 throughout: the sum of max r over
                    // the L <= 65535 steps fits 32 bits, and sum (s_i - smin) <
                    // B * 65536 is exact from the modular sum of starts.
                    const uint32_t L = (uint32_t)(nxt - k), s = (uint32_t)run_cnt;
                    const uint32_t m0 = (uint32_t)(k - smin + 1);     // max r at step k
                    const int32_t ext = smax - smin;                  // max r - min r
                    mad_wide(W, s, L * m0 + ((L * (L - 1u)) >> 1));
                    mad_wide(E, L, sum_st - s * (uint32_t)smin);
                    mad_wide(sumext, L, (uint32_t)ext);
                    maxext = max(maxext, ext);
                    viol += ext > alpha32 ? (int32_t)L : 0;
                    kvviol += kv_over ? (int32_t)L : 0;
                    Tb += (int32_t)L;
                    tok += (int32_t)(s * L);
                }
                k = nxt;
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
            R.ael = n > 0 ? __ddiv_rn((double)sumc, (double)n) : 0.0;
        }
        A.records[(int64_t)run * A.n_inst + inst] = R;
        if (status != ISJL_OK) atomicCAS(A.dev_status, 0, (int32_t)status);
    }
    __syncwarp();
}

// resident blocks per SM the register allocation is bounded for, per
// instantiation (measured on GB300): 4 (up to 128 registers) in general;
// SPL_BLOCKS16 for 16 register rows (B > 256), where shared memory already
// limits large instances to 2 blocks per SM and a tighter bound only spills;
// SPL_BLOCKS4_STEP for the step kernel with 4 rows (B <= 128)
#ifndef ISJL_SIM_MIN_BLOCKS
#define ISJL_SIM_MIN_BLOCKS 4
#endif
#ifndef ISJL_SIM_BLOCKS16
#define ISJL_SIM_BLOCKS16 3
#endif
#ifndef ISJL_SIM_BLOCKS4_STEP
#define ISJL_SIM_BLOCKS4_STEP 5
#endif
template <int SPL, bool EPOCH>
constexpr int sim_min_blocks() {
    return SPL >= 16 ? ISJL_SIM_BLOCKS16 : (SPL == 4 && !EPOCH ? ISJL_SIM_BLOCKS4_STEP : ISJL_SIM_MIN_BLOCKS);
}

template <int SPL, bool EPOCH>
__global__ void __launch_bounds__(kSimWarpsPerBlock * 32, sim_min_blocks<SPL, EPOCH>())
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
    S.srem = b + 4 * A.B;
    S.spsum = b + 5 * A.B;
    S.sres = b + 6 * A.B;
    S.pend0 = reinterpret_cast<uint32_t *>(b + 7 * A.B);
    S.pend1 = S.pend0 + A.words0;
    const int64_t gwarp = (int64_t)blockIdx.x * kSimWarpsPerBlock + wib;
    for (;;) {
        int t = 0;
        if (lane == 0) t = atomicAdd(A.task_counter, 1);
        t = __shfl_sync(kFull, t, 0);
        if ((int64_t)t >= n_tasks) break;
        // run-major: at any time the warps of an SM mostly run one policy's code
        const int64_t inst = t % A.n_inst;
        const int run = (int)(t / A.n_inst);
        switch (A.runs.policy[run]) {
            case ISJL_POLICY_FCFS: run_task<SPL, EPOCH, ISJL_POLICY_FCFS>(A, S, lane, gwarp, inst, run); break;
            case ISJL_POLICY_LJF:  run_task<SPL, EPOCH, ISJL_POLICY_LJF>(A, S, lane, gwarp, inst, run); break;
            case ISJL_POLICY_SJF:  run_task<SPL, EPOCH, ISJL_POLICY_SJF>(A, S, lane, gwarp, inst, run); break;
            default:               run_task<SPL, EPOCH, ISJL_POLICY_ISJL>(A, S, lane, gwarp, inst, run); break;
        }
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
    int bps = 0, sms = 0, dev = 0;
    size_t smem = 0;
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
