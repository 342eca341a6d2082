// prep_kernels.cu -- per-instance preparation and cross-instance summaries.
//
//   derive     o_i = prompt_i + output_i (Section 2), input validation and the
//              policy-independent totals O = sum o_i and
//              Q = sum o_i (o_i + 1) / 2 (Eq. intrinsic-resource-cost)
//   sort       the order o_1 >= o_2 >= ... of Algorithms 1 and 2 (ties by
//              index): a permutation, its inverse and the sorted lengths;
//              bitonic in shared memory for small instances, a stable
//              two-pass LSD radix sort for large ones
//   summarize  per-run totals over all instances, a fixed-order reduction
#include <climits>
#include <cstdint>

#include "sim_internal.cuh"

namespace isjl {
namespace {

constexpr int kDeriveThreads = 256;
constexpr int kSortThreads = 256;
constexpr int kSumThreads = 256;

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(kFull, v, s);
    return v;
}
template <typename T>
__device__ __forceinline__ T warp_max(T v) {
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) v = max(v, __shfl_xor_sync(kFull, v, s));
    return v;
}

// one block per instance
__global__ void __launch_bounds__(kDeriveThreads)
derive_kernel(const int32_t *__restrict__ arrival, const int32_t *__restrict__ prompt,
              const int32_t *__restrict__ output, const int32_t *__restrict__ count,
              const int32_t *__restrict__ slack, int32_t *__restrict__ o, int32_t *__restrict__ otrue,
              InstStats *inst, int32_t n_slots) {
    const int64_t base = (int64_t)blockIdx.x * n_slots;
    int64_t O = 0, Q = 0, sumA = 0;
    int32_t maxo = 0, maxA = 0, invalid = 0, infeasible = 0;
    int32_t n = count ? count[blockIdx.x] : n_slots;
    if (n < 0 || n > n_slots) { invalid = 1; n = 0; }
    for (int i = threadIdx.x; i < n; i += kDeriveThreads) {
        const int32_t a = arrival[base + i], p = prompt[base + i], q = output[base + i];
        const int32_t e = slack ? slack[base + i] : 0;
        const int64_t oi = (int64_t)p + q;
        const int64_t ui = oi + e;                  // planning length (Robust-ISJL's u_i)
        if (a < 0 || p < 0 || q < 0 || e < 0 || (i > 0 && arrival[base + i - 1] > a) || ui > ISJL_MAX_LEN)
            invalid = 1;
        else if (oi < 1) infeasible = 1;
        const bool ok = oi >= 0 && ui <= ISJL_MAX_LEN && e >= 0;
        const int32_t oc = ok ? (int32_t)oi : 0;
        const int32_t uc = ok ? (int32_t)ui : 0;
        o[base + i] = uc;
        if (otrue) otrue[base + i] = oc;
        O += oc;
        Q += (int64_t)oc * (oc + 1) / 2;
        sumA += a;
        maxo = max(maxo, uc);
        maxA = max(maxA, a);
    }
    O = warp_sum(O); Q = warp_sum(Q); sumA = warp_sum(sumA);
    maxo = warp_max(maxo); maxA = warp_max(maxA);
    invalid = warp_max(invalid); infeasible = warp_max(infeasible);
    __shared__ int64_t s64[3][kDeriveThreads / 32];
    __shared__ int32_t s32[4][kDeriveThreads / 32];
    const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        s64[0][wid] = O; s64[1][wid] = Q; s64[2][wid] = sumA;
        s32[0][wid] = maxo; s32[1][wid] = maxA; s32[2][wid] = invalid; s32[3][wid] = infeasible;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        InstStats st{};
        for (int w = 0; w < kDeriveThreads / 32; ++w) {
            st.O += s64[0][w]; st.Q += s64[1][w]; st.sumA += s64[2][w];
            st.maxo = max(st.maxo, s32[0][w]); st.maxA = max(st.maxA, s32[1][w]);
            invalid |= s32[2][w]; infeasible |= s32[3][w];
        }
        st.status = invalid ? ISJL_ERR_INVALID_ARG : (infeasible ? ISJL_ERR_INFEASIBLE : ISJL_OK);
        st.n = n;
        inst[blockIdx.x] = st;
    }
}

__device__ __forceinline__ uint32_t len_key(int32_t o) {   // larger o sorts first
    const int32_t c = o < 0 ? 0 : (o > ISJL_MAX_LEN ? ISJL_MAX_LEN : o);
    return (uint32_t)(ISJL_MAX_LEN - c);
}

// n <= 4096: keys (65535 - o) << 16 | index, bitonic sort in shared memory
__global__ void __launch_bounds__(kSortThreads)
sort_small_kernel(const int32_t *__restrict__ o, const InstStats *__restrict__ inst, int32_t *__restrict__ perm,
                  int32_t *__restrict__ osorted, int32_t *__restrict__ posof, int32_t n_slots, int32_t npow2) {
    extern __shared__ uint32_t key[];
    const int64_t base = (int64_t)blockIdx.x * n_slots;
    const int32_t n = inst[blockIdx.x].n;
    for (int t = threadIdx.x; t < npow2; t += kSortThreads)
        key[t] = t < n ? (len_key(o[base + t]) << 16) | (uint32_t)t : 0xffffffffu;
    for (int size = 2; size <= npow2; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            __syncthreads();
            for (int t = threadIdx.x; t < npow2; t += kSortThreads) {
                const int u = t ^ stride;
                if (u > t) {
                    const bool up = (t & size) == 0;
                    const uint32_t x = key[t], y = key[u];
                    if ((x > y) == up) { key[t] = y; key[u] = x; }
                }
            }
        }
    }
    __syncthreads();
    for (int p = threadIdx.x; p < n; p += kSortThreads) {
        const uint32_t k = key[p];
        const int idx = (int)(k & 0xffffu);
        perm[base + p] = idx;
        osorted[base + p] = ISJL_MAX_LEN - (int32_t)(k >> 16);
        posof[base + idx] = p;
    }
}

// large n: stable LSD radix sort on the 16-bit key, two 8-bit passes.  Each
// thread owns a contiguous chunk; per-(digit, thread) counts in shared memory
// (padded rows) give every element its stable output position.
constexpr int kCntStride = kRadixThreads + 1;

__global__ void __launch_bounds__(kRadixThreads)
sort_radix_kernel(const int32_t *__restrict__ o, const InstStats *__restrict__ inst, int32_t *__restrict__ perm,
                  int32_t *__restrict__ osorted, int32_t *__restrict__ posof, int32_t *__restrict__ tmp,
                  int32_t n_slots) {
    extern __shared__ uint32_t cnt[];             // [256][kCntStride]
    __shared__ uint32_t dbase[256];
    const int64_t base = (int64_t)blockIdx.x * n_slots;
    const int32_t n = inst[blockIdx.x].n;
    const int tid = threadIdx.x;
    const int chunk = (n + kRadixThreads - 1) / kRadixThreads;
    const int lo = min(n, tid * chunk), hi = min(n, lo + chunk);
    for (int pass = 0; pass < 2; ++pass) {
        const int shift = pass * 8;
        const int32_t *src = pass == 0 ? nullptr : tmp + base;
        int32_t *dst = pass == 0 ? tmp + base : perm + base;
        for (int d = 0; d < 256; ++d) cnt[d * kCntStride + tid] = 0u;
        __syncthreads();
        for (int j = lo; j < hi; ++j) {
            const int idx = src ? src[j] : j;
            const uint32_t d = (len_key(o[base + idx]) >> shift) & 255u;
            cnt[d * kCntStride + tid]++;
        }
        __syncthreads();
        for (int d = tid; d < 256; d += kRadixThreads) {
            uint32_t run = 0;
            for (int t = 0; t < kRadixThreads; ++t) {
                const uint32_t v = cnt[d * kCntStride + t];
                cnt[d * kCntStride + t] = run;
                run += v;
            }
            dbase[d] = run;
        }
        __syncthreads();
        if (tid == 0) {
            uint32_t run = 0;
            for (int d = 0; d < 256; ++d) { const uint32_t v = dbase[d]; dbase[d] = run; run += v; }
        }
        __syncthreads();
        for (int j = lo; j < hi; ++j) {
            const int idx = src ? src[j] : j;
            const uint32_t d = (len_key(o[base + idx]) >> shift) & 255u;
            const uint32_t pos = dbase[d] + cnt[d * kCntStride + tid]++;
            dst[pos] = idx;
        }
        __syncthreads();
    }
    for (int p = tid; p < n; p += kRadixThreads) {
        const int idx = perm[base + p];
        osorted[base + p] = ISJL_MAX_LEN - (int32_t)len_key(o[base + idx]);
        posof[base + idx] = p;
    }
}

// one block per run; fixed assignment of records to threads and a fixed tree
__global__ void __launch_bounds__(kSumThreads)
summarize_kernel(const isjl_record *__restrict__ rec, int64_t n_inst, RunList runs, int32_t kv_cap,
                 isjl_summary *out) {
    const int run = blockIdx.x;
    const isjl_record *R = rec + (int64_t)run * n_inst;
    constexpr int NI = 13, ND = 6;
    int64_t vi[NI] = {0};
    double vd[ND] = {0.0};
    int64_t maxext = 0, n_ok = 0, first_bad = INT64_MAX;
    for (int64_t i = threadIdx.x; i < n_inst; i += kSumThreads) {
        const isjl_record &r = R[i];
        vi[0] += r.T_make; vi[1] += r.T_busy; vi[2] += r.O; vi[3] += r.Q; vi[4] += r.W; vi[5] += r.E;
        vi[6] += r.token_adv; vi[7] += r.sum_completion; vi[8] += r.sum_latency; vi[9] += r.sum_extent;
        vi[10] += r.violations; vi[11] += r.kv_violations; vi[12] += 0;
        vd[0] += r.c_T; vd[1] += r.tau_Q; vd[2] += r.tau_E; vd[3] += r.cost; vd[4] += r.revenue; vd[5] += r.profit;
        maxext = max(maxext, r.max_extent);
        if (r.status == ISJL_OK) n_ok++; else first_bad = min(first_bad, i);
    }
    __shared__ int64_t si[kSumThreads];
    __shared__ double sd[kSumThreads];
    auto red_i = [&](int64_t v, int op) -> int64_t {   // op 0 sum, 1 max, 2 min
        si[threadIdx.x] = v;
        __syncthreads();
        for (int s = kSumThreads / 2; s > 0; s >>= 1) {
            if (threadIdx.x < s) {
                const int64_t a = si[threadIdx.x], b = si[threadIdx.x + s];
                si[threadIdx.x] = op == 0 ? a + b : (op == 1 ? max(a, b) : min(a, b));
            }
            __syncthreads();
        }
        const int64_t r = si[0];
        __syncthreads();
        return r;
    };
    auto red_d = [&](double v) -> double {
        sd[threadIdx.x] = v;
        __syncthreads();
        for (int s = kSumThreads / 2; s > 0; s >>= 1) {
            if (threadIdx.x < s) sd[threadIdx.x] = __dadd_rn(sd[threadIdx.x], sd[threadIdx.x + s]);
            __syncthreads();
        }
        const double r = sd[0];
        __syncthreads();
        return r;
    };
    isjl_summary S;
    S.T_make = red_i(vi[0], 0); S.T_busy = red_i(vi[1], 0); S.O = red_i(vi[2], 0); S.Q = red_i(vi[3], 0);
    S.W = red_i(vi[4], 0); S.E = red_i(vi[5], 0); S.token_adv = red_i(vi[6], 0);
    S.sum_completion = red_i(vi[7], 0); S.sum_latency = red_i(vi[8], 0); S.sum_extent = red_i(vi[9], 0);
    S.violations = red_i(vi[10], 0); S.kv_violations = red_i(vi[11], 0);
    S.max_extent = red_i(maxext, 1);
    S.n_ok = red_i(n_ok, 0);
    const int64_t fb = red_i(first_bad, 2);
    S.c_T = red_d(vd[0]); S.tau_Q = red_d(vd[1]); S.tau_E = red_d(vd[2]);
    S.cost = red_d(vd[3]); S.revenue = red_d(vd[4]); S.profit = red_d(vd[5]);
    if (threadIdx.x == 0) {
        S.policy = runs.policy[run];
        S.delta = runs.delta[run];
        S.kv_cap = kv_cap;
        S.n_instances = n_inst;
        S.status = fb == INT64_MAX ? ISJL_OK : (int32_t)R[fb].status;
        out[run] = S;
    }
}

}  // namespace

cudaError_t launch_derive(const int32_t *arrival, const int32_t *prompt, const int32_t *output,
                          const int32_t *count, const int32_t *slack, int32_t *o, int32_t *otrue,
                          InstStats *inst, int64_t n_inst, int32_t n, cudaStream_t s) {
    derive_kernel<<<(unsigned)n_inst, kDeriveThreads, 0, s>>>(arrival, prompt, output, count, slack, o, otrue,
                                                              inst, n);
    return cudaGetLastError();
}

cudaError_t launch_sort(const int32_t *o, const InstStats *inst, int32_t *perm, int32_t *osorted, int32_t *posof,
                        int32_t *tmp, int64_t n_inst, int32_t n, cudaStream_t s) {
    if (n <= kSortSmallMax) {
        int npow2 = 1;
        while (npow2 < n) npow2 <<= 1;
        sort_small_kernel<<<(unsigned)n_inst, kSortThreads, npow2 * sizeof(uint32_t), s>>>(o, inst, perm, osorted,
                                                                                         posof, n, npow2);
        return cudaGetLastError();
    }
    const size_t smem = 256 * kCntStride * sizeof(uint32_t);
    cudaError_t e = cudaFuncSetAttribute(sort_radix_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    sort_radix_kernel<<<(unsigned)n_inst, kRadixThreads, smem, s>>>(o, inst, perm, osorted, posof, tmp, n);
    return cudaGetLastError();
}

cudaError_t launch_summarize(const isjl_record *records, int64_t n_inst, int32_t n_runs, const RunList &runs,
                             int32_t kv_cap, isjl_summary *out, cudaStream_t s) {
    summarize_kernel<<<n_runs, kSumThreads, 0, s>>>(records, n_inst, runs, kv_cap, out);
    return cudaGetLastError();
}

}  // namespace isjl
