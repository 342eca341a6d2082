// sim_internal.cuh -- internal definitions shared by the simulator's kernels
// and its C-ABI host code (not part of the public interface).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "isjl_sim.h"

namespace isjl {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarp = 32;
constexpr int kSimWarpsPerBlock = 4;         // 128-thread blocks for the simulation kernel
constexpr int kSortSmallMax = 4096;           // bitonic in shared memory up to this n
constexpr int kRadixThreads = 128;            // threads of the large-n radix sort

// Per-instance facts derived once per call (policy independent).
struct InstStats {
    int64_t O;        // sum o_i (true lengths)
    int64_t Q;        // sum o_i (o_i + 1) / 2
    int64_t sumA;     // sum of arrivals
    int32_t maxo;     // largest planning length u_i (= o_i without slack): KV feasibility
    int32_t maxA;     // largest arrival
    int32_t status;   // ISJL_OK, ISJL_ERR_INVALID_ARG or ISJL_ERR_INFEASIBLE (o_i < 1)
    int32_t n;        // requests of this instance (its first n slots)
};

// (policy, delta) list of one sweep, passed by value to the kernel.
struct RunList {
    int32_t policy[ISJL_MAX_RUNS];
    int32_t delta[ISJL_MAX_RUNS];
    int32_t beta[ISJL_MAX_RUNS];    // ISJL packing slack: delta, or Algorithm "ISJL"'s beta
};

// floor((sqrt(17) - 1) / 4 * alpha) exactly: the largest m with (4m + alpha)^2 <= 17 alpha^2
inline int32_t isjl_beta(int32_t alpha) {
    if (alpha > 1000000) return alpha;   // no plan exists when alpha >= every length
    const int64_t a = alpha;
    int64_t m = (int64_t)(0.780776406404415 * (double)alpha);
    while (m > 0 && (4 * m + a) * (4 * m + a) > 17 * a * a) m--;
    while ((4 * (m + 1) + a) * (4 * (m + 1) + a) <= 17 * a * a) m++;
    return (int32_t)m;
}
inline int32_t run_beta(int32_t policy, int32_t delta) {
    return policy == ISJL_POLICY_ISJL_BETA ? isjl_beta(delta) : delta;
}

struct SimArgs {
    const int32_t *arrival;    // [N] instance-major
    const int32_t *o;          // [N] planning length u_i = prompt + output (+ slack)
    const int32_t *otrue;      // [N] true length o_i, or null when there is no slack
    const int32_t *perm;       // [N] sorted position -> request index within its instance
    const int32_t *osorted;    // [N] o at each sorted position (non-increasing)
    const int32_t *posof;      // [N] request index -> sorted position
    const InstStats *inst;     // [n_inst]
    int32_t *plan_next;        // [resident warps * n] ISJL plan links (scratch)
    isjl_record *records;      // [n_runs * n_inst]
    int32_t *start_out;        // [n_runs * N] or null
    int32_t *compl_out;        // [n_runs * N] or null
    int32_t *task_counter;     // work queue head, zeroed before each launch
    int32_t *dev_status;       // first nonzero status of the launch
    int64_t n_inst;
    int32_t n;
    int32_t B;
    int64_t kv_cap;
    int64_t max_steps;         // 0 = per-instance automatic bound
    int32_t n_runs;
    int32_t words0;            // ceil(n / 32): level-0 words of the pending bitset
    int32_t words1;            // ceil(words0 / 32): level-1 summary words
    double c, tau, p0;
    RunList runs;
};

// host-side launchers (defined in the .cu files)
cudaError_t launch_derive(const int32_t *arrival, const int32_t *prompt, const int32_t *output,
                          const int32_t *count, const int32_t *slack, int32_t *o, int32_t *otrue,
                          InstStats *inst, int64_t n_inst, int32_t n, cudaStream_t s);
cudaError_t launch_sort(const int32_t *o, const InstStats *inst, int32_t *perm, int32_t *osorted, int32_t *posof,
                        int32_t *tmp, int64_t n_inst, int32_t n, cudaStream_t s);
cudaError_t launch_sim(const SimArgs &args, bool epoch, int total_warps, cudaStream_t s);
cudaError_t launch_summarize(const isjl_record *records, int64_t n_inst, int32_t n_runs,
                             const RunList &runs, int32_t kv_cap, isjl_summary *out, cudaStream_t s);
// resident warps the simulation kernel is launched with for this B and n
int sim_resident_warps(int B, int n, bool epoch, int device);
size_t sim_smem_per_warp(int B, int n);
int slots_per_lane(int B);

}  // namespace isjl
