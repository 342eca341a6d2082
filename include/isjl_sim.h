/*
 * isjl_sim.h -- C ABI of the GB300 batched scheduling simulator.
 *
 * The library simulates, on one GPU, the token-step scheduling model of
 * "Efficiency and Cost Alignment in Batched LLM Serving via Resource-Fair
 * Scheduling" (Yao & Zhou) for many independent request instances at once:
 *
 *   - Section 2 (Model): request i needs o_i = prompt_i + output_i tokens and
 *     advances one token per step; at most B requests run in a step; the
 *     makespan counts steps.  Fairness, Eq. 1: over the running set,
 *     max a_i - min a_i <= delta (the paper's alpha), a_i = tokens processed.
 *   - Policies: FCFS (Section 2.1 and the continuous-batching remark),
 *     LJF (Algorithm 1), ISJL (Algorithm 2 with beta = alpha, in the rolling
 *     online form of Section 3.4 when requests have release times).
 *   - Cost (Section 5, Eq. batch-cost-progress): a nonempty step costs
 *     c + tau*|S|*max r_i with r_i = a_i + 1, decomposed as
 *     tau*Q + c*T + tau*E (Theorem "Profit decomposition"); revenue p0*sum o_i.
 *
 * Readings the library fixes where the paper is silent: a running request
 * reserves KV memory equal to its peak footprint o_i and a start needs
 * sum_{S} o_j + o_i <= kv_cap; the first start that does not fit ends the
 * starts of that step; "longest" means (o desc, index asc); a request started
 * in step k runs in step k and completes at (last step) + 1.
 *
 * Conventions for every entry point:
 *   - Pointers documented as "device" must be device memory of the current
 *     CUDA device; "host" pointers are ordinary (preferably pinned) memory.
 *   - Arrays are int32, structure of arrays, instance-major: element
 *     inst * n_per_instance + i is request i of instance inst.  Within an
 *     instance, arrivals are non-decreasing in i (index order = arrival order).
 *   - stream is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   - No entry point throws, traps or aborts; errors are returned as
 *     isjl_status.  Errors found on the device (an infeasible request, a step
 *     limit) are recorded per run and returned by isjl_sim_metrics().
 *   - A handle is not thread safe; use one handle per host thread.
 */
#ifndef ISJL_SIM_H
#define ISJL_SIM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    ISJL_OK = 0,
    ISJL_ERR_INVALID_ARG = 1,  /* bad argument, negative length, decreasing arrivals, o_i > ISJL_MAX_LEN */
    ISJL_ERR_INFEASIBLE = 2,   /* some o_i < 1 or o_i > kv_cap: the request can never start */
    ISJL_ERR_OOM = 3,          /* device or pinned-host allocation failed in create / first host call */
    ISJL_ERR_CUDA = 4,         /* a CUDA runtime call failed (launch, copy, sync) */
    ISJL_ERR_STEP_LIMIT = 5,   /* a simulation exceeded max_steps (defensive guard; never trapped) */
    ISJL_ERR_NOT_READY = 6,    /* metrics requested before any run */
    ISJL_ERR_INTERNAL = 7      /* an internal invariant of the simulation kernel failed (a library bug):
                                  the run stopped where it found it; its counters are partial and its
                                  per-request outputs -1 beyond what it had written */
} isjl_status;

typedef enum {
    ISJL_POLICY_FCFS = 0,       /* arrival order, continuous batching; ignores delta */
    ISJL_POLICY_LJF = 1,        /* Algorithm 1, static batches of the longest; ignores delta */
    ISJL_POLICY_ISJL = 2,       /* Algorithm 2 (beta = alpha = delta) */
    ISJL_POLICY_SJF = 3,        /* shortest first, continuous batching (Section 6 baseline); ignores delta */
    ISJL_POLICY_ISJL_BETA = 4   /* Algorithm "ISJL": beta = (sqrt(17) - 1) / 4 * delta replaces alpha in the
                                   packing thresholds (o_1 - o_j + beta); defined by the paper for B = 2 */
} isjl_policy;

#define ISJL_DELTA_INF 2147483647   /* fairness budget infinity: Eq. 1 is vacuous */
#define ISJL_KV_INF    2147483647   /* no KV cap: the paper's compute-bound model */
#define ISJL_MAX_B     512          /* largest batch-slot count B */
#define ISJL_MAX_LEN   65535        /* largest request length o_i */
#define ISJL_MAX_RUNS  32           /* largest (policy, delta) list of one sweep call */

/* config flags */
#define ISJL_FLAG_STEP_KERNEL 0u    /* default: per-step kernel, every running request advanced each step */
#define ISJL_FLAG_EPOCH_KERNEL 1u   /* event-driven kernel: closed-form cost between events; same results */
#define ISJL_FLAG_TIMING 2u         /* record CUDA events around each kernel (see isjl_sim_kernel_times) */

typedef struct {
    int64_t n_instances;     /* >= 1 */
    int32_t n_per_instance;  /* n >= 1 requests per instance */
    int32_t B;               /* batch slots, 1..ISJL_MAX_B */
    double c;                /* fixed cost of a nonempty step (paper: 0.0005) */
    double tau;              /* cost per unit of |S| * max r (paper: 1e-6) */
    double p0;               /* revenue per token (paper: 1/500) */
    int64_t max_steps;       /* step guard per run; 0 = sum o + max arrival + 1 (a proven bound) */
    uint32_t flags;          /* ISJL_FLAG_* */
} isjl_config;

/* Inputs: three device arrays of n_instances * n_per_instance int32 each,
 * plus an optional per-instance request count for ragged batches. */
typedef struct {
    const int32_t *arrival;  /* release step A_i >= 0, non-decreasing within an instance */
    const int32_t *prompt;   /* prompt tokens >= 0 */
    const int32_t *output;   /* output tokens >= 0; o_i = prompt + output must be 1..ISJL_MAX_LEN, and
                                per instance sum o_i + max A_i <= 2^30 - 2 (the range of the step
                                counter); an instance beyond either limit is INVALID_ARG */
    const int32_t *count;    /* device, n_instances entries or NULL: instance i uses its first
                                count[i] slots (0..n_per_instance; 0 = an empty instance, all
                                counters 0); NULL = every instance uses all n_per_instance.  A
                                count outside 0..n_per_instance makes that instance INVALID_ARG. */
    const int32_t *slack;    /* device, same shape as arrival, or NULL: upper-bound slack
                                e_i = u_i - o_i >= 0 of length predictions (Robust-ISJL, Section
                                3.3).  Every policy then plans with u_i = o_i + e_i (order, packing,
                                KV reservation) while request i still finishes after o_i tokens and
                                the fairness gate uses true progress.  NULL = exact lengths. */
} isjl_instances;

/* One result record per (run, instance).  Integers are exact; the doubles
 * are computed from them in the stated order without fused multiply-add. */
typedef struct {
    int64_t T_make;          /* makespan: max completion step */
    int64_t T_busy;          /* steps with a nonempty batch (the "batch-steps") */
    int64_t O;               /* sum o_i (revenue tokens) */
    int64_t Q;               /* sum o_i (o_i + 1) / 2, Eq. intrinsic-resource-cost */
    int64_t W;               /* sum over steps of |S| * max r  (= Q + E exactly) */
    int64_t E;               /* batching externality, Eq. batching-externality */
    int64_t token_adv;       /* sum over steps of |S|  (= O exactly) */
    int64_t sum_completion;  /* sum c_i (AEL numerator, Eq. ael) */
    int64_t sum_latency;     /* sum (c_i - A_i) */
    int64_t sum_extent;      /* sum over nonempty steps of max r - min r */
    int64_t max_extent;      /* max over steps of max r - min r */
    int64_t violations;      /* steps whose extent exceeds delta (0 for LJF and ISJL) */
    int64_t kv_violations;   /* steps whose reserved KV exceeds kv_cap (always 0) */
    int64_t peak_kv;         /* max reserved KV (sum of o over the running set) */
    int64_t peak_batch;      /* max |S| */
    int64_t status;          /* isjl_status of this run on this instance */
    double c_T;              /* c * T_busy */
    double tau_Q;            /* tau * Q */
    double tau_E;            /* tau * E */
    double cost;             /* (c_T + tau_Q) + tau_E */
    double revenue;          /* p0 * O */
    double profit;           /* revenue - cost */
    double throughput;       /* O / T_make, tokens per step */
    double ael;              /* sum_completion / n (0 for an empty instance) */
} isjl_record;

/* Where results go.  records: device, n_runs * n_instances entries,
 * run-major (record run * n_instances + inst).  start / completion: device
 * or NULL, n_runs * n_instances * n_per_instance int32 each, run-major; the
 * step a request started / completed, -1 for one that did not (an instance
 * with an error status, a run stopped by max_steps, the unused slots of a
 * ragged instance).  Output buffers are owned by the
 * caller and must stay valid until the run's work on the stream is done. */
typedef struct {
    isjl_record *records;
    int32_t *start;
    int32_t *completion;
} isjl_outputs;

/* Per-run totals over all instances (fixed-order reduction on the device). */
typedef struct {
    int32_t policy;
    int32_t delta;
    int32_t kv_cap;
    int32_t status;          /* first nonzero record status of the run, else 0 */
    int64_t n_instances;
    int64_t n_ok;            /* records with status 0 */
    int64_t T_make, T_busy, O, Q, W, E, token_adv;
    int64_t sum_completion, sum_latency, sum_extent, max_extent, violations, kv_violations;
    double c_T, tau_Q, tau_E, cost, revenue, profit;
} isjl_summary;

typedef struct isjl_sim isjl_sim;

/* Create a simulator for instances of the shape in *cfg on the current CUDA
 * device.  Allocates the device workspace (derived lengths, per-instance
 * sort, plan scratch, per-run summaries), about 16 bytes per request plus
 * n_per_instance * 4 bytes per resident warp.  Errors: INVALID_ARG (null
 * pointer, n_instances < 1, n_per_instance < 1, B outside 1..ISJL_MAX_B,
 * negative cost constants, unknown flags), OOM, CUDA.  On error *out is NULL. */
isjl_status isjl_sim_create(const isjl_config *cfg, isjl_sim **out);

/* Free everything create and the host entry point allocated.  Synchronizes
 * the device first.  NULL is ignored. */
void isjl_sim_destroy(isjl_sim *sim);

/* Simulate every instance under one policy.  delta: fairness budget >= 0
 * (ISJL_DELTA_INF = none; FCFS, LJF and SJF ignore it except for counting
 * violations).  kv_cap >= 1 (ISJL_KV_INF = none).  Asynchronous on stream:
 * validation of the lengths (INFEASIBLE / INVALID_ARG per instance) happens on
 * the device and is reported by isjl_sim_metrics and the records.
 * Synchronous errors: INVALID_ARG (null pointers, delta < 0, kv_cap < 1,
 * policy unknown), CUDA (launch failure). */
isjl_status isjl_sim_run(isjl_sim *sim, isjl_policy policy, int32_t delta, int32_t kv_cap,
                         const isjl_instances *in, const isjl_outputs *out, void *stream);

/* Simulate n_runs (policy, delta) pairs (host arrays of n_runs entries,
 * 1 <= n_runs <= ISJL_MAX_RUNS) over every instance with one derive/sort
 * pass and one simulation launch.  Results are identical to n_runs calls of
 * isjl_sim_run.  Same errors as isjl_sim_run. */
isjl_status isjl_sim_run_sweep(isjl_sim *sim, int32_t n_runs, const int32_t *policies,
                               const int32_t *deltas, int32_t kv_cap,
                               const isjl_instances *in, const isjl_outputs *out, void *stream);

/* The same sweep from and to HOST memory: copies the three input arrays
 * (n_instances * n_per_instance int32 each) and, when not NULL, the request
 * counts (n_instances int32, as isjl_instances.count) and the upper-bound
 * slack (n_instances * n_per_instance int32, as isjl_instances.slack) to the
 * device, simulates, and copies the n_runs * n_instances records back into
 * h_records, all on stream, then synchronizes it.  The first call allocates
 * the device input and record buffers, the first call with counts or slack
 * their buffers (kept until destroy).  Errors: as isjl_sim_run_sweep, plus OOM
 * on first use, plus the first device status (as isjl_sim_metrics). */
isjl_status isjl_sim_run_sweep_host(isjl_sim *sim, int32_t n_runs, const int32_t *policies,
                                    const int32_t *deltas, int32_t kv_cap,
                                    const int32_t *h_arrival, const int32_t *h_prompt,
                                    const int32_t *h_output, const int32_t *h_count,
                                    const int32_t *h_slack, isjl_record *h_records, void *stream);

/* Wait for the last run/sweep on its stream and copy its per-run summaries
 * into the host array out (capacity max_runs >= the last call's n_runs).
 * Returns the first nonzero device status of the last call (INFEASIBLE,
 * INVALID_ARG, STEP_LIMIT, INTERNAL), NOT_READY if nothing ran, CUDA on a
 * failed sync. */
isjl_status isjl_sim_metrics(isjl_sim *sim, isjl_summary *out, int32_t max_runs);

/* Number of kernels the last run/sweep call launched (0 if none). */
int32_t isjl_sim_last_launches(const isjl_sim *sim);

/* Device durations (milliseconds) of the kernels of the last run/sweep call,
 * in launch order: derive, sort, simulate, summarize.  Needs ISJL_FLAG_TIMING
 * at create; waits for the call's events.  Writes min(cap, 4) values to ms
 * (host) and returns how many it wrote; 0 without the flag or before a run,
 * -1 on a CUDA error. */
int32_t isjl_sim_kernel_times(const isjl_sim *sim, float *ms, int32_t cap);

/* The sweep of isjl_sim_run_sweep without any allocation and without a
 * handle.  The paper has no counterpart; this is a library service.
 *
 * For callers that cannot call cudaMalloc at the point of use: code running
 * inside an allocator or memory pool that owns all device memory, processes
 * under a fixed device-memory budget, and callers that must not let an
 * allocation or free synchronize the device.  The workspace (derived lengths,
 * sort arrays, plan links, work counter) lives in a fixed array of
 * ISJL_NOALLOC_SCRATCH_BYTES bytes of device memory that every GPU loading
 * this library holds until the process exits.  The caller passes the input
 * arrays and the output buffers exactly as for isjl_sim_run_sweep (records
 * required, start / completion optional, all device memory); no summaries are
 * produced and device-side errors appear only in the records' status fields.
 *
 * cfg: as for isjl_sim_create (ISJL_FLAG_TIMING not accepted).  The first
 * call with a given device current looks up the array's device address for
 * that device; make that first call before any stream capture.  All calls
 * share the one array and its contents persist between calls: calls whose
 * GPU work overlaps (other streams, other threads) race and must be
 * serialized by the caller.  Asynchronous on stream.
 *
 * Limit: the workspace needs 16 bytes per request (20 when
 * n_per_instance > 4096, and 4 more when in->slack is given, for the true
 * lengths), 40 bytes per instance, and n_per_instance * 16 bytes per block of
 * the simulation kernel; fewer blocks run when the array cannot hold all
 * resident ones.  That is about 3 to 4 million requests per call.
 * Errors: INVALID_ARG (as isjl_sim_run_sweep, or the problem does not fit the
 * fixed workspace), CUDA (symbol lookup or launch failure). */
#define ISJL_NOALLOC_SCRATCH_BYTES (64u << 20)
isjl_status isjl_sim_run_sweep_noalloc(const isjl_config *cfg, int32_t n_runs, const int32_t *policies,
                                       const int32_t *deltas, int32_t kv_cap, const isjl_instances *in,
                                       const isjl_outputs *out, void *stream);

/* Measurement helper; the paper has no counterpart.  The rate at which the
 * current GPU executes simple int32 instructions: the denominator of the
 * simulation kernels' roofline (they are bound by integer issue, not by memory
 * or tensor throughput).  kind 0: 32-bit adds; kind 1: 32-bit min / max (the
 * instructions of a step's extent).  One launch on stream that fills every SM
 * (256-thread blocks, as many per SM as fit), each thread running
 * iters x 128 instructions spread over 8 independent dependency chains; waits
 * for it.  Writes, to host memory, the int32 lane-instructions executed
 * (threads x iters x 128) to *lane_instructions and the launch's CUDA-event
 * time in milliseconds to *ms.  Errors: INVALID_ARG (kind not 0 or 1,
 * iters < 1, a null pointer), CUDA. */
isjl_status isjl_probe_int_rate(int32_t kind, int32_t iters, void *stream, double *lane_instructions, float *ms);

/* Static description of a status code (never NULL). */
const char *isjl_status_string(isjl_status status);

#ifdef __cplusplus
}
#endif

#endif /* ISJL_SIM_H */
