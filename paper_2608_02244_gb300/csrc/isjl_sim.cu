// isjl_sim.cu -- the C ABI (include/isjl_sim.h): handle, workspace, launches.
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <new>

#include "sim_internal.cuh"

using isjl::InstStats;
using isjl::RunList;
using isjl::SimArgs;

struct isjl_sim {
    isjl_config cfg;
    int device = 0;
    int64_t N = 0;                   // n_instances * n_per_instance
    int32_t *d_o = nullptr, *d_perm = nullptr, *d_osorted = nullptr, *d_posof = nullptr, *d_tmp = nullptr;
    int32_t *d_otrue = nullptr;      // true lengths, allocated on the first call with slack
    InstStats *d_inst = nullptr;
    int32_t *d_plan_next = nullptr;
    int total_warps = 0;
    int32_t *d_counter = nullptr, *d_status = nullptr;
    isjl_summary *d_summary = nullptr;
    // buffers of the host-memory entry point, allocated on first use
    int32_t *d_in[3] = {nullptr, nullptr, nullptr};
    int32_t *d_cnt_in = nullptr, *d_slack_in = nullptr;   // host-entry counts and slack
    isjl_record *d_rec_io = nullptr;
    // last call
    cudaStream_t last_stream = nullptr;
    int32_t last_runs = 0;
    int32_t last_launches = 0;
    bool ran = false;
    // optional per-kernel timing (ISJL_FLAG_TIMING)
    cudaEvent_t ev[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
    bool timed = false;
};

namespace {

template <typename T>
cudaError_t dalloc(T **p, size_t count) {
    return cudaMalloc(reinterpret_cast<void **>(p), count * sizeof(T) + 16);
}

void free_all(isjl_sim *s) {
    for (cudaEvent_t &e : s->ev)
        if (e) { cudaEventDestroy(e); e = nullptr; }
    void *ptrs[] = {s->d_o, s->d_otrue, s->d_perm, s->d_osorted, s->d_posof, s->d_tmp, s->d_inst, s->d_plan_next,
                    s->d_counter, s->d_status, s->d_summary, s->d_in[0], s->d_in[1], s->d_in[2], s->d_rec_io,
                    s->d_cnt_in, s->d_slack_in};
    for (void *p : ptrs)
        if (p) cudaFree(p);
}

bool valid_runs(int32_t n_runs, const int32_t *policies, const int32_t *deltas) {
    if (n_runs < 1 || n_runs > ISJL_MAX_RUNS || !policies || !deltas) return false;
    for (int i = 0; i < n_runs; ++i) {
        if (policies[i] < ISJL_POLICY_FCFS || policies[i] > ISJL_POLICY_ISJL_BETA) return false;
        if (deltas[i] < 0) return false;
    }
    return true;
}

}  // namespace

extern "C" {

const char *isjl_status_string(isjl_status st) {
    switch (st) {
        case ISJL_OK: return "ok";
        case ISJL_ERR_INVALID_ARG: return "invalid argument";
        case ISJL_ERR_INFEASIBLE: return "infeasible request (o_i < 1 or o_i > kv_cap)";
        case ISJL_ERR_OOM: return "out of memory";
        case ISJL_ERR_CUDA: return "CUDA runtime error";
        case ISJL_ERR_STEP_LIMIT: return "step limit exceeded";
        case ISJL_ERR_NOT_READY: return "no run to report";
        case ISJL_ERR_INTERNAL: return "internal invariant failed (library bug)";
    }
    return "unknown status";
}

isjl_status isjl_sim_create(const isjl_config *cfg, isjl_sim **out) {
    if (!out) return ISJL_ERR_INVALID_ARG;
    *out = nullptr;
    if (!cfg || cfg->n_instances < 1 || cfg->n_per_instance < 1 || cfg->B < 1 || cfg->B > ISJL_MAX_B ||
        !(cfg->c >= 0.0) || !(cfg->tau >= 0.0) || !(cfg->p0 >= 0.0) || cfg->max_steps < 0 ||
        (cfg->flags & ~(ISJL_FLAG_EPOCH_KERNEL | ISJL_FLAG_TIMING)) != 0u)
        return ISJL_ERR_INVALID_ARG;
    if (cfg->n_instances > INT32_MAX || cfg->n_instances * (int64_t)ISJL_MAX_RUNS > INT32_MAX)
        return ISJL_ERR_INVALID_ARG;   // task ids are int32
    isjl_sim *s = new (std::nothrow) isjl_sim();
    if (!s) return ISJL_ERR_OOM;
    s->cfg = *cfg;
    s->N = cfg->n_instances * (int64_t)cfg->n_per_instance;
    if (cudaGetDevice(&s->device) != cudaSuccess) { delete s; return ISJL_ERR_CUDA; }
    const int n = cfg->n_per_instance;
    const bool epoch = (cfg->flags & ISJL_FLAG_EPOCH_KERNEL) != 0u;
    s->total_warps = isjl::sim_resident_warps(cfg->B, n, epoch, s->device);
    if (s->total_warps < 1) { delete s; cudaGetLastError(); return ISJL_ERR_INVALID_ARG; }   // B, n too large for smem
    bool ok = dalloc(&s->d_o, s->N) == cudaSuccess && dalloc(&s->d_perm, s->N) == cudaSuccess &&
              dalloc(&s->d_osorted, s->N) == cudaSuccess && dalloc(&s->d_posof, s->N) == cudaSuccess &&
              dalloc(&s->d_inst, cfg->n_instances) == cudaSuccess &&
              dalloc(&s->d_plan_next, (size_t)s->total_warps * n) == cudaSuccess &&
              dalloc(&s->d_counter, 1) == cudaSuccess && dalloc(&s->d_status, 1) == cudaSuccess &&
              dalloc(&s->d_summary, ISJL_MAX_RUNS) == cudaSuccess;
    if (ok && n > isjl::kSortSmallMax) ok = dalloc(&s->d_tmp, s->N) == cudaSuccess;
    if (ok && (cfg->flags & ISJL_FLAG_TIMING))
        for (cudaEvent_t &e : s->ev) ok = ok && cudaEventCreate(&e) == cudaSuccess;
    if (!ok) {
        cudaGetLastError();
        free_all(s);
        delete s;
        return ISJL_ERR_OOM;
    }
    *out = s;
    return ISJL_OK;
}

void isjl_sim_destroy(isjl_sim *s) {
    if (!s) return;
    cudaDeviceSynchronize();
    free_all(s);
    delete s;
}

isjl_status isjl_sim_run_sweep(isjl_sim *s, int32_t n_runs, const int32_t *policies, const int32_t *deltas,
                               int32_t kv_cap, const isjl_instances *in, const isjl_outputs *out, void *stream) {
    if (!s || !in || !out || !in->arrival || !in->prompt || !in->output || !out->records || kv_cap < 1 ||
        !valid_runs(n_runs, policies, deltas))
        return ISJL_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const isjl_config &c = s->cfg;
    s->last_launches = 0;
    s->ran = false;
    s->timed = false;
    const bool timing = (c.flags & ISJL_FLAG_TIMING) != 0u;
    auto mark = [&](int i) { return !timing || cudaEventRecord(s->ev[i], st) == cudaSuccess; };
    RunList runs;
    std::memset(&runs, 0, sizeof(runs));
    for (int i = 0; i < n_runs; ++i) {
        runs.policy[i] = policies[i];
        runs.delta[i] = deltas[i];
        runs.beta[i] = isjl::run_beta(policies[i], deltas[i]);
    }

    if (cudaMemsetAsync(s->d_counter, 0, sizeof(int32_t), st) != cudaSuccess ||
        cudaMemsetAsync(s->d_status, 0, sizeof(int32_t), st) != cudaSuccess || !mark(0))
        return ISJL_ERR_CUDA;
    if (in->slack && !s->d_otrue && dalloc(&s->d_otrue, s->N) != cudaSuccess) {
        cudaGetLastError();
        s->d_otrue = nullptr;
        return ISJL_ERR_OOM;
    }
    int32_t *otrue = in->slack ? s->d_otrue : nullptr;
    if (isjl::launch_derive(in->arrival, in->prompt, in->output, in->count, in->slack, s->d_o, otrue, s->d_inst,
                            c.n_instances, c.n_per_instance, st) != cudaSuccess || !mark(1))
        return ISJL_ERR_CUDA;
    s->last_launches++;
    if (isjl::launch_sort(s->d_o, s->d_inst, s->d_perm, s->d_osorted, s->d_posof, s->d_tmp, c.n_instances,
                          c.n_per_instance, st) != cudaSuccess || !mark(2))
        return ISJL_ERR_CUDA;
    s->last_launches++;

    SimArgs a;
    std::memset(&a, 0, sizeof(a));
    a.arrival = in->arrival;
    a.o = s->d_o;
    a.otrue = otrue;
    a.perm = s->d_perm;
    a.osorted = s->d_osorted;
    a.posof = s->d_posof;
    a.inst = s->d_inst;
    a.plan_next = s->d_plan_next;
    a.records = out->records;
    a.start_out = out->start;
    a.compl_out = out->completion;
    a.task_counter = s->d_counter;
    a.dev_status = s->d_status;
    a.n_inst = c.n_instances;
    a.n = c.n_per_instance;
    a.B = c.B;
    a.kv_cap = kv_cap;
    a.max_steps = c.max_steps;
    a.n_runs = n_runs;
    a.words0 = (c.n_per_instance + 31) / 32;
    a.words1 = (a.words0 + 31) / 32;
    a.c = c.c;
    a.tau = c.tau;
    a.p0 = c.p0;
    a.runs = runs;
    const bool epoch = (c.flags & ISJL_FLAG_EPOCH_KERNEL) != 0u;
    if (isjl::launch_sim(a, epoch, s->total_warps, st) != cudaSuccess || !mark(3)) return ISJL_ERR_CUDA;
    s->last_launches++;
    if (isjl::launch_summarize(out->records, c.n_instances, n_runs, runs, kv_cap, s->d_summary, st) !=
            cudaSuccess || !mark(4))
        return ISJL_ERR_CUDA;
    s->timed = timing;
    s->last_launches++;
    s->last_stream = st;
    s->last_runs = n_runs;
    s->ran = true;
    return ISJL_OK;
}

isjl_status isjl_sim_run(isjl_sim *s, isjl_policy policy, int32_t delta, int32_t kv_cap,
                         const isjl_instances *in, const isjl_outputs *out, void *stream) {
    const int32_t p = (int32_t)policy, d = delta;
    return isjl_sim_run_sweep(s, 1, &p, &d, kv_cap, in, out, stream);
}

isjl_status isjl_sim_metrics(isjl_sim *s, isjl_summary *out, int32_t max_runs) {
    if (!s || !out) return ISJL_ERR_INVALID_ARG;
    if (!s->ran) return ISJL_ERR_NOT_READY;
    if (max_runs < s->last_runs) return ISJL_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(s->last_stream) != cudaSuccess) return ISJL_ERR_CUDA;
    int32_t dev_status = 0;
    if (cudaMemcpy(out, s->d_summary, sizeof(isjl_summary) * s->last_runs, cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemcpy(&dev_status, s->d_status, sizeof(int32_t), cudaMemcpyDeviceToHost) != cudaSuccess)
        return ISJL_ERR_CUDA;
    return (isjl_status)dev_status;
}

isjl_status isjl_sim_run_sweep_host(isjl_sim *s, int32_t n_runs, const int32_t *policies, const int32_t *deltas,
                                    int32_t kv_cap, const int32_t *h_arrival, const int32_t *h_prompt,
                                    const int32_t *h_output, const int32_t *h_count, const int32_t *h_slack,
                                    isjl_record *h_records, void *stream) {
    if (!s || !h_arrival || !h_prompt || !h_output || !h_records || !valid_runs(n_runs, policies, deltas) ||
        kv_cap < 1)
        return ISJL_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (!s->d_in[0]) {
        bool ok = dalloc(&s->d_in[0], s->N) == cudaSuccess && dalloc(&s->d_in[1], s->N) == cudaSuccess &&
                  dalloc(&s->d_in[2], s->N) == cudaSuccess &&
                  dalloc(&s->d_rec_io, (size_t)ISJL_MAX_RUNS * s->cfg.n_instances) == cudaSuccess;
        if (!ok) {
            cudaGetLastError();
            for (int i = 0; i < 3; ++i) { if (s->d_in[i]) cudaFree(s->d_in[i]); s->d_in[i] = nullptr; }
            if (s->d_rec_io) cudaFree(s->d_rec_io);
            s->d_rec_io = nullptr;
            return ISJL_ERR_OOM;
        }
    }
    if ((h_count && !s->d_cnt_in && dalloc(&s->d_cnt_in, (size_t)s->cfg.n_instances) != cudaSuccess) ||
        (h_slack && !s->d_slack_in && dalloc(&s->d_slack_in, s->N) != cudaSuccess)) {
        cudaGetLastError();
        return ISJL_ERR_OOM;
    }
    const size_t bytes = sizeof(int32_t) * (size_t)s->N;
    const int32_t *src[3] = {h_arrival, h_prompt, h_output};
    for (int i = 0; i < 3; ++i)
        if (cudaMemcpyAsync(s->d_in[i], src[i], bytes, cudaMemcpyHostToDevice, st) != cudaSuccess)
            return ISJL_ERR_CUDA;
    if (h_count && cudaMemcpyAsync(s->d_cnt_in, h_count, sizeof(int32_t) * (size_t)s->cfg.n_instances,
                                   cudaMemcpyHostToDevice, st) != cudaSuccess)
        return ISJL_ERR_CUDA;
    if (h_slack && cudaMemcpyAsync(s->d_slack_in, h_slack, bytes, cudaMemcpyHostToDevice, st) != cudaSuccess)
        return ISJL_ERR_CUDA;
    isjl_instances in{s->d_in[0], s->d_in[1], s->d_in[2], h_count ? s->d_cnt_in : nullptr,
                      h_slack ? s->d_slack_in : nullptr};
    isjl_outputs out{s->d_rec_io, nullptr, nullptr};
    isjl_status rs = isjl_sim_run_sweep(s, n_runs, policies, deltas, kv_cap, &in, &out, stream);
    if (rs != ISJL_OK) return rs;
    int32_t dev_status = 0;
    if (cudaMemcpyAsync(h_records, s->d_rec_io, sizeof(isjl_record) * (size_t)n_runs * s->cfg.n_instances,
                        cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaMemcpyAsync(&dev_status, s->d_status, sizeof(int32_t), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return ISJL_ERR_CUDA;
    return (isjl_status)dev_status;
}

int32_t isjl_sim_last_launches(const isjl_sim *s) { return s ? s->last_launches : 0; }

int32_t isjl_sim_kernel_times(const isjl_sim *s, float *ms, int32_t cap) {
    if (!s || !ms || cap < 1 || !s->timed) return 0;
    if (cudaEventSynchronize(s->ev[4]) != cudaSuccess) return -1;
    int32_t k = 0;
    for (; k < 4 && k < cap; ++k)
        if (cudaEventElapsedTime(&ms[k], s->ev[k], s->ev[k + 1]) != cudaSuccess) return -1;
    return k;
}

}  // extern "C"
