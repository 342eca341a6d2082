// noalloc.cu -- the sweep without any allocation (isjl_sim_run_sweep_noalloc).
//
// Some callers cannot allocate device memory at the point where they need a
// simulation: code running inside a memory pool or arena that owns every
// allocation, a host process under a strict allocation budget, or a caller
// that must not synchronize the device (cudaMalloc and cudaFree can).  For
// them this file holds a fixed workspace in a file-scope device array and runs
// the same derive / sort / simulate kernels out of it.  The caller still
// passes the inputs and the output buffers.
//
// The array exists once per GPU that loads the library, for the life of the
// process.  Its device address is looked up once per device, on the first
// call made with that device current; that first call should therefore come
// before any stream capture.  Every call uses the same array, so calls whose
// work overlaps on the GPU (two streams, or two host threads) race and must
// be serialized by the caller.  The array keeps the previous call's contents:
// the work counter and status word are zeroed on the stream at each call;
// everything else is written before it is read.
#include <cstdint>
#include <cstring>
#include <mutex>

#include "sim_internal.cuh"

namespace {

constexpr size_t kScratchBytes = ISJL_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mu;
void *g_ptr[kMaxDevices] = {nullptr};

// device address of g_scratch for the current device (looked up once per device)
cudaError_t scratch_ptr(unsigned char **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_scratch);
        if (e != cudaSuccess) return e;
        g_ptr[dev] = p;
    }
    *out = static_cast<unsigned char *>(g_ptr[dev]);
    return cudaSuccess;
}

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

extern "C" isjl_status isjl_sim_run_sweep_noalloc(const isjl_config *cfg, int32_t n_runs, const int32_t *policies,
                                                  const int32_t *deltas, int32_t kv_cap,
                                                  const isjl_instances *in, const isjl_outputs *out,
                                                  void *stream) {
    if (!cfg || !in || !out || !in->arrival || !in->prompt || !in->output || !out->records || kv_cap < 1)
        return ISJL_ERR_INVALID_ARG;
    if (cfg->n_instances < 1 || cfg->n_per_instance < 1 || cfg->B < 1 || cfg->B > ISJL_MAX_B ||
        !(cfg->c >= 0.0) || !(cfg->tau >= 0.0) || !(cfg->p0 >= 0.0) || cfg->max_steps < 0 ||
        (cfg->flags & ~ISJL_FLAG_EPOCH_KERNEL) != 0u || cfg->n_instances > INT32_MAX ||
        cfg->n_instances * (int64_t)ISJL_MAX_RUNS > INT32_MAX)
        return ISJL_ERR_INVALID_ARG;
    if (n_runs < 1 || n_runs > ISJL_MAX_RUNS || !policies || !deltas) return ISJL_ERR_INVALID_ARG;
    for (int i = 0; i < n_runs; ++i)
        if (policies[i] < ISJL_POLICY_FCFS || policies[i] > ISJL_POLICY_ISJL_BETA || deltas[i] < 0)
            return ISJL_ERR_INVALID_ARG;

    // workspace layout inside the fixed array
    const int64_t N = cfg->n_instances * (int64_t)cfg->n_per_instance;
    const int n = cfg->n_per_instance;
    const bool big = n > isjl::kSortSmallMax;
    size_t off = 0;
    const size_t o_off = off;        off = align256(off + sizeof(int32_t) * N);
    const size_t perm_off = off;     off = align256(off + sizeof(int32_t) * N);
    const size_t os_off = off;       off = align256(off + sizeof(int32_t) * N);
    const size_t pos_off = off;      off = align256(off + sizeof(int32_t) * N);
    const size_t tmp_off = off;      if (big) off = align256(off + sizeof(int32_t) * N);
    const size_t ot_off = off;       if (in->slack) off = align256(off + sizeof(int32_t) * N);
    const size_t inst_off = off;     off = align256(off + sizeof(isjl::InstStats) * cfg->n_instances);
    const size_t ctr_off = off;      off = align256(off + 2 * sizeof(int32_t));
    const size_t plan_off = off;
    if (off >= kScratchBytes) return ISJL_ERR_INVALID_ARG;   // too large for the fixed workspace
    const bool epoch = (cfg->flags & ISJL_FLAG_EPOCH_KERNEL) != 0u;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return ISJL_ERR_CUDA;
    int warps = isjl::sim_resident_warps(cfg->B, n, epoch, dev);
    if (warps < 1) return ISJL_ERR_INVALID_ARG;
    const int64_t fit = (int64_t)((kScratchBytes - plan_off) / (sizeof(int32_t) * (size_t)n));
    if (fit < warps) warps = (int)(fit / isjl::kSimWarpsPerBlock) * isjl::kSimWarpsPerBlock;
    if (warps < isjl::kSimWarpsPerBlock) return ISJL_ERR_INVALID_ARG;   // plan scratch for one block does not fit

    unsigned char *base = nullptr;
    if (scratch_ptr(&base) != cudaSuccess) return ISJL_ERR_CUDA;
    int32_t *d_o = reinterpret_cast<int32_t *>(base + o_off);
    int32_t *d_perm = reinterpret_cast<int32_t *>(base + perm_off);
    int32_t *d_os = reinterpret_cast<int32_t *>(base + os_off);
    int32_t *d_pos = reinterpret_cast<int32_t *>(base + pos_off);
    int32_t *d_tmp = big ? reinterpret_cast<int32_t *>(base + tmp_off) : nullptr;
    int32_t *d_ot = in->slack ? reinterpret_cast<int32_t *>(base + ot_off) : nullptr;
    isjl::InstStats *d_inst = reinterpret_cast<isjl::InstStats *>(base + inst_off);
    int32_t *d_ctr = reinterpret_cast<int32_t *>(base + ctr_off);
    int32_t *d_plan = reinterpret_cast<int32_t *>(base + plan_off);

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(d_ctr, 0, 2 * sizeof(int32_t), st) != cudaSuccess) return ISJL_ERR_CUDA;
    if (isjl::launch_derive(in->arrival, in->prompt, in->output, in->count, in->slack, d_o, d_ot, d_inst,
                            cfg->n_instances, n, st) != cudaSuccess)
        return ISJL_ERR_CUDA;
    if (isjl::launch_sort(d_o, d_inst, d_perm, d_os, d_pos, d_tmp, cfg->n_instances, n, st) != cudaSuccess)
        return ISJL_ERR_CUDA;

    isjl::SimArgs a;
    std::memset(&a, 0, sizeof(a));
    a.arrival = in->arrival;
    a.o = d_o;
    a.otrue = d_ot;
    a.perm = d_perm;
    a.osorted = d_os;
    a.posof = d_pos;
    a.inst = d_inst;
    a.plan_next = d_plan;
    a.records = out->records;
    a.start_out = out->start;
    a.compl_out = out->completion;
    a.task_counter = d_ctr;
    a.dev_status = d_ctr + 1;
    a.n_inst = cfg->n_instances;
    a.n = n;
    a.B = cfg->B;
    a.kv_cap = kv_cap;
    a.max_steps = cfg->max_steps;
    a.n_runs = n_runs;
    a.words0 = (n + 31) / 32;
    a.words1 = (a.words0 + 31) / 32;
    a.c = cfg->c;
    a.tau = cfg->tau;
    a.p0 = cfg->p0;
    for (int i = 0; i < n_runs; ++i) {
        a.runs.policy[i] = policies[i];
        a.runs.delta[i] = deltas[i];
        a.runs.beta[i] = isjl::run_beta(policies[i], deltas[i]);
    }
    if (isjl::launch_sim(a, epoch, warps, st) != cudaSuccess) return ISJL_ERR_CUDA;
    return ISJL_OK;
}
