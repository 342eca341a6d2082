// probe.cu -- measured integer issue rates, the denominators of the
// simulation kernels' roofline.  Not a step of the simulated method: the
// simulator is bound by simple int32 instructions (adds for progress and cost
// counters, min / max for the step's extent), and the GPU's rate for them is
// measured here instead of taken from a nominal lane count.
//
// Every thread of a full-occupancy grid runs 8 independent dependency chains
// of one PTX integer instruction each, so no instruction can be folded into
// another:
//   kind 0 (add):    four coupled pairs x += w; w += x  (each add feeds the
//                    next, and every intermediate value is used)
//   kind 1 (minmax): two 4-cycles a = max(a, b); b = min(b, c); c = max(c, d);
//                    d = min(d, a)
// The rate is (threads x iterations x 128 instructions) / CUDA-event time.
#include <cstdint>

#include <cuda_runtime.h>

#include "isjl_sim.h"

namespace {

constexpr int kProbeThreads = 256;
constexpr int kProbeUnroll = 16;          // 16 x 8 = 128 chain instructions per loop iteration

__device__ int32_t g_probe_sink;          // keeps the chains' results live

__device__ __forceinline__ void add_pair(int32_t &x, int32_t &w) {
    asm volatile("add.s32 %0, %0, %1;" : "+r"(x) : "r"(w));
    asm volatile("add.s32 %0, %0, %1;" : "+r"(w) : "r"(x));
}

__device__ __forceinline__ void minmax_cycle(int32_t &a, int32_t &b, int32_t &c, int32_t &d) {
    asm volatile("max.s32 %0, %0, %1;" : "+r"(a) : "r"(b));
    asm volatile("min.s32 %0, %0, %1;" : "+r"(b) : "r"(c));
    asm volatile("max.s32 %0, %0, %1;" : "+r"(c) : "r"(d));
    asm volatile("min.s32 %0, %0, %1;" : "+r"(d) : "r"(a));
}

template <int KIND>
__global__ void __launch_bounds__(kProbeThreads) int_rate_kernel(int32_t iters, int32_t seed) {
    const int32_t t = (int32_t)(blockIdx.x * blockDim.x + threadIdx.x);
    int32_t v[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) v[c] = seed * (c + 3) + t * (2 * c + 1);
    for (int32_t it = 0; it < iters; ++it) {
#pragma unroll
        for (int u = 0; u < kProbeUnroll; ++u) {
            if (KIND == 0) {
                add_pair(v[0], v[1]);
                add_pair(v[2], v[3]);
                add_pair(v[4], v[5]);
                add_pair(v[6], v[7]);
            } else {
                minmax_cycle(v[0], v[1], v[2], v[3]);
                minmax_cycle(v[4], v[5], v[6], v[7]);
            }
        }
    }
    int32_t acc = 0;
#pragma unroll
    for (int c = 0; c < 8; ++c) acc ^= v[c];
    if (acc == seed) g_probe_sink = acc;   // practically never; the compiler cannot know
}

}  // namespace

extern "C" isjl_status isjl_probe_int_rate(int32_t kind, int32_t iters, void *stream, double *lane_instructions,
                                           float *ms) {
    if ((kind != 0 && kind != 1) || iters < 1 || !lane_instructions || !ms) return ISJL_ERR_INVALID_ARG;
    int dev = 0, sms = 0, per_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return ISJL_ERR_CUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return ISJL_ERR_CUDA;
    const void *k = kind == 0 ? reinterpret_cast<const void *>(&int_rate_kernel<0>)
                              : reinterpret_cast<const void *>(&int_rate_kernel<1>);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kProbeThreads, 0) != cudaSuccess || per_sm < 1)
        return ISJL_ERR_CUDA;
    const unsigned blocks = (unsigned)(sms * per_sm);   // one full wave: every SM fully occupied
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    if (cudaEventCreate(&e0) != cudaSuccess) return ISJL_ERR_CUDA;
    if (cudaEventCreate(&e1) != cudaSuccess) { cudaEventDestroy(e0); return ISJL_ERR_CUDA; }
    int32_t seed = 0x2545F491;
    void *params[] = {&iters, &seed};
    cudaError_t err = cudaEventRecord(e0, st);
    if (err == cudaSuccess) err = cudaLaunchKernel(k, dim3(blocks), dim3(kProbeThreads), params, 0, st);
    if (err == cudaSuccess) err = cudaEventRecord(e1, st);
    if (err == cudaSuccess) err = cudaEventSynchronize(e1);
    float t = 0.f;
    if (err == cudaSuccess) err = cudaEventElapsedTime(&t, e0, e1);
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    if (err != cudaSuccess) return ISJL_ERR_CUDA;
    *ms = t;
    *lane_instructions = (double)blocks * kProbeThreads * (double)iters * (kProbeUnroll * 8);
    return ISJL_OK;
}
