// Measurement tooling, not part of libposeidon: poseidon_probe_int32 times
// the relaxation the makespan kernels are built from,
// finish = max(pred + edge, clock) + weight (one add, one max, one add:
// 3 int32 ops; the add-max fused into one instruction as the kernels do), with enough independent chains per thread and threads per
// SM that no dependency or latency limits it.  The result checks the
// roofline denominator the benchmark uses for the ALU-bound kernels
// (SMs x 128 int32 lanes x clock).  Built into libposeidon_probe.so.
#include <cuda_runtime.h>

#include "../../include/poseidon_probe.h"

namespace {

constexpr int kProbeChains = 8;    // independent relaxation chains per thread
constexpr int kProbeThreads = 256;
constexpr int kProbeBlocksPerSm = 8;

__global__ void __launch_bounds__(kProbeThreads) int32_probe_kernel(int iters, int32_t seed,
                                                                     int32_t *out) {
    int32_t x[kProbeChains], y[kProbeChains], e[kProbeChains], w[kProbeChains];
    const int32_t t = (int32_t)(blockIdx.x * blockDim.x + threadIdx.x);
#pragma unroll
    for (int k = 0; k < kProbeChains; ++k) {
        x[k] = seed ^ (t * 7 + k);
        y[k] = seed + t + 3 * k;
        e[k] = (seed >> 3) + k;
        w[k] = (seed >> 5) - k;
    }
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int k = 0; k < kProbeChains; ++k) {
            // two chained relaxations per chain and iteration (6 int32 ops),
            // the add-max fused as in the makespan kernels (__viaddmax_s32)
            x[k] = __viaddmax_s32(y[k], e[k], x[k]) + w[k];
            y[k] = __viaddmax_s32(x[k], w[k], y[k]) + e[k];
        }
    }
    int32_t acc = 0;
#pragma unroll
    for (int k = 0; k < kProbeChains; ++k) acc ^= x[k] ^ y[k];
    if (acc == seed) out[0] = acc;  // keeps the chains live; practically never taken
}

}  // namespace

extern "C" int poseidon_probe_int32(void *stream, int64_t *ops, double *ms) {
    if (!ops || !ms) return (int)cudaErrorInvalidValue;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return (int)e;
    const int blocks = sms * kProbeBlocksPerSm;
    const int iters = 4096;
    int32_t *d_out = nullptr;
    e = cudaMallocAsync(reinterpret_cast<void **>(&d_out), sizeof(int32_t), s);
    if (e != cudaSuccess) return (int)e;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    e = cudaEventCreate(&e0);
    if (e == cudaSuccess) e = cudaEventCreate(&e1);
    if (e == cudaSuccess) {
        int32_probe_kernel<<<blocks, kProbeThreads, 0, s>>>(iters, 0x2f6e2b1, d_out);
        e = cudaEventRecord(e0, s);
    }
    if (e == cudaSuccess) {
        int32_probe_kernel<<<blocks, kProbeThreads, 0, s>>>(iters, 0x1b873593, d_out);
        e = cudaEventRecord(e1, s);
    }
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaEventSynchronize(e1);
    float t = 0.f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t, e0, e1);
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    const cudaError_t e2 = cudaFreeAsync(d_out, s);
    if (e != cudaSuccess) return (int)e;
    if (e2 != cudaSuccess) return (int)e2;
    *ops = (int64_t)blocks * kProbeThreads * iters * kProbeChains * 6;
    *ms = t;
    return 0;
}
