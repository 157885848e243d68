// poseidon_argmin_noalloc: the argmin of poseidon_argmin without any device
// allocation.  Some callers cannot allocate device memory during a call: a
// process whose device memory is owned by another allocator (a framework's
// caching allocator that has reserved the free memory, or a service that
// reserves everything at start-up and forbids allocation afterwards) gets
// an out-of-memory error or an unwanted allocation from the stream-ordered
// scratch that poseidon_argmin takes per call.  This variant keeps its
// per-block partial results in a fixed array in device global memory that
// the library holds on every GPU that loads it, until the process exits.
#include <mutex>

#include "common.cuh"

namespace pos {

// the two kernels of poseidon_argmin (defined in eval.cu)
__global__ void argmin_partial(const int32_t *T, const uint8_t *F, int64_t n, int32_t *part_t,
                               long long *part_i);
__global__ void argmin_final(const int32_t *part_t, const long long *part_i, int parts,
                             int64_t *out);

constexpr int kNoAllocParts = 4096;  // partial results the fixed scratch holds

// 4096 x (int32 makespan, padded to 8 bytes) + 4096 x int64 index = 64 KB
static __device__ __align__(256) unsigned char g_argmin_scratch[kNoAllocParts * 16];

constexpr int kMaxDevices = 64;
static std::mutex g_scratch_mutex;
static void *g_scratch_addr[kMaxDevices];  // device address of the array, per device

// The name g_argmin_scratch in host code is only a host-side stand-in for
// the array; its device address comes from cudaGetSymbolAddress, taken once
// per device with that device current and kept for the life of the
// process.  After cudaDeviceReset the module is loaded again and the array
// may move, so the library must not be used across a device reset.
static pos_status scratch_address(void **out) {
    int dev = 0;
    POS_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kMaxDevices) return fail(POS_EINVAL, "device index above 63");
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        POS_CUDA(cudaGetSymbolAddress(&p, g_argmin_scratch));
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return POS_OK;
}

}  // namespace pos

extern "C" pos_status poseidon_argmin_noalloc(const int32_t *d_makespan,
                                              const uint8_t *d_feasible, int64_t n,
                                              int64_t *d_out, void *stream) {
    if (n < 0 || !d_out || (n > 0 && (!d_makespan || !d_feasible)))
        return pos::fail(POS_EINVAL, "bad argmin arguments");
    const int64_t parts = std::max<int64_t>(
        1, std::min<int64_t>((n + pos::kArgminThreads - 1) / pos::kArgminThreads,
                             4LL * pos::sm_count()));
    if (parts > pos::kNoAllocParts)
        return pos::fail(POS_EINVAL,
                         "poseidon_argmin_noalloc: this GPU needs more than 4096 partial "
                         "results (more than 1024 SMs); use poseidon_argmin");
    void *scratch = nullptr;
    const pos_status st = pos::scratch_address(&scratch);
    if (st != POS_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int32_t *pt = static_cast<int32_t *>(scratch);
    long long *pi =
        reinterpret_cast<long long *>(static_cast<char *>(scratch) + pos::kNoAllocParts * 8);
    // every slot the final kernel reads is written by the partial kernel of
    // the same call, so nothing has to be cleared between calls
    pos::argmin_partial<<<(int)parts, pos::kArgminThreads, 0, s>>>(d_makespan, d_feasible, n, pt,
                                                                     pi);
    pos::argmin_final<<<1, 32, 0, s>>>(pt, pi, (int)parts, d_out);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return pos::cuda_fail(e, "argmin_noalloc launch");
    return POS_OK;
}
