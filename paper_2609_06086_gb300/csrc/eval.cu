// poseidon_eval_batch, poseidon_eval_batch_host and poseidon_argmin (hot-path
// step a9).  The evaluation kernels live in eval_kernel.cuh and the
// eval_range_*.cu instantiation units.
#include "eval_kernel.cuh"

namespace pos {

// ---------------------------------------------------------------------------
// argmin over (makespan, index) among feasible entries, ties -> lowest index
// ---------------------------------------------------------------------------
constexpr int kArgThreads = 256;

__device__ __forceinline__ void better_of(int32_t &bt, long long &bi, int32_t t, long long i) {
    if (i >= 0 && (bi < 0 || t < bt || (t == bt && i < bi))) {
        bt = t;
        bi = i;
    }
}

__global__ void argmin_partial(const int32_t *T, const uint8_t *F, int64_t n, int32_t *part_t,
                               long long *part_i) {
    int32_t bt = 0;
    long long bi = -1;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        if (F[i] == POS_FEAS_YES) better_of(bt, bi, T[i], i);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int32_t ot = __shfl_down_sync(0xffffffffu, bt, o);
        const long long oi = __shfl_down_sync(0xffffffffu, bi, o);
        better_of(bt, bi, ot, oi);
    }
    __shared__ int32_t st[kArgThreads / 32];
    __shared__ long long si[kArgThreads / 32];
    if ((threadIdx.x & 31) == 0) {
        st[threadIdx.x >> 5] = bt;
        si[threadIdx.x >> 5] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < (int)(blockDim.x >> 5); ++w) better_of(bt, bi, st[w], si[w]);
        part_t[blockIdx.x] = bt;
        part_i[blockIdx.x] = bi;
    }
}

__global__ void argmin_final(const int32_t *part_t, const long long *part_i, int parts,
                             int64_t *out) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    int32_t bt = 0;
    long long bi = -1;
    for (int q = 0; q < parts; ++q) better_of(bt, bi, part_t[q], part_i[q]);
    *out = bi;
}

pos_status launch_eval(Handle *h, const pos_candidate *d_cands, int64_t n, int32_t *d_T,
                       uint8_t *d_F, cudaStream_t stream) {
    if (n == 0) return POS_OK;
    EvalParams p;
    p.cands = reinterpret_cast<const uint4 *>(d_cands);
    p.n = n;
    p.T = d_T;
    p.F = d_F;
    p.blob = h->d_blob;
    p.lay = h->lay;
    p.gA = h->guard_A;
    p.gD = h->guard_D;
    p.gP = h->guard_P;
    const int smem = eval_smem_bytes(h->lay);
    pos_status st;
    if ((st = eval_fast_1_4(p, smem, stream)) != POS_OK) return st;
    if ((st = eval_fast_5_8(p, smem, stream)) != POS_OK) return st;
    if ((st = eval_fast_9_12(p, smem, stream)) != POS_OK) return st;
    if ((st = eval_fast_13_16(p, smem, stream)) != POS_OK) return st;
    if ((st = eval_generic_2_8(p, smem, stream)) != POS_OK) return st;
    return eval_generic_9_16(p, smem, stream);
}

}  // namespace pos

extern "C" {

pos_status poseidon_eval_batch(void *handle, const pos_candidate *d_cands, int64_t n,
                               int32_t *d_makespan, uint8_t *d_feasible, void *stream) {
    if (!handle) return pos::fail(POS_EINVAL, "handle is NULL");
    if (n < 0) return pos::fail(POS_EINVAL, "n < 0");
    if (n > 0 && (!d_cands || !d_makespan || !d_feasible))
        return pos::fail(POS_EINVAL, "NULL buffer");
    if ((reinterpret_cast<uintptr_t>(d_cands) & 15) != 0)
        return pos::fail(POS_EINVAL, "candidates must be 16-byte aligned");
    return pos::launch_eval(static_cast<pos::Handle *>(handle), d_cands, n, d_makespan,
                            d_feasible, static_cast<cudaStream_t>(stream));
}

pos_status poseidon_eval_batch_host(void *handle, const pos_candidate *cands, int64_t n,
                                    int32_t *makespan, uint8_t *feasible) {
    if (!handle) return pos::fail(POS_EINVAL, "handle is NULL");
    if (n < 0) return pos::fail(POS_EINVAL, "n < 0");
    if (n == 0) return POS_OK;
    if (!cands || !makespan || !feasible) return pos::fail(POS_EINVAL, "NULL buffer");
    void *d = nullptr;
    const size_t bc = sizeof(pos_candidate) * (size_t)n, bt = sizeof(int32_t) * (size_t)n;
    POS_CUDA(cudaMalloc(&d, bc + bt + (size_t)n));
    pos_candidate *dc = static_cast<pos_candidate *>(d);
    int32_t *dt = reinterpret_cast<int32_t *>(static_cast<char *>(d) + bc);
    uint8_t *df = reinterpret_cast<uint8_t *>(static_cast<char *>(d) + bc + bt);
    pos_status st = POS_OK;
    cudaError_t e = cudaMemcpy(dc, cands, bc, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) {
        st = pos::launch_eval(static_cast<pos::Handle *>(handle), dc, n, dt, df, 0);
        if (st == POS_OK) e = cudaMemcpy(makespan, dt, bt, cudaMemcpyDeviceToHost);
        if (st == POS_OK && e == cudaSuccess)
            e = cudaMemcpy(feasible, df, (size_t)n, cudaMemcpyDeviceToHost);
    }
    cudaFree(d);
    if (e != cudaSuccess) return pos::cuda_fail(e, "eval_batch_host copies");
    return st;
}

pos_status poseidon_argmin(const int32_t *d_makespan, const uint8_t *d_feasible, int64_t n,
                           int64_t *d_out, void *stream) {
    if (n < 0 || !d_out || (n > 0 && (!d_makespan || !d_feasible)))
        return pos::fail(POS_EINVAL, "bad argmin arguments");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int parts = (int)std::max<int64_t>(
        1, std::min<int64_t>((n + pos::kArgThreads - 1) / pos::kArgThreads,
                             4LL * pos::sm_count()));
    void *scratch = nullptr;
    POS_CUDA(cudaMallocAsync(&scratch, (size_t)parts * 16, s));
    int32_t *pt = static_cast<int32_t *>(scratch);
    long long *pi = reinterpret_cast<long long *>(static_cast<char *>(scratch) + parts * 8);
    pos::argmin_partial<<<parts, pos::kArgThreads, 0, s>>>(d_makespan, d_feasible, n, pt, pi);
    pos::argmin_final<<<1, 32, 0, s>>>(pt, pi, parts, d_out);
    const cudaError_t e = cudaGetLastError();
    const cudaError_t e2 = cudaFreeAsync(scratch, s);
    if (e != cudaSuccess) return pos::cuda_fail(e, "argmin launch");
    if (e2 != cudaSuccess) return pos::cuda_fail(e2, "argmin free");
    return POS_OK;
}

}  // extern "C"
