// Evaluation kernel family of poseidon_eval_batch (hot-path steps a2-a5).
//
// One thread evaluates one candidate.  The makespan loop costs ~6*S*M
// integer ops and its live registers grow with S (about 7*S), so a batch is
// evaluated by a family of kernels, each owning the candidates of one S
// range and either M >= S (fully unrolled fast path) or M < S (predicated
// path), each with launch bounds matched to its register need.  Every
// kernel walks the batch in tiles of kEvalTile candidates, sorts the
// candidates it owns by (S, M/4) in shared memory (counting sort), and lets
// every warp evaluate 32 consecutive sorted entries: S is then warp-uniform
// (one template instance per warp) and M nearly uniform.  Results go back
// to input order through shared memory.
#pragma once
#include <algorithm>

#include "common.cuh"

namespace pos {

constexpr int kEvalThreads = 256;
constexpr int kEvalTile = 2048;
constexpr int kBinsPad = 1040;  // >= 16*64 + 1 bins, multiple of 16

struct EvalParams {
    const uint4 *cands;
    int64_t n;
    int32_t *T;
    uint8_t *F;
    const void *blob;
    BlobLayout lay;
    int64_t gA, gD, gP;
};

__host__ __device__ inline int eval_smem_bytes(const BlobLayout &ly) {
    return ly.bytes + kEvalTile * 4 /*keys*/ + kBinsPad * 4 /*hist*/ + kEvalTile * 2 /*order*/ +
           kEvalTile * 4 /*T*/ + kEvalTile /*F*/;
}

// Exclusive prefix sum of a[0..n) in shared memory by the whole block.
__device__ __forceinline__ void block_exclusive_scan(uint32_t *a, int n, uint32_t *warp_tot) {
    const int per = (n + blockDim.x - 1) / blockDim.x;
    const int lo = threadIdx.x * per, hi = min(n, lo + per);
    uint32_t sum = 0;
    for (int i = lo; i < hi; ++i) sum += a[i];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
    }
    if (lane == 31) warp_tot[wid] = incl;
    __syncthreads();
    if (wid == 0) {
        const int nw = blockDim.x >> 5;
        uint32_t v = lane < nw ? warp_tot[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t u = __shfl_up_sync(0xffffffffu, v, o);
            if (lane >= o) v += u;
        }
        if (lane < nw) warp_tot[lane] = v;  // inclusive warp totals
    }
    __syncthreads();
    uint32_t run = (wid > 0 ? warp_tot[wid - 1] : 0) + incl - sum;
    for (int i = lo; i < hi; ++i) {
        const uint32_t v = a[i];
        a[i] = run;
        run += v;
    }
    __syncthreads();
}

template <int PATH>
struct EvalWith {
    template <int S>
    struct One {
        static __device__ __forceinline__ void run(const Tab &t, const uint4 &rec,
                                                   const EvalParams &p, int32_t &T, uint8_t &F) {
            const uint64_t rank = (uint64_t)rec.x | ((uint64_t)rec.y << 32);
            const uint32_t tcode = rec.z;
            const int M = (rec.w >> 8) & 0xff;
            const int tp = (rec.w >> 16) & 0xff;
            bool ok = M >= 1 && S <= t.L() && tp < t.n_tp() && rank < binom(t, t.L() - 1, S - 1);
            int cls[S];
#pragma unroll
            for (int s = 0; s < S; ++s) {
                const int ty = (tcode >> (2 * s)) & 3;
                ok &= ty < t.n_types();
                cls[s] = ty * t.n_tp() + tp;
            }
            if (!ok) {
                T = -1;
                F = POS_FEAS_INVALID;
                return;
            }
            if (guard_trips(p.gA, p.gD, p.gP, S, M)) {
                T = -1;
                F = POS_FEAS_OVERFLOW;
                return;
            }
            int cut[S + 1];
            unrank_cuts<S>(t, rank, cut);
            // memory first, so that its inputs are dead before the wavefront
            F = plan_fits<S>(t, M, cut, cls) ? POS_FEAS_YES : POS_FEAS_NO;
            StageW<S> w;
            stage_weights<S>(t, cut, cls, w);
            T = makespan_1f1b<S, PATH>(w, M);
        }
    };
};

template <int SLO, int SHI, int PATH>
__device__ __forceinline__ void dispatch_range(int S, const Tab &t, const uint4 &rec,
                                               const EvalParams &p, int32_t &T, uint8_t &F) {
#define POS_EV(n)                                                                              \
    if (n >= SLO && n <= SHI && S == n) {                                                      \
        EvalWith<PATH>::template One<(n >= SLO && n <= SHI) ? n : SLO>::run(t, rec, p, T, F); \
        return;                                                                                \
    }
    POS_EV(1) POS_EV(2) POS_EV(3) POS_EV(4) POS_EV(5) POS_EV(6) POS_EV(7) POS_EV(8)
    POS_EV(9) POS_EV(10) POS_EV(11) POS_EV(12) POS_EV(13) POS_EV(14) POS_EV(15) POS_EV(16)
#undef POS_EV
}

// Candidates owned by kernel <SLO, SHI, PATH>: S in [SLO, SHI] and M >= S
// (fast) or M < S (generic).  Records with S outside 1..16 or M = 0 belong
// to the first fast kernel, which flags them invalid.
template <int SLO, int SHI, int PATH>
__device__ __forceinline__ bool owns(int S, int M, bool &invalid) {
    invalid = S < 1 || S > POS_MAX_STAGES || M < 1;
    if (invalid) return SLO == 1 && PATH == kPathFast;
    return S >= SLO && S <= SHI && (PATH == kPathFast ? M >= S : M < S);
}

template <int SLO, int SHI, int PATH, int MINB>
__global__ void __launch_bounds__(kEvalThreads, MINB) eval_kernel(EvalParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    const BlobLayout &ly = p.lay;
    uint32_t *keys = reinterpret_cast<uint32_t *>(sm + ly.bytes);
    uint32_t *hist = keys + kEvalTile;
    uint16_t *order = reinterpret_cast<uint16_t *>(hist + kBinsPad);
    int32_t *outT = reinterpret_cast<int32_t *>(order + kEvalTile);
    uint8_t *outF = reinterpret_cast<uint8_t *>(outT + kEvalTile);
    __shared__ uint32_t warp_tot[32];
    __shared__ uint32_t n_owned;
    constexpr int kBins = (SHI - SLO + 1) * 64 + 1;
    constexpr uint32_t kNone = 0xffffffffu;

    stage_blob(sm, p.blob, ly.bytes);
    __syncthreads();
    const Tab t = tab_at(sm, ly);
    const int64_t n_tiles = (p.n + kEvalTile - 1) / kEvalTile;

    for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        const int64_t base = tile * kEvalTile;
        const int cnt = (int)(p.n - base < kEvalTile ? p.n - base : (int64_t)kEvalTile);
        for (int i = threadIdx.x; i < kBinsPad; i += blockDim.x) hist[i] = 0;
        __syncthreads();
        // 1. counting sort of the owned candidates by (S, M/4)
        for (int i = threadIdx.x; i < cnt; i += blockDim.x) {
            const uint32_t w = __ldg(&p.cands[base + i].w);
            const int S = w & 0xff, M = (w >> 8) & 0xff;
            bool invalid;
            uint32_t key = kNone;
            if (owns<SLO, SHI, PATH>(S, M, invalid)) {
                key = invalid ? kBins - 1 : (S - SLO) * 64 + (M >> 2);
                atomicAdd(&hist[key], 1u);
            }
            keys[i] = key;
        }
        __syncthreads();
        const uint32_t last_bin = hist[kBins - 1];
        block_exclusive_scan(hist, kBins, warp_tot);
        if (threadIdx.x == 0) n_owned = hist[kBins - 1] + last_bin;
        for (int i = threadIdx.x; i < cnt; i += blockDim.x) {
            if (keys[i] != kNone) {
                const uint32_t pos = atomicAdd(&hist[keys[i]], 1u);
                order[pos] = (uint16_t)i;
            }
        }
        __syncthreads();
        const int owned = (int)n_owned;
        // 2. evaluate in sorted order; every lane of a warp takes part in the
        //    ballots, so the loop runs over the owned count rounded up to 32
        const int own32 = (owned + 31) & ~31;
        for (int j = threadIdx.x; j < own32; j += blockDim.x) {
            const bool active = j < owned;
            const int i = active ? order[j] : 0;
            const uint32_t key = active ? keys[i] : (uint32_t)(kBins - 1);
            const int S = key == (uint32_t)(kBins - 1) ? 0 : (int)(key >> 6) + SLO;
            uint4 rec = make_uint4(0, 0, 0, 0);
            if (active) rec = __ldg(&p.cands[base + i]);
            int32_t T = -1;
            uint8_t F = POS_FEAS_INVALID;
            unsigned pending = __ballot_sync(0xffffffffu, active);
            while (pending) {
                const int leader = __ffs(pending) - 1;
                const int Sg = __shfl_sync(0xffffffffu, S, leader);
                const bool mine = active && S == Sg;
                const unsigned grp = __ballot_sync(0xffffffffu, mine);
                if (mine && Sg > 0) dispatch_range<SLO, SHI, PATH>(Sg, t, rec, p, T, F);
                pending &= ~grp;
            }
            if (active) {
                outT[i] = T;
                outF[i] = F;
            }
        }
        __syncthreads();
        // 3. write back the owned results in input order
        for (int i = threadIdx.x; i < cnt; i += blockDim.x) {
            if (keys[i] != kNone) {
                p.T[base + i] = outT[i];
                p.F[base + i] = outF[i];
            }
        }
        __syncthreads();
    }
}

template <int SLO, int SHI, int PATH, int MINB>
pos_status launch_eval_range(const EvalParams &p, int smem, cudaStream_t stream) {
    auto kern = eval_kernel<SLO, SHI, PATH, MINB>;
    POS_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    int per_sm = 0;
    POS_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kEvalThreads, smem));
    if (per_sm < 1) return fail(POS_ECUDA, "eval kernel does not fit on an SM");
    const int64_t tiles = (p.n + kEvalTile - 1) / kEvalTile;
    const int grid = (int)std::min<int64_t>(tiles, (int64_t)per_sm * sm_count());
    kern<<<grid, kEvalThreads, smem, stream>>>(p);
    POS_CUDA(cudaGetLastError());
    return POS_OK;
}

// one launcher per instantiation unit (eval_range_*.cu)
pos_status eval_fast_1_4(const EvalParams &p, int smem, cudaStream_t s);
pos_status eval_fast_5_8(const EvalParams &p, int smem, cudaStream_t s);
pos_status eval_fast_9_12(const EvalParams &p, int smem, cudaStream_t s);
pos_status eval_fast_13_16(const EvalParams &p, int smem, cudaStream_t s);
pos_status eval_generic_2_8(const EvalParams &p, int smem, cudaStream_t s);
pos_status eval_generic_9_16(const EvalParams &p, int smem, cudaStream_t s);

}  // namespace pos
