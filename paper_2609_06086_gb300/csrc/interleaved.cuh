// Interleaved 1F1B evaluation (Sec. 4.1.4): N devices each hold V model
// chunks, so the pipeline has J = N*V virtual stages (virtual stage j is
// chunk j / N on device j % N) and the DAG 2VNM compute nodes.  One thread
// evaluates one candidate with all state in registers:
//   * weights: F_j, B_j of every virtual stage (prefix-sum differences on
//     its device's class), the transfer times pf_d = p2p_f[k_d][k_{d+1}] and
//     pb_d = p2p_b[k_{d+1}][k_d] (an edge j -> j+1 always joins device j % N
//     to device (j+1) % N), and each device's all-reduce time summed over
//     its chunks;
//   * makespan: the ops in the static order of interleaved_order.h, where
//     each op is one relaxation finish = max(device clock, finish of the
//     latest op of its kind on the neighbouring virtual stage + edge) +
//     weight, and T = max_d (clock_d + allreduce_d) (the last op of device d
//     is B of chunk 0 on the last micro-batch, which feeds R_d);
//   * memory: the largest activation footprint over device d's chain plus
//     its resident bytes must fit its class's capacity.  The footprint after
//     each op adds the chunk's activations on a forward and releases them on
//     a backward; it is largest after a forward, and in the steady phase its
//     values after the forwards repeat with period NV (every NV consecutive
//     forwards, and backwards, cover each chunk N times), so the warm-up
//     footprint (from per-chunk forward counts) and at most one period,
//     scanned in runs of fixed chunks, decide it.
#pragma once
#include "eval_kernel.cuh"
#include "interleaved_order.h"

namespace pos {

// The interleaved key region follows the 1F1B keys: record (N, V, M) with
// V >= 2, N*V <= 16 and M = q*N has key kKeys + kIlKeyOf[N-1][V] + q.
constexpr int kKeysIl = kKeys + IlPair<kIlPairs>::key;

template <int N, int V>
struct IlState {
    static constexpr int J = N * V;
    int32_t Fo[J], Bo[J], clk[N];  // latest forward / backward finish per virtual stage
    int32_t F[J], B[J], pf[N], pb[N];
};

template <int N, int V, int OP>
__device__ __forceinline__ void il_relax(IlState<N, V> &s) {
    constexpr int J = N * V, j = OP & 15, d = j % N;
    if constexpr ((OP & 0x80) == 0) {
        int32_t t = s.clk[d];
        if constexpr (j > 0) t = add_max(s.Fo[j - 1], s.pf[(j - 1) % N], t);
        s.Fo[j] = t + s.F[j];
        s.clk[d] = s.Fo[j];
    } else {
        int32_t t = s.clk[d];
        if constexpr (j + 1 < J) t = add_max(s.Bo[j + 1], s.pb[d], t);
        s.Bo[j] = t + s.B[j];
        s.clk[d] = s.Bo[j];
    }
}

// part 0 = P, 1 = Body, 2 = E, 3 = Short
template <int N, int V, int PART, int I>
__device__ __forceinline__ constexpr int il_op() {
    using O = IlOrder<N, V>;
    if constexpr (PART == 0) return O::P[I];
    else if constexpr (PART == 1) return O::Body[I];
    else if constexpr (PART == 2) return O::E[I];
    else return O::Short[I];
}

template <int N, int V, int PART, int... I>
__device__ __forceinline__ void il_run(IlState<N, V> &s, std::integer_sequence<int, I...>) {
    (il_relax<N, V, il_op<N, V, PART, I>()>(s), ...);
}

template <int N, int V>
__device__ __forceinline__ void il_makespan_ops(IlState<N, V> &s, int q) {
    using O = IlOrder<N, V>;
#pragma unroll
    for (int d = 0; d < N; ++d) s.clk[d] = 0;
    if (q < O::q0) {
        il_run<N, V, 3>(s, std::make_integer_sequence<int, O::nShort>{});
        return;
    }
    il_run<N, V, 0>(s, std::make_integer_sequence<int, O::nP>{});
#pragma unroll 1
    for (int r = O::q0; r < q; ++r) il_run<N, V, 1>(s, std::make_integer_sequence<int, O::nBody>{});
    il_run<N, V, 2>(s, std::make_integer_sequence<int, O::nE>{});
}

// Forwards of chunk c among a device's first k forwards: forward f runs
// chunk (f mod NV) / N, so every NV consecutive forwards hold N of each
// chunk.
__host__ __device__ constexpr int il_fwd_count(int N, int V, int k, int c) {
    const int part = k % (N * V) - c * N;
    return (k / (N * V)) * N + (part < 0 ? 0 : part > N ? N : part);
}

// Largest footprint after a forward over the steady pairs (F_{W+i}, B_i),
// i < STEPS, from `held` after the W warm-up forwards.  The forward's chunk
// changes when (W + i) mod N = 0 and the backward's when i mod N = 0; in a
// run between two changes both are fixed, the footprint after the run's
// k-th forward is h0 + k (aF - aB), and its largest value is at the run's
// first or last forward.
template <int N, int V, int W, int STEPS>
__device__ __forceinline__ int64_t il_steady_peak(const int64_t (&act)[V], int64_t held) {
    constexpr int NV = N * V;
    int64_t peak = 0, h0 = 0;
    int first = 0;
#pragma unroll
    for (int i = 0; i < STEPS; ++i) {
        const int64_t aF = act[((W + i) % NV) / N], aB = act[V - 1 - (i % NV) / N];
        const bool start = i == 0 || (W + i) % N == 0 || i % N == 0;
        const bool end = i == STEPS - 1 || (W + i + 1) % N == 0 || (i + 1) % N == 0;
        if (start) {
            h0 = held + aF;
            first = i;
        }
        if (end) {
            const int64_t span = (int64_t)(i - first) * (aF - aB);
            peak = max(peak, max(h0, h0 + span));
            held = h0 + span - aB;
        }
    }
    return peak;
}

// Does device d (class k) fit?  act[c]: activations of its chunk c per
// micro-batch; resident: its weights and optimizer state over all chunks.
template <int N, int V, int d>
__device__ __forceinline__ bool il_device_fits(const int64_t (&act)[V], int64_t resident,
                                               int64_t cap, int q) {
    constexpr int NV = N * V;
    int64_t peak;
    if (q == 1) {  // M = N: every forward runs before the first backward
        int64_t all = 0;
#pragma unroll
        for (int c = 0; c < V; ++c) all += act[c];
        peak = (int64_t)N * all;
    } else {
        constexpr int w = 2 * (N - d - 1) + (V - 1) * N;  // warm-up forwards (< VM for q >= 2)
        int64_t held = 0;
#pragma unroll
        for (int c = 0; c < V; ++c) held += (int64_t)il_fwd_count(N, V, w, c) * act[c];
        // steady pairs (F_{w+i}, B_i): all of one period for q >= 3, the
        // 2NV - w pairs there are for q = 2 when fewer
        constexpr int steady2 = 2 * NV - w;
        if (q >= 3 || steady2 >= NV) peak = il_steady_peak<N, V, w, NV>(act, held);
        else peak = il_steady_peak<N, V, w, (steady2 < NV ? steady2 : NV)>(act, held);
    }
    return peak + resident <= cap;
}

template <int N, int V, int... D>
__device__ __forceinline__ bool il_fits_all(const Tab &t, const int (&cut)[N * V + 1],
                                            const int (&cls)[N], int q,
                                            std::integer_sequence<int, D...>) {
    bool ok = true;
    (
        [&] {
            constexpr int d = D;
            const int k = cls[d];
            int64_t act[V], resident = 0;
#pragma unroll
            for (int c = 0; c < V; ++c) {
                const int j = c * N + d;
                act[c] = Pa(t, k, cut[j + 1]) - Pa(t, k, cut[j]);
                resident += Pw(t, k, cut[j + 1]) - Pw(t, k, cut[j]);
            }
            ok &= il_device_fits<N, V, d>(act, resident, cap_of(t, k), q);
        }(),
        ...);
    return ok;
}

// Makespan and feasibility of one decoded interleaved candidate: S = N
// devices, pad byte V, cut positions of the J virtual stages packed by the
// decode pass.
template <int N, int V>
__device__ __forceinline__ void il_eval_one(const Tab &t, const uint4 &rec, const uint4 &packed,
                                            int32_t &T, uint8_t &feasible) {
    constexpr int J = N * V;
    const uint32_t tcode = rec.z;
    const int M = (rec.w >> 8) & 0xff;
    const int tp = (rec.w >> 16) & 0xff;
    const int q = M / N;
    int cls[N], cut[J + 1];
#pragma unroll
    for (int d = 0; d < N; ++d) cls[d] = stage_class(tcode, rec.x, tp, t.n_tp(), d);
    const uint32_t pw[4] = {packed.x, packed.y, packed.z, packed.w};
    cut[0] = 0;
#pragma unroll
    for (int j = 0; j < J - 1; ++j) cut[j + 1] = (pw[j / 4] >> (8 * (j % 4))) & 0xff;
    cut[J] = t.L();
    feasible = il_fits_all<N, V>(t, cut, cls, q, std::make_integer_sequence<int, N>{})
                   ? POS_FEAS_YES
                   : POS_FEAS_NO;
    IlState<N, V> s;
    int32_t dsum[N];
#pragma unroll
    for (int d = 0; d < N; ++d) {
        dsum[d] = 0;
        s.pf[d] = p2f(t, cls[d], cls[(d + 1) % N]);
        s.pb[d] = p2b(t, cls[(d + 1) % N], cls[d]);
    }
#pragma unroll
    for (int j = 0; j < J; ++j) {
        const int k = cls[j % N];
        s.F[j] = Pf(t, k, cut[j + 1]) - Pf(t, k, cut[j]);
        s.B[j] = Pb(t, k, cut[j + 1]) - Pb(t, k, cut[j]);
        dsum[j % N] += Pd(t, k, cut[j + 1]) - Pd(t, k, cut[j]);
    }
    il_makespan_ops<N, V>(s, q);
    int32_t best = 0;
#pragma unroll
    for (int d = 0; d < N; ++d) best = max(best, s.clk[d] + dsum[d]);
    T = best;
}

template <int PLO, int PHI>
__device__ __forceinline__ void il_dispatch(int N, int V, const Tab &t, const uint4 &rec,
                                            const uint4 &packed, int32_t &T, uint8_t &feasible) {
    if constexpr (PLO <= PHI) {
        if (N == IlPair<PLO>::N && V == IlPair<PLO>::V) {
            il_eval_one<IlPair<PLO>::N, IlPair<PLO>::V>(t, rec, packed, T, feasible);
            return;
        }
        il_dispatch<PLO + 1, PHI>(N, V, t, rec, packed, T, feasible);
    }
}

// Evaluates the sorted range of pairs PLO..PHI (their key blocks are
// contiguous); warps split by (N, V) like eval_kernel splits by S.
template <int PLO, int PHI, int MINB>
__global__ void __launch_bounds__(kEvalThreads, MINB) il_eval_kernel(EvalParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    // the key offsets come from the sort's scan, two or more kernels back
    const int64_t begin = p.offs[kKeys + IlPair<PLO>::key], end = p.offs[kKeys + IlPair<PHI + 1>::key];
    // blocks with no record (all of them when the range is empty) leave
    // without staging the tables, after the decode pass has completed
    if ((int64_t)blockIdx.x * blockDim.x >= end - begin) {
        grid_dep_wait();
        return;
    }
    stage_blob(sm, p.blob, p.lay.bytes);
    __syncthreads();
    grid_dep_wait();  // the decoded records
    grid_dep_trigger();
    const Tab t = tab_at(sm, p.lay);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t span = ((end - begin) + 31) & ~(int64_t)31;
    int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    // the next decoded record is loaded one iteration ahead, so its memory
    // latency overlaps the current candidate's wavefront
    const uint4 none = make_uint4(0, 0, 0, 1u << 24);
    uint4 next_packed = none, next_meta = none;
    if (j < end - begin) {
        next_packed = __ldcs(p.cuts + 2 * (begin + j));
        next_meta = __ldcs(p.cuts + 2 * (begin + j) + 1);
    }
    for (; j < span; j += stride) {
        bool active = j < end - begin;
        uint32_t i = 0;
        uint4 rec = make_uint4(0, 0, 0, 0);
        const uint4 packed = next_packed, meta = next_meta;
        next_packed = none;
        if (j + stride < end - begin) {
            next_packed = __ldcs(p.cuts + 2 * (begin + j + stride));
            next_meta = __ldcs(p.cuts + 2 * (begin + j + stride) + 1);
        }
        if (active) {
            active = (packed.w >> 24) == 0;  // not answered by the decode pass
            i = meta.x;
            rec = make_uint4(meta.w, 0u, meta.y, meta.z);
        }
        const int g = active ? (int)(rec.w & 0xff) * 32 + (int)(rec.w >> 24) : 0;  // N*32 + V
        int32_t T = -1;
        uint8_t feasible = POS_FEAS_INVALID;
        unsigned pending = __ballot_sync(0xffffffffu, active);
        while (pending) {
            const int leader = __ffs(pending) - 1;
            const int gg = __shfl_sync(0xffffffffu, g, leader);
            const bool mine = active && g == gg;
            const unsigned grp = __ballot_sync(0xffffffffu, mine);
            if (mine) il_dispatch<PLO, PHI>(gg >> 5, gg & 31, t, rec, packed, T, feasible);
            pending &= ~grp;
        }
        if (active) {
            p.T[i] = T;
            p.F[i] = feasible;
        }
    }
}

template <int PLO, int PHI, int MINB>
pos_status launch_il_range(const EvalParams &p, cudaStream_t stream) {
    auto kern = il_eval_kernel<PLO, PHI, MINB>;
    const int smem = p.lay.bytes;
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(kern), smem));
    int per_sm = 0;
    POS_TRY(blocks_per_sm(reinterpret_cast<const void *>(kern), kEvalThreads, smem, &per_sm));
    if (per_sm < 1) return fail(POS_ECUDA, "interleaved eval kernel does not fit on an SM");
    const int64_t blocks = (p.n + kEvalThreads - 1) / kEvalThreads;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(blocks, (int64_t)per_sm * sm_count()));
    POS_CUDA(launch_dependent(kern, grid, kEvalThreads, smem, stream, p));
    return POS_OK;
}

// one launcher per instantiation unit (eval_il_*.cu), pairs by index
pos_status eval_il_0_11(const EvalParams &p, cudaStream_t s);
pos_status eval_il_12_22(const EvalParams &p, cudaStream_t s);
pos_status eval_il_23_29(const EvalParams &p, cudaStream_t s);
pos_status eval_il_30_31(const EvalParams &p, cudaStream_t s);
pos_status eval_il_32_33(const EvalParams &p, cudaStream_t s);

inline pos_status eval_interleaved(const EvalParams &p, cudaStream_t s) {
    POS_TRY(eval_il_0_11(p, s));
    POS_TRY(eval_il_12_22(p, s));
    POS_TRY(eval_il_23_29(p, s));
    POS_TRY(eval_il_30_31(p, s));
    return eval_il_32_33(p, s);
}

}  // namespace pos
