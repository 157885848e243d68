// Shared internals of libposeidon: error state, the device table blob and
// the per-candidate device routines (composition unranking/ranking, stage
// weights, memory feasibility, the 1F1B makespan wavefront).
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <utility>
#include <vector>

#include "../../include/poseidon.h"

namespace pos {

// ---------------------------------------------------------------------------
// Error state (per host thread)
// ---------------------------------------------------------------------------
void set_error(const std::string &msg);
pos_status fail(pos_status st, const std::string &msg);
pos_status cuda_fail(cudaError_t e, const char *what);
// Raises a kernel's dynamic shared-memory limit to `smem` on the current
// device unless an earlier call already set at least that much (the
// attribute call costs host time that a launch-bound pipeline feels).
pos_status ensure_smem(const void *kernel, int smem);
// Resident blocks per SM of `kernel` at (threads, smem), from the occupancy
// calculator once per device and configuration, then from a cache (the
// query costs host time on every launch otherwise).
pos_status blocks_per_sm(const void *kernel, int threads, int smem, int *out);

// Programmatic dependent launch (sm_90 and later).  A kernel launched by
// launch_dependent may be scheduled while the kernel queued before it on
// the stream is still running; before it reads anything that kernel wrote
// it executes grid_dep_wait(), which returns once that grid has completed
// and its memory is visible.  It then calls grid_dep_trigger(), which lets
// the next such kernel be scheduled: a kernel's pre-wait part can therefore
// only overlap the post-wait part of its predecessor, so it may read
// whatever was written two or more kernels earlier (the cost tables, slice
// records and bound tables of a search).  Every block of such a kernel
// executes grid_dep_wait() before it exits, even when it has no work: a grid
// completes only after its predecessor has, which keeps the chain's order
// transitive for the kernels after it.  Without the launch attribute the two
// instructions do nothing.
__device__ __forceinline__ void grid_dep_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void grid_dep_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent(void (*kern)(KArgs...), int grid, int block, int smem,
                                    cudaStream_t stream, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)block);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

#define POS_CUDA(call)                                           \
    do {                                                         \
        cudaError_t e_ = (call);                                 \
        if (e_ != cudaSuccess) return pos::cuda_fail(e_, #call); \
    } while (0)

// Propagate a non-OK pos_status.
#define POS_TRY(call)                             \
    do {                                          \
        const pos_status st_ = (call);            \
        if (st_ != POS_OK) return st_;            \
    } while (0)

// ---------------------------------------------------------------------------
// Table blob: one contiguous device buffer, staged whole into shared memory
// by every kernel.  Offsets are bytes from the blob start, 16-byte aligned.
//   binom  u64 [16][128]        C(n, k) at [k][n], k <= 15 (0 for n < k)
//   Pw, Pa i64 [K][L+1] each    exclusive prefix sums of mem_w, mem_a
//   cap    i64 [K]
//   Pf, Pb, Pd i32 [K][L+1]     exclusive prefix sums of fwd, bwd, dsync
//   p2f, p2b   i32 [K][K]       transfer times [src class][dst class]
// ---------------------------------------------------------------------------
constexpr int kBinomN = 128;
constexpr int kBinomK = 16;

struct BlobLayout {
    int L, K, n_types, n_tp;
    int sched;  // POS_SCHED_* (stage chains, in-flight counts; Interleaved 1F1B
                // evaluates records with V < 2 as 1F1B)
    int off_binom, off_Pw, off_Pa, off_cap, off_Pf, off_Pb, off_Pd, off_p2f, off_p2b;
    int bytes;  // multiple of 16
};

BlobLayout make_layout(int L, int n_types, int n_tp);
// The timing part of a blob (Pf, Pb, Pd, p2f, p2b: its last five tables),
// rebased to start at byte 0, for kernels that read nothing else; the
// timing part starts at byte ly.off_Pf of the full blob.
BlobLayout timing_layout(const BlobLayout &ly);
// The memory part (Pw, Pa, cap: the three tables after the binomials),
// rebased likewise; it starts at byte ly.off_Pw of the full blob.
BlobLayout memory_layout(const BlobLayout &ly);

struct Handle {
    int device;
    BlobLayout lay;
    void *d_blob;  // device copy of the blob
    // overflow guard terms: sum_l max_k(fwd+bwd), sum_l max_k dsync, max p2p
    int64_t guard_A, guard_D, guard_P;
    // memory-limit table of the evaluation's decode pass (after the blob in
    // the same allocation, byte lim_off): lim[k][w-1][a] = the largest b with
    // sum_{l in [a,b)} (mem_w + w mem_a) <= cap[k] (a when no layer fits), for
    // w = 1..lim_w in-flight micro-batches; lim_bytes = 0 when the table
    // would exceed kLimMaxBytes and the pass checks the sums directly
    int lim_off, lim_w, lim_bytes;
};
constexpr int kLimMaxBytes = 32768;
// Threads per block of the argmin partial kernel (poseidon_argmin and
// poseidon_argmin_noalloc): its shared arrays hold one entry per warp of a
// block of this size, so every launch must use exactly this many threads.
constexpr int kArgminThreads = 256;

pos_status validate_tables(const pos_tables *t);
pos_status create_handle(const pos_tables *t, int sched, Handle **out);
// host part of create_handle: validated blob with raw rows, plus guard terms
pos_status build_blob(const pos_tables *t, int sched, std::vector<unsigned char> &host,
                      BlobLayout &ly, int64_t &guard_A, int64_t &guard_D, int64_t &guard_P);
// device part: per-class prefix sums in place, asynchronous on `stream`
pos_status launch_prefix_rows(void *d_blob, const BlobLayout &ly, cudaStream_t stream);
void destroy_handle(Handle *h);
int sm_count();

// View of the blob staged in shared memory.  It keeps the shared-memory
// base and a pointer to the layout in kernel parameter space; every access
// adds an offset read from there, so no table pointer occupies a register.
struct Tab {
    const unsigned char *base;  // the staged blob (dynamic shared memory)
    const BlobLayout *ly;       // points into kernel parameter space
    __device__ __forceinline__ int L() const { return ly->L; }
    __device__ __forceinline__ int Lp1() const { return ly->L + 1; }
    __device__ __forceinline__ int K() const { return ly->K; }
    __device__ __forceinline__ int n_tp() const { return ly->n_tp; }
    __device__ __forceinline__ int n_types() const { return ly->n_types; }
};

__device__ __forceinline__ int32_t ld32(const unsigned char *base, uint32_t off) {
    return *reinterpret_cast<const int32_t *>(base + off);
}
__device__ __forceinline__ int64_t ld64(const unsigned char *base, uint32_t off) {
    return *reinterpret_cast<const int64_t *>(base + off);
}

__device__ __forceinline__ Tab tab_at(const unsigned char *base, const BlobLayout &ly) {
    Tab t;
    t.base = base;
    t.ly = &ly;
    return t;
}

__device__ __forceinline__ int32_t Pf(const Tab &t, int k, int c) {
    return ld32(t.base, t.ly->off_Pf + 4u * (uint32_t)(k * (t.ly->L + 1) + c));
}
__device__ __forceinline__ int32_t Pb(const Tab &t, int k, int c) {
    return ld32(t.base, t.ly->off_Pb + 4u * (uint32_t)(k * (t.ly->L + 1) + c));
}
__device__ __forceinline__ int32_t Pd(const Tab &t, int k, int c) {
    return ld32(t.base, t.ly->off_Pd + 4u * (uint32_t)(k * (t.ly->L + 1) + c));
}
__device__ __forceinline__ int64_t Pw(const Tab &t, int k, int c) {
    return ld64(t.base, t.ly->off_Pw + 8u * (uint32_t)(k * (t.ly->L + 1) + c));
}
__device__ __forceinline__ int64_t Pa(const Tab &t, int k, int c) {
    return ld64(t.base, t.ly->off_Pa + 8u * (uint32_t)(k * (t.ly->L + 1) + c));
}
__device__ __forceinline__ int64_t cap_of(const Tab &t, int k) {
    return ld64(t.base, t.ly->off_cap + 8u * (uint32_t)k);
}
__device__ __forceinline__ int32_t p2f(const Tab &t, int a, int b) {
    return ld32(t.base, t.ly->off_p2f + 4u * (uint32_t)(a * t.ly->K + b));
}
__device__ __forceinline__ int32_t p2b(const Tab &t, int a, int b) {
    return ld32(t.base, t.ly->off_p2b + 4u * (uint32_t)(a * t.ly->K + b));
}
// stored k-major ([k][n]) as 64-bit words, so that a warp reading
// C(n_lane, k) for one k touches consecutive 8-byte words
__device__ __forceinline__ uint64_t binom(const Tab &t, int n, int k) {
    return (uint64_t)ld64(t.base, t.ly->off_binom + 8u * (uint32_t)(k * kBinomN + n));
}

// One stage of the combinatorial-number-system unranking.  With rem layers
// left for k+1 stages (k >= 1), the remaining rank is carried as
// Y = C(rem-1, k) - rank, 1 <= Y <= C(rem-1, k).  The stage takes rem - j
// layers, j the smallest value in [k, rem-1] with C(j, k) >= Y; the next
// stage's Y (rem' = j layers, k' = k-1) is Y - C(j-1, k), since
// C(j, k) = C(j-1, k) + C(j-1, k-1) (Pascal's rule) puts it in
// [1, C(j-1, k-1)].  So a stage reads only C(j-1, k) and C(j, k).
//
// j is first estimated from C(x, k) ~ m^k / k! * exp(-k(k^2-1) / (12 m^2)),
// m = x - (k-1)/2 (the product of the k factors m +- d around their mean):
// m0 = (Y k!)^(1/k), x ~ m0 + (k-1)/2 + (k^2-1) / (24 m0) (half the
// second-order term, which over-corrects), and j = ceil(x - 0.01) (a margin
// for rounding error), taken as the nearest integer to x + 0.49.  Over
// uniform ranks of 64 layers in 2..16 stages this lands on j in about 99 %
// of the stages (else one step low); exact comparisons then move it to the
// answer whatever the estimate.
struct UnrankCoef {
    float log2_fact;  // log2(k!)
    float inv_k;      // 1/k
    float shift;      // (k-1)/2 + 0.49
    float corr;       // (k^2-1)/24
};
__device__ __constant__ static const UnrankCoef kUnrankCoef[16] = {
    {0.000000000f, 0.000000000f, 0.00f, 0.000000000f},
    {0.000000000f, 1.000000000f, 0.49f, 0.000000000f},
    {1.000000000f, 0.500000000f, 0.99f, 0.125000000f},
    {2.584962501f, 0.333333333f, 1.49f, 0.333333333f},
    {4.584962501f, 0.250000000f, 1.99f, 0.625000000f},
    {6.906890596f, 0.200000000f, 2.49f, 1.000000000f},
    {9.491853096f, 0.166666667f, 2.99f, 1.458333333f},
    {12.299208018f, 0.142857143f, 3.49f, 2.000000000f},
    {15.299208018f, 0.125000000f, 3.99f, 2.625000000f},
    {18.469133020f, 0.111111111f, 4.49f, 3.333333333f},
    {21.791061115f, 0.100000000f, 4.99f, 4.125000000f},
    {25.250492733f, 0.090909091f, 5.49f, 5.000000000f},
    {28.835455234f, 0.083333333f, 5.99f, 5.958333333f},
    {32.535894952f, 0.076923077f, 6.49f, 7.000000000f},
    {36.343249874f, 0.071428571f, 6.99f, 8.125000000f},
    {40.250140470f, 0.066666667f, 7.49f, 9.333333333f}};

// the hardware's approximate base-2 logarithm, power and reciprocal (PTX
// lg2 / ex2 / rcp .approx): an estimate only, the comparisons fix any error
__device__ __forceinline__ float approx_lg2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float approx_ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float approx_rcp(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ int unrank_guess(uint64_t Y, int k, int rem) {
    const UnrankCoef c = kUnrankCoef[k];
    // Y as a float from its two 32-bit words: a 64-bit integer conversion
    // issues to the FP64 pipe, a small fraction of the FP32 rate here
    const float yf = __fmaf_rz(__uint2float_rz((uint32_t)(Y >> 32)), 4294967296.0f,
                               __uint2float_rz((uint32_t)Y));
    const float lg = approx_lg2(yf);
    const float m0 = approx_ex2((lg + c.log2_fact) * c.inv_k);
    const float x = m0 + c.shift + c.corr * approx_rcp(m0);
    // nearest integer by the float adder: 1.5 * 2^23 + x (0 <= x < 2^22)
    // has unit spacing, so its low bits are round(x)
    const int j = __float_as_int(x + 12582912.0f) - 0x4B400000;
    return min(max(j, k), rem - 1);
}

__device__ __forceinline__ int unrank_step(const Tab &t, int rem, int k, uint64_t &Y) {
    int j = unrank_guess(Y, k, rem);
    uint64_t below = binom(t, j - 1, k), at = binom(t, j, k);
    while (below >= Y) {  // stops at j = k at the latest: C(k-1, k) = 0 < Y
        --j;
        at = below;
        below = binom(t, j - 1, k);
    }
    while (at < Y && j < rem - 1) {  // C(rem-1, k) >= Y stops it first
        ++j;
        below = at;
        at = binom(t, j, k);
    }
    Y -= below;
    return j;
}

// Cooperative 16-byte copy of the blob into shared memory, four loads in
// flight per thread (a load-store pair per iteration would wait a full
// memory latency each time).
__device__ __forceinline__ void stage_blob(unsigned char *dst, const void *src, int bytes) {
    const uint4 *s = reinterpret_cast<const uint4 *>(src);
    uint4 *d = reinterpret_cast<uint4 *>(dst);
    const int n = bytes / 16, bd = blockDim.x;
    int i = threadIdx.x;
    for (; i + 3 * bd < n; i += 4 * bd) {
        const uint4 a = __ldg(s + i), b = __ldg(s + i + bd), c = __ldg(s + i + 2 * bd),
                    e = __ldg(s + i + 3 * bd);
        d[i] = a;
        d[i + bd] = b;
        d[i + 2 * bd] = c;
        d[i + 3 * bd] = e;
    }
    for (; i < n; i += bd) d[i] = __ldg(s + i);
}

// Bulk copies global -> this CTA's shared memory on the TMA engine
// (cp.async.bulk), completion counted in bytes on one mbarrier.  Thread 0
// calls bulk_begin with the total byte count, then issues the copies
// (16-byte aligned addresses, sizes multiples of 16); then every thread of
// the block calls bulk_wait, which returns the same value in all threads:
// false if the copies did not complete within kBulkWaitLimit polls.  That is
// a last-resort exit (2^24 polls, far beyond any copy of at most a few
// hundred KB): the caller counts it and leaves, the search then reports
// POS_ETIMEOUT, and a copy still in flight may land in shared memory that
// the block no longer owns; nothing exercises it on a GPU.
constexpr int kBulkWaitLimit = 1 << 24;

__device__ __forceinline__ void bulk_begin(uint64_t *bar, uint32_t total_bytes) {
    const uint32_t b = (uint32_t)__cvta_generic_to_shared(bar);
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(b) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b),
                 "r"(total_bytes)
                 : "memory");
}

__device__ __forceinline__ void bulk_copy(void *dst_smem, const void *src, uint32_t bytes,
                                          uint64_t *bar) {
    const uint32_t b = (uint32_t)__cvta_generic_to_shared(bar);
    const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst_smem);
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(d),
        "l"(src), "r"(bytes), "r"(b)
        : "memory");
}

__device__ __forceinline__ bool bulk_wait(uint64_t *bar) {
    __syncthreads();  // the barrier is initialised before anyone polls it
    const uint32_t b = (uint32_t)__cvta_generic_to_shared(bar);
    uint32_t done = 0;
    for (int it = 0; it < kBulkWaitLimit && !done; ++it) {
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n"
            " selp.u32 %0, 1, 0, p;\n}"
            : "=r"(done)
            : "r"(b)
            : "memory");
    }
    return __syncthreads_and(done) != 0;
}

// The whole blob (or a rebased part of it) by one bulk copy.
__device__ __forceinline__ bool stage_blob_bulk(unsigned char *dst, const void *src, int bytes,
                                                uint64_t *bar) {
    if (threadIdx.x == 0) {
        bulk_begin(bar, (uint32_t)bytes);
        bulk_copy(dst, src, (uint32_t)bytes, bar);
    }
    return bulk_wait(bar);
}

// ---------------------------------------------------------------------------
// Composition <-> lexicographic rank (combinatorial number system).
// With p stages left and rem layers left, the compositions whose current
// stage takes fewer than v layers number C(rem-1, p-1) - C(rem-v, p-1)
// (hockey-stick sum of C(rem-u-1, p-2) over u < v).
// cut[0] = 0, cut[s+1] = layers of stages 0..s, cut[S] = L.
// ---------------------------------------------------------------------------
// Rank of the composition given by cut[0..S] (the numbering unrank_step
// walks stage by stage).
template <int S>
__device__ __forceinline__ uint64_t rank_cuts(const Tab &t, const int (&cut)[S + 1]) {
    uint64_t r = 0;
#pragma unroll
    for (int s = 0; s < S - 1; ++s) {
        const int rem = t.L() - cut[s];
        const int l = cut[s + 1] - cut[s];
        const int k = S - s - 1;
        r += binom(t, rem - 1, k) - binom(t, rem - l, k);
    }
    return r;
}

// ---------------------------------------------------------------------------
// Stage weights (Sec. 4.1.3) from prefix-sum differences; memory (Sec. 3.2).
// ---------------------------------------------------------------------------
// max(a + b, c) as one fused integer add-max (the CUDA intrinsic
// __viaddmax_s32); the makespan relaxations are built from it.
__device__ __forceinline__ int32_t add_max(int32_t a, int32_t b, int32_t c) {
    return __viaddmax_s32(a, b, c);
}

template <int S>
struct StageW {
    int32_t F[S], B[S], d[S];
    int32_t pf[S], pb[S];  // pf[s]: F edge s->s+1; pb[s]: B edge s+1->s
};

// In-flight micro-batches of 0-based stage s under 1F1B: min(S - s, M).
// Micro-batches a 0-based stage s holds at once = its warm-up forwards:
// N-s+1 (1F1B) or 2(N-s)+1 (Eager 1F1B) in 1-based numbering, at most M.
__host__ __device__ __forceinline__ int inflight(int sched, int S, int M, int s) {
    const int w = sched == POS_SCHED_EAGER_1F1B ? 2 * (S - 1 - s) + 1 : S - s;
    return w < M ? w : M;
}

// Does 0-based stage s of an S-stage pipeline on class k fit layers [a, b)?
// ... with w micro-batches in flight
__device__ __forceinline__ bool stage_fits_w(const Tab &t, int w, int k, int a, int b) {
    const int64_t need = (Pw(t, k, b) - Pw(t, k, a)) + (int64_t)w * (Pa(t, k, b) - Pa(t, k, a));
    return need <= cap_of(t, k);
}
__device__ __forceinline__ bool stage_fits(const Tab &t, int S, int M, int s, int k, int a,
                                           int b) {
    return stage_fits_w(t, inflight(t.ly->sched, S, M, s), k, a, b);
}

template <int S>
__device__ __forceinline__ void stage_weights(const Tab &t, const int (&cut)[S + 1],
                                              const int (&cls)[S], StageW<S> &w) {
#pragma unroll
    for (int s = 0; s < S; ++s) {
        w.F[s] = Pf(t, cls[s], cut[s + 1]) - Pf(t, cls[s], cut[s]);
        w.B[s] = Pb(t, cls[s], cut[s + 1]) - Pb(t, cls[s], cut[s]);
        w.d[s] = Pd(t, cls[s], cut[s + 1]) - Pd(t, cls[s], cut[s]);
    }
#pragma unroll
    for (int s = 0; s < S; ++s) {
        w.pf[s] = (s + 1 < S) ? p2f(t, cls[s], cls[s + 1 < S ? s + 1 : s]) : 0;
        w.pb[s] = (s + 1 < S) ? p2b(t, cls[s + 1 < S ? s + 1 : s], cls[s]) : 0;
    }
}

template <int S>
__device__ __forceinline__ bool plan_fits(const Tab &t, int M, const int (&cut)[S + 1],
                                          const int (&cls)[S]) {
    bool ok = true;
#pragma unroll
    for (int s = 0; s < S; ++s) ok &= stage_fits(t, S, M, s, cls[s], cut[s], cut[s + 1]);
    return ok;
}

// ---------------------------------------------------------------------------
// 1F1B makespan as a max-plus wavefront (Sec. 4.1, longest path by DP).
//
// Stage s (1-based) runs W_s = min(S-s+1, M) forwards, then (B_i, F_{W+i})
// pairs, then the remaining backwards.  Every op is one relaxation
//     finish = max(finish of the stage's previous op,
//                  finish of the inter-stage predecessor + edge) + weight.
// The ops are visited in the level order of the unit-weight schedule,
//     F_{s,m}: m + s - 1 (m <= W_s), 2m + s - 2 (m > W_s);
//     B_{s,m}: 2S - s + 2m - 1,
// a topological order with at most one op per stage per level in which,
// visiting the stages of a level in descending order, the inter-stage
// predecessor of an op is always the latest op of that kind on the
// neighbouring stage.  So per stage only the finish of its last forward (Fo)
// and last backward (Bo) are kept, in registers.  For M >= S the levels
// split into a ramp-up (levels 1..2S-1), M-S steady two-level steps in which
// every stage does one F and one B, and a ramp-down (levels 2M..2M+2S-2);
// the ramps depend on S only and are fully unrolled.  M < S takes a
// separate instantiation (kPathGeneric) whose schedule is unrolled for
// each M in 1..S-1.
// ---------------------------------------------------------------------------
// Paths: 1F1B with M >= S (ramps + steady loop), 1F1B with M < S (unrolled
// per M), Eager 1F1B with M >= 2S-1 (ramps + steady loop), Eager 1F1B with
// M < 2S-1 as a level program (the search's leaf kernel) or unrolled per M
// (the evaluator).
enum { kPathFast = 0, kPathGeneric = 1, kPathEager = 2, kPathEagerShort = 3, kPathEagerUnrolled = 4 };

// Op of 1-based stage s1 at ramp-up level t (1 <= t <= 2S-1) and at
// ramp-down level 2M + tau (0 <= tau <= 2S-2), for M >= S: 0 none, 1 F, 2 B.
__host__ __device__ constexpr int ramp_up_op(int S, int s1, int t) {
    return (t >= s1 && t <= S) ? 1
           : ((t >= 2 * S - s1 + 2) && ((t + s1) & 1) == 0) ? 1
           : ((t >= 2 * S - s1 + 1) && ((t + s1) & 1) == 1) ? 2
                                                              : 0;
}
__host__ __device__ constexpr int ramp_down_op(int S, int s1, int tau) {
    return ((tau <= s1 - 2) && ((tau + s1) & 1) == 0) ? 1
           : ((tau <= 2 * S - s1 - 1) && ((tau + s1) & 1) == 1) ? 2
                                                                : 0;
}
// Was the last op of stage s1 before ramp-up level t a backward?  (No op
// yet counts as a forward: Fo starts at 0, the finish time of node S.)
__host__ __device__ constexpr bool up_last_is_b(int S, int s1, int t) {
    for (int u = t - 1; u >= 1; --u)
        if (ramp_up_op(S, s1, u)) return ramp_up_op(S, s1, u) == 2;
    return false;
}
// Same before ramp-down level 2M + tau; at the end of the steady state odd
// stages (1-based) last ran F and even stages B.
__host__ __device__ constexpr bool down_last_is_b(int S, int s1, int tau) {
    for (int u = tau - 1; u >= 0; --u)
        if (ramp_down_op(S, s1, u)) return ramp_down_op(S, s1, u) == 2;
    return (s1 & 1) == 0;
}

// One relaxation of stage s (0-based) on the forward or backward side:
// finish = max(stage clock, predecessor's finish + edge) + node weight, the
// add-max fused into one integer instruction (add_max).  Every time is >= 0
// (non-negative weights from time 0), so a stage without an inter-stage
// predecessor takes its clock alone.
template <int S, int s>
__device__ __forceinline__ void relax_f(int32_t (&Fo)[S], const StageW<S> &w, int32_t clock) {
    if constexpr (s > 0) Fo[s] = add_max(Fo[s - 1], w.pf[s - 1], clock) + w.F[s];
    else Fo[s] = clock + w.F[s];
}
template <int S, int s>
__device__ __forceinline__ void relax_b(int32_t (&Bo)[S], const StageW<S> &w, int32_t clock) {
    if constexpr (s + 1 < S) Bo[s] = add_max(Bo[s + 1], w.pb[s], clock) + w.B[s];
    else Bo[s] = clock + w.B[s];
}

// Ramp op of 1-based stage s1 at level t (UP) or at level 2M + t (DOWN);
// the clock is the finish of the stage's last op, known at compile time.
template <int S, bool UP, int t, int s1>
__device__ __forceinline__ void ramp_op(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w) {
    constexpr int op = UP ? ramp_up_op(S, s1, t) : ramp_down_op(S, s1, t);
    constexpr bool last_b = UP ? up_last_is_b(S, s1, t) : down_last_is_b(S, s1, t);
    constexpr int s = s1 - 1;
    if constexpr (op == 1) relax_f<S, s>(Fo, w, last_b ? Bo[s] : Fo[s]);
    else if constexpr (op == 2) relax_b<S, s>(Bo, w, last_b ? Bo[s] : Fo[s]);
}
// one level, stages in descending order (i = 0 is stage S)
template <int S, bool UP, int t, int... i>
__device__ __forceinline__ void ramp_level(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w,
                                           std::integer_sequence<int, i...>) {
    (ramp_op<S, UP, t, S - i>(Fo, Bo, w), ...);
}
template <int S, bool UP, int T0, int... t>
__device__ __forceinline__ void ramp(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w,
                                     std::integer_sequence<int, t...>) {
    (ramp_level<S, UP, T0 + t>(Fo, Bo, w, std::make_integer_sequence<int, S>{}), ...);
}
// steady level: at level parity P (0 even) stage s1 runs F when s1 has the
// same parity, B otherwise; an F follows the stage's B and vice versa
template <int S, int P, int i>
__device__ __forceinline__ void steady_op(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w) {
    constexpr int s1 = S - i, s = s1 - 1;
    if constexpr ((s1 & 1) == P) relax_f<S, s>(Fo, w, Bo[s]);
    else relax_b<S, s>(Bo, w, Fo[s]);
}
template <int S, int P, int... i>
__device__ __forceinline__ void steady_level(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w,
                                             std::integer_sequence<int, i...>) {
    (steady_op<S, P, i>(Fo, Bo, w), ...);
}

// M < S: the same level order, with W_s = min(S-s1+1, M); every op and the
// type of each stage's previous op are known at compile time for a given
// (S, M), so the whole schedule is unrolled (M < S <= 16 keeps it small).
__host__ __device__ constexpr int short_op(int S, int M, int s1, int t) {
    const int ws = S - s1 + 1 < M ? S - s1 + 1 : M;
    const bool odd = ((t + s1) & 1) != 0;
    if ((t >= s1 && t <= s1 + ws - 1) || (!odd && t >= 2 * ws + s1 && t <= 2 * M + s1 - 2))
        return 1;
    if (odd && t >= 2 * S - s1 + 1 && t <= 2 * S - s1 + 2 * M - 1) return 2;
    return 0;
}
__host__ __device__ constexpr bool short_last_is_b(int S, int M, int s1, int t) {
    for (int u = t - 1; u >= 1; --u)
        if (short_op(S, M, s1, u)) return short_op(S, M, s1, u) == 2;
    return false;
}
template <int S, int M, int t, int s1>
__device__ __forceinline__ void short_step(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w) {
    constexpr int op = short_op(S, M, s1, t);
    constexpr bool last_b = short_last_is_b(S, M, s1, t);
    constexpr int s = s1 - 1;
    if constexpr (op == 1) relax_f<S, s>(Fo, w, last_b ? Bo[s] : Fo[s]);
    else if constexpr (op == 2) relax_b<S, s>(Bo, w, last_b ? Bo[s] : Fo[s]);
}
template <int S, int M, int t, int... i>
__device__ __forceinline__ void short_level(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w,
                                            std::integer_sequence<int, i...>) {
    (short_step<S, M, t, S - i>(Fo, Bo, w), ...);
}
template <int S, int M, int... t>
__device__ __forceinline__ void short_all(int32_t (&Fo)[S], int32_t (&Bo)[S], const StageW<S> &w,
                                          std::integer_sequence<int, t...>) {
    (short_level<S, M, t + 1>(Fo, Bo, w, std::make_integer_sequence<int, S>{}), ...);
}
template <int S, int M>
__device__ __forceinline__ int32_t makespan_short(const StageW<S> &w) {
    int32_t Fo[S], Bo[S];
#pragma unroll
    for (int s = 0; s < S; ++s) {
        Fo[s] = 0;
        Bo[s] = 0;
    }
    short_all<S, M>(Fo, Bo, w, std::make_integer_sequence<int, 2 * (M + S - 1)>{});
    int32_t T = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) T = max(T, Bo[s] + w.d[s]);
    return T;
}
// runtime M in 1..S-1 -> its unrolled instance
template <int S, int... m>
__device__ __forceinline__ int32_t makespan_short_dispatch(const StageW<S> &w, int M,
                                                           std::integer_sequence<int, m...>) {
    int32_t T = -1;
    ((M == m + 1 ? (T = makespan_short<S, m + 1>(w), 0) : 0), ...);
    return T;
}

template <int S, int PATH>
__device__ __forceinline__ int32_t makespan_1f1b(const StageW<S> &w, int M) {
    int32_t Fo[S], Bo[S];
#pragma unroll
    for (int s = 0; s < S; ++s) {
        Fo[s] = 0;
        Bo[s] = 0;
    }
    if constexpr (PATH == kPathFast) {
        // ramp-up: levels 1 .. 2S-1
        ramp<S, true, 1>(Fo, Bo, w, std::make_integer_sequence<int, 2 * S - 1>{});
        // steady state: M - S steps of two levels (even, then odd)
        for (int j = 0; j < M - S; ++j) {
            steady_level<S, 0>(Fo, Bo, w, std::make_integer_sequence<int, S>{});
            steady_level<S, 1>(Fo, Bo, w, std::make_integer_sequence<int, S>{});
        }
        // ramp-down: levels 2M + tau, tau = 0 .. 2S-2
        ramp<S, false, 0>(Fo, Bo, w, std::make_integer_sequence<int, 2 * S - 1>{});
    } else {
        // M < S (kPathGeneric): fully unrolled instance for this M
        if constexpr (S > 1) return makespan_short_dispatch<S>(w, M, std::make_integer_sequence<int, S - 1>{});
    }
    int32_t T = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) T = max(T, Bo[s] + w.d[s]);
    return T;
}

// ---------------------------------------------------------------------------
// Eager 1F1B (App. B): stage s (1-based) runs W_s = min(2(S-s)+1, M)
// forwards, then (B_i, F_{W_s+i}) pairs, then the remaining backwards.  In
// the unit-weight level order (stages descending within a level)
//     F_{s,m}: s + m - 1 (m <= W_s), 2m - 2S + 3s - 2 (m > W_s);
//     B_{s,m}: 2S - s + 2m - 1,
// each stage runs at most one op per level, but a stage can be two forwards
// ahead of the next one: the forward predecessor of F_{s,m} is the latest
// or the previous forward of stage s-1 (its lag, 1 or 2, is known at
// compile time).  So each stage keeps Fo (last forward), Fp (the one before)
// and Bo.  For M >= 2S-1 the levels split into a ramp-up (levels 1..2S-1),
// M-2S+1 steady two-level steps in which every stage alternates B and F
// (lag 2), and a ramp-down (levels 2M+tau, tau = -2S+2..2S-2).
// ---------------------------------------------------------------------------
__host__ __device__ constexpr int eager_up_op(int S, int s1, int t) {
    return (t >= s1 && t <= 2 * S - s1) ? 1
           : (t >= 2 * S - s1 + 1 && ((t + s1) & 1) == 1) ? 2
           : (t >= 2 * S - s1 + 2 && ((t + s1) & 1) == 0) ? 1
                                                            : 0;
}
__host__ __device__ constexpr int eager_down_op(int S, int s1, int tau) {
    return ((((tau + s1) % 2) + 2) % 2 == 0 && tau <= 3 * s1 - 2 * S - 2) ? 1
           : ((((tau + s1) % 2) + 2) % 2 == 1 && tau <= 2 * S - s1 - 1) ? 2
                                                                          : 0;
}
__host__ __device__ constexpr bool eager_up_last_is_b(int S, int s1, int t) {
    for (int u = t - 1; u >= 1; --u)
        if (eager_up_op(S, s1, u)) return eager_up_op(S, s1, u) == 2;
    return false;
}
// before the ramp-down, the last steady level 2M-2S+1 ran F on odd stages
__host__ __device__ constexpr bool eager_down_last_is_b(int S, int s1, int tau) {
    for (int u = tau - 1; u >= -2 * S + 2; --u)
        if (eager_down_op(S, s1, u)) return eager_down_op(S, s1, u) == 2;
    return (s1 & 1) == 0;
}
// forwards of stage s1 in ramp-up levels < t / ramp-down levels < 2M+tau
__host__ __device__ constexpr int eager_up_nf(int S, int s1, int t) {
    int n = 0;
    for (int u = 1; u < t; ++u) n += eager_up_op(S, s1, u) == 1;
    return n;
}
__host__ __device__ constexpr int eager_down_nf(int S, int s1, int tau) {
    int n = 0;
    for (int u = -2 * S + 2; u < tau; ++u) n += eager_down_op(S, s1, u) == 1;
    return n;
}
// forwards stage s1-1 has done beyond stage s1 before this op (1 or 2)
__host__ __device__ constexpr int eager_up_lag(int S, int s1, int t) {
    return eager_up_nf(S, s1 - 1, t) - eager_up_nf(S, s1, t);
}
__host__ __device__ constexpr int eager_down_lag(int S, int s1, int tau) {
    return (eager_down_nf(S, s1, 2 * S - 1) - eager_down_nf(S, s1 - 1, 2 * S - 1)) +
           eager_down_nf(S, s1 - 1, tau) - eager_down_nf(S, s1, tau);
}

template <int S, int s, int LAG>
__device__ __forceinline__ void relax_f_lag(int32_t (&Fo)[S], int32_t (&Fp)[S],
                                            const StageW<S> &w, int32_t clock) {
    Fp[s] = Fo[s];
    if constexpr (s > 0) {
        static_assert(LAG == 1 || LAG == 2, "forward lag");
        Fo[s] = add_max(LAG == 2 ? Fp[s - 1] : Fo[s - 1], w.pf[s - 1], clock) + w.F[s];
    } else {
        Fo[s] = clock + w.F[s];
    }
}

template <int S, bool UP, int t, int s1>
__device__ __forceinline__ void eager_ramp_op(int32_t (&Fo)[S], int32_t (&Fp)[S], int32_t (&Bo)[S],
                                              const StageW<S> &w) {
    constexpr int op = UP ? eager_up_op(S, s1, t) : eager_down_op(S, s1, t);
    constexpr bool last_b = UP ? eager_up_last_is_b(S, s1, t) : eager_down_last_is_b(S, s1, t);
    constexpr int s = s1 - 1;
    if constexpr (op == 1) {
        constexpr int lag = s1 == 1 ? 1 : (UP ? eager_up_lag(S, s1, t) : eager_down_lag(S, s1, t));
        relax_f_lag<S, s, lag>(Fo, Fp, w, last_b ? Bo[s] : Fo[s]);
    } else if constexpr (op == 2) {
        relax_b<S, s>(Bo, w, last_b ? Bo[s] : Fo[s]);
    }
}
template <int S, bool UP, int t, int... i>
__device__ __forceinline__ void eager_ramp_level(int32_t (&Fo)[S], int32_t (&Fp)[S],
                                                 int32_t (&Bo)[S], const StageW<S> &w,
                                                 std::integer_sequence<int, i...>) {
    (eager_ramp_op<S, UP, t, S - i>(Fo, Fp, Bo, w), ...);
}
template <int S, bool UP, int T0, int... t>
__device__ __forceinline__ void eager_ramp(int32_t (&Fo)[S], int32_t (&Fp)[S], int32_t (&Bo)[S],
                                           const StageW<S> &w, std::integer_sequence<int, t...>) {
    (eager_ramp_level<S, UP, T0 + t>(Fo, Fp, Bo, w, std::make_integer_sequence<int, S>{}), ...);
}
// steady level of parity P: stage s1 with the parity of P runs F (after its
// B, forward lag 2), the others B (after their F)
template <int S, int P, int i>
__device__ __forceinline__ void eager_steady_op(int32_t (&Fo)[S], int32_t (&Fp)[S],
                                                int32_t (&Bo)[S], const StageW<S> &w) {
    constexpr int s1 = S - i, s = s1 - 1;
    if constexpr ((s1 & 1) == P) relax_f_lag<S, s, 2>(Fo, Fp, w, Bo[s]);
    else relax_b<S, s>(Bo, w, Fo[s]);
}
template <int S, int P, int... i>
__device__ __forceinline__ void eager_steady_level(int32_t (&Fo)[S], int32_t (&Fp)[S],
                                                   int32_t (&Bo)[S], const StageW<S> &w,
                                                   std::integer_sequence<int, i...>) {
    (eager_steady_op<S, P, i>(Fo, Fp, Bo, w), ...);
}

// Eager 1F1B, M >= 2S-1
template <int S>
__device__ __forceinline__ int32_t makespan_eager(const StageW<S> &w, int M) {
    int32_t Fo[S], Fp[S], Bo[S];
#pragma unroll
    for (int s = 0; s < S; ++s) {
        Fo[s] = 0;
        Fp[s] = 0;
        Bo[s] = 0;
    }
    eager_ramp<S, true, 1>(Fo, Fp, Bo, w, std::make_integer_sequence<int, 2 * S - 1>{});
    for (int j = 0; j < M - 2 * S + 1; ++j) {
        eager_steady_level<S, 0>(Fo, Fp, Bo, w, std::make_integer_sequence<int, S>{});
        eager_steady_level<S, 1>(Fo, Fp, Bo, w, std::make_integer_sequence<int, S>{});
    }
    eager_ramp<S, false, -2 * S + 2>(Fo, Fp, Bo, w, std::make_integer_sequence<int, 4 * S - 3>{});
    int32_t T = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) T = max(T, Bo[s] + w.d[s]);
    return T;
}

// Eager 1F1B with M < 2S-1: the unit-weight ASAP level order has no closed
// form, so it is computed at compile time for each (S, M) and unrolled like
// the ramps.  Stage s (0-based) runs W = min(2(S-1-s)+1, M) forwards, then
// (B_i, F_{W+i}) pairs, then the remaining backwards; an op's level is one
// more than the later of its stage's previous op and its inter-stage
// predecessor (F_{s-1,m} for F_{s,m}, B_{s+1,m} for B_{s,m}).  Within a
// level the stages are visited in descending order, as in the ramps, and
// while the program is built every op is checked to read the finish it
// depends on: F_{s-1,m} from stage s-1's latest forward (lag 1) or the one
// before (lag 2), B_{s+1,m} from stage s+1's latest backward.
struct EagerShortOp {
    int kind;      // 0 none, 1 forward, 2 backward
    int lag;       // forward of a stage s > 0: 1 or 2
    bool clock_b;  // the stage's previous op is a backward (else a forward)
};
template <int S, int M>
struct EagerShortProgram {
    static constexpr int kMaxLevels = 2 * (M + S) + 2;
    EagerShortOp op[kMaxLevels][S];
    int n_levels;
    bool ok;
    __host__ __device__ constexpr EagerShortProgram() : op{}, n_levels(0), ok(true) {
        int kind[S][2 * M] = {}, mb[S][2 * M] = {};  // chains: op kind and micro-batch
        for (int s = 0; s < S; ++s) {
            const int W = 2 * (S - 1 - s) + 1 < M ? 2 * (S - 1 - s) + 1 : M;
            int n = 0;
            for (int m = 0; m < W; ++m) kind[s][n] = 1, mb[s][n++] = m;
            for (int i = 0; i < M - W; ++i) {
                kind[s][n] = 2, mb[s][n++] = i;
                kind[s][n] = 1, mb[s][n++] = W + i;
            }
            for (int m = M - W; m < M; ++m) kind[s][n] = 2, mb[s][n++] = m;
        }
        int lf[S][M] = {}, lb[S][M] = {};  // ASAP levels (1-based)
        for (bool changed = true; changed;) {
            changed = false;
            for (int s = 0; s < S; ++s) {
                int prev = 0;
                for (int n = 0; n < 2 * M; ++n) {
                    const int m = mb[s][n];
                    int p = prev;
                    if (kind[s][n] == 2 && s + 1 < S && lb[s + 1][m] > p) p = lb[s + 1][m];
                    if (kind[s][n] == 1 && s > 0 && lf[s - 1][m] > p) p = lf[s - 1][m];
                    int &v = kind[s][n] == 2 ? lb[s][m] : lf[s][m];
                    if (v != p + 1) {
                        v = p + 1;
                        changed = true;
                    }
                    prev = p + 1;
                }
            }
        }
        for (int s = 0; s < S; ++s)
            for (int m = 0; m < M; ++m) {
                if (lf[s][m] > n_levels) n_levels = lf[s][m];
                if (lb[s][m] > n_levels) n_levels = lb[s][m];
            }
        if (n_levels > kMaxLevels) {
            ok = false;
            n_levels = kMaxLevels;
        }
        // registers: the micro-batch whose finish Fo / Fp / Bo of a stage
        // holds (-1: none yet) and whether its last op was a backward
        int fo[S] = {}, fp[S] = {}, bo[S] = {};
        bool last_b[S] = {};
        for (int s = 0; s < S; ++s) fo[s] = fp[s] = bo[s] = -1;
        for (int l = 1; l <= n_levels; ++l)
            for (int s = S - 1; s >= 0; --s) {
                int k = 0, m = -1;
                for (int u = 0; u < M; ++u) {
                    if (lf[s][u] == l) k = k ? 3 : 1, m = u;
                    if (lb[s][u] == l) k = k ? 3 : 2, m = u;
                }
                if (k == 3) ok = false;  // two ops of one stage in a level
                if (k == 1) {
                    int lag = 1;
                    if (s > 0) {
                        if (fo[s - 1] == m) lag = 1;
                        else if (fp[s - 1] == m) lag = 2;
                        else ok = false;
                    }
                    op[l - 1][s] = EagerShortOp{1, lag, last_b[s]};
                    fp[s] = fo[s];
                    fo[s] = m;
                    last_b[s] = false;
                } else if (k == 2) {
                    if (s + 1 < S && bo[s + 1] != m) ok = false;
                    op[l - 1][s] = EagerShortOp{2, 0, last_b[s]};
                    bo[s] = m;
                    last_b[s] = true;
                }
            }
    }
};
template <int S, int M>
struct EagerShortTab {
    static constexpr EagerShortProgram<S, M> value{};
    static_assert(value.ok, "Eager 1F1B short level order: an op would read the wrong finish");
};

template <int S, int M, int l, int i>
__device__ __forceinline__ void eager_short_op(int32_t (&Fo)[S], int32_t (&Fp)[S],
                                               int32_t (&Bo)[S], const StageW<S> &w) {
    constexpr int s = S - 1 - i;
    constexpr EagerShortOp o = EagerShortTab<S, M>::value.op[l][s];
    if constexpr (o.kind == 1)
        relax_f_lag<S, s, (s > 0 ? o.lag : 1)>(Fo, Fp, w, o.clock_b ? Bo[s] : Fo[s]);
    else if constexpr (o.kind == 2)
        relax_b<S, s>(Bo, w, o.clock_b ? Bo[s] : Fo[s]);
}
template <int S, int M, int l, int... i>
__device__ __forceinline__ void eager_short_level(int32_t (&Fo)[S], int32_t (&Fp)[S],
                                                  int32_t (&Bo)[S], const StageW<S> &w,
                                                  std::integer_sequence<int, i...>) {
    (eager_short_op<S, M, l, i>(Fo, Fp, Bo, w), ...);
}
template <int S, int M, int... l>
__device__ __forceinline__ void eager_short_all(int32_t (&Fo)[S], int32_t (&Fp)[S],
                                                int32_t (&Bo)[S], const StageW<S> &w,
                                                std::integer_sequence<int, l...>) {
    (eager_short_level<S, M, l>(Fo, Fp, Bo, w, std::make_integer_sequence<int, S>{}), ...);
}
template <int S, int M>
__device__ __forceinline__ int32_t makespan_eager_short(const StageW<S> &w) {
    int32_t Fo[S], Fp[S], Bo[S];
#pragma unroll
    for (int s = 0; s < S; ++s) {
        Fo[s] = 0;
        Fp[s] = 0;
        Bo[s] = 0;
    }
    eager_short_all<S, M>(Fo, Fp, Bo, w,
                          std::make_integer_sequence<int, EagerShortTab<S, M>::value.n_levels>{});
    int32_t T = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) T = max(T, Bo[s] + w.d[s]);
    return T;
}
// runtime M in 1..2S-2 -> its unrolled instance
template <int S, int... m>
__device__ __forceinline__ int32_t makespan_eager_short_dispatch(const StageW<S> &w, int M,
                                                                 std::integer_sequence<int, m...>) {
    int32_t T = -1;
    ((M == m + 1 ? (T = makespan_eager_short<S, m + 1>(w), 0) : 0), ...);
    return T;
}

// Level program of one (schedule, S, M): per level one 64-bit word, bit s of
// bits 0-15 = stage s runs a forward, bits 16-31 = a backward, bits 32-47 =
// that forward's predecessor is the previous forward of stage s-1 (lag 2).
// Built on the host from the unit-weight ASAP levels of the schedule's
// chains (schedules.cu); used for Eager 1F1B with M < 2S-1.
template <int S>
__device__ __forceinline__ int32_t makespan_program(const StageW<S> &w, const uint64_t *prog,
                                                    int n_levels) {
    // A stage's last op finished at max(Fo, Bo) (finishes grow along its
    // chain), so no separate clock is kept.  The ops of one level are
    // independent (at most one per stage, and an op's inter-stage
    // predecessor lies on an earlier level), so a level's forwards run
    // first and its backwards second, each phase skipped when empty.
    int32_t Fo[S], Fp[S], Bo[S];
#pragma unroll
    for (int s = 0; s < S; ++s) {
        Fo[s] = 0;
        Fp[s] = 0;
        Bo[s] = 0;
    }
    // the next level's word is loaded one level ahead, so the load latency
    // overlaps the current level's relaxations
    uint64_t next = n_levels > 0 ? __ldg(prog) : 0ull;
#pragma unroll 1
    for (int l = 0; l < n_levels; ++l) {
        const uint64_t word = next;
        if (l + 1 < n_levels) next = __ldg(prog + l + 1);
        const uint32_t fm = (uint32_t)word & 0xffffu, bm = (uint32_t)(word >> 16) & 0xffffu;
        const uint32_t lm = (uint32_t)(word >> 32) & 0xffffu;
        if (fm) {
#pragma unroll
            for (int s = S - 1; s >= 0; --s) {
                if ((fm >> s) & 1u) {
                    int32_t start = max(Fo[s], Bo[s]);
                    if (s > 0)
                        start = max(start, (((lm >> s) & 1u) ? Fp[s > 0 ? s - 1 : 0]
                                                             : Fo[s > 0 ? s - 1 : 0]) +
                                               w.pf[s > 0 ? s - 1 : 0]);
                    Fp[s] = Fo[s];
                    Fo[s] = start + w.F[s];
                }
            }
        }
        if (bm) {
#pragma unroll
            for (int s = S - 1; s >= 0; --s) {
                if ((bm >> s) & 1u) {
                    int32_t start = max(Fo[s], Bo[s]);
                    if (s + 1 < S) start = max(start, Bo[s + 1 < S ? s + 1 : s] + w.pb[s]);
                    Bo[s] = start + w.B[s];
                }
            }
        }
    }
    int32_t T = 0;
#pragma unroll
    for (int s = 0; s < S; ++s) T = max(T, Bo[s] + w.d[s]);
    return T;
}

// Level programs on the device: index[(S-1)*32 + M] = (first word, levels)
// for the (S, M) pairs a schedule's short path covers.
struct Programs {
    const uint64_t *words;
    const uint2 *index;
};
// Programs of a schedule on the current device (built and uploaded on first
// use, kept for the process); words = index = NULL for 1F1B.
pos_status schedule_programs(int sched, Programs *out);

// Makespan of one decoded plan on path PATH.
template <int S, int PATH>
__device__ __forceinline__ int32_t makespan_path(const StageW<S> &w, int M, const Programs &pg) {
    if constexpr (PATH == kPathEager) {
        return makespan_eager<S>(w, M);
    } else if constexpr (PATH == kPathEagerShort) {
        const uint2 ix = __ldg(pg.index + (S - 1) * 32 + M);
        return makespan_program<S>(w, pg.words + ix.x, (int)ix.y);
    } else if constexpr (PATH == kPathEagerUnrolled) {
        if constexpr (S > 1)
            return makespan_eager_short_dispatch<S>(w, M, std::make_integer_sequence<int, 2 * S - 2>{});
        else
            return -1;  // S = 1 has no short case
    } else {
        return makespan_1f1b<S, PATH>(w, M);
    }
}

// Path of (schedule, S, M) and the first M of the fast path.
__host__ __device__ __forceinline__ int fast_min_m(int sched, int S) {
    return sched == POS_SCHED_EAGER_1F1B ? 2 * S - 1 : S;
}
__host__ __device__ __forceinline__ int path_of(int sched, int S, int M) {
    const bool fast = M >= fast_min_m(sched, S);
    return sched == POS_SCHED_EAGER_1F1B ? (fast ? kPathEager : kPathEagerShort)
                                         : (fast ? kPathFast : kPathGeneric);
}

// ---------------------------------------------------------------------------
// Layer-level pruning (Theorem 2): for each device type the layer counts of
// its stages, in stage order, rise and then fall ("ridge-like").  A partial
// plan keeps one byte per type: bits 0-6 = layers of the type's last placed
// stage (0 = none yet), bit 7 = its counts have fallen; a type whose counts
// have fallen caps its next stage at its last count.
// ---------------------------------------------------------------------------
__host__ __device__ __forceinline__ int ridge_cap(uint32_t state, int type) {
    const uint32_t b = (state >> (8 * type)) & 0xffu;
    return (b & 0x80u) ? (int)(b & 0x7fu) : 127;
}
__host__ __device__ __forceinline__ uint32_t ridge_next(uint32_t state, int type, int l) {
    const uint32_t b = (state >> (8 * type)) & 0xffu, last = b & 0x7fu;
    const uint32_t fallen = (b & 0x80u) | ((last != 0u && (uint32_t)l < last) ? 0x80u : 0u);
    return (state & ~(0xffu << (8 * type))) | ((fallen | (uint32_t)l) << (8 * type));
}
// Is a complete plan ridge-like?  cut[0..S], cls[s] = type * n_tp + tp.
template <int S>
__device__ __forceinline__ bool ridge_plan_ok(const int (&cut)[S + 1], const int (&cls)[S],
                                              int n_tp) {
    uint32_t st = 0;
    bool ok = true;
#pragma unroll
    for (int s = 0; s < S; ++s) {
        const int ty = cls[s] / n_tp, l = cut[s + 1] - cut[s];
        ok &= l <= ridge_cap(st, ty);
        st = ridge_next(st, ty, l);
    }
    return ok;
}

// Overflow guard U(S, M) >= 2^31 ?
__host__ __device__ __forceinline__ bool guard_trips(int64_t A, int64_t D, int64_t P, int S,
                                                     int M) {
    const int64_t U = (int64_t)M * A + D + 2 * (int64_t)M * (S - 1) * P;
    return U >= ((int64_t)1 << 31);
}

}  // namespace pos
