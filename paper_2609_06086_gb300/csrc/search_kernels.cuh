// Device side of poseidon_search (hot-path steps a2-a8): shared types, the
// incumbent, and the leaf-evaluation kernel templated on the stage count.
#pragma once
#include "common.cuh"

namespace pos {

// Packed incumbent: compared as (obj, idx) -- the scaled objective
// T * Q/(D*M) first, then the global index -- and updated with a 128-bit
// compare-and-swap, so concurrent updates always keep the true minimum.
struct __align__(16) Key128 {
    unsigned long long idx;
    unsigned long long obj;
};

// One slice = (M, TP index, stage-type placement).
struct SliceRec {
    uint64_t ordinal;  // (m_idx*n_tp + tp_idx)*n_place + place_rank
    uint64_t scale;    // Q / (D*M): T * scale orders plans by T/(D*M)
    uint8_t cls[16];   // class of each stage
    int32_t M;
    uint32_t gid;      // row of this slice in the feasibility table
    uint32_t vslot;    // row of this slice in the completion-bound tables (prune mode 2)
    uint32_t pad;
};
static_assert(sizeof(SliceRec) == 48, "SliceRec layout");

// Partial plan at depth x: stages 0..x-1 placed; cut[i] = layers of stages
// 0..i.  slice indexes the current batch's slice table; 0xffff = hole.
// A and Bm are the two partial sums of Eq. 2 over the placed stages,
//   A = sum_{i<x} F_i,   Bm = max_{i<x} (sum_{j=i}^{x-1} B_j + d_i)
// (Bm = -1 at depth 0; every d is >= 0), so that for a new stage x with
// totals (F, B, d):  g(S_{x+1}) = A + M (F + B) + max(Bm, d).
struct Prefix {
    uint16_t slice;
    uint8_t cut[14];
    int32_t A, Bm;
    uint32_t pad[2];
};
static_assert(sizeof(Prefix) == 32, "Prefix layout");

// Complete plan: cut[0..S-2]; slice indexes the slice table of the launch.
struct Leaf {
    uint32_t slice;
    uint8_t cut[16];
    uint32_t pad[3];
};
static_assert(sizeof(Leaf) == 32, "Leaf layout");

// 32-byte entries move as two 16-byte vectors; byte I of an entry is
// addressed at compile time (word I/4, shift 8*(I%4)).
struct Vec32 {
    uint4 a, b;
};

__device__ __forceinline__ Vec32 load32(const void *ptr) {
    const uint4 *q = static_cast<const uint4 *>(ptr);
    Vec32 v;
    v.a = __ldg(q);
    v.b = __ldg(q + 1);
    return v;
}
__device__ __forceinline__ void store32(void *ptr, const Vec32 &v) {
    uint4 *q = static_cast<uint4 *>(ptr);
    q[0] = v.a;
    q[1] = v.b;
}
__device__ __forceinline__ uint32_t &word_of(Vec32 &v, int w) {
    return w == 0 ? v.a.x : w == 1 ? v.a.y : w == 2 ? v.a.z : w == 3 ? v.a.w
         : w == 4 ? v.b.x : w == 5 ? v.b.y : w == 6 ? v.b.z : v.b.w;
}
template <int I>
__device__ __forceinline__ uint32_t get_byte(const Vec32 &v) {
    const uint32_t w = (I / 4) == 0 ? v.a.x : (I / 4) == 1 ? v.a.y : (I / 4) == 2 ? v.a.z
                     : (I / 4) == 3 ? v.a.w : (I / 4) == 4 ? v.b.x : (I / 4) == 5 ? v.b.y
                     : (I / 4) == 6 ? v.b.z : v.b.w;
    return (w >> (8 * (I % 4))) & 0xffu;
}
template <int I>
__device__ __forceinline__ void set_byte(Vec32 &v, uint32_t b) {
    uint32_t &w = word_of(v, I / 4);
    w = (w & ~(0xffu << (8 * (I % 4)))) | ((b & 0xffu) << (8 * (I % 4)));
}

constexpr uint32_t kLeafHole = 0xffffffffu;
constexpr uint16_t kPrefixHole = 0xffff;

// device counters / statistics (uint64 each)
enum {
    kStPrefixes = 0,
    kStPrunedBound,
    kStPrunedMemory,
    kStEvaluated,
    kStTimeout,
    kStRelaxations,
    kStParentsExpand,
    kStParentsComplete,
    kStLeaves,
    kStPrunedRidge,   // children cut by the layer-level (ridge) rule
    kStBulkTimeout,   // blocks whose table staging (TMA bulk copy) wait ran out
    kStDepthParents,                                // + x: parents read at depth x
    kStDepthChildren = kStDepthParents + POS_MAX_STAGES,  // + x: children (plans) written
    kStCount = kStDepthChildren + POS_MAX_STAGES
};

constexpr int kCasLimit = 1 << 20;  // default rounds of the incumbent's CAS loop

__device__ __forceinline__ bool key_less(unsigned long long ao, unsigned long long ai,
                                         unsigned long long bo, unsigned long long bi) {
    return ao < bo || (ao == bo && ai < bi);
}

// Lower the incumbent to (obj, idx) if that is smaller.  Bounded loop: every
// failed CAS means another thread lowered the key; after `limit` rounds
// (kCasLimit unless the problem sets another) the timeout counter is raised
// and the update is abandoned.
__device__ __forceinline__ void incumbent_update(Key128 *inc, unsigned long long obj,
                                                 unsigned long long idx,
                                                 unsigned long long *stats, int limit) {
    Key128 cur;
    cur.obj = __ldcg(&inc->obj);
    cur.idx = __ldcg(&inc->idx);
    for (int it = 0; it < limit; ++it) {
        if (!key_less(obj, idx, cur.obj, cur.idx)) return;
        Key128 want;
        want.obj = obj;
        want.idx = idx;
        const Key128 prev = atomicCAS(inc, cur, want);
        if (prev.obj == cur.obj && prev.idx == cur.idx) return;
        cur = prev;
    }
    atomicAdd(stats + kStTimeout, 1ull);
}

struct LeafParams {
    const Leaf *leaves;
    const unsigned long long *count;  // device count of written leaf slots
    unsigned long long cap;
    const SliceRec *slices;
    int M;
    uint64_t n_map;
    Key128 *inc;
    unsigned long long *stats;
    unsigned long long *slice_best;  // optional per-slice minimum objective
    const void *blob;
    BlobLayout lay;
    Programs pg;  // level programs of the schedule's short path
    int ridge;    // 1: only ridge-like plans may lower the incumbent (warm-up plans)
    int cas_limit;  // rounds of the incumbent's CAS loop
};

// leaf byte 4+s holds cut[s+1] (layers of stages 0..s)
template <int S, int... s>
__device__ __forceinline__ void leaf_cuts_i(const Vec32 &v, int (&cut)[S + 1],
                                            std::integer_sequence<int, s...>) {
    ((cut[s + 1] = (int)get_byte<4 + s>(v)), ...);
}
template <int S>
__device__ __forceinline__ void leaf_cuts(const Vec32 &v, int (&cut)[S + 1]) {
    leaf_cuts_i<S>(v, cut, std::make_integer_sequence<int, S - 1>{});
}

// blocks per SM: the Eager paths keep three registers per stage, not two
__host__ __device__ constexpr int leaf_min_blocks(int S, int path) {
    return (path == kPathEager || path == kPathEagerShort)
               ? (S <= 4 ? 4 : S <= 6 ? 3 : S <= 12 ? 2 : 1)
               : (S <= 4 ? 4 : S <= 8 ? 3 : 2);
}

template <int S, int PATH>
__global__ void __launch_bounds__(256, leaf_min_blocks(S, PATH)) leaf_kernel(LeafParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ uint64_t bar;
    // the tables were written before the previous kernel: staged while it
    // finishes; the plans and their count only after it has completed
    if (!stage_blob_bulk(sm, p.blob, p.lay.bytes, &bar)) {
        if (threadIdx.x == 0) atomicAdd(p.stats + kStBulkTimeout, 1ull);
        grid_dep_wait();  // a block never leaves before its predecessor has completed
        return;
    }
    grid_dep_wait();
    grid_dep_trigger();
    const unsigned long long c0 = __ldcg(p.count);
    const unsigned long long n = c0 < p.cap ? c0 : p.cap;
    if ((unsigned long long)blockIdx.x * blockDim.x >= n) return;  // no plan for this block
    const Tab t = tab_at(sm, p.lay);
    const int L = p.lay.L;
    unsigned long long evaluated = 0;
    const unsigned long long stride = (unsigned long long)gridDim.x * blockDim.x;
    // all lanes of a warp iterate together (the warp minimum uses shuffles)
    const unsigned long long n_round = (n + 31) & ~31ull;
    const Vec32 none = {make_uint4(kLeafHole, 0, 0, 0), make_uint4(0, 0, 0, 0)};
    unsigned long long i = blockIdx.x * (unsigned long long)blockDim.x + threadIdx.x;
    // the next plan's record is loaded one iteration ahead, so its memory
    // latency overlaps the current plan's wavefront
    Vec32 next = i < n ? load32(p.leaves + i) : none;
    for (; i < n_round; i += stride) {
        unsigned long long obj = ~0ull, idx = ~0ull;
        const Vec32 lv = next;
        next = i + stride < n ? load32(p.leaves + i + stride) : none;
        const uint32_t sl = lv.a.x;
        bool cand = false;
        if (sl != kLeafHole) {
            const SliceRec &sr = p.slices[sl];
            int cut[S + 1], cls[S];
            cut[0] = 0;
            leaf_cuts<S>(lv, cut);
            cut[S] = L;
#pragma unroll
            for (int s = 0; s < S; ++s) cls[s] = __ldg(&sr.cls[s]);
            const uint64_t scale = __ldg(&sr.scale);
            // enumerated plans are ridge-like already; warm-up plans may not be
            cand = !p.ridge || ridge_plan_ok<S>(cut, cls, t.n_tp());
            StageW<S> w;
            stage_weights<S>(t, cut, cls, w);
            const int32_t T = makespan_path<S, PATH>(w, p.M, p.pg);
            obj = (unsigned long long)T * scale;
            ++evaluated;
            if (p.slice_best) atomicMin(p.slice_best + sl, obj);  // ordering hint only
        }
        // A plan whose objective is above the incumbent's cannot lower it
        // (the incumbent only decreases, so a stale read lets more through,
        // never fewer): most warps stop here, and only the candidates pay
        // for their global index (the composition's rank) and the warp
        // minimum.
        cand = cand && obj <= __ldcg(&p.inc->obj);
        if (!__any_sync(0xffffffffu, cand)) continue;
        if (cand) {
            int cut[S + 1];
            cut[0] = 0;
            leaf_cuts<S>(lv, cut);
            cut[S] = L;
            idx = __ldg(&p.slices[sl].ordinal) * p.n_map + rank_cuts<S>(t, cut);
        } else {
            obj = ~0ull;
        }
        // warp minimum, then one CAS attempt per warp
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const unsigned long long oo = __shfl_xor_sync(0xffffffffu, obj, o);
            const unsigned long long oi = __shfl_xor_sync(0xffffffffu, idx, o);
            if (key_less(oo, oi, obj, idx)) {
                obj = oo;
                idx = oi;
            }
        }
        if ((threadIdx.x & 31) == 0 && obj != ~0ull) incumbent_update(p.inc, obj, idx, p.stats, p.cas_limit);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) evaluated += __shfl_xor_sync(0xffffffffu, evaluated, o);
    if ((threadIdx.x & 31) == 0 && evaluated) {
        atomicAdd(p.stats + kStEvaluated, evaluated);
        atomicAdd(p.stats + kStRelaxations, evaluated * 2ull * S * (unsigned long long)p.M);
    }
}

template <int S, int PATH>
pos_status launch_leaf_t(const LeafParams &p, int grid, cudaStream_t s) {
    auto kern = leaf_kernel<S, PATH>;
    const int smem = p.lay.bytes;
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(kern), smem));
    POS_CUDA(launch_dependent(kern, grid, 256, smem, s, p));
    return POS_OK;
}

// Launch of leaf_kernel<S, path> for a runtime path of one schedule family
// (instantiated by the search_leaf_*.cu units; S = 1 has only fast paths).
template <int S, bool EAGER>
pos_status launch_leaf_s(int path, const LeafParams &p, int grid, cudaStream_t s) {
    if constexpr (EAGER) {
        if (path == kPathEager) return launch_leaf_t<S, kPathEager>(p, grid, s);
        if constexpr (S > 1)
            if (path == kPathEagerShort) return launch_leaf_t<S, kPathEagerShort>(p, grid, s);
    } else {
        if (path == kPathFast) return launch_leaf_t<S, kPathFast>(p, grid, s);
        if constexpr (S > 1)
            if (path == kPathGeneric) return launch_leaf_t<S, kPathGeneric>(p, grid, s);
    }
    return fail(POS_EINVAL, "no such path for this stage count");
}

// per-unit dispatchers (search_leaf_*.cu): 1F1B or Eager paths, S in the
// unit's range
pos_status launch_leaf_1f1b_1_6(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_1f1b_7_10(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_1f1b_11_12(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_1f1b_13_14(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_1f1b_15_15(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_1f1b_16_16(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_eager_1_8(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_eager_9_12(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_eager_13_14(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_eager_15_15(int S, int path, const LeafParams &p, int grid, cudaStream_t s);
pos_status launch_leaf_eager_16_16(int S, int path, const LeafParams &p, int grid, cudaStream_t s);

inline pos_status launch_leaf(int S, int path, const LeafParams &p, int grid, cudaStream_t s) {
    if (path == kPathEager || path == kPathEagerShort) {
        if (S <= 8) return launch_leaf_eager_1_8(S, path, p, grid, s);
        if (S <= 12) return launch_leaf_eager_9_12(S, path, p, grid, s);
        if (S <= 14) return launch_leaf_eager_13_14(S, path, p, grid, s);
        if (S == 15) return launch_leaf_eager_15_15(S, path, p, grid, s);
        return launch_leaf_eager_16_16(S, path, p, grid, s);
    }
    if (S <= 6) return launch_leaf_1f1b_1_6(S, path, p, grid, s);
    if (S <= 10) return launch_leaf_1f1b_7_10(S, path, p, grid, s);
    if (S <= 12) return launch_leaf_1f1b_11_12(S, path, p, grid, s);
    if (S <= 14) return launch_leaf_1f1b_13_14(S, path, p, grid, s);
    if (S == 15) return launch_leaf_1f1b_15_15(S, path, p, grid, s);
    return launch_leaf_1f1b_16_16(S, path, p, grid, s);
}

}  // namespace pos
