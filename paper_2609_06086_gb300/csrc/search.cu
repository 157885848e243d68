// poseidon_search: exact parallelism search of Sec. 4.2.3 on the GPU.
//
//  1. slices (m_idx, tp_idx, placement) in global-index order; per slice a
//     suffix-feasibility table feas[x] = bitset of c such that layers [c, L)
//     can be split over stages x..S-1 within memory (exact memory cut);
//  2. warm-up (Sec. 4.2.3): random memory-feasible plans seed the incumbent
//     T_min and give every sampled slice a first objective;
//  3. slices are taken in batches, most promising first; per batch the
//     layer compositions are enumerated level by level (stage 1, 2, ...):
//     every prefix S_x that survives the memory cut and the prune
//     g(S_x) > T_min (Eq. 2, Theorem 1) is written to the next frontier,
//     the last two stages are completed in one kernel, and complete plans
//     are evaluated by the templated leaf kernel, which lowers the incumbent.
//     Frontiers have a fixed capacity; warps whose children do not fit are
//     deferred and re-expanded after the part that fit has been finished.
#include <algorithm>
#include <chrono>
#include <mutex>
#include <new>
#include <cstring>
#include <numeric>
#include <vector>

#include "search_host.h"

namespace pos {

constexpr int kThreads = 256;
constexpr int32_t kNoCompletion = 0x7fffffff;  // completion-bound entry without a completion
constexpr int kVbSlotsSmem = 64;  // batches up to this many slots stage their bound rows
                                  // in shared memory; larger ones read them from L2

// 128-bit set of cut positions 0..127.
struct Bits128 {
    uint32_t w[4];
};

__device__ __forceinline__ Bits128 range_bits(int lo, int hi) {  // positions lo..hi
    Bits128 r;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int a = max(lo - 32 * i, 0), b = min(hi - 32 * i, 31);
        r.w[i] = (a > b) ? 0u : ((b == 31 ? 0xffffffffu : ((1u << (b + 1)) - 1u)) & ~((1u << a) - 1u));
    }
    return r;
}

__device__ __forceinline__ int popc128(const Bits128 &b) {
    return __popc(b.w[0]) + __popc(b.w[1]) + __popc(b.w[2]) + __popc(b.w[3]);
}

// ---------------------------------------------------------------------------
// suffix feasibility: one block per slice, thread c
// ---------------------------------------------------------------------------
// Also fills lim[(gid*S + x)*128 + c] = the largest l such that stage x
// holds layers [c, c+l) within memory (0 if none), capped at L - c, and
// root[gid] = 1 when the slice has a memory-feasible plan.
__global__ void feas_kernel(const SliceRec *slices, int n_slices, int S, uint4 *feas,
                            uint8_t *lim, uint8_t *root, const void *blob, BlobLayout lay,
                            unsigned long long *stats) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ uint32_t prev[4], cur[4];
    __shared__ uint64_t bar;
    if (!stage_blob_bulk(sm, blob, lay.bytes, &bar)) {
        if (threadIdx.x == 0) atomicAdd(stats + kStBulkTimeout, 1ull);
        return;
    }
    const Tab t = tab_at(sm, lay);
    const int L = lay.L, c = threadIdx.x;
    for (int sl = blockIdx.x; sl < n_slices; sl += gridDim.x) {
        const SliceRec &sr = slices[sl];
        const int M = sr.M;
        uint4 *row = feas + (size_t)sr.gid * (S + 1);
        // x = S: only the empty suffix starting at c = L
        if (c < 4) prev[c] = (L >> 5) == c ? (1u << (L & 31)) : 0u;
        __syncthreads();
        if (c == 0) row[S] = make_uint4(prev[0], prev[1], prev[2], prev[3]);
        for (int x = S - 1; x >= 0; --x) {
            bool ok = false;
            int most = 0;
            if (c < L) {
                // memory grows with the layer count: binary search for the
                // largest l that fits, then any suffix start in (c, c+l]
                const int k = sr.cls[x];
                int lo = 0, hi = L - c;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (stage_fits(t, S, M, x, k, c, c + mid)) lo = mid;
                    else hi = mid - 1;
                }
                most = lo;
                const Bits128 win = range_bits(c + 1, c + most);
                ok = ((prev[0] & win.w[0]) | (prev[1] & win.w[1]) | (prev[2] & win.w[2]) |
                      (prev[3] & win.w[3])) != 0u;
            }
            if (c < 128) lim[((size_t)sr.gid * S + x) * 128 + c] = (uint8_t)most;
            const unsigned b = __ballot_sync(0xffffffffu, ok);
            if ((c & 31) == 0) cur[c >> 5] = b;
            __syncthreads();
            if (c < 4) prev[c] = cur[c];
            __syncthreads();
            if (c == 0) row[x] = make_uint4(prev[0], prev[1], prev[2], prev[3]);
        }
        // root[gid] = the whole model fits the slice's stages (bit c = 0 of row 0)
        if (c == 0) root[sr.gid] = (uint8_t)(prev[0] & 1u);
        __syncthreads();
    }
}


// ---------------------------------------------------------------------------
// completion bounds (prune mode 2).  For a complete plan and 0-based stages
// i <= y, the DAG path through the first micro-batch's forwards up to stage
// y, stage y's whole chain, the last micro-batch's backwards down to stage i
// and R_i has length
//   P(y, i) = sum_{j<y} (F_j + pf_j) + M (F_y + B_y) + sum_{j=i}^{y-1} (B_j + pb_j) + d_i,
// so T >= P(y, i).  Eq. 2 is max_i P(x, i) without the edges.  Over the
// stages y >= x that a prefix has not placed yet, with A = sum_{j<x}
// (F_j + pf_j) and Bm = max_{i<x} (sum_{j=i}^{x-1} (B_j + pb_j) + d_i):
//   max_{y>=x} P(y, y)          = A + V1,
//   max_{y>=x, i<x} P(y, i)     = A + Bm + V2,
// where, for the stages x..S-1 covering layers [c, L),
//   V1 = max_y (sum_{x<=j<y} (F_j + pf_j) + M (F_y + B_y) + d_y),
//   V2 = max_y (sum_{x<=j<y} (F_j + pf_j + B_j + pb_j) + M (F_y + B_y)).
// V1[x][c] and V2[x][c] hold their minima over every memory-feasible
// completion, by the recursion over stage x's layer count l
//   V1[x][c] = min_l max(M (F + B) + d, F + pf_x + V1[x+1][c+l]),
//   V2[x][c] = min_l max(M (F + B),     F + pf_x + B + pb_x + V2[x+1][c+l]).
// A prefix whose A + V1 or A + Bm + V2 exceeds the incumbent has no
// completion that beats it.  Each finite entry is at most the makespan of
// a feasible plan, so it fits in int32 under the overflow guard.
// One block per memory-feasible slice, four threads per start c (each
// takes every fourth layer count, then the four minima are combined by
// shuffles).  vb[(x*n_rows + vslot)*128 + c]; arg[x][c] (shared memory)
// keeps the smallest l attaining V1[x][c], and thread 0 follows it from
// (0, 0) to write the slice's argmin completion as a plan: a memory-feasible
// plan whose makespan is usually close to the slice's best (warm-up seed).
// root_lb[slice] = V1[0][0] * scale, a lower bound on the slice's objective.
constexpr int kBoundThreads = 512;

// rows = NULL: row r is slice r, for every slice (n_rows = the slice count);
// a slice whose root is infeasible (root[r] == 0) then gets a hole for its
// greedy plan and an infinite root bound, and no table rows.
__global__ void __launch_bounds__(kBoundThreads) bound_kernel(
    const SliceRec *slices, const uint32_t *rows, const uint8_t *root, int n_rows, int S,
    const uint8_t *lim, int2 *vb, Leaf *greedy, unsigned long long *root_lb, const void *blob,
    BlobLayout lay, unsigned long long *stats) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ int2 nxt[128];
    __shared__ uint8_t arg[POS_MAX_STAGES][128];
    __shared__ uint64_t bar;
    if (!stage_blob_bulk(sm, blob, lay.bytes, &bar)) {
        if (threadIdx.x == 0) atomicAdd(stats + kStBulkTimeout, 1ull);
        grid_dep_wait();  // a block never leaves before its predecessor has completed
        return;
    }
    grid_dep_wait();  // the memory-limit rows and root bits (feasibility kernel)
    grid_dep_trigger();
    const Tab t = tab_at(sm, lay);
    const int L = lay.L, c = threadIdx.x >> 2, part = threadIdx.x & 3;
    for (int r = blockIdx.x; r < n_rows; r += gridDim.x) {
        const uint32_t sl = rows ? rows[r] : (uint32_t)r;
        if (!rows && !root[sl]) {  // the same for the whole block
            if (threadIdx.x == 0) {
                const Vec32 hole = {make_uint4(kLeafHole, 0, 0, 0), make_uint4(0, 0, 0, 0)};
                store32(greedy + r, hole);
                root_lb[sl] = ~0ull;
            }
            continue;
        }
        const SliceRec &sr = slices[sl];
        const int M = sr.M;
        const uint32_t vslot = sr.vslot;
        for (int x = S - 1; x >= 0; --x) {
            const int k = sr.cls[x];
            const int32_t pf = x + 1 < S ? p2f(t, k, sr.cls[x + 1]) : 0;
            const int32_t pb = x + 1 < S ? p2b(t, sr.cls[x + 1], k) : 0;
            int64_t v1 = INT64_MAX, v2 = INT64_MAX;
            int best_l = 0;
            if (c < L) {
                const int most = lim[((size_t)sr.gid * S + x) * 128 + c];
                const int32_t f0 = Pf(t, k, c), b0 = Pb(t, k, c), d0 = Pd(t, k, c);
                const int l_lo = x == S - 1 ? L - c : 1;
                const int l_hi = x == S - 1 ? L - c : min(most, L - c - (S - 1 - x));
                for (int l = l_lo + part; l <= l_hi && l <= most; l += 4) {
                    const int c2 = c + l;
                    const int64_t F = Pf(t, k, c2) - f0, B = Pb(t, k, c2) - b0;
                    const int64_t d = Pd(t, k, c2) - d0;
                    const int64_t a = (int64_t)M * (F + B);
                    int64_t w1, w2;
                    if (x == S - 1) {
                        w1 = a + d;
                        w2 = a;
                    } else {
                        const int2 n = nxt[c2];
                        if (n.x == kNoCompletion) continue;
                        w1 = max(a + d, F + pf + n.x);
                        w2 = max(a, F + pf + B + pb + n.y);
                    }
                    if (w1 < v1) {  // l increases: the first strict minimum is the smallest l
                        v1 = w1;
                        best_l = l;
                    }
                    v2 = min(v2, w2);
                }
            }
            // combine the four partial minima of start c (lanes 4c .. 4c+3);
            // ties in V1 go to the smallest l
#pragma unroll
            for (int o = 1; o < 4; o <<= 1) {
                const int64_t o1 = __shfl_xor_sync(0xffffffffu, v1, o);
                const int64_t o2 = __shfl_xor_sync(0xffffffffu, v2, o);
                const int ol = __shfl_xor_sync(0xffffffffu, best_l, o);
                if (o1 < v1 || (o1 == v1 && ol < best_l)) {
                    v1 = o1;
                    best_l = ol;
                }
                v2 = min(v2, o2);
            }
            __syncthreads();  // every thread has read row x+1
            if (part == 0) {
                const int2 out = v1 == INT64_MAX ? make_int2(kNoCompletion, kNoCompletion)
                                                 : make_int2((int32_t)v1, (int32_t)v2);
                nxt[c] = out;
                arg[x][c] = (uint8_t)best_l;
                vb[((size_t)x * n_rows + vslot) * 128 + c] = out;
            }
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            // the root of a memory-feasible slice always has a completion
            uint32_t cw[4] = {0u, 0u, 0u, 0u};  // cut[x] in byte x
            int cc = 0;
            for (int x = 0; x < S - 1; ++x) {
                cc += arg[x][cc];
                const uint32_t v = (uint32_t)cc << (8 * (x % 4));
#pragma unroll
                for (int wi = 0; wi < 4; ++wi) cw[wi] |= (x / 4 == wi) ? v : 0u;
            }
            const Vec32 lf = {make_uint4(sl, cw[0], cw[1], cw[2]), make_uint4(cw[3], 0u, 0u, 0u)};
            store32(greedy + r, lf);
            // the slice's root bound V1[0][0] = min over plans of max_y P(y, y),
            // as an objective (orders the slices)
            root_lb[sl] = (unsigned long long)nxt[0].x * sr.scale;
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// warm-up sampler (Sec. 4.2.3): random memory-feasible plans.  splitmix64
// (Steele, Lea & Flood, 2014) on the counter (seed, sample index).
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t splitmix64_next(uint64_t &s) {
    uint64_t z = (s += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}


// Position of the r-th (0-based) set bit of a 128-bit set with more than r
// set bits.
__device__ __forceinline__ int nth_set(const Bits128 &b, int r) {
    int base = 0;
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const int p = __popc(b.w[i]);
        if (base == 32 * i && r >= p) {
            r -= p;
            base = 32 * (i + 1);
        }
    }
    const uint32_t word = base == 0 ? b.w[0] : base == 32 ? b.w[1] : base == 64 ? b.w[2] : b.w[3];
    return base + (int)__fns(word, 0, r + 1);
}

// One thread per sample: stage by stage, the layer count is drawn uniformly
// among the counts l that fit the stage's memory (l <= lim) and leave a
// memory-feasible suffix (feasibility bit of c + l), i.e. the set bits of
// one 128-bit window, picked with a popcount and a select.
__global__ void sample_kernel(const SliceRec *slices, const uint32_t *feasible, int n_feasible,
                              int n_samples, int S, uint64_t seed, const uint4 *feas,
                              const uint8_t *lim, Leaf *out, int L) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n_samples;
         i += gridDim.x * blockDim.x) {
        uint64_t st = seed ^ ((uint64_t)i * 0xD1B54A32D192ED03ull);
        const uint32_t sl = feasible[splitmix64_next(st) % (uint64_t)n_feasible];
        const SliceRec &sr = slices[sl];
        const uint32_t gid = sr.gid;
        uint32_t cw[4] = {0u, 0u, 0u, 0u};  // cut[0..15], byte x = cut[x]
        int c = 0;
        for (int x = 0; x < S - 1; ++x) {
            const int hi = min((int)__ldg(lim + ((size_t)gid * S + x) * 128 + c),
                               L - c - (S - x - 1));
            const uint4 f = __ldg(feas + (size_t)gid * (S + 1) + x + 1);
            const Bits128 win = range_bits(c + 1, c + hi);
            const Bits128 ok = {{f.x & win.w[0], f.y & win.w[1], f.z & win.w[2], f.w & win.w[3]}};
            const int n_ok = popc128(ok);
            const int r = (int)(splitmix64_next(st) % (uint64_t)max(n_ok, 1));
            c = n_ok > 0 ? nth_set(ok, r) : c + 1;
            const uint32_t v = (uint32_t)c << (8 * (x % 4));
#pragma unroll
            for (int wi = 0; wi < 4; ++wi) cw[wi] |= (x / 4 == wi) ? v : 0u;
        }
        // leaf: slice in bytes 0-3, cut[x] in byte 4 + x
        const Vec32 lf = {make_uint4(sl, cw[0], cw[1], cw[2]), make_uint4(cw[3], 0u, 0u, 0u)};
        store32(out + i, lf);
    }
}

// ---------------------------------------------------------------------------
// level expansion and completion (Sec. 4.2.1 prune, Sec. 3.2 memory cut)
// ---------------------------------------------------------------------------
struct ExpandParams {
    const Prefix *in;
    long long n_in;
    const unsigned long long *n_in_dev;  // if set: n_in = min(*n_in_dev, cap), read on the device
    const uint32_t *groups;  // work list of 32-parent groups, or NULL = all groups
    long long n_groups;
    int x;                   // depth of the parents (stages 0..x-1 placed)
    int S, M;
    int prune;
    int ridge;               // 1: layer-level (ridge) pruning
    int exact;               // 1: host-driven pass (lane-per-parent mode with deferral lists)
    const SliceRec *slices;
    const uint4 *feas;
    const uint8_t *lim;      // per (slice, stage, start) memory limit, see feas_kernel
    const int2 *vb;          // prune 2: completion bounds per (batch slot, stage, start)
    int vb_smem;             // 1: stage this depth's rows of all nb slots in shared memory
    int nb;                  // slots in the batch
    int n_vrows;             // rows per depth of vb (vb[(x*n_vrows + vslot)*128 + c])
    Prefix *out;             // expand: children at depth x+1
    Leaf *leaves;            // complete: full plans
    unsigned long long *out_count;
    unsigned long long cap;
    uint32_t *deferred;
    unsigned long long *n_deferred;
    const Key128 *inc;
    unsigned long long *stats;
    const void *blob;
    BlobLayout lay;
};


// Largest l in [0, hi] with pred(l), for pred true up to some l and false
// after (pred(0) is taken as true).
template <class Pred>
__device__ __forceinline__ int last_true(int hi, Pred pred) {
    int lo = 0;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (pred(mid)) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

// Per-parent quantities shared by the search for children and the writes:
// parent cut c, class k of the new stage, prefix sums at c.
struct ParentCtx {
    int c, k;
    int32_t f0, b0, d0;
    int32_t pf, pb;  // prune 2: F and B edge between the new stage and the next one
    // ridge rule: state of the prefix, device types of the new and the next
    // stage, most layers the new stage may take (127: no cap)
    uint32_t rstate;
    int rta, rtb, rcap;
};

// Ridge fields of a parent (when the rule is on): its state word, the types
// of stages X and X+1, and the cap on stage X's layers.
__device__ __forceinline__ void ridge_ctx(ParentCtx &q, bool on, uint32_t state, int ka, int kb,
                                          int n_tp) {
    if (!on) return;
    q.rstate = state;
    q.rta = ka / n_tp;
    q.rtb = kb / n_tp;
    q.rcap = ridge_cap(state, q.rta);
}

__device__ __forceinline__ ParentCtx parent_ctx(const Tab &t, int k, int c) {
    ParentCtx q;
    q.c = c;
    q.k = k;
    q.f0 = Pf(t, k, c);
    q.b0 = Pb(t, k, c);
    q.d0 = Pd(t, k, c);
    q.pf = 0;
    q.pb = 0;
    q.rstate = 0;
    q.rta = q.rtb = 0;
    q.rcap = 127;
    return q;
}

// Children of one parent, as the set of new cut positions c2 = c + l.
// Expansion (parent depth x <= S-3): stage x takes l layers.  Its memory
// need and g(S_{x+1}) both grow with l, so the admissible l form a prefix
// [1, hi] found by binary search; the children are the positions in
// (c, c+hi] from which the remaining layers still fit the remaining stages
// (feasibility bits).
__device__ __forceinline__ int expand_set(const ExpandParams &p, const Tab &t, int64_t A,
                                          int64_t Bm, const ParentCtx &q, uint32_t gid,
                                          const int2 *vrow, uint64_t scale,
                                          uint64_t thr, Bits128 &acc, unsigned long long &cut_b,
                                          unsigned long long &cut_m, unsigned long long &cut_r) {
    const int S = p.S, M = p.M, x = p.x, L = t.L();
    const int lmax = L - q.c - (S - x - 1);
    const int hi_mem0 = min(lmax, (int)__ldg(p.lim + ((size_t)gid * S + x) * 128 + q.c));
    const int hi_mem = min(hi_mem0, q.rcap);  // ridge rule: a cap on the layer count
    cut_r += (unsigned long long)(hi_mem0 - hi_mem);
    int hi = hi_mem;
    if (p.prune) {  // g(S_{x+1}) grows with l: binary search for the last l within the bound
        int lo = 0;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1, c2 = q.c + mid;
            const int64_t F = Pf(t, q.k, c2) - q.f0, B = Pb(t, q.k, c2) - q.b0;
            const int64_t d = Pd(t, q.k, c2) - q.d0;
            if ((uint64_t)(A + (int64_t)M * (F + B) + max(Bm, d)) * scale <= thr) lo = mid;
            else hi = mid - 1;
        }
    }
    const uint4 f = __ldg(p.feas + (size_t)gid * (S + 1) + x + 1);
    const Bits128 win = range_bits(q.c + 1, q.c + hi);
    acc.w[0] = f.x & win.w[0];
    acc.w[1] = f.y & win.w[1];
    acc.w[2] = f.z & win.w[2];
    acc.w[3] = f.w & win.w[3];
    int n = popc128(acc);
    cut_m += (unsigned long long)(lmax - hi_mem0) + (unsigned long long)(hi - n);
    cut_b += (unsigned long long)(hi_mem - hi);
    if (p.prune == 2 && n > 0) {
        // completion terms: the bound is not monotone in l, so every
        // candidate child is tested on its own
#pragma unroll
        for (int wd = 0; wd < 4; ++wd) {
            uint32_t m = acc.w[wd];
            while (m) {
                // up to four candidates at a time, their table loads in flight together
                int bb[4];
                int2 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    bb[u] = m ? __ffs(m) - 1 : -1;
                    m &= m - 1;
                }
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (bb[u] >= 0) v[u] = vrow[32 * wd + bb[u]];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    if (bb[u] < 0) continue;
                    const int c2 = 32 * wd + bb[u];
                    const int64_t F = Pf(t, q.k, c2) - q.f0, B = Pb(t, q.k, c2) - q.b0;
                    const int64_t d = Pd(t, q.k, c2) - q.d0;
                    const int64_t A2 = A + F + q.pf, Bm2 = max(Bm, d) + B + q.pb;
                    if (v[u].x == kNoCompletion || (uint64_t)(A2 + v[u].x) * scale > thr ||
                        (uint64_t)(A2 + Bm2 + v[u].y) * scale > thr) {
                        acc.w[wd] &= ~(1u << bb[u]);
                        --n;
                        ++cut_b;
                    }
                }
            }
        }
    }
    return n;
}

// Completion (parent depth S-2): stage a = S-2 takes l layers, stage
// b = S-1 the rest.  Stage a's memory and g(S_{S-1}) bound l from above,
// stage b's memory from below (fewer layers as l grows); inside that window
// each l is checked against g(S_S).
__device__ __forceinline__ int complete_set(const ExpandParams &p, const Tab &t, int64_t A,
                                            int64_t Bm, const ParentCtx &q, int kb, uint32_t gid,
                                            uint64_t scale,
                                            uint64_t thr, Bits128 &acc, unsigned long long &cut_b,
                                            unsigned long long &cut_m, unsigned long long &cut_r) {
    const int S = p.S, M = p.M, L = t.L(), a = S - 2, b = S - 1;
    const int c = q.c;
    const int lmax = L - c - 1;
    const int hi_mem0 = min(lmax, (int)__ldg(p.lim + ((size_t)gid * S + a) * 128 + c));
    const int hi_mem = min(hi_mem0, q.rcap);
    cut_r += (unsigned long long)(hi_mem0 - hi_mem);
    int hi = hi_mem;
    if (p.prune) {  // g(S_{S-1}) grows with l
        int lo = 0;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1, c2 = c + mid;
            const int64_t F = Pf(t, q.k, c2) - q.f0, B = Pb(t, q.k, c2) - q.b0;
            const int64_t d = Pd(t, q.k, c2) - q.d0;
            if ((uint64_t)(A + (int64_t)M * (F + B) + max(Bm, d)) * scale <= thr) lo = mid;
            else hi = mid - 1;
        }
    }
    // stage b fits [c2, L) exactly for the set feasibility bits of depth b,
    // a suffix of positions: the smallest l is the first set bit above c
    const uint4 fb = __ldg(p.feas + (size_t)gid * (S + 1) + b);
    const Bits128 above = range_bits(c + 1, L - 1);
    const uint32_t m0 = fb.x & above.w[0], m1 = fb.y & above.w[1], m2 = fb.z & above.w[2],
                   m3 = fb.w & above.w[3];
    const int first = m0 ? __ffs(m0) - 1 : m1 ? 31 + __ffs(m1) : m2 ? 63 + __ffs(m2)
                    : m3 ? 95 + __ffs(m3) : 128;
    const int lo = first - c;
    for (int i = 0; i < 4; ++i) acc.w[i] = 0;
    int n = 0;
    const int32_t fbL = Pf(t, kb, L), bbL = Pb(t, kb, L), dbL = Pd(t, kb, L);
    for (int l = lo; l <= hi; ++l) {
        const int c2 = c + l;
        // ridge rule for the last stage, after this one took l layers
        if (p.ridge && L - c2 > ridge_cap(ridge_next(q.rstate, q.rta, l), q.rtb)) {
            ++cut_r;
            continue;
        }
        if (p.prune) {
            const int64_t Fa = Pf(t, q.k, c2) - q.f0, Ba = Pb(t, q.k, c2) - q.b0;
            const int64_t da = Pd(t, q.k, c2) - q.d0;
            const int64_t Fb = fbL - Pf(t, kb, c2), Bb = bbL - Pb(t, kb, c2);
            const int64_t db = dbL - Pd(t, kb, c2);
            const int64_t g =
                A + Fa + q.pf + (int64_t)M * (Fb + Bb) + max(max(Bm, da) + Ba + q.pb, db);
            if ((uint64_t)g * scale > thr) {
                ++cut_b;
                continue;
            }
        }
#pragma unroll
        for (int wd = 0; wd < 4; ++wd) acc.w[wd] |= (c2 >> 5) == wd ? 1u << (c2 & 31) : 0u;
        ++n;
    }
    cut_m += (unsigned long long)(lmax - hi_mem0) + (unsigned long long)(lo - 1 < hi ? lo - 1 : hi);
    cut_b += (unsigned long long)(hi_mem - hi);
    return n;
}

// Small frontiers: one warp per parent.  Lane j tests the layer counts
// l = 1 + j + 32 r (r = 0..3) of the new stage X at once: memory (l <= the
// memory limit row), Eq. 2 for the child, the feasibility bit of c + l and
// the per-candidate test (completion bounds when expanding under prune
// mode 2, g(S_S) when completing); four ballots hold the survivors, one
// atomic reserves their slots.  Only the pipelined pass uses this mode; on
// overflow it counts the parent as deferred without listing it (the batch
// is then run again by the host-driven path).  Statistics are kept by
// lane 0.
template <bool COMPLETE, int X>
__device__ __forceinline__ void level_warp_mode(const ExpandParams &p, const Tab &t,
                                                long long n_in, const int2 *vsm,
                                                const int2 *vdepth, uint64_t thr,
                                                unsigned long long &emitted,
                                                unsigned long long &cb, unsigned long long &cm,
                                                unsigned long long &cr,
                                                unsigned long long &written) {
    const int lane = threadIdx.x & 31;
    const unsigned lt_mask = (1u << lane) - 1u;
    const long long warp = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
    const long long n_warps = ((long long)gridDim.x * blockDim.x) >> 5;
    const int S = p.S, M = p.M, L = t.L();
    for (long long i = warp; i < n_in; i += n_warps) {
        const Vec32 pv = load32(p.in + i);  // one address: a broadcast
        const uint32_t slice = pv.a.x & 0xffffu;
        if (slice == kPrefixHole) continue;
        const SliceRec &sr = p.slices[slice];
        const int c = X > 0 ? (int)get_byte<(X > 0 ? X + 1 : 2)>(pv) : 0;
        ParentCtx q = parent_ctx(t, sr.cls[X], c);
        const int kb = sr.cls[X + 1];  // X + 1 <= S - 1
        ridge_ctx(q, p.ridge != 0, pv.b.z, q.k, kb, t.n_tp());
        const int32_t pf = p.prune == 2 ? p2f(t, q.k, kb) : 0;
        const int32_t pb = p.prune == 2 ? p2b(t, kb, q.k) : 0;
        const uint64_t scale = sr.scale;
        const uint32_t gid = sr.gid;
        const int64_t A = (int32_t)pv.b.x, Bm = (int32_t)pv.b.y;
        const int lmax = COMPLETE ? L - c - 1 : L - c - (S - X - 1);
        const int hi_mem0 = min(lmax, (int)__ldg(p.lim + ((size_t)gid * S + X) * 128 + c));
        const int hi_mem = min(hi_mem0, q.rcap);  // ridge rule: a cap on the layer count
        // expansion: the next stage must fit from c + l (row X+1); completion:
        // stage S-1 must hold [c + l, L) (row S-1)
        const uint4 f = __ldg(p.feas + (size_t)gid * (S + 1) + (COMPLETE ? S - 1 : X + 1));
        const int2 *vrow = vsm ? vsm + (size_t)slice * 128
                               : (vdepth ? vdepth + (size_t)sr.vslot * 128 : nullptr);
        unsigned pass[4];
        int n_bound = 0, n_win = 0, n_fail = 0, n_ridge_b = 0;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int l = 1 + lane + 32 * r;
            const int c2 = c + l;
            const bool in_mem = l <= hi_mem;
            bool g_ok = false, cand = false, ok = false;
            if (in_mem) {
                const int64_t F = Pf(t, q.k, c2) - q.f0, B = Pb(t, q.k, c2) - q.b0;
                const int64_t d = Pd(t, q.k, c2) - q.d0;
                g_ok = !p.prune ||
                       (uint64_t)(A + (int64_t)M * (F + B) + max(Bm, d)) * scale <= thr;
                const uint32_t word2 = (c2 >> 5) == 0 ? f.x : (c2 >> 5) == 1 ? f.y
                                     : (c2 >> 5) == 2 ? f.z : f.w;
                cand = g_ok && ((word2 >> (c2 & 31)) & 1u);
                // ridge rule for the last stage, after this one took l layers
                if (COMPLETE && cand && p.ridge &&
                    L - c2 > ridge_cap(ridge_next(q.rstate, q.rta, l), q.rtb))
                    cand = false, ++n_ridge_b;
                ok = cand;
                if (cand) {
                    const int64_t A2 = A + F + pf, Bm2 = max(Bm, d) + B + pb;
                    if (COMPLETE) {
                        if (p.prune) {
                            const int64_t Fb = Pf(t, kb, L) - Pf(t, kb, c2);
                            const int64_t Bb = Pb(t, kb, L) - Pb(t, kb, c2);
                            const int64_t db = Pd(t, kb, L) - Pd(t, kb, c2);
                            ok = (uint64_t)(A2 + (int64_t)M * (Fb + Bb) + max(Bm2, db)) * scale <=
                                 thr;
                        }
                    } else if (p.prune == 2) {
                        const int2 v = vrow[c2];
                        ok = v.x != kNoCompletion && (uint64_t)(A2 + v.x) * scale <= thr &&
                             (uint64_t)(A2 + Bm2 + v.y) * scale <= thr;
                    }
                }
            }
            pass[r] = __ballot_sync(0xffffffffu, ok);
            n_bound += __popc(__ballot_sync(0xffffffffu, in_mem && g_ok));
            n_win += __popc(__ballot_sync(0xffffffffu, cand));
            n_fail += __popc(__ballot_sync(0xffffffffu, cand && !ok));
        }
        const int total = __popc(pass[0]) + __popc(pass[1]) + __popc(pass[2]) + __popc(pass[3]);
        // lanes cut by the last-stage ridge test, summed over the warp
        int r_sum = n_ridge_b;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) r_sum += __shfl_xor_sync(0xffffffffu, r_sum, o);
        if (lane == 0) {
            cm += (unsigned long long)(lmax - hi_mem0) + (unsigned long long)(n_bound - n_win - r_sum);
            cb += (unsigned long long)(hi_mem - n_bound) + (unsigned long long)n_fail;
            cr += (unsigned long long)(hi_mem0 - hi_mem) + (unsigned long long)r_sum;
            written += 1;
        }
        if (total == 0) continue;
        unsigned long long base = 0;
        if (lane == 0) base = atomicAdd(p.out_count, (unsigned long long)total);
        base = __shfl_sync(0xffffffffu, base, 0);
        if (base + (unsigned long long)total > p.cap) {
            // no room: reserved slots below the capacity become holes
            const Vec32 hole = {make_uint4(COMPLETE ? kLeafHole : kPrefixHole, 0, 0, 0),
                                make_uint4(0, 0, 0, 0)};
            for (unsigned long long e = base + lane; e < base + (unsigned long long)total && e < p.cap;
                 e += 32) {
                if (COMPLETE) store32(p.leaves + e, hole);
                else store32(p.out + e, hole);
            }
            if (lane == 0) atomicAdd(p.n_deferred, 1ull);
            continue;
        }
        unsigned long long pos = base;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            if ((pass[r] >> lane) & 1u) {
                const int c2 = c + 1 + lane + 32 * r;
                const unsigned long long at = pos + (unsigned long long)__popc(pass[r] & lt_mask);
                Vec32 out;
                if (COMPLETE) {
                    // leaf: slice in bytes 0-3, cut[i] in byte 4+i; the
                    // parent's cuts (bytes 2..15) move up two bytes
                    out.a.x = slice;
                    out.a.y = __funnelshift_r(pv.a.x, pv.a.y, 16);
                    out.a.z = __funnelshift_r(pv.a.y, pv.a.z, 16);
                    out.a.w = __funnelshift_r(pv.a.z, pv.a.w, 16);
                    out.b = make_uint4(pv.a.w >> 16, 0u, 0u, 0u);
                    set_byte<4 + X>(out, (uint32_t)c2);
                    store32(p.leaves + at, out);
                } else {
                    const int32_t F = Pf(t, q.k, c2) - q.f0, B = Pb(t, q.k, c2) - q.b0;
                    const int32_t d = Pd(t, q.k, c2) - q.d0;
                    out.a = pv.a;
                    out.b = make_uint4((uint32_t)((int32_t)pv.b.x + F + pf),
                                       (uint32_t)(max((int32_t)pv.b.y, d) + B + pb),
                                       p.ridge ? ridge_next(q.rstate, q.rta, c2 - c) : 0u, 0u);
                    set_byte<2 + (X < 14 ? X : 0)>(out, (uint32_t)c2);
                    store32(p.out + at, out);
                }
            }
            pos += (unsigned long long)__popc(pass[r]);
        }
        if (lane == 0) emitted += (unsigned long long)total;
    }
}

// One warp per group of 32 consecutive parents: each lane finds its
// parent's children (a 128-bit set of cut positions), the warp reserves
// output slots with one atomic and writes them -- or, when the output is
// full, marks its reserved slots as holes and defers the group.
template <bool COMPLETE, int X>
__global__ void __launch_bounds__(kThreads, 3) level_kernel(ExpandParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    // timing tables and, when expanding under prune mode 2, the
    // completion-bound rows of depth X+1 of every slot (contiguous), by TMA;
    // all written before the previous kernel, so staged while it finishes
    __shared__ uint64_t bar;
    const bool use_v = !COMPLETE && p.prune == 2;
    const bool stage_v = use_v && p.vb_smem;
    // depth X+1 of the bound tables: the row of table row v is vdepth + 128 v
    const int2 *vdepth = use_v ? p.vb + (size_t)(X + 1) * p.n_vrows * 128 : nullptr;
    if (threadIdx.x == 0) {
        const uint32_t vbytes = stage_v ? (uint32_t)p.nb * 128u * 8u : 0u;
        bulk_begin(&bar, (uint32_t)p.lay.bytes + vbytes);
        bulk_copy(sm, p.blob, (uint32_t)p.lay.bytes, &bar);
    }
    if (stage_v) {
        __syncthreads();  // the barrier is armed before the other copies start
        if (threadIdx.x < 32)
            for (int slot = threadIdx.x; slot < p.nb; slot += 32)
                bulk_copy(sm + p.lay.bytes + (size_t)slot * 1024,
                          vdepth + (size_t)__ldg(&p.slices[slot].vslot) * 128, 1024u, &bar);
    }
    if (!bulk_wait(&bar)) {
        if (threadIdx.x == 0) atomicAdd(p.stats + kStBulkTimeout, 1ull);
        grid_dep_wait();  // a block never leaves before its predecessor has completed
        return;
    }
    // the frontier, its count and the incumbent only after the previous
    // kernel has completed
    grid_dep_wait();
    grid_dep_trigger();
    long long n_in = p.n_in;
    if (p.n_in_dev) {
        const unsigned long long c0 = __ldcg(p.n_in_dev);
        n_in = (long long)(c0 < p.cap ? c0 : p.cap);
    }
    const long long n_work = p.groups ? p.n_groups : (n_in + 31) / 32;
    const long long n_warps = ((long long)gridDim.x * blockDim.x) >> 5;
    // small frontier in the pipelined pass: one warp per parent
    const bool warp_mode = !p.exact && !p.groups && n_in <= n_warps;
    if ((long long)blockIdx.x * (kThreads / 32) >= (warp_mode ? n_in : n_work)) return;
    const int2 *vsm = stage_v ? reinterpret_cast<const int2 *>(sm + p.lay.bytes) : nullptr;
    const Tab t = tab_at(sm, p.lay);
    const uint64_t thr = p.prune ? __ldcg(&p.inc->obj) : ~0ull;
    const int lane = threadIdx.x & 31;
    const long long warp = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
    unsigned long long emitted = 0, cb = 0, cm = 0, cr = 0, written_parents = 0;
    if (warp_mode)
        level_warp_mode<COMPLETE, X>(p, t, n_in, vsm, vdepth, thr, emitted, cb, cm, cr,
                                     written_parents);
    for (long long w = warp; !warp_mode && w < n_work; w += n_warps) {
        const long long g = p.groups ? (long long)p.groups[w] : w;
        const long long i = g * 32 + lane;
        Vec32 pv = {make_uint4(kPrefixHole, 0, 0, 0), make_uint4(0, 0, 0, 0)};
        if (i < n_in) pv = load32(p.in + i);
        const uint32_t slice = pv.a.x & 0xffffu;
        const bool live = slice != kPrefixHole;
        Bits128 acc = {{0u, 0u, 0u, 0u}};
        unsigned long long lb = 0, lm = 0, lr = 0;
        int n = 0;
        ParentCtx q = {0, 0, 0, 0, 0};
        if (live) {
            const SliceRec &sr = p.slices[slice];
            // X = depth of the parents = index of the stage placed here;
            // parent byte 2+i holds cut[i]
            const int c = X > 0 ? (int)get_byte<(X > 0 ? X + 1 : 2)>(pv) : 0;
            q = parent_ctx(t, sr.cls[X], c);
            ridge_ctx(q, p.ridge != 0, pv.b.z, sr.cls[X], sr.cls[X + 1], t.n_tp());
            if (p.prune == 2) {  // X + 1 <= S - 1: the next stage exists
                q.pf = p2f(t, sr.cls[X], sr.cls[X + 1]);
                q.pb = p2b(t, sr.cls[X + 1], sr.cls[X]);
            }
            const uint64_t scale = sr.scale;
            const int64_t A = (int32_t)pv.b.x, Bm = (int32_t)pv.b.y;
            n = COMPLETE ? complete_set(p, t, A, Bm, q, sr.cls[X + 1], sr.gid, scale, thr, acc, lb,
                                        lm, lr)
                         : expand_set(p, t, A, Bm, q, sr.gid,
                                      vsm ? vsm + (size_t)slice * 128
                                          : (vdepth ? vdepth + (size_t)sr.vslot * 128 : nullptr),
                                      scale, thr, acc, lb, lm, lr);
        }
        int incl = n;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        const int total = __shfl_sync(0xffffffffu, incl, 31);
        unsigned long long base = 0;
        if (lane == 0 && total > 0) base = atomicAdd(p.out_count, (unsigned long long)total);
        base = __shfl_sync(0xffffffffu, base, 0);
        if (total == 0) {
            cb += lb;
            cm += lm;
            cr += lr;
            written_parents += live;
            continue;
        }
        unsigned long long pos = base + (unsigned long long)(incl - n);
        if (base + (unsigned long long)total <= p.cap) {
#pragma unroll
            for (int wd = 0; wd < 4; ++wd) {
                uint32_t m = acc.w[wd];
                while (m) {
                    const int c2 = 32 * wd + __ffs(m) - 1;
                    m &= m - 1;
                    if (COMPLETE) {
                        // leaf: slice in bytes 0-3, cut[i] in byte 4+i; the
                        // parent's cuts (bytes 2..15) move up two bytes
                        Vec32 lf;
                        lf.a.x = slice;
                        lf.a.y = __funnelshift_r(pv.a.x, pv.a.y, 16);
                        lf.a.z = __funnelshift_r(pv.a.y, pv.a.z, 16);
                        lf.a.w = __funnelshift_r(pv.a.z, pv.a.w, 16);
                        lf.b = make_uint4(pv.a.w >> 16, 0u, 0u, 0u);
                        set_byte<4 + X>(lf, (uint32_t)c2);
                        store32(p.leaves + pos++, lf);
                    } else {
                        Vec32 ch = pv;
                        set_byte<2 + (X < 14 ? X : 0)>(ch, (uint32_t)c2);
                        ch.b.x = (uint32_t)((int32_t)pv.b.x + (Pf(t, q.k, c2) - q.f0) + q.pf);
                        ch.b.y = (uint32_t)(max((int32_t)pv.b.y, Pd(t, q.k, c2) - q.d0) +
                                            (Pb(t, q.k, c2) - q.b0) + q.pb);
                        ch.b.z = p.ridge ? ridge_next(q.rstate, q.rta, c2 - q.c) : 0u;
                        store32(p.out + pos++, ch);
                    }
                }
            }
            emitted += n;
            cb += lb;
            cm += lm;
            cr += lr;
            written_parents += live;
        } else {
            // no room: mark this warp's reserved slots below cap as holes
            const Vec32 hole = {make_uint4(COMPLETE ? kLeafHole : kPrefixHole, 0, 0, 0),
                                make_uint4(0, 0, 0, 0)};
            for (unsigned long long e = pos; e < pos + (unsigned long long)n && e < p.cap; ++e) {
                if (COMPLETE) store32(p.leaves + e, hole);
                else store32(p.out + e, hole);
            }
            if (lane == 0) {
                const unsigned long long d = atomicAdd(p.n_deferred, 1ull);
                p.deferred[d] = (uint32_t)g;
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        emitted += __shfl_xor_sync(0xffffffffu, emitted, o);
        cb += __shfl_xor_sync(0xffffffffu, cb, o);
        cm += __shfl_xor_sync(0xffffffffu, cm, o);
        cr += __shfl_xor_sync(0xffffffffu, cr, o);
        written_parents += __shfl_xor_sync(0xffffffffu, written_parents, o);
    }
    if (lane == 0) {
        if (cr) atomicAdd(p.stats + kStPrunedRidge, cr);
        if (emitted) atomicAdd(p.stats + (COMPLETE ? kStLeaves : kStPrefixes), emitted);
        if (cb) atomicAdd(p.stats + kStPrunedBound, cb);
        if (cm) atomicAdd(p.stats + kStPrunedMemory, cm);
        if (written_parents) {
            atomicAdd(p.stats + (COMPLETE ? kStParentsComplete : kStParentsExpand), written_parents);
            atomicAdd(p.stats + kStDepthParents + X, written_parents);
        }
        if (emitted) atomicAdd(p.stats + kStDepthChildren + X, emitted);
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
constexpr int kMaxDevices = 64;
static std::mutex g_ws_mutex;
static Workspace *g_ws[kMaxDevices];

pos_status get_workspace(Workspace **out) {
    int dev = 0;
    POS_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kMaxDevices) return fail(POS_EINVAL, "device index above 63");
    std::lock_guard<std::mutex> lock(g_ws_mutex);
    if (!g_ws[dev]) {
        Workspace *w = new (std::nothrow) Workspace();
        if (!w) return fail(POS_ENOMEM, "host allocation failed");
        cudaError_t e = cudaStreamCreateWithFlags(&w->stream, cudaStreamNonBlocking);
        for (int i = 0; i < 3 && e == cudaSuccess; ++i) e = cudaEventCreate(&w->ev[i]);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&w->ev_lb, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&w->side, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&w->ev_fork, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&w->ev_join, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaMallocHost(&w->h_cnt, 64 * sizeof(unsigned long long));
        if (e != cudaSuccess) {
            delete w;
            return cuda_fail(e, "search workspace");
        }
        g_ws[dev] = w;
    }
    *out = g_ws[dev];
    return POS_OK;
}

struct Search {
    Workspace &ws;
    explicit Search(Workspace &w) : ws(w), stream(w.stream), ev(w.ev), d_slices(w.d_slices),
        d_feas(w.d_feas), d_batch(w.d_batch), d_inc(w.d_inc), d_ctr(w.d_ctr), d_best(w.d_best),
        d_feasible(w.d_feasible), d_leaves(w.d_leaves), d_roots(w.d_roots), d_root(w.d_root),
        d_front(w.d_front), d_defer(w.d_defer) {}
    const pos_problem *pb = nullptr;
    Handle hd{};
    Handle *h = &hd;
    cudaStream_t stream;
    cudaEvent_t (&ev)[3];
    int S = 0, L = 0, n_tp = 0;
    uint64_t n_map = 0;
    long long cap = 0;
    int grid_level = 0;
    const SliceSpace *sp = nullptr;  // the slices' identities, global-index order
    std::vector<SliceRec> slices;
    DevBuf &d_slices, &d_feas, &d_batch, &d_inc, &d_ctr, &d_best, &d_feasible, &d_leaves,
        &d_roots, &d_root;
    DevBuf (&d_front)[POS_MAX_STAGES + 1];
    DevBuf (&d_defer)[2 * (POS_MAX_STAGES + 1)];
    unsigned long long *ctr = nullptr;  // device counters, see search_impl
    unsigned long long *stats = nullptr;
    uint64_t launches = 0;
    double ms_expand = 0, ms_complete = 0, ms_leaf = 0, ms_bound = 0;
    double ms_depth[POS_MAX_STAGES] = {};
    uint64_t launches_depth[POS_MAX_STAGES] = {};
    uint64_t n_expand = 0, n_complete = 0, n_leaf = 0, n_bound = 0, reruns = 0;
    int cur_nb = 0;    // slots of the batch being enumerated
    Programs pg{};     // level programs of the schedule's short path
    size_t stage_off = 0;  // bytes of the staging area used by this search
    int n_vrows = 0;   // rows of the completion-bound tables (memory-feasible slices)
};

static pos_status validate_problem(const pos_problem *p) {
    if (!p) return fail(POS_EINVAL, "problem is NULL");
    if (p->schedule != POS_SCHED_1F1B && p->schedule != POS_SCHED_EAGER_1F1B &&
        p->schedule != POS_SCHED_INTERLEAVED_1F1B)
        return fail(POS_ENOTIMPL, "unknown schedule");
    if (p->schedule == POS_SCHED_INTERLEAVED_1F1B && p->ridge)
        return fail(POS_EINVAL, "layer-level (ridge) pruning is defined for 1F1B and Eager 1F1B "
                                "plans only");
    if (p->S < 1 || p->S > POS_MAX_STAGES) return fail(POS_EINVAL, "S must be in 1..16");
    if (p->S > p->tables.L) return fail(POS_EINVAL, "S > L");
    if (p->n_M < 1 || !p->M_list) return fail(POS_EINVAL, "empty M_list");
    for (int i = 0; i < p->n_M; ++i)
        if (p->M_list[i] < 1 || p->M_list[i] > 255) return fail(POS_EINVAL, "M out of 1..255");
    if (!p->tp_list) return fail(POS_EINVAL, "tp_list is NULL");
    if (p->placement != POS_PLACE_FREE && p->placement != POS_PLACE_EXACT &&
        p->placement != POS_PLACE_DEVICES)
        return fail(POS_EINVAL, "unknown placement rule");
    if (p->placement == POS_PLACE_DEVICES) {
        if (!p->D_list || p->n_D < 1) return fail(POS_EINVAL, "D_list is empty");
        for (int i = 0; i < p->n_D; ++i)
            if (p->D_list[i] < 1) return fail(POS_EINVAL, "D must be >= 1");
        for (int i = 0; i < p->tables.n_tp; ++i)
            if (p->tp_list[i] < 1) return fail(POS_EINVAL, "TP degrees must be >= 1");
        if (!p->type_counts) return fail(POS_EINVAL, "type_counts is NULL");
        for (int i = 0; i < p->tables.n_types; ++i)
            if (p->type_counts[i] < 0 || p->type_counts[i] > 65536)
                return fail(POS_EINVAL, "device counts must be in 0..65536");
        if (p->ridge)
            return fail(POS_EINVAL, "layer-level (ridge) pruning is not defined for per-stage TP");
        if (p->schedule == POS_SCHED_INTERLEAVED_1F1B && p->tables.n_tp > 4)
            return fail(POS_EINVAL, "Interleaved 1F1B with a TP index per device needs n_tp <= 4");
    } else {
        if (!p->dp_list) return fail(POS_EINVAL, "dp_list is NULL");
        for (int i = 0; i < p->tables.n_tp; ++i)
            if (p->dp_list[i] < 1) return fail(POS_EINVAL, "D must be >= 1");
    }
    if (p->placement == POS_PLACE_EXACT) {
        if (!p->type_counts) return fail(POS_EINVAL, "type_counts is NULL");
        int sum = 0;
        for (int i = 0; i < p->tables.n_types; ++i) {
            if (p->type_counts[i] < 0) return fail(POS_EINVAL, "negative type count");
            sum += p->type_counts[i];
        }
        if (sum != p->S) return fail(POS_EINVAL, "type_counts must sum to S");
    }
    if (p->warmup < 0) return fail(POS_EINVAL, "warmup < 0");
    if (p->prune < 0 || p->prune > 2) return fail(POS_EINVAL, "prune must be 0, 1 or 2");
    if (p->ridge != 0 && p->ridge != 1) return fail(POS_EINVAL, "ridge must be 0 or 1");
    if (p->frontier_cap < 0) return fail(POS_EINVAL, "frontier_cap < 0");
    if (p->schedule == POS_SCHED_INTERLEAVED_1F1B && (p->V < 2 || p->S * p->V > POS_MAX_STAGES))
        return fail(POS_EINVAL, "Interleaved 1F1B needs V >= 2 and S*V <= 16");
    return POS_OK;
}

// POS_PLACE_DEVICES: the class sequences of one D in lexicographic order,
// by a depth-first walk that keeps only prefixes with a completion: the
// remaining r stages can use up every type's remaining devices iff there
// are counts n_t (sum r) such that each remainder, in units of D, is a sum
// of exactly n_t TP degrees (reach[n][v]).
static pos_status device_sequences(const pos_problem *p, int units, int D,
                                   std::vector<uint8_t> &out, uint64_t *total) {
    const int T = p->tables.n_types, n_tp = p->tables.n_tp, K = T * n_tp;
    const uint64_t limit = 1ull << 22;
    int bud[POS_MAX_TYPES];
    int vmax = 0;
    for (int t = 0; t < T; ++t) {
        if (p->type_counts[t] % D != 0) return POS_OK;  // no stage split uses them up
        bud[t] = p->type_counts[t] / D;
        vmax = std::max(vmax, bud[t]);
    }
    // reach[v], bit n: v is a sum of exactly n TP degrees (n <= units)
    std::vector<uint32_t> reach((size_t)vmax + 1, 0u);
    reach[0] = 1u;
    for (int v = 1; v <= vmax; ++v)
        for (int j = 0; j < n_tp; ++j) {
            const int d = p->tp_list[j];
            if (d <= v) reach[v] |= (reach[v - d] << 1) & ((2u << units) - 1u);
        }
    // completes(r): the remaining budgets bud[] split over exactly r stages;
    // memoised over (r, budgets) when that table is small
    size_t states = (size_t)units + 1;
    int radix[POS_MAX_TYPES];
    for (int t = 0; t < T; ++t) {
        radix[t] = bud[t] + 1;
        states = states <= ((size_t)1 << 24) / (size_t)radix[t] ? states * radix[t] : 0;
        if (states == 0) break;
    }
    std::vector<uint8_t> memo(states, 0);  // 0 unknown, 1 no, 2 yes
    auto completes = [&](int r) -> bool {
        size_t key = 0;
        if (!memo.empty()) {
            for (int t = T - 1; t >= 0; --t) key = key * radix[t] + bud[t];
            key = key * (units + 1) + r;
            if (memo[key]) return memo[key] == 2;
        }
        uint32_t mask = 1u;  // bit n: n stages used by the types seen so far
        for (int t = 0; t < T && mask; ++t) {
            uint32_t next = 0, m = reach[bud[t]] & ((2u << r) - 1u);
            while (m) {
                next |= mask << __builtin_ctz(m);
                m &= m - 1u;
            }
            mask = next & ((2u << r) - 1u);
        }
        const bool ok = (mask >> r) & 1u;
        if (!memo.empty()) memo[key] = ok ? 2 : 1;
        return ok;
    };
    if (!completes(units)) return POS_OK;
    uint8_t seq[POS_MAX_STAGES];
    int k_at[POS_MAX_STAGES];
    int u = 0;
    k_at[0] = -1;
    while (u >= 0) {  // iterative depth-first walk, classes in ascending order
        if (u == units - 1) {
            // the last stage takes what is left: the one type with a budget
            // left, with a TP degree equal to it (the prefix was kept only if
            // such a class exists)
            int t = 0;
            while (t < T && bud[t] == 0) ++t;
            for (int j = 0; t < T && j < n_tp; ++j) {
                if (p->tp_list[j] != bud[t]) continue;
                seq[u] = (uint8_t)(t * n_tp + j);
                const size_t at = out.size();
                out.resize(at + units);
                std::memcpy(out.data() + at, seq, units);
                if (++*total > limit) return fail(POS_EINVAL, "more than 2^22 class sequences");
            }
            --u;  // the parent's class is undone on its next step
            continue;
        }
        int k = k_at[u] + 1;
        if (k_at[u] >= 0) bud[k_at[u] / n_tp] += p->tp_list[k_at[u] % n_tp];  // undo
        for (; k < K; ++k) {
            const int t = k / n_tp, d = p->tp_list[k % n_tp];
            if (bud[t] < d) continue;
            bud[t] -= d;
            if (completes(units - u - 1)) break;
            bud[t] += d;
        }
        if (k == K) {  // no further class at this position: back up
            k_at[u] = -1;
            --u;
            continue;
        }
        k_at[u] = k;
        seq[u] = (uint8_t)k;
        k_at[++u] = -1;
    }
    return POS_OK;
}

pos_status build_slice_space(const pos_problem *p, int units, SliceSpace &sp) {
    const int T = p->tables.n_types, n_tp = p->tables.n_tp;
    const uint64_t limit = 1ull << 22;
    sp = SliceSpace();
    sp.units = units;
    sp.per_stage = p->placement == POS_PLACE_DEVICES;
    sp.n_grp = sp.per_stage ? p->n_D : n_tp;
    if (sp.per_stage) {
        uint64_t total = 0;
        sp.seqs.resize(p->n_D);
        for (int g = 0; g < p->n_D; ++g) {
            POS_TRY(device_sequences(p, units, p->D_list[g], sp.seqs[g], &total));
            sp.D.push_back(p->D_list[g]);
        }
    } else {
        sp.seqs.resize(1);
        std::vector<uint8_t> &places = sp.seqs[0];
        std::vector<uint8_t> seq;
        if (p->placement == POS_PLACE_EXACT) {
            // the distinct permutations of the multiset, in lexicographic order
            int sum = 0;
            for (int ty = 0; ty < T; ++ty) sum += p->type_counts[ty];
            if (sum != units) return fail(POS_EINVAL, "type_counts must sum to S");
            for (int ty = 0; ty < T; ++ty) seq.insert(seq.end(), p->type_counts[ty], (uint8_t)ty);
            do {
                places.insert(places.end(), seq.begin(), seq.end());
                if (places.size() > limit * units) return fail(POS_EINVAL, "too many placements");
            } while (std::next_permutation(seq.begin(), seq.end()));
        } else {
            // every sequence in T^S, as an odometer (last stage fastest)
            double total = 1;
            for (int x = 0; x < units; ++x) total *= T;
            if (total > (double)limit) return fail(POS_EINVAL, "too many placements");
            seq.assign(units, 0);
            for (;;) {
                places.insert(places.end(), seq.begin(), seq.end());
                int x = units - 1;
                while (x >= 0 && seq[x] == T - 1) seq[x--] = 0;
                if (x < 0) break;
                seq[x]++;
            }
        }
        for (int g = 0; g < n_tp; ++g) sp.D.push_back(p->dp_list[g]);
    }
    sp.grp_off.assign(sp.n_grp + 1, 0);
    for (int g = 0; g < sp.n_grp; ++g) sp.grp_off[g + 1] = sp.grp_off[g] + sp.n_seq(g);
    sp.per_m = sp.grp_off[sp.n_grp];
    if ((uint64_t)p->n_M * sp.per_m > limit) return fail(POS_EINVAL, "more than 2^22 slices");
    return POS_OK;
}

void plan_slice_fields(const pos_problem *p, const SliceSpace &sp, uint64_t ord, pos_plan *out) {
    int mi = 0, g = 0;
    uint64_t pr = 0;
    sp.decode(ord, &mi, &g, &pr);
    const int n_tp = p->tables.n_tp;
    out->m_idx = mi;
    out->M = p->M_list[mi];
    out->D = sp.D[g];
    out->place_rank = pr;
    out->tp_idx = sp.per_stage ? -1 : g;
    out->tp = sp.per_stage ? -1 : p->tp_list[g];
    out->d_idx = sp.per_stage ? g : -1;
    for (int x = 0; x < POS_MAX_STAGES; ++x) {
        const int k = x < sp.units ? sp.cls(g, pr, x, n_tp) : -1;
        out->type[x] = k < 0 ? -1 : k / n_tp;
        out->tp_stage[x] = k < 0 ? -1 : k % n_tp;
    }
}

// Size limits of the search space that do not need the slices, checked on
// the host before the device is touched: the global index (slices x
// compositions) below 2^64 and the objective scale (lcm of every D*M) below
// 2^32.
static pos_status validate_space(const pos_problem *p, const SliceSpace &sp) {
    const int S = p->S;
    const uint64_t n_slices = (uint64_t)p->n_M * sp.per_m;
    const int J = p->schedule == POS_SCHED_INTERLEAVED_1F1B ? S * p->V : S;
    const uint64_t n_map = host_binom(p->tables.L - 1, J - 1);
    if (n_map && n_slices > ~0ull / n_map) return fail(POS_EINVAL, "global index overflows");
    uint64_t Q = 1;
    for (int i = 0; i < p->n_M; ++i)
        for (int32_t D : sp.D) {
            const uint64_t dm = (uint64_t)D * p->M_list[i];
            Q = Q / gcd64(Q, dm) * dm;
            if (Q >= (1ull << 32)) return fail(POS_EINVAL, "lcm of D*M reaches 2^32");
        }
    return POS_OK;
}

// Q = lcm of every D*M: T * Q / (D*M) orders plans by time per sample
static uint64_t objective_scale(const pos_problem *p, const SliceSpace &sp) {
    uint64_t Q = 1;
    for (int i = 0; i < p->n_M; ++i)
        for (int32_t D : sp.D) {
            const uint64_t dm = (uint64_t)D * p->M_list[i];
            Q = Q / gcd64(Q, dm) * dm;
        }
    return Q;
}

static pos_status sync_read(Search &s, void *dst, const void *src, size_t bytes) {
    if (bytes <= 64 * sizeof(unsigned long long)) {  // small reads through pinned memory
        POS_CUDA(cudaMemcpyAsync(s.ws.h_cnt, src, bytes, cudaMemcpyDeviceToHost, s.stream));
        POS_CUDA(cudaStreamSynchronize(s.stream));
        std::memcpy(dst, s.ws.h_cnt, bytes);
        return POS_OK;
    }
    if (bytes > s.ws.h_read_cap) {  // no copy is in flight: the old area can go
        if (s.ws.h_read) cudaFreeHost(s.ws.h_read);
        s.ws.h_read = nullptr;
        s.ws.h_read_cap = 0;
        POS_CUDA(cudaMallocHost(&s.ws.h_read, bytes + bytes / 2));
        s.ws.h_read_cap = bytes + bytes / 2;
    }
    POS_CUDA(cudaMemcpyAsync(s.ws.h_read, src, bytes, cudaMemcpyDeviceToHost, s.stream));
    POS_CUDA(cudaStreamSynchronize(s.stream));
    std::memcpy(dst, s.ws.h_read, bytes);
    return POS_OK;
}

// Several device-to-host copies behind one synchronisation (each
// synchronisation leaves the device idle for a host round trip).
struct ReadPart {
    void *dst;
    const void *src;
    size_t bytes;
};
static pos_status sync_read_many(Search &s, const ReadPart *parts, int n) {
    size_t total = 0;
    for (int i = 0; i < n; ++i) total += (parts[i].bytes + 15) & ~(size_t)15;
    if (total > s.ws.h_read_cap) {  // no copy is in flight: the old area can go
        if (s.ws.h_read) cudaFreeHost(s.ws.h_read);
        s.ws.h_read = nullptr;
        s.ws.h_read_cap = 0;
        POS_CUDA(cudaMallocHost(&s.ws.h_read, total + total / 2));
        s.ws.h_read_cap = total + total / 2;
    }
    size_t off = 0;
    for (int i = 0; i < n; ++i) {
        POS_CUDA(cudaMemcpyAsync(s.ws.h_read + off, parts[i].src, parts[i].bytes,
                                 cudaMemcpyDeviceToHost, s.stream));
        off += (parts[i].bytes + 15) & ~(size_t)15;
    }
    POS_CUDA(cudaStreamSynchronize(s.stream));
    off = 0;
    for (int i = 0; i < n; ++i) {
        std::memcpy(parts[i].dst, s.ws.h_read + off, parts[i].bytes);
        off += (parts[i].bytes + 15) & ~(size_t)15;
    }
    return POS_OK;
}

// Enqueues an upload through the workspace's pinned staging area (an
// upload straight from pageable memory makes the host wait while the
// driver stages it).  The area is sized at the start of a search and only
// reused after that search has synchronised; if it is full the copy goes
// from pageable memory.
static pos_status upload(Search &s, void *dst, const void *src, size_t bytes) {
    const size_t off = (s.stage_off + 255) & ~(size_t)255;
    if (off + bytes > s.ws.h_stage_cap) {
        POS_CUDA(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, s.stream));
        return POS_OK;
    }
    std::memcpy(s.ws.h_stage + off, src, bytes);
    POS_CUDA(cudaMemcpyAsync(dst, s.ws.h_stage + off, bytes, cudaMemcpyHostToDevice, s.stream));
    s.stage_off = off + bytes;
    return POS_OK;
}

static pos_status reserve_stage(Search &s, size_t bytes) {
    s.stage_off = 0;
    if (bytes <= s.ws.h_stage_cap) return POS_OK;
    if (s.ws.h_stage) cudaFreeHost(s.ws.h_stage);  // the previous search has synchronised
    s.ws.h_stage = nullptr;
    s.ws.h_stage_cap = 0;
    POS_CUDA(cudaMallocHost(&s.ws.h_stage, bytes));
    s.ws.h_stage_cap = bytes;
    return POS_OK;
}

static pos_status ensure_depth(Search &s, int depth) {
    POS_CUDA(s.d_front[depth].reserve(sizeof(Prefix) * (size_t)s.cap));
    return POS_OK;
}

static pos_status ensure_defer(Search &s, int depth, long long groups) {
    const size_t b = sizeof(uint32_t) * (size_t)std::max<long long>(groups, 1);
    POS_CUDA(s.d_defer[2 * depth].reserve(b));
    POS_CUDA(s.d_defer[2 * depth + 1].reserve(b));
    return POS_OK;
}

static ExpandParams base_params(Search &s, const SliceRec *batch, int M) {
    ExpandParams p;
    std::memset(&p, 0, sizeof(p));
    p.S = s.S;
    p.M = M;
    p.prune = s.pb->prune;
    p.ridge = s.pb->ridge;
    p.slices = batch;
    p.feas = static_cast<const uint4 *>(s.d_feas.p);
    p.lim = static_cast<const uint8_t *>(s.ws.d_lim.p);
    p.vb = static_cast<const int2 *>(s.ws.d_vb.p);
    p.nb = s.cur_nb;
    p.n_vrows = s.n_vrows;
    p.cap = (unsigned long long)s.cap;
    p.inc = static_cast<const Key128 *>(s.d_inc.p);
    p.stats = s.stats;
    // level kernels read only the timing tables: stage that part alone
    p.blob = static_cast<const unsigned char *>(s.h->d_blob) + s.h->lay.off_Pf;
    p.lay = timing_layout(s.h->lay);
    return p;
}

static pos_status run_leaves(Search &s, const Leaf *leaves, unsigned long long *count,
                             const SliceRec *table, int M, unsigned long long *slice_best,
                             cudaStream_t stream = nullptr) {
    LeafParams lp;
    lp.leaves = leaves;
    lp.count = count;
    lp.cap = (unsigned long long)s.cap;
    lp.slices = table;
    lp.M = M;
    lp.n_map = s.n_map;
    lp.inc = static_cast<Key128 *>(s.d_inc.p);
    lp.stats = s.stats;
    lp.slice_best = slice_best;
    lp.blob = s.h->d_blob;
    lp.lay = s.h->lay;
    s.launches++;
    lp.pg = s.pg;
    lp.ridge = s.pb->ridge;
    lp.cas_limit = s.pb->cas_limit == 0 ? kCasLimit : std::max(0, s.pb->cas_limit);
    // as many blocks as the launch bounds keep resident on every SM
    const int path = path_of(s.pb->schedule, s.S, M);
    return launch_leaf(s.S, path, lp, leaf_min_blocks(s.S, path) * sm_count(),
                       stream ? stream : s.stream);
}

template <bool COMPLETE, int X>
static pos_status launch_level_t(const ExpandParams &p, int grid, int smem, cudaStream_t st) {
    auto kern = level_kernel<COMPLETE, X>;
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(kern), smem));
    POS_CUDA(launch_dependent(kern, grid, kThreads, smem, st, p));
    return POS_OK;
}

template <int... X>
static pos_status launch_level_x(bool complete, int x, const ExpandParams &p, int grid, int smem,
                                 cudaStream_t st, std::integer_sequence<int, X...>) {
    pos_status r = fail(POS_EINVAL, "depth out of range");
    ((x == X ? (r = complete ? launch_level_t<true, X>(p, grid, smem, st)
                             : launch_level_t<false, X>(p, grid, smem, st),
                0)
             : 0),
     ...);
    return r;
}

// parents at depth x = 0..14 (completion: x = S-2)
static pos_status launch_level(bool complete, int x, const ExpandParams &p, int grid, int smem,
                               cudaStream_t st) {
    return launch_level_x(complete, x, p, grid, smem, st, std::make_integer_sequence<int, 15>{});
}

// Enumerate everything below the prefixes in[0..n_in) (depth x).
static pos_status process(Search &s, const SliceRec *batch, int M, int x, const Prefix *in,
                          long long n_in) {
    const int S = s.S;
    const bool last = (x == S - 2);
    const long long all_groups = (n_in + 31) / 32;
    pos_status st = ensure_defer(s, x, all_groups);
    if (st != POS_OK) return st;
    if (!last && (st = ensure_depth(s, x + 1)) != POS_OK) return st;
    // (children count, deferred groups) of this depth, adjacent: one read
    unsigned long long *out_count = s.ctr + 2 * x;
    unsigned long long *n_def = out_count + 1;
    const uint32_t *work = nullptr;
    long long n_work = all_groups;
    int flip = 0;
    for (;;) {
        POS_CUDA(cudaMemsetAsync(out_count, 0, 2 * sizeof(unsigned long long), s.stream));
        ExpandParams p = base_params(s, batch, M);
        p.exact = 1;
        p.in = in;
        p.n_in = n_in;
        p.groups = work;
        p.n_groups = n_work;
        p.x = x;
        p.out = last ? nullptr : static_cast<Prefix *>(s.d_front[x + 1].p);
        p.leaves = last ? static_cast<Leaf *>(s.d_leaves.p) : nullptr;
        p.out_count = out_count;
        p.deferred = static_cast<uint32_t *>(s.d_defer[2 * x + flip].p);
        p.n_deferred = n_def;
        const int smem = p.lay.bytes;
        const long long blocks_needed = (n_work * 32 + kThreads - 1) / kThreads;
        const int grid = (int)std::max<long long>(1, std::min<long long>(blocks_needed,
                                                                         s.grid_level));
        s.launches++;
        const bool prof = s.pb->profile != 0;
        if (prof) POS_CUDA(cudaEventRecord(s.ev[0], s.stream));
        if ((st = launch_level(last, x, p, grid, smem, s.stream)) != POS_OK) return st;
        (last ? s.n_complete : s.n_expand)++;
        s.launches_depth[x]++;
        if (prof) POS_CUDA(cudaEventRecord(s.ev[1], s.stream));
        if (last) {
            // evaluate the leaves that fit; the count stays on the device
            if ((st = run_leaves(s, p.leaves, out_count, batch, M, nullptr)) != POS_OK) return st;
            s.n_leaf++;
            if (prof) POS_CUDA(cudaEventRecord(s.ev[2], s.stream));
        }
        unsigned long long cnt[2];
        if ((st = sync_read(s, cnt, out_count, sizeof(cnt))) != POS_OK) return st;
        if (prof) {
            float ms_k = 0;
            POS_CUDA(cudaEventElapsedTime(&ms_k, s.ev[0], s.ev[1]));
            s.ms_depth[x] += ms_k;
            if (last) {
                s.ms_complete += ms_k;
                float ms_l = 0;
                POS_CUDA(cudaEventElapsedTime(&ms_l, s.ev[1], s.ev[2]));
                s.ms_leaf += ms_l;
            } else {
                s.ms_expand += ms_k;
            }
        }
        if (!last) {
            const long long n_out = (long long)std::min<unsigned long long>(cnt[0], s.cap);
            if (n_out > 0) {
                st = process(s, batch, M, x + 1, static_cast<const Prefix *>(s.d_front[x + 1].p),
                             n_out);
                if (st != POS_OK) return st;
            }
        }
        if (cnt[1] == 0) break;
        if ((long long)cnt[1] >= n_work)
            return fail(POS_ENOMEM, "frontier capacity too small to make progress");
        work = static_cast<const uint32_t *>(s.d_defer[2 * x + flip].p);
        n_work = (long long)cnt[1];
        flip ^= 1;
    }
    return POS_OK;
}

static double ms_since(std::chrono::steady_clock::time_point t0) {
    return std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0)
        .count();
}

static pos_status search_impl(Search &s, pos_plan *out, pos_search_stats *stats) {
    const auto t_start = std::chrono::steady_clock::now();
    const pos_problem *p = s.pb;
    pos_status st = validate_problem(p);
    if (st != POS_OK) return st;
    s.S = p->S;
    s.L = p->tables.L;
    s.n_tp = p->tables.n_tp;
    s.n_map = host_binom(s.L - 1, s.S - 1);
    // a warp group of 32 parents has at most 32*L children, so a buffer of
    // at least that size always accepts the first group of a pass: every
    // deferral pass makes progress
    s.cap = p->frontier_cap > 0 ? p->frontier_cap : (1ll << 24);
    s.cap = std::max<long long>(s.cap, 32LL * s.L);
    const SliceSpace &sp = *s.sp;
    const uint64_t n_slices64 = (uint64_t)p->n_M * sp.per_m;
    if (n_slices64 > (1ull << 22)) return fail(POS_EINVAL, "more than 2^22 slices");
    const int n_slices = (int)n_slices64;
    if (s.n_map && n_slices64 > ~0ull / s.n_map) return fail(POS_EINVAL, "global index overflows");
    if ((st = schedule_programs(p->schedule, &s.pg)) != POS_OK) return st;
    // after the side-stream work of an earlier search (which may have
    // returned early), since this one reuses its buffers
    POS_CUDA(cudaStreamWaitEvent(s.stream, s.ws.ev_join, 0));
    // pinned staging for this search's uploads (tables, slice records, lists)
    if ((st = reserve_stage(s, ((size_t)256 << 10) + (size_t)n_slices * 320 +
                                   (size_t)p->n_M * 16)) != POS_OK)
        return st;
    {
        std::vector<unsigned char> host;
        st = build_blob(&p->tables, p->schedule, host, s.hd.lay, s.hd.guard_A, s.hd.guard_D,
                        s.hd.guard_P);
        if (st != POS_OK) return st;
        POS_CUDA(cudaGetDevice(&s.hd.device));
        POS_CUDA(s.ws.blob.reserve(s.hd.lay.bytes));
        s.hd.d_blob = s.ws.blob.p;
        POS_TRY(upload(s, s.hd.d_blob, host.data(), s.hd.lay.bytes));
        if ((st = launch_prefix_rows(s.hd.d_blob, s.hd.lay, s.stream)) != POS_OK) return st;
    }
    // overflow guard for every M (Sec. 4.1 path-length bound)
    for (int i = 0; i < p->n_M; ++i)
        if (guard_trips(s.h->guard_A, s.h->guard_D, s.h->guard_P, s.S, p->M_list[i]))
            return fail(POS_EOVERFLOW, "makespan bound reaches 2^31 for some M");
    // objective scale: Q = lcm(D*M); T*Q/(D*M) orders plans by time per sample
    const uint64_t Q = objective_scale(p, sp);
    s.slices.resize(n_slices);
    {
        uint64_t ord = 0;
        for (int mi = 0; mi < p->n_M; ++mi)
            for (int g = 0; g < sp.n_grp; ++g)
                for (uint64_t pr = 0; pr < sp.n_seq(g); ++pr, ++ord) {
                    SliceRec &r = s.slices[ord];
                    std::memset(&r, 0, sizeof(r));
                    r.ordinal = ord;
                    r.M = p->M_list[mi];
                    r.scale = Q / ((uint64_t)sp.D[g] * p->M_list[mi]);
                    r.gid = (uint32_t)ord;
                    r.vslot = (uint32_t)ord;  // bound-table row when every slice has one
                    for (int x = 0; x < s.S; ++x) r.cls[x] = (uint8_t)sp.cls(g, pr, x, s.n_tp);
                }
    }
    const int smem = s.h->lay.bytes;
    int per_sm = 0;
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(level_kernel<false, 0>), smem));
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(feas_kernel), smem));
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(bound_kernel), smem));
    POS_TRY(blocks_per_sm(reinterpret_cast<const void *>(level_kernel<false, 0>), kThreads,
                          timing_layout(s.h->lay).bytes, &per_sm));
    s.grid_level = std::max(1, per_sm) * sm_count();

    POS_CUDA(s.d_slices.reserve(sizeof(SliceRec) * n_slices));
    POS_CUDA(s.d_feas.reserve(sizeof(uint4) * (size_t)n_slices * (s.S + 1)));
    POS_CUDA(s.ws.d_lim.reserve((size_t)n_slices * s.S * 128));
    POS_CUDA(s.d_inc.reserve(sizeof(Key128)));
    POS_CUDA(s.d_ctr.reserve(sizeof(unsigned long long) * 128));
    POS_CUDA(s.d_best.reserve(sizeof(unsigned long long) * n_slices));
    POS_CUDA(s.d_leaves.reserve(sizeof(Leaf) * (size_t)s.cap));
    s.ctr = static_cast<unsigned long long *>(s.d_ctr.p);
    s.stats = s.ctr + 40;  // ctr[0..33]: per-depth counters, ctr[36]: leaf count
    static_assert(40 + kStCount <= 128, "counter block");
    POS_TRY(upload(s, s.d_slices.p, s.slices.data(), sizeof(SliceRec) * n_slices));
    POS_CUDA(cudaMemsetAsync(s.d_inc.p, 0xff, sizeof(Key128), s.stream));
    POS_CUDA(cudaMemsetAsync(s.d_ctr.p, 0, sizeof(unsigned long long) * 128, s.stream));
    POS_CUDA(cudaMemsetAsync(s.d_best.p, 0xff, sizeof(unsigned long long) * n_slices, s.stream));
    const SliceRec *d_all = static_cast<const SliceRec *>(s.d_slices.p);
    DevBuf &d_root = s.d_root;
    POS_CUDA(d_root.reserve(n_slices));
    {
        // the memory tables alone (Pw, Pa, cap) are staged per block
        const BlobLayout ml = memory_layout(s.h->lay);
        POS_TRY(ensure_smem(reinterpret_cast<const void *>(feas_kernel), ml.bytes));
        feas_kernel<<<std::min(n_slices, 16 * sm_count()), 128, ml.bytes, s.stream>>>(
            d_all, n_slices, s.S, static_cast<uint4 *>(s.d_feas.p),
            static_cast<uint8_t *>(s.ws.d_lim.p), static_cast<uint8_t *>(d_root.p),
            static_cast<const unsigned char *>(s.h->d_blob) + s.h->lay.off_Pw, ml, s.stats);
    }
    POS_CUDA(cudaGetLastError());
    s.launches++;
    std::vector<uint8_t> root(n_slices);
    std::vector<std::vector<uint32_t>> feas_by_m(p->n_M);  // feasible slices per M index
    uint64_t n_feasible = 0;
    auto list_feasible = [&]() {
        for (int i = 0; i < n_slices; ++i)
            if (root[i]) {
                feas_by_m[i / sp.per_m].push_back((uint32_t)i);
                ++n_feasible;
            }
    };
    uint64_t warm_evals = 0;
    // prune mode 2 with tables for every slice small enough (up to 256 MB):
    // the completion bounds of all slices right after the feasibility kernel
    // (the infeasible ones skip out), no host round trip in between; the
    // root bits come back with the root bounds
    const bool bound_all = p->prune == 2 && (uint64_t)n_slices * s.S * 1024 <= (256ull << 20);
    if (bound_all) {
        s.n_vrows = n_slices;  // table row = slice index (vslot = gid)
        POS_CUDA(s.ws.d_vb.reserve(sizeof(int2) * 128 * (size_t)s.S * n_slices));
        POS_CUDA(s.ws.d_greedy.reserve(sizeof(Leaf) * n_slices));
        POS_CUDA(s.ws.d_lb.reserve(sizeof(unsigned long long) * n_slices));
        const BlobLayout tl = timing_layout(s.h->lay);
        POS_TRY(ensure_smem(reinterpret_cast<const void *>(bound_kernel), tl.bytes));
        if (p->profile) POS_CUDA(cudaEventRecord(s.ev[0], s.stream));
        POS_CUDA(launch_dependent(
            bound_kernel, std::min(n_slices, 8 * sm_count()), kBoundThreads, tl.bytes, s.stream,
            d_all, static_cast<const uint32_t *>(nullptr),
            static_cast<const uint8_t *>(d_root.p), n_slices, s.S,
            static_cast<const uint8_t *>(s.ws.d_lim.p), static_cast<int2 *>(s.ws.d_vb.p),
            static_cast<Leaf *>(s.ws.d_greedy.p), static_cast<unsigned long long *>(s.ws.d_lb.p),
            static_cast<const void *>(static_cast<const unsigned char *>(s.h->d_blob) +
                                      s.h->lay.off_Pf),
            tl, s.stats));
        if (p->profile) POS_CUDA(cudaEventRecord(s.ev[1], s.stream));
        s.launches++;
        s.n_bound++;
        // the greedy plans of each M index (holes for the infeasible slices),
        // on the side stream: they only lower the incumbent, which the
        // enumeration reads after the join below
        std::vector<unsigned long long> gc(p->n_M, (unsigned long long)sp.per_m);
        POS_CUDA(s.ws.d_wcnt.reserve(sizeof(unsigned long long) * p->n_M));
        POS_TRY(upload(s, s.ws.d_wcnt.p, gc.data(), sizeof(unsigned long long) * p->n_M));
        POS_CUDA(cudaEventRecord(s.ws.ev_fork, s.stream));
        POS_CUDA(cudaStreamWaitEvent(s.ws.side, s.ws.ev_fork, 0));
        for (int mi = 0; mi < p->n_M && st == POS_OK; ++mi)
            st = run_leaves(s, static_cast<const Leaf *>(s.ws.d_greedy.p) + mi * sp.per_m,
                            static_cast<unsigned long long *>(s.ws.d_wcnt.p) + mi, d_all,
                            p->M_list[mi], static_cast<unsigned long long *>(s.d_best.p),
                            s.ws.side);
        // recorded also after a failed launch: the next search waits on it
        POS_CUDA(cudaEventRecord(s.ws.ev_join, s.ws.side));
        if (st != POS_OK) return st;
        if ((size_t)n_slices > s.ws.h_lb_cap) {
            POS_CUDA(cudaStreamSynchronize(s.stream));  // no copy into the old area in flight
            if (s.ws.h_lb) cudaFreeHost(s.ws.h_lb);
            s.ws.h_lb = nullptr;
            s.ws.h_lb_cap = 0;
            POS_CUDA(cudaMallocHost(&s.ws.h_lb, sizeof(unsigned long long) * n_slices));
            s.ws.h_lb_cap = (size_t)n_slices;
        }
        const ReadPart parts[2] = {{root.data(), d_root.p, (size_t)n_slices},
                                   {s.ws.h_lb, s.ws.d_lb.p, sizeof(unsigned long long) * n_slices}};
        if ((st = sync_read_many(s, parts, 2)) != POS_OK) return st;
        list_feasible();
        for (int mi = 0; mi < p->n_M; ++mi) warm_evals += feas_by_m[mi].size();
    } else {
        if ((st = sync_read(s, root.data(), d_root.p, n_slices)) != POS_OK) return st;
        list_feasible();
    }
    const double ms_setup = ms_since(t_start);

    // prune mode 2: completion-bound tables of every memory-feasible slice
    // (one launch), and each slice's argmin completion as a warm-up plan
    const auto t_warm = std::chrono::steady_clock::now();
    std::vector<size_t> feas_off(p->n_M + 1, 0);  // first row of each M index
    for (int mi = 0; mi < p->n_M; ++mi) feas_off[mi + 1] = feas_off[mi] + feas_by_m[mi].size();
    if (p->prune == 2 && n_feasible > 0 && !bound_all) {
        std::vector<uint32_t> rows;
        rows.reserve(n_feasible);
        for (int mi = 0; mi < p->n_M; ++mi)
            for (uint32_t g : feas_by_m[mi]) {
                s.slices[g].vslot = (uint32_t)rows.size();
                rows.push_back(g);
            }
        s.n_vrows = (int)rows.size();
        POS_CUDA(s.ws.d_rows.reserve(sizeof(uint32_t) * rows.size()));
        POS_CUDA(s.ws.d_vb.reserve(sizeof(int2) * 128 * (size_t)s.S * rows.size()));
        POS_CUDA(s.ws.d_greedy.reserve(sizeof(Leaf) * rows.size()));
        POS_CUDA(s.ws.d_lb.reserve(sizeof(unsigned long long) * n_slices));
        POS_TRY(upload(s, s.ws.d_rows.p, rows.data(), sizeof(uint32_t) * rows.size()));
        POS_TRY(upload(s, s.d_slices.p, s.slices.data(), sizeof(SliceRec) * n_slices));
        const BlobLayout tl = timing_layout(s.h->lay);
        POS_TRY(ensure_smem(reinterpret_cast<const void *>(bound_kernel), tl.bytes));
        if (p->profile) POS_CUDA(cudaEventRecord(s.ev[0], s.stream));
        bound_kernel<<<(int)std::min<size_t>(rows.size(), 8 * sm_count()), kBoundThreads, tl.bytes,
                       s.stream>>>(
            d_all, static_cast<const uint32_t *>(s.ws.d_rows.p), nullptr, (int)rows.size(), s.S,
            static_cast<const uint8_t *>(s.ws.d_lim.p), static_cast<int2 *>(s.ws.d_vb.p),
            static_cast<Leaf *>(s.ws.d_greedy.p), static_cast<unsigned long long *>(s.ws.d_lb.p),
            static_cast<const unsigned char *>(s.h->d_blob) + s.h->lay.off_Pf, tl, s.stats);
        POS_CUDA(cudaGetLastError());
        if (p->profile) POS_CUDA(cudaEventRecord(s.ev[1], s.stream));
        s.launches++;
        s.n_bound++;
        // the root bounds order the slices: their copy to the host is queued
        // here and waited for alone, so the warm-up kernels queued next run
        // while the host plans the batches
        if ((size_t)n_slices > s.ws.h_lb_cap) {
            POS_CUDA(cudaStreamSynchronize(s.stream));  // no copy into the old area in flight
            if (s.ws.h_lb) cudaFreeHost(s.ws.h_lb);
            s.ws.h_lb = nullptr;
            s.ws.h_lb_cap = 0;
            POS_CUDA(cudaMallocHost(&s.ws.h_lb, sizeof(unsigned long long) * n_slices));
            s.ws.h_lb_cap = (size_t)n_slices;
        }
        POS_CUDA(cudaMemcpyAsync(s.ws.h_lb, s.ws.d_lb.p, sizeof(unsigned long long) * n_slices,
                                 cudaMemcpyDeviceToHost, s.stream));
        POS_CUDA(cudaEventRecord(s.ws.ev_lb, s.stream));
        // counts of the greedy plans per M index, then one leaf launch each
        std::vector<unsigned long long> gc(p->n_M);
        for (int mi = 0; mi < p->n_M; ++mi) gc[mi] = feas_by_m[mi].size();
        POS_CUDA(s.ws.d_wcnt.reserve(sizeof(unsigned long long) * p->n_M));
        POS_TRY(upload(s, s.ws.d_wcnt.p, gc.data(), sizeof(unsigned long long) * p->n_M));
        for (int mi = 0; mi < p->n_M; ++mi) {
            if (gc[mi] == 0) continue;
            if ((st = run_leaves(s, static_cast<const Leaf *>(s.ws.d_greedy.p) + feas_off[mi],
                                 static_cast<unsigned long long *>(s.ws.d_wcnt.p) + mi, d_all,
                                 p->M_list[mi], static_cast<unsigned long long *>(s.d_best.p))) !=
                POS_OK)
                return st;
            warm_evals += gc[mi];
        }
    }
    // warm-up sampling (Sec. 4.2.3), split over the M values in proportion
    // to their feasible slices
    if (p->warmup > 0 && n_feasible > 0) {
        POS_CUDA(s.d_feasible.reserve(sizeof(uint32_t) * n_feasible));
        for (int mi = 0; mi < p->n_M; ++mi) {
            const auto &fl = feas_by_m[mi];
            if (fl.empty()) continue;
            const long long n_s = std::min<long long>(
                s.cap, std::max<long long>(1, (long long)p->warmup * (long long)fl.size() /
                                                  (long long)n_feasible));
            POS_TRY(upload(s, s.d_feasible.p, fl.data(), sizeof(uint32_t) * fl.size()));
            sample_kernel<<<(int)std::min<long long>((n_s + 255) / 256, 4 * sm_count()), 256, 0,
                            s.stream>>>(
                d_all, static_cast<const uint32_t *>(s.d_feasible.p), (int)fl.size(), (int)n_s,
                s.S, p->seed + 0x632BE59BD9B4E019ull * (uint64_t)mi,
                static_cast<const uint4 *>(s.d_feas.p), static_cast<const uint8_t *>(s.ws.d_lim.p),
                static_cast<Leaf *>(s.d_leaves.p), s.L);
            POS_CUDA(cudaGetLastError());
            s.launches++;
            const unsigned long long cnt = (unsigned long long)n_s;
            POS_TRY(upload(s, s.ctr + 36, &cnt, 8));
            if ((st = run_leaves(s, static_cast<const Leaf *>(s.d_leaves.p), s.ctr + 36, d_all,
                                 p->M_list[mi], static_cast<unsigned long long *>(s.d_best.p))) !=
                POS_OK)
                return st;
            warm_evals += (uint64_t)n_s;
        }
    }
    // the greedy plans' makespans (side stream) before anything that reads
    // the incumbent or the per-slice bests
    POS_CUDA(cudaStreamWaitEvent(s.stream, s.ws.ev_join, 0));
    // slice order: with the completion bounds, by each slice's root lower
    // bound (the slice most likely to hold the optimum first), waiting for
    // their copy only; otherwise by the best warm-up plan of the slice,
    // after the warm-up
    const bool by_bound = p->prune == 2 && n_feasible > 0;
    std::vector<unsigned long long> key(n_slices);
    if (by_bound) {
        if (!bound_all) POS_CUDA(cudaEventSynchronize(s.ws.ev_lb));  // else read already
        std::memcpy(key.data(), s.ws.h_lb, sizeof(unsigned long long) * n_slices);
    } else if ((st = sync_read(s, key.data(), s.d_best.p,
                               sizeof(unsigned long long) * n_slices)) != POS_OK) {
        return st;
    }
    if (p->profile && s.n_bound) {
        float ms_b = 0;
        POS_CUDA(cudaEventElapsedTime(&ms_b, s.ev[0], s.ev[1]));
        s.ms_bound += ms_b;
    }
    const double ms_warm = ms_since(t_warm);

    // batches of slices, most promising first
    const auto t_search = std::chrono::steady_clock::now();
    struct Group {
        int mi;
        unsigned long long best;
    };
    std::vector<Group> groups;
    for (int mi = 0; mi < p->n_M; ++mi) {
        if (feas_by_m[mi].empty()) continue;
        auto &fl = feas_by_m[mi];
        std::stable_sort(fl.begin(), fl.end(),
                         [&](uint32_t a, uint32_t b) { return key[a] < key[b]; });
        groups.push_back({mi, key[fl[0]]});
    }
    std::stable_sort(groups.begin(), groups.end(),
                     [](const Group &a, const Group &b) { return a.best < b.best; });
    // every batch, in processing order, uploaded once
    struct Batch {
        int M;
        size_t off, nb;
    };
    std::vector<SliceRec> ordered;
    std::vector<Batch> batches;
    size_t max_nb = 1;
    for (const Group &g : groups) {
        const auto &fl = feas_by_m[g.mi];
        // Eq. 2 alone: eight batches, best first, so that the incumbent
        // improves between them.  With the completion bounds the warm-up
        // already holds each slice's argmin completion and every launch
        // costs more than a little extra pruning saves: a first batch of
        // the 1/16 of the slices with the smallest root bounds (most likely
        // to hold the optimum), then the rest in one batch.
        const size_t bsz = p->prune == 2
                               ? std::min<size_t>(65535, fl.size())
                               : std::min<size_t>(65535, std::max<size_t>(32, (fl.size() + 7) / 8));
        const size_t first = p->prune == 2 ? (fl.size() + 15) / 16 : bsz;
        for (size_t b0 = 0; b0 < fl.size();) {
            const size_t nb = std::min(b0 == 0 ? first : bsz, fl.size() - b0);
            batches.push_back({p->M_list[g.mi], ordered.size(), nb});
            for (size_t j = 0; j < nb; ++j) ordered.push_back(s.slices[fl[b0 + j]]);
            max_nb = std::max(max_nb, nb);
            b0 += nb;
        }
    }
    POS_CUDA(s.d_batch.reserve(sizeof(SliceRec) * std::max<size_t>(1, ordered.size())));
    if (!ordered.empty())
        POS_TRY(upload(s, s.d_batch.p, ordered.data(), sizeof(SliceRec) * ordered.size()));
    // roots: slot j of a batch, no stage placed (the first nb serve a batch of nb)
    std::vector<Prefix> roots(max_nb);
    for (size_t j = 0; j < max_nb; ++j) {
        std::memset(&roots[j], 0, sizeof(Prefix));
        roots[j].slice = (uint16_t)j;
        roots[j].A = 0;
        roots[j].Bm = -1;
    }
    POS_CUDA(s.d_roots.reserve(sizeof(Prefix) * max_nb));
    POS_TRY(upload(s, s.d_roots.p, roots.data(), sizeof(Prefix) * max_nb));
    const SliceRec *d_ordered = static_cast<const SliceRec *>(s.d_batch.p);
    const Prefix *d_rootp = static_cast<const Prefix *>(s.d_roots.p);

    Key128 inc;
    unsigned long long hs[kStCount];
    bool have_results = false;  // inc and hs read after the last launch
    if (s.S == 1) {
        // the single stage takes every layer: each feasible slice is one plan
        for (const Batch &b : batches) {
            std::vector<Leaf> lv(b.nb);
            for (size_t j = 0; j < b.nb; ++j) {
                std::memset(&lv[j], 0, sizeof(Leaf));
                lv[j].slice = (uint32_t)j;
            }
            POS_TRY(upload(s, s.d_leaves.p, lv.data(), sizeof(Leaf) * b.nb));
            const unsigned long long cnt = b.nb;
            POS_TRY(upload(s, s.ctr + 36, &cnt, 8));
            if ((st = run_leaves(s, static_cast<const Leaf *>(s.d_leaves.p), s.ctr + 36,
                                 d_ordered + b.off, b.M, nullptr)) != POS_OK)
                return st;
            POS_CUDA(cudaStreamSynchronize(s.stream));
        }
    } else {
        // Optimistic pass: every batch runs as one stream-ordered pipeline
        // (completion bounds, one level kernel per depth, the completion
        // kernel, the leaf kernel); each kernel reads its input count from
        // the counter the previous one filled, so the host never waits.
        // Per batch and depth x: bctr[2x] = entries written (uncapped),
        // bctr[2x+1] = warp groups that did not fit.
        const int S = s.S;
        for (int x = 1; x <= S - 2; ++x)
            if ((st = ensure_depth(s, x)) != POS_OK) return st;
        for (int x = 0; x <= S - 2; ++x)
            if ((st = ensure_defer(s, x, (s.cap + 31) / 32 + 1)) != POS_OK) return st;
        const size_t n_b = batches.size();
        POS_CUDA(s.ws.d_bctr.reserve(sizeof(unsigned long long) * 32 * std::max<size_t>(1, n_b)));
        unsigned long long *bctr = static_cast<unsigned long long *>(s.ws.d_bctr.p);
        POS_CUDA(cudaMemsetAsync(bctr, 0, sizeof(unsigned long long) * 32 * n_b, s.stream));
        // timing events (profile only), S + 1 per batch: before level 0,
        // after each level kernel, after the leaf kernel
        const bool prof = p->profile != 0;
        const size_t n_ev = prof ? n_b * (S + 1) : 0;
        while (s.ws.evs.size() < n_ev) {
            cudaEvent_t e;
            POS_CUDA(cudaEventCreate(&e));
            s.ws.evs.push_back(e);
        }
        for (size_t bi = 0; bi < n_b; ++bi) {
            const Batch &b = batches[bi];
            s.cur_nb = (int)b.nb;
            cudaEvent_t *ev = prof ? s.ws.evs.data() + bi * (S + 1) : nullptr;
            unsigned long long *bc = bctr + 32 * bi;
            if (prof) POS_CUDA(cudaEventRecord(ev[0], s.stream));
            for (int x = 0; x <= S - 2; ++x) {
                const bool last = x == S - 2;
                ExpandParams ep = base_params(s, d_ordered + b.off, b.M);
                ep.in = x == 0 ? d_rootp : static_cast<const Prefix *>(s.d_front[x].p);
                ep.n_in = x == 0 ? (long long)b.nb : 0;
                ep.n_in_dev = x == 0 ? nullptr : bc + 2 * (x - 1);
                ep.x = x;
                ep.out = last ? nullptr : static_cast<Prefix *>(s.d_front[x + 1].p);
                ep.leaves = last ? static_cast<Leaf *>(s.d_leaves.p) : nullptr;
                ep.out_count = bc + 2 * x;
                ep.deferred = static_cast<uint32_t *>(s.d_defer[2 * x].p);
                ep.n_deferred = bc + 2 * x + 1;
                ep.nb = (int)b.nb;
                ep.vb_smem = p->prune == 2 && !last && b.nb <= kVbSlotsSmem;
                const int smem_l = ep.lay.bytes + (ep.vb_smem ? (int)b.nb * 128 * 8 : 0);
                // depth 0: the batch's nb roots, one warp each (the kernel
                // takes the warp-per-parent mapping when the grid has a warp
                // per parent); deeper frontiers are sized on the device
                const int grid = x == 0 ? (int)std::max<long long>(
                                              1, std::min<long long>(
                                                     ((long long)b.nb + kThreads / 32 - 1) /
                                                         (kThreads / 32),
                                                     s.grid_level))
                                        : s.grid_level;
                s.launches++;
                if ((st = launch_level(last, x, ep, grid, smem_l, s.stream)) != POS_OK)
                    return st;
                (last ? s.n_complete : s.n_expand)++;
                s.launches_depth[x]++;
                if (prof) POS_CUDA(cudaEventRecord(ev[x + 1], s.stream));
            }
            if ((st = run_leaves(s, static_cast<const Leaf *>(s.d_leaves.p), bc + 2 * (S - 2),
                                 d_ordered + b.off, b.M, nullptr)) != POS_OK)
                return st;
            s.n_leaf++;
            if (prof) POS_CUDA(cudaEventRecord(ev[S], s.stream));
        }
        // the passes' counters, the incumbent and the statistics in one read
        std::vector<unsigned long long> hb(32 * n_b);
        {
            const ReadPart parts[3] = {{hb.data(), bctr, sizeof(unsigned long long) * hb.size()},
                                       {&inc, s.d_inc.p, sizeof(inc)},
                                       {hs, s.stats, sizeof(hs)}};
            if ((st = sync_read_many(s, parts, 3)) != POS_OK) return st;
            have_results = true;
        }
        for (size_t bi = 0; bi < n_b && prof; ++bi) {
            cudaEvent_t *ev = s.ws.evs.data() + bi * (S + 1);
            for (int x = 0; x <= S - 1; ++x) {
                float ms = 0;
                POS_CUDA(cudaEventElapsedTime(&ms, ev[x], ev[x + 1]));
                if (x <= S - 2) s.ms_depth[x] += ms;
                if (x < S - 2) s.ms_expand += ms;
                else if (x == S - 2) s.ms_complete += ms;
                else s.ms_leaf += ms;
            }
        }
        // A batch in which some frontier overflowed lost the children that
        // did not fit: run it again with the exact, host-driven deferral.
        // Plans it evaluated twice do not change the incumbent.
        for (size_t bi = 0; bi < n_b; ++bi) {
            bool overflow = false;
            for (int x = 0; x <= S - 2; ++x) overflow |= hb[32 * bi + 2 * x + 1] != 0;
            if (!overflow) continue;
            s.reruns++;
            have_results = false;
            const Batch &b = batches[bi];
            s.cur_nb = (int)b.nb;
            st = process(s, d_ordered + b.off, b.M, 0, d_rootp, (long long)b.nb);
            if (st != POS_OK) return st;
        }
    }
    if (!have_results) {
        const ReadPart parts[2] = {{&inc, s.d_inc.p, sizeof(inc)}, {hs, s.stats, sizeof(hs)}};
        if ((st = sync_read_many(s, parts, 2)) != POS_OK) return st;
    }
    const double ms_search = ms_since(t_search);

    if (hs[kStTimeout])
        return fail(POS_ETIMEOUT, "the incumbent's compare-and-swap loop hit its iteration "
                                  "limit (pos_problem.cas_limit rounds)");
    if (hs[kStBulkTimeout])
        return fail(POS_ETIMEOUT, "a block's cost-table staging (TMA bulk copy) did not "
                                  "complete within its poll limit");

    std::memset(out, 0, sizeof(*out));
    if (stats) {
        std::memset(stats, 0, sizeof(*stats));
        stats->evaluated = hs[kStEvaluated];
        stats->warmup_evaluated = warm_evals;
        stats->prefixes = hs[kStPrefixes];
        stats->pruned_bound = hs[kStPrunedBound];
        stats->pruned_memory = hs[kStPrunedMemory];
        stats->pruned_ridge = hs[kStPrunedRidge];
        stats->relaxations = hs[kStRelaxations];
        stats->slices = (uint64_t)n_slices;
        stats->slices_feasible = n_feasible;
        stats->launches = s.launches;
        stats->ms_setup = ms_setup;
        stats->ms_warmup = ms_warm;
        stats->ms_search = ms_search;
        stats->ms_expand = s.ms_expand;
        stats->ms_complete = s.ms_complete;
        stats->ms_leaf = s.ms_leaf;
        stats->expand_launches = s.n_expand;
        stats->complete_launches = s.n_complete;
        stats->leaf_launches = s.n_leaf;
        stats->parents_expand = hs[kStParentsExpand];
        stats->parents_complete = hs[kStParentsComplete];
        stats->leaves = hs[kStLeaves];
        stats->ms_bound = s.ms_bound;
        for (int x = 0; x < POS_MAX_STAGES; ++x) {
            stats->ms_depth[x] = s.ms_depth[x];
            stats->launches_depth[x] = s.launches_depth[x];
            stats->parents_depth[x] = hs[kStDepthParents + x];
            stats->children_depth[x] = hs[kStDepthChildren + x];
        }
        stats->bound_launches = s.n_bound;
        stats->reruns = s.reruns;
    }
    if (inc.obj == ~0ull) {
        if (stats) stats->ms_total = ms_since(t_start);
        return fail(POS_EINFEASIBLE, "no memory-feasible plan");
    }
    const uint64_t ord = inc.idx / s.n_map;
    const SliceRec &sr = s.slices[ord];
    out->found = 1;
    out->map_rank = inc.idx % s.n_map;
    plan_slice_fields(p, sp, ord, out);
    out->S = s.S;
    out->makespan = (int32_t)(inc.obj / sr.scale);
    out->global_index = inc.idx;
    for (int x = 0; x < POS_MAX_STAGES; ++x) out->layers[x] = 0;
    host_unrank(s.L, s.S, out->map_rank, out->layers);
    if (stats) stats->ms_total = ms_since(t_start);
    return POS_OK;
}

}  // namespace pos

extern "C" pos_status poseidon_search(const pos_problem *problem, pos_plan *out,
                                      pos_search_stats *stats) {
    if (!out) return pos::fail(POS_EINVAL, "plan out-pointer is NULL");
    pos::set_error("");
    pos_status st = pos::validate_problem(problem);  // before touching the device
    if (st == POS_OK) st = pos::validate_tables(&problem->tables);
    if (st != POS_OK) return st;
    pos::SliceSpace sp;
    try {
        st = pos::build_slice_space(problem, problem->S, sp);
    } catch (...) {
        return pos::fail(POS_ENOMEM, "host exception (allocation failure)");
    }
    if (st == POS_OK) st = pos::validate_space(problem, sp);
    if (st != POS_OK) return st;
    pos::Workspace *ws = nullptr;
    st = pos::get_workspace(&ws);
    if (st != POS_OK) return st;
    std::lock_guard<std::mutex> lock(ws->mu);
    try {
        if (problem->schedule == POS_SCHED_INTERLEAVED_1F1B)
            return pos::search_interleaved(*ws, problem, sp, out, stats);
        pos::Search s(*ws);
        s.pb = problem;
        s.sp = &sp;
        return pos::search_impl(s, out, stats);
    } catch (...) {
        return pos::fail(POS_ENOMEM, "host exception (allocation failure)");
    }
}
