// poseidon_search under Interleaved 1F1B (Sec. 4.1.4 model, Sec. 4.2.3
// search order).  The S = N devices hold V model chunks each, so a plan is
// a slice (M, TP index, device-type placement over the N devices) and a
// composition of the L layers into the J = N*V virtual stages; virtual
// stage j is chunk j / N on device j % N.  M values that are not multiples
// of N have no interleaved schedule and are skipped (their index still
// counts in the global numbering).
//
//  1. seeds: per slice, the composition that minimises the largest virtual
//     stage time M (F + B) (a dynamic program over (stage, first layer));
//     evaluated like every complete plan, they give the first incumbent;
//  2. enumeration, level by level over the virtual stages (one thread per
//     partial plan, 32-parent groups reserve their output with one atomic):
//     the layer counts l of the next virtual stage that keep its device's
//     resident bytes within capacity and the prefix's lower bound within
//     the incumbent form a range [1, hi] (both grow with l); the last two
//     stages are completed together and each completion is tested;
//  3. complete plans are written as decoded interleaved records and
//     evaluated by the evaluator's interleaved makespan kernels (exact
//     activation check included), then a kernel lowers the incumbent with
//     the (objective, global index) key.
// Frontiers have a fixed capacity; 32-parent groups whose children do not
// fit are deferred and re-expanded after the part that fit has been
// finished (depth first over chunks), so memory stays bounded.
//
// Lower bounds of a prefix (each term is the length of a DAG path of every
// completion; weights are non-negative, so placing more layers never lowers
// a term):
//   prune 1: max over devices d of M * sum (F + B) + sum dsync over the
//            chunks of d placed so far (d runs its 2VM ops one at a time and
//            R_d follows its last op);
//   prune 2: for a device d whose first chunk is placed (virtual stage d),
//            the first micro-batch reaches d's first op F_{d,0} through the
//            forwards and transfers of virtual stages 0..d-1, d runs its
//            chain, and its last op B_{d,M-1} (chunk 0) either feeds R_d or
//            the backwards of virtual stages d-1..0 down to R_0:
//              A_d + M sum (F + B) + max(dsync_d, Bs_d + dsync_0),
//            A_d = sum_{i<d} (F_i + pf_i), Bs_d = sum_{i<d} (B_i + pb_i).
#include <algorithm>
#include <chrono>
#include <cstring>
#include <vector>

#include "interleaved.cuh"
#include "search_host.h"

namespace pos {

namespace {

constexpr int kIlThreads = 256;
constexpr uint32_t kIlHole = 0xffffffffu;

// byte 4 + i of a 32-byte entry = cut[i + 1] (end of virtual stage i), for
// a runtime i in 0..14
__device__ __forceinline__ int cut_byte(const Vec32 &v, int i) {
    const int p = 4 + i, w = p >> 2;
    const uint32_t word = w == 1 ? v.a.y : w == 2 ? v.a.z : w == 3 ? v.a.w : v.b.x;
    return (int)((word >> (8 * (p & 3))) & 0xffu);
}

__device__ __forceinline__ void put_cut(Vec32 &v, int i, int c) {
    const int p = 4 + i, w = p >> 2, sh = 8 * (p & 3);
    const uint32_t m = ~(0xffu << sh), b = (uint32_t)c << sh;
    if (w == 1) v.a.y = (v.a.y & m) | b;
    else if (w == 2) v.a.z = (v.a.z & m) | b;
    else if (w == 3) v.a.w = (v.a.w & m) | b;
    else v.b.x = (v.b.x & m) | b;
}

// Per-device sums over the virtual stages placed so far (stages 0..placed-1).
template <int N>
struct IlAcc {
    int32_t ser[N];  // M * sum (F + B) over the device's placed chunks
    int32_t ds[N];   // sum dsync over them
    int64_t wt[N];   // resident bytes (weights, optimizer state) over them
    int32_t A[N], Bs[N];  // prune 2: fill and drain sums before the device's first chunk
    int32_t runF, runB;   // running sums over the placed chunk-0 stages
    int placed;
};

// Adds virtual stage i = layers [c0, c1) to the sums (device i % N).
template <int N>
__device__ __forceinline__ void il_add(IlAcc<N> &a, const Tab &t, const int (&cls)[N], int M,
                                       int i, int c0, int c1) {
    const int d = i % N;
    int k = cls[0];
#pragma unroll
    for (int dd = 1; dd < N; ++dd) k = dd == d ? cls[dd] : k;
    const int32_t F = Pf(t, k, c1) - Pf(t, k, c0), B = Pb(t, k, c1) - Pb(t, k, c0);
    const int32_t D = Pd(t, k, c1) - Pd(t, k, c0);
    const int64_t W = Pw(t, k, c1) - Pw(t, k, c0);
#pragma unroll
    for (int dd = 0; dd < N; ++dd)
        if (dd == d) {
            a.ser[dd] += M * (F + B);
            a.ds[dd] += D;
            a.wt[dd] += W;
            if (i < N) {
                a.A[dd] = a.runF;
                a.Bs[dd] = a.runB;
            }
        }
    if (i < N) {
        // the edge from virtual stage i (device d) to i + 1 (device (d+1) % N)
        int kn = cls[0];
#pragma unroll
        for (int dd = 0; dd < N; ++dd) kn = dd == (d + 1) % N ? cls[dd] : kn;
        a.runF += F + p2f(t, k, kn);
        a.runB += B + p2b(t, kn, k);
    }
    a.placed = i + 1;
}

template <int N>
__device__ __forceinline__ void il_init(IlAcc<N> &a) {
#pragma unroll
    for (int dd = 0; dd < N; ++dd) {
        a.ser[dd] = a.ds[dd] = a.A[dd] = a.Bs[dd] = 0;
        a.wt[dd] = 0;
    }
    a.runF = a.runB = 0;
    a.placed = 0;
}

// Lower bound of every completion of the placed stages.
template <int N>
__device__ __forceinline__ int64_t il_bound(const IlAcc<N> &a, int prune) {
    int64_t lb = 0;
#pragma unroll
    for (int dd = 0; dd < N; ++dd) {
        int64_t v = (int64_t)a.ser[dd] + a.ds[dd];
        if (prune == 2 && dd < a.placed)
            v = (int64_t)a.A[dd] + a.ser[dd] + max((int64_t)a.ds[dd], (int64_t)a.Bs[dd] + a.ds[0]);
        lb = max(lb, v);
    }
    return lb;
}

template <int N>
__device__ __forceinline__ int64_t il_weight(const IlAcc<N> &a, int d) {
    int64_t w = a.wt[0];
#pragma unroll
    for (int dd = 1; dd < N; ++dd) w = dd == d ? a.wt[dd] : w;
    return w;
}

}  // namespace

// ---------------------------------------------------------------------------
// level kernel: parents at depth x (virtual stages 0..x-1 placed)
// ---------------------------------------------------------------------------
struct IlLevelParams {
    const Vec32 *in;          // parents: slice in bytes 0-3, cut[i+1] in byte 4+i
    long long n_in;
    const uint32_t *groups;   // work list of 32-parent groups, or NULL = all groups
    long long n_groups;
    int x;                    // depth of the parents
    int J, V, prune;
    const SliceRec *slices;
    Vec32 *out;               // expansion (x < J-2): children at depth x+1
    uint4 *rec;               // completion (x = J-2): decoded records, two uint4 per plan
    uint32_t *leaf_slice;     // completion: slice of each record (kIlHole: none)
    unsigned long long *out_count;
    unsigned long long cap;
    uint32_t *deferred;
    unsigned long long *n_deferred;
    const Key128 *inc;
    unsigned long long *stats;
    const void *blob;
    BlobLayout lay;
};

// Largest l in [0, hi] with pred(l), pred true up to some l and false after.
template <class Pred>
__device__ __forceinline__ int il_last_true(int hi, Pred pred) {
    int lo = 0;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (pred(mid)) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

// The decoded record's second word of a slice's plans, as the interleaved
// makespan kernels read it: (slot, type code with 2 bits per device,
// S = N | M << 8 | tp << 16 | V << 24, per-device TP code).  The class of
// device d is type_d * n_tp + tp + its field of the TP code: with at most
// four TP indices each device's index goes in the TP code (tp = 0), which
// holds a TP index per device (POS_PLACE_DEVICES); above four every device
// shares one index (checked on the host), carried by tp.
__device__ __forceinline__ uint4 il_meta_pack(uint32_t tcode, uint32_t tpc, int cls0, int N,
                                              int n_tp, int M, int V, uint32_t slot) {
    const uint32_t tp = n_tp <= 4 ? 0u : (uint32_t)(cls0 % n_tp);
    const uint32_t word = (uint32_t)N | ((uint32_t)M << 8) | (tp << 16) | ((uint32_t)V << 24);
    return make_uint4(slot, tcode, word, n_tp <= 4 ? tpc : 0u);
}
template <int N>
__device__ __forceinline__ uint4 il_meta(const int (&cls)[N], int n_tp, int M, int V,
                                         uint32_t slot) {
    uint32_t tcode = 0, tpc = 0;
#pragma unroll
    for (int d = 0; d < N; ++d) {
        tcode |= (uint32_t)(cls[d] / n_tp) << (2 * d);
        tpc |= (uint32_t)(cls[d] % n_tp) << (2 * d);
    }
    return il_meta_pack(tcode, tpc, cls[0], N, n_tp, M, V, slot);
}
// the same from a slice record (runtime N)
__device__ __forceinline__ uint4 il_meta_rt(const uint8_t *cls, int N, int n_tp, int M, int V,
                                            uint32_t slot) {
    uint32_t tcode = 0, tpc = 0;
    for (int d = 0; d < N; ++d) {
        tcode |= (uint32_t)(cls[d] / n_tp) << (2 * d);
        tpc |= (uint32_t)(cls[d] % n_tp) << (2 * d);
    }
    return il_meta_pack(tcode, tpc, cls[0], N, n_tp, M, V, slot);
}

template <int N>
__global__ void __launch_bounds__(kIlThreads) il_level_kernel(IlLevelParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ uint64_t bar;
    const long long n_in = p.n_in;
    const long long n_work = p.groups ? p.n_groups : (n_in + 31) / 32;
    // blocks without work leave before staging the tables
    if ((long long)blockIdx.x * (kIlThreads / 32) >= n_work) return;
    if (!stage_blob_bulk(sm, p.blob, p.lay.bytes, &bar)) {
        if (threadIdx.x == 0) atomicAdd(p.stats + kStBulkTimeout, 1ull);
        return;
    }
    const Tab t = tab_at(sm, p.lay);
    const int L = t.L(), J = p.J, x = p.x, n_tp = t.n_tp();
    const bool complete = x == J - 2;
    const uint64_t thr = p.prune ? __ldcg(&p.inc->obj) : ~0ull;
    const int lane = threadIdx.x & 31;
    const long long warp = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
    const long long n_warps = ((long long)gridDim.x * blockDim.x) >> 5;
    unsigned long long emitted = 0, cut_b = 0, cut_m = 0, parents = 0;
    for (long long w = warp; w < n_work; w += n_warps) {
        const long long g = p.groups ? (long long)p.groups[w] : w;
        const long long i = g * 32 + lane;
        Vec32 pv = {make_uint4(kIlHole, 0, 0, 0), make_uint4(0, 0, 0, 0)};
        if (i < n_in) pv = load32(p.in + i);
        const uint32_t sl = pv.a.x;
        const bool live = sl != kIlHole;
        int n = 0, c = 0, hi = 0, M = 0;
        uint32_t pass[4] = {0u, 0u, 0u, 0u};  // completion: bit l-1 = l layers pass
        int cls[N];
#pragma unroll
        for (int d = 0; d < N; ++d) cls[d] = 0;
        unsigned long long lb = 0, lm = 0;
        if (live) {
            const SliceRec &sr = p.slices[sl];
            M = sr.M;
            const uint64_t scale = sr.scale;
#pragma unroll
            for (int d = 0; d < N; ++d) cls[d] = sr.cls[d];
            IlAcc<N> a;
            il_init(a);
            for (int s = 0; s < x; ++s) {
                const int c1 = cut_byte(pv, s);
                il_add(a, t, cls, M, s, c, c1);
                c = c1;
            }
            const int dn = x % N;
            int kn = cls[0];
#pragma unroll
            for (int d = 1; d < N; ++d) kn = d == dn ? cls[d] : kn;
            const int64_t w0 = il_weight(a, dn) - Pw(t, kn, c), capn = cap_of(t, kn);
            if (!complete) {
                // resident bytes and the bound both grow with l: [1, hi]
                const int lmax = L - c - (J - x - 1);
                const int hi_mem =
                    il_last_true(lmax, [&](int l) { return w0 + Pw(t, kn, c + l) <= capn; });
                hi = hi_mem;
                if (p.prune)
                    hi = il_last_true(hi_mem, [&](int l) {
                        IlAcc<N> b = a;
                        il_add(b, t, cls, M, x, c, c + l);
                        return (uint64_t)il_bound(b, p.prune) * scale <= thr;
                    });
                n = hi;
                lm += (unsigned long long)(lmax - hi_mem);
                lb += (unsigned long long)(hi_mem - hi);
            } else {
                // stage x = J-2 takes l layers, stage J-1 the rest; each l is
                // tested (the last stage's terms shrink as l grows)
                const int db = (J - 1) % N;
                int kb = cls[0];
#pragma unroll
                for (int d = 1; d < N; ++d) kb = d == db ? cls[d] : kb;
                const int64_t capb = cap_of(t, kb);
                for (int l = 1; l <= L - c - 1; ++l) {
                    IlAcc<N> b = a;
                    il_add(b, t, cls, M, x, c, c + l);
                    il_add(b, t, cls, M, J - 1, c + l, L);
                    if (il_weight(b, dn) > capn || il_weight(b, db) > capb) {
                        ++lm;
                        continue;
                    }
                    if (p.prune && (uint64_t)il_bound(b, p.prune) * scale > thr) {
                        ++lb;
                        continue;
                    }
                    pass[(l - 1) >> 5] |= 1u << ((l - 1) & 31);
                    ++n;
                }
            }
        }
        int incl = n;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        const int total = __shfl_sync(0xffffffffu, incl, 31);
        cut_b += lb;
        cut_m += lm;
        if (total == 0) {
            parents += live;
            continue;
        }
        unsigned long long base = 0;
        if (lane == 0) base = atomicAdd(p.out_count, (unsigned long long)total);
        base = __shfl_sync(0xffffffffu, base, 0);
        unsigned long long pos = base + (unsigned long long)(incl - n);
        if (base + (unsigned long long)total <= p.cap) {
            if (!complete) {
                for (int l = 1; l <= hi; ++l) {
                    Vec32 ch = pv;
                    put_cut(ch, x, c + l);
                    store32(p.out + pos++, ch);
                }
            } else {
#pragma unroll
                for (int wd = 0; wd < 4; ++wd) {
                    uint32_t m = pass[wd];
                    while (m) {
                        const int l = 32 * wd + __ffs(m);
                        m &= m - 1;
                        Vec32 lf = pv;
                        put_cut(lf, x, c + l);
                        // cut[1..J-1] in bytes 0..14 of the record's first word;
                        // byte 15 = 0: not answered yet
                        p.rec[2 * pos] = make_uint4(lf.a.y, lf.a.z, lf.a.w, lf.b.x & 0x00ffffffu);
                        p.rec[2 * pos + 1] = il_meta(cls, n_tp, M, p.V, (uint32_t)pos);
                        p.leaf_slice[pos] = sl;
                        ++pos;
                    }
                }
            }
            emitted += (unsigned long long)n;
            parents += live;
        } else {
            // no room: the reserved slots below the capacity become holes and
            // the group is deferred
            for (unsigned long long e = pos; e < pos + (unsigned long long)n && e < p.cap; ++e) {
                if (complete) {
                    p.rec[2 * e] = make_uint4(0u, 0u, 0u, 1u << 24);  // answered: skipped
                    p.rec[2 * e + 1] = make_uint4((uint32_t)e, 0u, 0u, 0u);
                    p.leaf_slice[e] = kIlHole;
                } else {
                    const Vec32 hole = {make_uint4(kIlHole, 0, 0, 0), make_uint4(0, 0, 0, 0)};
                    store32(p.out + e, hole);
                }
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
        cut_b += __shfl_xor_sync(0xffffffffu, cut_b, o);
        cut_m += __shfl_xor_sync(0xffffffffu, cut_m, o);
        parents += __shfl_xor_sync(0xffffffffu, parents, o);
    }
    if (lane == 0) {
        if (emitted) {
            atomicAdd(p.stats + (complete ? kStLeaves : kStPrefixes), emitted);
            atomicAdd(p.stats + kStDepthChildren + x, emitted);
        }
        if (cut_b) atomicAdd(p.stats + kStPrunedBound, cut_b);
        if (cut_m) atomicAdd(p.stats + kStPrunedMemory, cut_m);
        if (parents) {
            atomicAdd(p.stats + (complete ? kStParentsComplete : kStParentsExpand), parents);
            atomicAdd(p.stats + kStDepthParents + x, parents);
        }
    }
}

// ---------------------------------------------------------------------------
// complete plans: key offsets for the interleaved makespan kernels, and the
// incumbent update
// ---------------------------------------------------------------------------
// The makespan kernels evaluate the records of each (N, V) key block
// [offs[kKeys + first key of the pair], offs[kKeys + first key of the next
// pair]); all of this search's records belong to one pair, so every offset
// up to that pair's first key is 0 and every later one the record count.
__global__ void il_offs_kernel(uint32_t *offs, int n_offs, int pair_key,
                               const unsigned long long *count, unsigned long long cap) {
    const unsigned long long c0 = __ldcg(count);
    const uint32_t n = (uint32_t)(c0 < cap ? c0 : cap);
    for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < n_offs; k += gridDim.x * blockDim.x)
        offs[k] = k <= pair_key ? 0u : n;
}

// Lowers the incumbent with every memory-feasible evaluated plan: objective
// T * Q/(D*M), global index slice ordinal * C(L-1, J-1) + composition rank.
__global__ void __launch_bounds__(kIlThreads) il_consider_kernel(
    const uint4 *rec, const uint32_t *leaf_slice, const int32_t *T, const uint8_t *F,
    const unsigned long long *count, unsigned long long cap, const SliceRec *slices,
    uint64_t n_map, int J, Key128 *inc, unsigned long long *stats, int cas_limit,
    const void *blob, BlobLayout lay) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ uint64_t bar;
    const unsigned long long c0 = __ldcg(count);
    const unsigned long long n = c0 < cap ? c0 : cap;
    if ((unsigned long long)blockIdx.x * blockDim.x >= n) return;
    // the binomials (composition ranks) are part of the staged blob
    if (!stage_blob_bulk(sm, blob, lay.bytes, &bar)) {
        if (threadIdx.x == 0) atomicAdd(stats + kStBulkTimeout, 1ull);
        return;
    }
    const Tab t = tab_at(sm, lay);
    const int L = t.L();
    const unsigned long long stride = (unsigned long long)gridDim.x * blockDim.x;
    const unsigned long long n_round = (n + 31) & ~31ull;
    unsigned long long evaluated = 0, relax = 0;
    for (unsigned long long i = blockIdx.x * (unsigned long long)blockDim.x + threadIdx.x;
         i < n_round; i += stride) {
        unsigned long long obj = ~0ull, idx = ~0ull;
        const uint32_t sl = i < n ? __ldg(leaf_slice + i) : kIlHole;
        if (sl != kIlHole) {
            const SliceRec &sr = slices[sl];
            ++evaluated;
            relax += 2ull * (unsigned long long)J * (unsigned long long)__ldg(&sr.M);
            if (__ldg(F + i) == POS_FEAS_YES) {
                const uint4 pk = __ldg(rec + 2 * i);
                const uint32_t pw[4] = {pk.x, pk.y, pk.z, pk.w};
                uint64_t r = 0;
                int c = 0;
                for (int s = 0; s < J - 1; ++s) {
                    const int c1 = (int)((pw[s >> 2] >> (8 * (s & 3))) & 0xffu);
                    const int rem = L - c, k = J - s - 1;
                    r += binom(t, rem - 1, k) - binom(t, L - c1, k);
                    c = c1;
                }
                obj = (unsigned long long)__ldg(T + i) * __ldg(&sr.scale);
                idx = __ldg(&sr.ordinal) * n_map + r;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const unsigned long long oo = __shfl_xor_sync(0xffffffffu, obj, o);
            const unsigned long long oi = __shfl_xor_sync(0xffffffffu, idx, o);
            if (key_less(oo, oi, obj, idx)) {
                obj = oo;
                idx = oi;
            }
        }
        if ((threadIdx.x & 31) == 0 && obj != ~0ull) incumbent_update(inc, obj, idx, stats, cas_limit);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        evaluated += __shfl_xor_sync(0xffffffffu, evaluated, o);
        relax += __shfl_xor_sync(0xffffffffu, relax, o);
    }
    if ((threadIdx.x & 31) == 0 && evaluated) {
        atomicAdd(stats + kStEvaluated, evaluated);
        atomicAdd(stats + kStRelaxations, relax);
    }
}

// ---------------------------------------------------------------------------
// seeds: per slice, the composition minimising the largest virtual-stage
// time M (F + B), by a dynamic program over (virtual stage j, first layer c)
//   best[j][c] = min over l of max(M (F + B)[c, c+l) on j's device class,
//                                  best[j+1][c+l]),
// one warp per slice (lanes over c), rows in shared memory after the blob.
// ---------------------------------------------------------------------------
constexpr int kSeedWarps = 4;
constexpr int32_t kSeedInf = 0x7fffffff;

__global__ void __launch_bounds__(32 * kSeedWarps) il_seed_kernel(
    const SliceRec *slices, int n_slices, int N, int J, int V, uint4 *rec, uint32_t *leaf_slice,
    const void *blob, BlobLayout lay, int row_bytes, unsigned long long *stats) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ uint64_t bar;
    if (blockIdx.x * kSeedWarps >= n_slices) return;
    if (!stage_blob_bulk(sm, blob, lay.bytes, &bar)) {
        if (threadIdx.x == 0) atomicAdd(stats + kStBulkTimeout, 1ull);
        return;
    }
    const Tab t = tab_at(sm, lay);
    const int L = t.L(), lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    int32_t *best = reinterpret_cast<int32_t *>(sm + ((lay.bytes + 15) & ~15) + wib * row_bytes);
    uint8_t *arg = reinterpret_cast<uint8_t *>(best + (J + 1) * (L + 1));
    for (int sl = blockIdx.x * kSeedWarps + wib; sl < n_slices; sl += gridDim.x * kSeedWarps) {
        const SliceRec &sr = slices[sl];
        const int M = sr.M;
        for (int j = J - 1; j >= 0; --j) {
            const int k = sr.cls[j % N];
            for (int c = lane; c <= L; c += 32) {
                int32_t v = kSeedInf;
                int al = 0;
                const int32_t f0 = Pf(t, k, c < L ? c : L), b0 = Pb(t, k, c < L ? c : L);
                if (j == J - 1) {
                    if (c < L) {
                        v = M * (Pf(t, k, L) - f0 + Pb(t, k, L) - b0);
                        al = L - c;
                    }
                } else {
                    const int lmax = L - c - (J - j - 1);
                    for (int l = 1; l <= lmax; ++l) {
                        const int32_t nb = best[(j + 1) * (L + 1) + c + l];
                        if (nb == kSeedInf) continue;
                        const int32_t m =
                            max(M * (Pf(t, k, c + l) - f0 + Pb(t, k, c + l) - b0), nb);
                        if (m < v) {
                            v = m;
                            al = l;
                        }
                    }
                }
                best[j * (L + 1) + c] = v;
                arg[j * (L + 1) + c] = (uint8_t)al;
            }
            __syncwarp();
        }
        if (lane == 0) {
            Vec32 lf = {make_uint4((uint32_t)sl, 0, 0, 0), make_uint4(0, 0, 0, 0)};
            int c = 0;
            for (int j = 0; j < J - 1; ++j) {
                c += arg[j * (L + 1) + c];
                put_cut(lf, j, c);
            }
            rec[2 * sl] = make_uint4(lf.a.y, lf.a.z, lf.a.w, lf.b.x & 0x00ffffffu);
            rec[2 * sl + 1] = il_meta_rt(sr.cls, N, t.n_tp(), M, V, (uint32_t)sl);
            leaf_slice[sl] = (uint32_t)sl;
        }
        __syncwarp();
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
namespace {

template <int P = 0>
int il_pair_key(int N, int V) {
    if constexpr (P < kIlPairs) {
        if (IlPair<P>::N == N && IlPair<P>::V == V) return IlPair<P>::key;
        return il_pair_key<P + 1>(N, V);
    } else {
        return -1;
    }
}

struct IlRun {
    Workspace &ws;
    const pos_problem *p;
    cudaStream_t st;
    BlobLayout lay{};
    void *blob = nullptr;
    int N = 0, V = 0, J = 0, L = 0, n_tp = 0, pair_key = 0;
    long long cap = 0;
    uint64_t n_map = 0;
    int grid_level = 0, grid_consider = 0;
    unsigned long long *ctr = nullptr, *stats = nullptr;
    const SliceRec *d_slices = nullptr;
    uint64_t launches = 0, n_expand = 0, n_complete = 0, n_leaf = 0;
    uint64_t launches_depth[POS_MAX_STAGES] = {};
    double ms_expand = 0, ms_complete = 0, ms_leaf = 0;
    double ms_depth[POS_MAX_STAGES] = {};
    explicit IlRun(Workspace &w) : ws(w), st(w.stream) {}
};

pos_status il_read(IlRun &r, void *dst, const void *src, size_t bytes) {
    POS_CUDA(cudaMemcpyAsync(r.ws.h_cnt, src, bytes, cudaMemcpyDeviceToHost, r.st));
    POS_CUDA(cudaStreamSynchronize(r.st));
    std::memcpy(dst, r.ws.h_cnt, bytes);
    return POS_OK;
}

// Evaluates the complete plans written so far (count on the device) and
// lowers the incumbent.
pos_status il_leaves(IlRun &r, const unsigned long long *count) {
    il_offs_kernel<<<(kKeysIl + 1 + 255) / 256, 256, 0, r.st>>>(
        static_cast<uint32_t *>(r.ws.il_offs.p), kKeysIl + 1, kKeys + r.pair_key, count,
        (unsigned long long)r.cap);
    POS_CUDA(cudaGetLastError());
    EvalParams ep;
    std::memset(&ep, 0, sizeof(ep));
    ep.n = r.cap;
    ep.T = static_cast<int32_t *>(r.ws.il_T.p);
    ep.F = static_cast<uint8_t *>(r.ws.il_F.p);
    ep.offs = static_cast<const uint32_t *>(r.ws.il_offs.p);
    ep.cuts = static_cast<uint4 *>(r.ws.il_rec.p);
    ep.blob = r.blob;
    ep.lay = r.lay;
    ep.nkeys = kKeysIl;
    POS_TRY(eval_interleaved(ep, r.st));
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(il_consider_kernel), r.lay.bytes));
    const int cas = r.p->cas_limit == 0 ? kCasLimit : std::max(0, r.p->cas_limit);
    il_consider_kernel<<<r.grid_consider, kIlThreads, r.lay.bytes, r.st>>>(
        static_cast<const uint4 *>(r.ws.il_rec.p), static_cast<const uint32_t *>(r.ws.il_slice.p),
        static_cast<const int32_t *>(r.ws.il_T.p), static_cast<const uint8_t *>(r.ws.il_F.p), count,
        (unsigned long long)r.cap, r.d_slices, r.n_map, r.J, static_cast<Key128 *>(r.ws.d_inc.p),
        r.stats, cas, r.blob, r.lay);
    POS_CUDA(cudaGetLastError());
    r.launches += 7;  // offsets, five makespan ranges, incumbent
    r.n_leaf++;
    return POS_OK;
}

template <int N>
pos_status il_launch_level_n(const IlLevelParams &lp, int grid, int smem, cudaStream_t st) {
    auto kern = il_level_kernel<N>;
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(kern), smem));
    kern<<<grid, kIlThreads, smem, st>>>(lp);
    POS_CUDA(cudaGetLastError());
    return POS_OK;
}

pos_status il_launch_level(int N, const IlLevelParams &lp, int grid, int smem, cudaStream_t st) {
    switch (N) {
        case 1: return il_launch_level_n<1>(lp, grid, smem, st);
        case 2: return il_launch_level_n<2>(lp, grid, smem, st);
        case 3: return il_launch_level_n<3>(lp, grid, smem, st);
        case 4: return il_launch_level_n<4>(lp, grid, smem, st);
        case 5: return il_launch_level_n<5>(lp, grid, smem, st);
        case 6: return il_launch_level_n<6>(lp, grid, smem, st);
        case 7: return il_launch_level_n<7>(lp, grid, smem, st);
        case 8: return il_launch_level_n<8>(lp, grid, smem, st);
        default: return fail(POS_EINVAL, "Interleaved 1F1B search: N must be 1..8");
    }
}

// Enumerates everything below the partial plans in[0..n_in) at depth x:
// children that fit are finished depth first, then the deferred groups are
// expanded again, until none is left.
pos_status il_process(IlRun &r, int x, const Vec32 *in, long long n_in) {
    const bool last = x == r.J - 2;
    const long long all_groups = (n_in + 31) / 32;
    POS_CUDA(r.ws.d_defer[2 * x].reserve(sizeof(uint32_t) * (size_t)std::max<long long>(all_groups, 1)));
    POS_CUDA(r.ws.d_defer[2 * x + 1].reserve(sizeof(uint32_t) * (size_t)std::max<long long>(all_groups, 1)));
    if (!last) POS_CUDA(r.ws.d_front[x + 1].reserve(sizeof(Vec32) * (size_t)r.cap));
    unsigned long long *out_count = r.ctr + 2 * x, *n_def = out_count + 1;
    const uint32_t *work = nullptr;
    long long n_work = all_groups;
    int flip = 0;
    const bool prof = r.p->profile != 0;
    for (;;) {
        POS_CUDA(cudaMemsetAsync(out_count, 0, 2 * sizeof(unsigned long long), r.st));
        IlLevelParams lp;
        std::memset(&lp, 0, sizeof(lp));
        lp.in = in;
        lp.n_in = n_in;
        lp.groups = work;
        lp.n_groups = n_work;
        lp.x = x;
        lp.J = r.J;
        lp.V = r.V;
        lp.prune = r.p->prune;
        lp.slices = r.d_slices;
        lp.out = last ? nullptr : static_cast<Vec32 *>(r.ws.d_front[x + 1].p);
        lp.rec = static_cast<uint4 *>(r.ws.il_rec.p);
        lp.leaf_slice = static_cast<uint32_t *>(r.ws.il_slice.p);
        lp.out_count = out_count;
        lp.cap = (unsigned long long)r.cap;
        lp.deferred = static_cast<uint32_t *>(r.ws.d_defer[2 * x + flip].p);
        lp.n_deferred = n_def;
        lp.inc = static_cast<const Key128 *>(r.ws.d_inc.p);
        lp.stats = r.stats;
        lp.blob = r.blob;
        lp.lay = r.lay;
        const long long blocks = (n_work * 32 + kIlThreads - 1) / kIlThreads;
        const int grid = (int)std::max<long long>(1, std::min<long long>(blocks, r.grid_level));
        if (prof) POS_CUDA(cudaEventRecord(r.ws.ev[0], r.st));
        POS_TRY(il_launch_level(r.N, lp, grid, r.lay.bytes, r.st));
        r.launches++;
        r.launches_depth[x]++;
        (last ? r.n_complete : r.n_expand)++;
        if (prof) POS_CUDA(cudaEventRecord(r.ws.ev[1], r.st));
        if (last) {
            POS_TRY(il_leaves(r, out_count));
            if (prof) POS_CUDA(cudaEventRecord(r.ws.ev[2], r.st));
        }
        unsigned long long cnt[2];
        POS_TRY(il_read(r, cnt, out_count, sizeof(cnt)));
        if (prof) {
            float ms_k = 0;
            POS_CUDA(cudaEventElapsedTime(&ms_k, r.ws.ev[0], r.ws.ev[1]));
            r.ms_depth[x] += ms_k;
            if (last) {
                r.ms_complete += ms_k;
                float ms_l = 0;
                POS_CUDA(cudaEventElapsedTime(&ms_l, r.ws.ev[1], r.ws.ev[2]));
                r.ms_leaf += ms_l;
            } else {
                r.ms_expand += ms_k;
            }
        }
        if (!last) {
            const long long n_out = (long long)std::min<unsigned long long>(cnt[0], r.cap);
            if (n_out > 0)
                POS_TRY(il_process(r, x + 1, static_cast<const Vec32 *>(r.ws.d_front[x + 1].p),
                                   n_out));
        }
        if (cnt[1] == 0) break;
        if ((long long)cnt[1] >= n_work)
            return fail(POS_ENOMEM, "frontier capacity too small to make progress");
        work = static_cast<const uint32_t *>(r.ws.d_defer[2 * x + flip].p);
        n_work = (long long)cnt[1];
        flip ^= 1;
    }
    return POS_OK;
}

double il_ms_since(std::chrono::steady_clock::time_point t0) {
    return std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
}

}  // namespace

// Exact search over Interleaved 1F1B plans (poseidon_search with
// POS_SCHED_INTERLEAVED_1F1B); the problem has been validated.
pos_status search_interleaved(Workspace &ws, const pos_problem *p, const SliceSpace &sp,
                              pos_plan *out, pos_search_stats *stats) {
    const auto t_start = std::chrono::steady_clock::now();
    IlRun r(ws);
    r.p = p;
    r.N = p->S;
    r.V = p->V;
    r.J = r.N * r.V;
    r.L = p->tables.L;
    r.n_tp = p->tables.n_tp;
    if (r.J > r.L) return fail(POS_EINVAL, "S*V > L: a virtual stage would hold no layer");
    r.pair_key = il_pair_key(r.N, r.V);
    if (r.pair_key < 0) return fail(POS_EINVAL, "Interleaved 1F1B needs V >= 2 and S*V <= 16");
    r.n_map = host_binom(r.L - 1, r.J - 1);
    const int N = r.N;  // the slices (sp) are over the N devices
    // tables: raw rows uploaded, prefix sums built on the device
    std::vector<unsigned char> host;
    int64_t gA = 0, gD = 0, gP = 0;
    POS_TRY(build_blob(&p->tables, POS_SCHED_INTERLEAVED_1F1B, host, r.lay, gA, gD, gP));
    for (int i = 0; i < p->n_M; ++i)
        if (p->M_list[i] % N == 0 && guard_trips(gA, gD, gP, r.J, p->M_list[i]))
            return fail(POS_EOVERFLOW, "makespan bound reaches 2^31 for some M");
    // after the side-stream work of an earlier search, whose buffers this
    // one reuses
    POS_CUDA(cudaStreamWaitEvent(r.st, ws.ev_join, 0));
    POS_CUDA(ws.blob.reserve(r.lay.bytes));
    r.blob = ws.blob.p;
    POS_CUDA(cudaMemcpyAsync(r.blob, host.data(), r.lay.bytes, cudaMemcpyHostToDevice, r.st));
    POS_TRY(launch_prefix_rows(r.blob, r.lay, r.st));
    // slices: M values that are multiples of N, then the groups (TP index or
    // D) and their sequences in global-index order
    uint64_t Q = 1;
    for (int i = 0; i < p->n_M; ++i)
        for (int32_t D : sp.D) {
            const uint64_t dm = (uint64_t)D * p->M_list[i];
            Q = Q / gcd64(Q, dm) * dm;
        }
    std::vector<SliceRec> slices;
    for (int mi = 0; mi < p->n_M; ++mi) {
        if (p->M_list[mi] % N != 0) continue;
        uint64_t ord = (uint64_t)mi * sp.per_m;
        for (int g = 0; g < sp.n_grp; ++g)
            for (uint64_t pr = 0; pr < sp.n_seq(g); ++pr, ++ord) {
                SliceRec sr;
                std::memset(&sr, 0, sizeof(sr));
                sr.ordinal = ord;
                sr.M = p->M_list[mi];
                sr.scale = Q / ((uint64_t)sp.D[g] * p->M_list[mi]);
                sr.gid = (uint32_t)slices.size();
                for (int d = 0; d < N; ++d) sr.cls[d] = (uint8_t)sp.cls(g, pr, d, r.n_tp);
                slices.push_back(sr);
            }
    }
    const long long n_slices = (long long)slices.size();
    r.cap = p->frontier_cap > 0 ? p->frontier_cap : (1ll << 24);
    r.cap = std::max<long long>({r.cap, 32LL * r.L, n_slices});
    std::memset(out, 0, sizeof(*out));
    if (stats) std::memset(stats, 0, sizeof(*stats));
    if (n_slices == 0) return fail(POS_EINFEASIBLE, "no M value is a multiple of S");
    POS_CUDA(ws.d_slices.reserve(sizeof(SliceRec) * n_slices));
    POS_CUDA(ws.d_inc.reserve(sizeof(Key128)));
    POS_CUDA(ws.d_ctr.reserve(sizeof(unsigned long long) * 128));
    POS_CUDA(ws.il_rec.reserve(2 * sizeof(uint4) * (size_t)r.cap));
    POS_CUDA(ws.il_slice.reserve(sizeof(uint32_t) * (size_t)r.cap));
    POS_CUDA(ws.il_T.reserve(sizeof(int32_t) * (size_t)r.cap));
    POS_CUDA(ws.il_F.reserve((size_t)r.cap));
    POS_CUDA(ws.il_offs.reserve(sizeof(uint32_t) * (kKeysIl + 1)));
    POS_CUDA(ws.d_front[0].reserve(sizeof(Vec32) * n_slices));
    POS_CUDA(cudaMemcpyAsync(ws.d_slices.p, slices.data(), sizeof(SliceRec) * n_slices,
                             cudaMemcpyHostToDevice, r.st));
    POS_CUDA(cudaMemsetAsync(ws.d_inc.p, 0xff, sizeof(Key128), r.st));
    POS_CUDA(cudaMemsetAsync(ws.d_ctr.p, 0, sizeof(unsigned long long) * 128, r.st));
    r.d_slices = static_cast<const SliceRec *>(ws.d_slices.p);
    r.ctr = static_cast<unsigned long long *>(ws.d_ctr.p);
    r.stats = r.ctr + 40;
    int per_sm = 0;
    {
        const void *lk = nullptr;
        switch (N) {
            case 1: lk = reinterpret_cast<const void *>(il_level_kernel<1>); break;
            case 2: lk = reinterpret_cast<const void *>(il_level_kernel<2>); break;
            case 3: lk = reinterpret_cast<const void *>(il_level_kernel<3>); break;
            case 4: lk = reinterpret_cast<const void *>(il_level_kernel<4>); break;
            case 5: lk = reinterpret_cast<const void *>(il_level_kernel<5>); break;
            case 6: lk = reinterpret_cast<const void *>(il_level_kernel<6>); break;
            case 7: lk = reinterpret_cast<const void *>(il_level_kernel<7>); break;
            default: lk = reinterpret_cast<const void *>(il_level_kernel<8>); break;
        }
        POS_TRY(ensure_smem(lk, r.lay.bytes));
        POS_TRY(blocks_per_sm(lk, kIlThreads, r.lay.bytes, &per_sm));
        r.grid_level = std::max(1, per_sm) * sm_count();
        POS_TRY(ensure_smem(reinterpret_cast<const void *>(il_consider_kernel), r.lay.bytes));
        POS_TRY(blocks_per_sm(reinterpret_cast<const void *>(il_consider_kernel), kIlThreads,
                              r.lay.bytes, &per_sm));
        r.grid_consider = std::max(1, per_sm) * sm_count();
    }
    const double ms_setup = il_ms_since(t_start);

    // seeds: one plan per slice, evaluated like every complete plan
    const auto t_warm = std::chrono::steady_clock::now();
    {
        const int row_bytes = ((4 * (r.J + 1) * (r.L + 1) + r.J * (r.L + 1)) + 15) & ~15;
        const int smem = ((r.lay.bytes + 15) & ~15) + kSeedWarps * row_bytes;
        POS_TRY(ensure_smem(reinterpret_cast<const void *>(il_seed_kernel), smem));
        const int grid = (int)std::min<long long>((n_slices + kSeedWarps - 1) / kSeedWarps,
                                                  8LL * sm_count());
        il_seed_kernel<<<grid, 32 * kSeedWarps, smem, r.st>>>(
            r.d_slices, (int)n_slices, N, r.J, r.V, static_cast<uint4 *>(ws.il_rec.p),
            static_cast<uint32_t *>(ws.il_slice.p), r.blob, r.lay, row_bytes, r.stats);
        POS_CUDA(cudaGetLastError());
        r.launches++;
        ws.h_cnt[0] = (unsigned long long)n_slices;
        POS_CUDA(cudaMemcpyAsync(r.ctr + 36, ws.h_cnt, sizeof(unsigned long long),
                                 cudaMemcpyHostToDevice, r.st));
        POS_TRY(il_leaves(r, r.ctr + 36));
    }
    const double ms_warm = il_ms_since(t_warm);

    // enumeration from the roots (one per slice, no stage placed)
    const auto t_search = std::chrono::steady_clock::now();
    {
        std::vector<Vec32> roots(n_slices);
        for (long long i = 0; i < n_slices; ++i) {
            std::memset(&roots[i], 0, sizeof(Vec32));
            roots[i].a.x = (uint32_t)i;
        }
        POS_CUDA(cudaMemcpyAsync(ws.d_front[0].p, roots.data(), sizeof(Vec32) * n_slices,
                                 cudaMemcpyHostToDevice, r.st));
        POS_TRY(il_process(r, 0, static_cast<const Vec32 *>(ws.d_front[0].p), n_slices));
    }
    POS_CUDA(cudaStreamSynchronize(r.st));
    const double ms_search = il_ms_since(t_search);

    Key128 inc;
    unsigned long long hs[kStCount];
    POS_CUDA(cudaMemcpy(&inc, ws.d_inc.p, sizeof(inc), cudaMemcpyDeviceToHost));
    POS_CUDA(cudaMemcpy(hs, r.stats, sizeof(hs), cudaMemcpyDeviceToHost));
    if (hs[kStTimeout])
        return fail(POS_ETIMEOUT, "the incumbent's compare-and-swap loop hit its iteration "
                                  "limit (pos_problem.cas_limit rounds)");
    if (hs[kStBulkTimeout])
        return fail(POS_ETIMEOUT, "a block's cost-table staging (TMA bulk copy) did not "
                                  "complete within its poll limit");
    if (stats) {
        stats->evaluated = hs[kStEvaluated];
        stats->warmup_evaluated = (uint64_t)n_slices;
        stats->prefixes = hs[kStPrefixes];
        stats->pruned_bound = hs[kStPrunedBound];
        stats->pruned_memory = hs[kStPrunedMemory];
        stats->relaxations = hs[kStRelaxations];
        stats->slices = (uint64_t)n_slices;
        stats->slices_feasible = (uint64_t)n_slices;
        stats->launches = r.launches;
        stats->ms_setup = ms_setup;
        stats->ms_warmup = ms_warm;
        stats->ms_search = ms_search;
        stats->ms_expand = r.ms_expand;
        stats->ms_complete = r.ms_complete;
        stats->ms_leaf = r.ms_leaf;
        stats->expand_launches = r.n_expand;
        stats->complete_launches = r.n_complete;
        stats->leaf_launches = r.n_leaf;
        stats->parents_expand = hs[kStParentsExpand];
        stats->parents_complete = hs[kStParentsComplete];
        stats->leaves = hs[kStLeaves];
        for (int x = 0; x < POS_MAX_STAGES; ++x) {
            stats->ms_depth[x] = r.ms_depth[x];
            stats->launches_depth[x] = r.launches_depth[x];
            stats->parents_depth[x] = hs[kStDepthParents + x];
            stats->children_depth[x] = hs[kStDepthChildren + x];
        }
    }
    if (inc.obj == ~0ull) {
        if (stats) stats->ms_total = il_ms_since(t_start);
        return fail(POS_EINFEASIBLE, "no memory-feasible plan");
    }
    const uint64_t ord = inc.idx / r.n_map;
    out->found = 1;
    out->map_rank = inc.idx % r.n_map;
    plan_slice_fields(p, sp, ord, out);
    out->S = N;
    out->makespan = (int32_t)(inc.obj / (Q / ((uint64_t)out->D * out->M)));
    out->global_index = inc.idx;
    for (int x = 0; x < POS_MAX_STAGES; ++x) out->layers[x] = 0;
    host_unrank(r.L, r.J, out->map_rank, out->layers);
    if (stats) stats->ms_total = il_ms_since(t_start);
    return POS_OK;
}

}  // namespace pos
