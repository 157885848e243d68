// Evaluation kernels of poseidon_eval_batch (hot-path steps a2-a5).
//
// One thread evaluates one candidate, in two passes: a decode pass (field
// checks, overflow guard, unranking, memory check; few registers, so the
// latency of its dependent shared-memory lookups is hidden by many warps)
// writes every candidate's cut positions to its place in the (S, M)-sorted
// order, and the makespan pass reads them coalesced.  The makespan loop
// costs ~6*S*M integer ops and its live registers grow with S (about 7*S),
// so the batch is first counting-sorted by exact (S, M) (stream-ordered
// scratch: every candidate's sorted position), and then a family of
// kernels, each owning the candidates of one S range and either M >= S
// (ramps unrolled, steady loop) or M < S (the whole schedule unrolled per
// (S, M)), walks its contiguous range of the sorted records with launch
// bounds matched to its register need.  Warps therefore see one (S, M)
// except at bucket boundaries, and no kernel waits at a block barrier after
// staging the cost tables.
//
// Sort keys: fast path (M >= S for 1F1B, M >= 2S-1 for Eager 1F1B) ->
// (S-1)*256 + M (the other slots of each S stay empty); short path ->
// 4096 + (S-1)*32 + M; Interleaved 1F1B records with V >= 2 get keys after
// those (interleaved.cuh); records with S outside 1..16 or M = 0 are flagged
// invalid by the sort pass and get no key.
#pragma once
#include <algorithm>

#include "common.cuh"

namespace pos {

constexpr int kKeys = 4096 + 16 * 32;  // fast keys, then short-path keys
constexpr int kEvalThreads = 128;

__host__ __device__ inline int fast_key_begin(int S) { return (S - 1) * 256; }
__host__ __device__ inline int generic_key_begin(int S) { return 4096 + (S - 1) * 32; }

struct EvalParams {
    const uint4 *cands;    // 16-byte records (poseidon_eval_batch), or
    const uint2 *cands_ex; // 24-byte records with a TP index per stage
                           // (poseidon_eval_batch_ex; cands is then NULL)
    int64_t n;
    int32_t *T;
    uint8_t *F;
    const uint32_t *dest;  // sorted position of every candidate (kNoDest:
                           // no key, answered by the histogram pass)
    const uint32_t *offs;  // [nkeys + 1] start of every key in sorted order
    uint4 *cuts;           // per sorted position j, two 16-byte words (read once,
                           // with evict-first loads, so that the outputs'
                           // sectors stay in L2):
                           // cuts[2j]: the cut positions (push_cut's layout;
                           // ascending bytes 0..14 for interleaved records),
                           // byte 15 = 1 when the result is already written;
                           // cuts[2j+1]: (candidate index, type_code, the
                           // record's S|M|tp|V word, per-stage TP code), so the makespan
                           // kernels read 32 contiguous bytes and no record
    const void *blob;
    BlobLayout lay;
    // guard_m[J]: the smallest M (1..255; 256 for none) at which the
    // overflow guard (guard_trips) trips for J (virtual) stages: U(J, M)
    // grows with M since every cost is non-negative
    uint16_t guard_m[POS_MAX_STAGES + 1];
    Programs pg;           // level programs of the schedule's short path
    int nkeys;             // kKeys, or kKeysIl under Interleaved 1F1B
    int per_stage_tp;      // 1: records carry a TP index per stage (n_tp <= 4)
    // the handle's memory-limit table (Handle::lim_*): the decode pass stages
    // the binomials and this table and checks memory with one byte per stage
    int lim_off, lim_w, lim_bytes;
};

// The record fields every pass reads, in the 16-byte record's word layout:
// x, y = composition rank, z = type code, w = S | M << 8 | tp << 16 | V << 24
// (tp = 0 for a 24-byte record), plus the per-stage TP code of a 24-byte
// record (TP index of stage s in bits [2s, 2s+2); 0 for 16-byte records).
struct RecView {
    uint4 rec;
    uint32_t tpc;
};
__device__ __forceinline__ RecView load_record(const EvalParams &p, uint32_t i) {
    RecView v;
    if (p.per_stage_tp) {
        // 24 bytes: u64 rank, u32 type code, u32 TP code, u8 S, M, V, pad, u32 pad
        const uint2 a = __ldg(p.cands_ex + 3 * (size_t)i), b = __ldg(p.cands_ex + 3 * (size_t)i + 1),
                    c = __ldg(p.cands_ex + 3 * (size_t)i + 2);
        v.rec = make_uint4(a.x, a.y, b.x, (c.x & 0xffffu) | ((c.x & 0xff0000u) << 8));
        v.tpc = b.y;
    } else {
        v.rec = __ldg(p.cands + i);
        v.tpc = 0;
    }
    return v;
}

// Class of stage s: type_s * n_tp + its TP index, which is tp for a 16-byte
// record (whose per-stage TP code reads 0) and the stage's field of the TP
// code for a 24-byte record (whose tp reads 0), so no select is needed.
__device__ __forceinline__ int stage_class(uint32_t tcode, uint32_t tpc, int tp, int n_tp, int s) {
    return (int)((tcode >> (2 * s)) & 3u) * n_tp + tp + (int)((tpc >> (2 * s)) & 3u);
}

// Are the 2-bit type fields of stages 0..S-1 (1 <= S <= 16) all below
// n_types (1..4)?  A field is >= n_types when its high bit is set
// (n_types <= 2), when both bits are set (n_types = 3), or, for one type,
// when it is not zero.
__device__ __forceinline__ bool types_ok(uint32_t tcode, int S, int n_types) {
    const uint32_t mask = S >= 16 ? 0xffffffffu : (1u << (2 * S)) - 1u;
    const uint32_t f = tcode & mask;
    const uint32_t bad = n_types >= 4   ? 0u
                         : n_types == 3 ? (f & (f >> 1) & 0x55555555u)
                         : n_types == 2 ? (f & 0xaaaaaaaau)
                                        : f;
    return bad == 0u;
}

// The decode pass packs the cut positions of a (non-interleaved) record
// (each below 256) into the bytes of a 16-byte word by shifting them in from
// the bottom: after pushing
// cut[1], ..., cut[n-1] (n - 1 <= 15 pushes), cut[q] sits in byte n-1-q and
// byte 15 is still 0 (the "answered by the decode pass" flag).  A push is
// three funnel shifts and a shift-or, whatever the stage index.
__device__ __forceinline__ void push_cut(uint4 &v, int c) {
    v.w = __funnelshift_l(v.z, v.w, 8);
    v.z = __funnelshift_l(v.y, v.z, 8);
    v.y = __funnelshift_l(v.x, v.y, 8);
    v.x = (v.x << 8) | (uint32_t)c;
}

// cut[q] (1 <= q <= n-1) of n stages from the packed word (n a constant
// after unrolling, so this is a constant shift of a constant word)
__device__ __forceinline__ int packed_cut(const uint32_t (&pw)[4], int n, int q) {
    const int b = n - 1 - q;
    return (int)((pw[b >> 2] >> (8 * (b & 3))) & 0xffu);
}

// Decode pass for an Interleaved 1F1B record (pad byte V >= 2, S = N
// devices): checks its fields (N*V <= 16 virtual stages, at most L, M a
// multiple of N) and the overflow guard over the N*V virtual stages, and
// unranks the composition of L layers into the virtual stages.  Memory is
// checked by the makespan kernel (it needs the device chains).
__device__ __forceinline__ uint4 decode_il(const Tab &t, const uint4 &rec, uint32_t tpc,
                                           const EvalParams &p, uint32_t i) {
    const uint64_t rank = (uint64_t)rec.x | ((uint64_t)rec.y << 32);
    const uint32_t tcode = rec.z;
    const int S = rec.w & 0xff;
    const int M = (rec.w >> 8) & 0xff;
    const int tp = (rec.w >> 16) & 0xff;
    const int V = (int)(rec.w >> 24);
    const int J = S * V, L = t.L();
    bool ok = S >= 1 && J <= POS_MAX_STAGES && J <= L && M >= 1 && M % S == 0 &&
              tp < t.n_tp();
    const uint64_t n_map = ok ? binom(t, L - 1, J - 1) : 0;
    ok = ok && rank < n_map;
    ok = ok && types_ok(tcode, S, t.n_types()) &&
         types_ok(tpc, S, t.n_tp());  // tpc = 0 for 16-byte records
    const uint4 done = make_uint4(0, 0, 0, 1u << 24);
    if (!ok) {
        p.T[i] = -1;
        p.F[i] = POS_FEAS_INVALID;
        return done;
    }
    if (M >= (int)p.guard_m[J]) {  // the overflow guard
        p.T[i] = -1;
        p.F[i] = POS_FEAS_OVERFLOW;
        return done;
    }
    // cut[1..J-1] in ascending bytes 0..14, the layout the interleaved
    // search writes its leaf records in
    uint64_t Y = n_map - rank;
    uint64_t lo8 = 0, hi8 = 0;
    int c = 0;
#pragma unroll 1
    for (int j = 0; j < J - 1; ++j) {
        const int rem = L - c, k = J - j - 1;
        c += rem - unrank_step(t, rem, k, Y);
        if (j < 8) lo8 |= (uint64_t)c << (8 * j);
        else hi8 |= (uint64_t)c << (8 * (j - 8));
    }
    return make_uint4((uint32_t)lo8, (uint32_t)(lo8 >> 32), (uint32_t)hi8,
                      (uint32_t)(hi8 >> 32) & 0x00ffffffu);
}

// Decode pass for one candidate: checks its fields and the overflow guard,
// unranks the composition stage by stage (unrank_step, carrying Y),
// checks each stage's memory as soon as its cut is known (LIM: by the
// memory-limit table staged at `lim`), and packs the cut positions
// (push_cut).  Invalid and overflowing candidates are answered here.  S is
// a runtime value and the stage loop is not unrolled, which keeps the
// kernel small enough to run many warps per SM.
template <bool LIM>
__device__ __forceinline__ uint4 decode_one(const Tab &t, const uint4 &rec, uint32_t tpc,
                                            const EvalParams &p, uint32_t i,
                                            const uint8_t *lim) {
    const uint64_t rank = (uint64_t)rec.x | ((uint64_t)rec.y << 32);
    const uint32_t tcode = rec.z;
    const int S = rec.w & 0xff;
    const int M = (rec.w >> 8) & 0xff;
    const int tp = (rec.w >> 16) & 0xff;
    const int L = t.L();
    if (t.ly->sched == POS_SCHED_INTERLEAVED_1F1B && (rec.w >> 24) >= 2)
        return decode_il(t, rec, tpc, p, i);
    bool ok = S >= 1 && S <= POS_MAX_STAGES && M >= 1 && S <= L && tp < t.n_tp();
    const uint64_t n_map = ok ? binom(t, L - 1, S - 1) : 0;
    ok = ok && rank < n_map;
    ok = ok && types_ok(tcode, S, t.n_types()) &&
         (!p.per_stage_tp || types_ok(tpc, S, t.n_tp()));  // tpc = 0 for 16-byte records
    const uint4 done = make_uint4(0, 0, 0, 1u << 24);  // byte 15 = 1: answered here
    if (!ok) {
        p.T[i] = -1;
        p.F[i] = POS_FEAS_INVALID;
        return done;
    }
    if (M >= (int)p.guard_m[S]) {  // the overflow guard
        p.T[i] = -1;
        p.F[i] = POS_FEAS_OVERFLOW;
        return done;
    }
    uint64_t Y = n_map - rank;
    uint4 cuts = make_uint4(0, 0, 0, 0);
    const int n_tp = t.n_tp();
    // in-flight micro-batches of stage s before the cap at M: S - s under
    // 1F1B, 2(S-1-s)+1 under Eager 1F1B (inflight()), stepped per stage
    const bool eager = t.ly->sched == POS_SCHED_EAGER_1F1B;
    const int dw = eager ? 2 : 1;
    int wl = eager ? 2 * S - 1 : S;
    // the stage's memory check, with the type and TP fields shifted down as
    // the stages go
    uint32_t tc = tcode, tq = tpc;
    auto fits_stage = [&](int a, int b) {
        const int cls = (int)(tc & 3u) * n_tp + tp + (int)(tq & 3u);  // stage_class
        const int w = min(wl, M);
        tc >>= 2;
        tq >>= 2;
        wl -= dw;
        if constexpr (LIM) return b <= (int)lim[(cls * p.lim_w + w - 1) * (L + 1) + a];
        else return stage_fits_w(t, w, cls, a, b);
    };
    bool fits = true;
    int c = 0;
    // stages 0..S-2 (k stages after each), then the last one up to L
#pragma unroll 1
    for (int k = S - 1; k >= 1; --k) {
        const int rem = L - c;
        const int c2 = c + (rem - unrank_step(t, rem, k, Y));
        push_cut(cuts, c2);
        fits &= fits_stage(c, c2);
        c = c2;
    }
    fits &= fits_stage(c, L);
    p.F[i] = fits ? POS_FEAS_YES : POS_FEAS_NO;
    return cuts;
}

template <int PATH>
struct EvalWith {
    template <int S>
    struct One {
        // makespan of a decoded candidate (cuts packed by the decode pass)
        static __device__ __forceinline__ void run(const Tab &t, const uint4 &rec,
                                                   const uint4 &packed, const Programs &pg,
                                                   int32_t &T) {
            // rec: x = per-stage TP code (0 for 16-byte records), z = type
            // code, w = S | M << 8 | tp << 16 | V << 24 (tp = 0 for 24-byte
            // records)
            const uint32_t tcode = rec.z;
            const int M = (rec.w >> 8) & 0xff;
            const int tp = (rec.w >> 16) & 0xff;
            int cls[S], cut[S + 1];
#pragma unroll
            for (int s = 0; s < S; ++s)
                cls[s] = stage_class(tcode, rec.x, tp, t.n_tp(), s);
            const uint32_t pw[4] = {packed.x, packed.y, packed.z, packed.w};
            cut[0] = 0;
#pragma unroll
            for (int s = 0; s < S - 1; ++s) cut[s + 1] = packed_cut(pw, S, s + 1);
            cut[S] = t.L();
            StageW<S> w;
            stage_weights<S>(t, cut, cls, w);
            T = makespan_path<S, PATH>(w, M, pg);
        }
    };
};

template <int SLO, int SHI, int PATH>
__device__ __forceinline__ void dispatch_range(int S, const Tab &t, const uint4 &rec,
                                               const uint4 &packed, const Programs &pg,
                                               int32_t &T) {
#define POS_EV(n)                                                                            \
    if (n >= SLO && n <= SHI && S == n) {                                                    \
        EvalWith<PATH>::template One<(n >= SLO && n <= SHI) ? n : SLO>::run(t, rec, packed, pg, T); \
        return;                                                                              \
    }
    POS_EV(1) POS_EV(2) POS_EV(3) POS_EV(4) POS_EV(5) POS_EV(6) POS_EV(7) POS_EV(8)
    POS_EV(9) POS_EV(10) POS_EV(11) POS_EV(12) POS_EV(13) POS_EV(14) POS_EV(15) POS_EV(16)
#undef POS_EV
}

// Evaluates the sorted positions [offs[key_lo], offs[key_hi]): all
// candidates with S in [SLO, SHI] on path PATH.
template <int SLO, int SHI, int PATH, int MINB>
__global__ void __launch_bounds__(kEvalThreads, MINB) eval_kernel(EvalParams p) {
    extern __shared__ __align__(16) unsigned char sm[];
    constexpr bool kFast = PATH == kPathFast || PATH == kPathEager;
    const int key_lo = kFast ? fast_key_begin(SLO) : generic_key_begin(SLO);
    const int key_hi = kFast ? fast_key_begin(SHI + 1) : generic_key_begin(SHI + 1);
    // the key offsets come from the sort's scan, two or more kernels back
    const int64_t begin = p.offs[key_lo], end = p.offs[key_hi];
    // blocks with no candidate (all of them when the range is empty) leave
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
    // whole warps iterate together (ballots below)
    const int64_t span = ((end - begin) + 31) & ~(int64_t)31;
    for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < span; j += stride) {
        bool active = j < end - begin;
        uint32_t i = 0;
        uint4 rec = make_uint4(0, 0, 0, 0), packed = make_uint4(0, 0, 0, 0);
        if (active) {
            packed = __ldcs(p.cuts + 2 * (begin + j));
            const uint4 meta = __ldcs(p.cuts + 2 * (begin + j) + 1);
            active = (packed.w >> 24) == 0;  // not answered by the decode pass
            i = meta.x;
            rec = make_uint4(meta.w, 0u, meta.y, meta.z);
        }
        const int S = active ? (int)(rec.w & 0xff) : 0;
        int32_t T = -1;
        unsigned pending = __ballot_sync(0xffffffffu, active);
        while (pending) {
            const int leader = __ffs(pending) - 1;
            const int Sg = __shfl_sync(0xffffffffu, S, leader);
            const bool mine = active && S == Sg;
            const unsigned grp = __ballot_sync(0xffffffffu, mine);
            if (mine) dispatch_range<SLO, SHI, PATH>(Sg, t, rec, packed, p.pg, T);
            pending &= ~grp;
        }
        if (active) p.T[i] = T;
    }
}

template <int SLO, int SHI, int PATH, int MINB>
pos_status launch_eval_range(const EvalParams &p, cudaStream_t stream) {
    auto kern = eval_kernel<SLO, SHI, PATH, MINB>;
    const int smem = p.lay.bytes;
    POS_TRY(ensure_smem(reinterpret_cast<const void *>(kern), smem));
    int per_sm = 0;
    POS_TRY(blocks_per_sm(reinterpret_cast<const void *>(kern), kEvalThreads, smem, &per_sm));
    if (per_sm < 1) return fail(POS_ECUDA, "eval kernel does not fit on an SM");
    const int64_t blocks = (p.n + kEvalThreads - 1) / kEvalThreads;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(blocks, (int64_t)per_sm * sm_count()));
    POS_CUDA(launch_dependent(kern, grid, kEvalThreads, smem, stream, p));
    return POS_OK;
}

pos_status launch_decode(const EvalParams &p, cudaStream_t stream);

// one launcher per instantiation unit (eval_range_*.cu)
pos_status eval_fast_1_4(const EvalParams &p, cudaStream_t s);
pos_status eval_fast_5_8(const EvalParams &p, cudaStream_t s);
pos_status eval_fast_9_12(const EvalParams &p, cudaStream_t s);
pos_status eval_fast_13_16(const EvalParams &p, cudaStream_t s);
pos_status eval_generic_2_8(const EvalParams &p, cudaStream_t s);
pos_status eval_generic_9_12(const EvalParams &p, cudaStream_t s);
pos_status eval_generic_13_14(const EvalParams &p, cudaStream_t s);
pos_status eval_generic_15_15(const EvalParams &p, cudaStream_t s);
pos_status eval_generic_16_16(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_1_6(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_7_10(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_11_13(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_14_16(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_short_2_8(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_short_9_10(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_short_11_12(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_short_13_13(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_short_14_14(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_short_15_15(const EvalParams &p, cudaStream_t s);
pos_status eval_eager_short_16_16(const EvalParams &p, cudaStream_t s);

}  // namespace pos
