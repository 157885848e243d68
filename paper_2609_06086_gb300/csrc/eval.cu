// poseidon_eval_batch, poseidon_eval_batch_host and poseidon_argmin (hot-path
// step a9).  The evaluation kernels live in eval_kernel.cuh and the
// eval_range_*.cu instantiation units.
#include <mutex>
#include <utility>

#include "interleaved.cuh"

namespace pos {

// ---------------------------------------------------------------------------
// argmin over (makespan, index) among feasible entries, ties -> lowest index
// ---------------------------------------------------------------------------
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
    __shared__ int32_t st[kArgminThreads / 32];
    __shared__ long long si[kArgminThreads / 32];
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

// ---------------------------------------------------------------------------
// counting sort of the candidates by (S, M) key
// ---------------------------------------------------------------------------
// il_key: kIlKeyOf staged in shared memory (a __constant__ read whose index
// differs between the lanes of a warp is served one address at a time)
__device__ __forceinline__ int eval_key(int sched, uint32_t w, const int16_t *il_key) {
    const int S = w & 0xff, M = (w >> 8) & 0xff, V = (int)(w >> 24);
    if (S < 1 || S > POS_MAX_STAGES || M < 1) return -1;
    if (sched == POS_SCHED_INTERLEAVED_1F1B && V >= 2) {
        // N = S devices, V chunks each: key block of (N, V), index q = M / N
        if (S * V > POS_MAX_STAGES || M % S != 0) return -1;
        return kKeys + il_key[(S - 1) * 17 + V] + M / S;
    }
    return M >= fast_min_m(sched, S) ? fast_key_begin(S) + M : generic_key_begin(S) + M;
}

// global key histogram; invalid records are answered right here
// 2-byte key per candidate, written by the histogram pass and read by the
// scatter pass (instead of the 16-byte record, twice)
constexpr uint16_t kNoKey = 0xffff;

// The S | M << 8 | tp << 16 | V << 24 word of record i (24-byte records:
// S, M, V at bytes 16..18, tp = 0).
__device__ __forceinline__ uint32_t record_word(const EvalParams &p, int64_t i) {
    if (p.per_stage_tp) {
        const uint32_t w = __ldg(reinterpret_cast<const uint32_t *>(p.cands_ex) + 6 * i + 4);
        return (w & 0xffffu) | ((w & 0xff0000u) << 8);
    }
    return __ldg(&p.cands[i].w);
}

template <int NK>
__global__ void sort_hist_kernel(EvalParams p, int64_t n, uint32_t *hist, uint16_t *keys,
                                 int32_t *T, uint8_t *F) {
    const int sched = p.lay.sched;
    __shared__ uint32_t h[NK];
    __shared__ int16_t il_key[8 * 17];
    for (int i = threadIdx.x; i < NK; i += blockDim.x) h[i] = 0;
    if (sched == POS_SCHED_INTERLEAVED_1F1B)
        for (int i = threadIdx.x; i < 8 * 17; i += blockDim.x) il_key[i] = kIlKeyOf[i / 17][i % 17];
    __syncthreads();
    // four record words in flight per thread (the pass is bound by HBM
    // latency: one load per thread and iteration kept too few bytes in flight)
    const int64_t bd = blockDim.x;
    for (int64_t i0 = blockIdx.x * 4 * bd + threadIdx.x; i0 < n; i0 += (int64_t)gridDim.x * 4 * bd) {
        uint32_t wv[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) wv[u] = i0 + u * bd < n ? record_word(p, i0 + u * bd) : 0u;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t i = i0 + u * bd;
            if (i >= n) break;
            const int k = eval_key(sched, wv[u], il_key);
            keys[i] = k >= 0 ? (uint16_t)k : kNoKey;
            if (k >= 0) {
                atomicAdd(&h[k], 1u);
            } else {
                T[i] = -1;
                F[i] = POS_FEAS_INVALID;
            }
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < NK; i += blockDim.x)
        if (h[i]) atomicAdd(&hist[i], h[i]);
}

// exclusive prefix sum of the histogram (one block); cursor = offs copy
template <int NK>
// (1024 threads: each sums a run of keys; the run totals are scanned within
// each warp by shuffles, then across the 32 warp totals by the first warp)
__global__ void __launch_bounds__(1024) sort_scan_kernel(const uint32_t *hist, uint32_t *offs,
                                                        uint32_t *cursor) {
    __shared__ uint32_t warp_total[32];
    grid_dep_wait();  // the histogram
    grid_dep_trigger();
    const int per = (NK + blockDim.x - 1) / blockDim.x;
    const int lo = threadIdx.x * per, hi = min(NK, lo + per);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint32_t sum = 0;
    for (int i = lo; i < hi; ++i) sum += hist[i];
    uint32_t incl = sum;  // inclusive scan over the warp's lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
    }
    if (lane == 31) warp_total[wid] = incl;
    __syncthreads();
    if (wid == 0) {
        const uint32_t t = lane < (int)(blockDim.x >> 5) ? warp_total[lane] : 0u;
        uint32_t ti = t;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t v = __shfl_up_sync(0xffffffffu, ti, o);
            if (lane >= o) ti += v;
        }
        warp_total[lane] = ti - t;  // exclusive prefix of the warp totals
        if (lane == 31) offs[NK] = ti;
    }
    __syncthreads();
    uint32_t run = warp_total[wid] + incl - sum;
    for (int i = lo; i < hi; ++i) {
        offs[i] = run;
        cursor[i] = run;
        run += hist[i];
    }
}

// Each block takes chunks of `chunk` candidates: counts their keys, reserves
// one range per key with a single atomic, then gives every candidate its
// sorted position (written in input order, so coalesced).  Chunks of up to
// 16384 for large batches (measured against 4096, 8192 and 32768: within
// 0.5 % of a config-5 call, 16384 the fastest), smaller ones (down to 1024)
// so that small batches still spread over the SMs.
// Within a chunk the candidates of one key get consecutive positions, so
// the decode pass's scattered record writes come in short runs.
__host__ inline int64_t scatter_chunk(int64_t n, int sms) {
    int64_t c = (n / (8 * (int64_t)sms) + 511) & ~(int64_t)511;
    return c < 1024 ? 1024 : (c > 16384 ? 16384 : c);
}

constexpr uint32_t kNoDest = 0xffffffffu;

template <int NK>
__global__ void sort_scatter_kernel(const uint16_t *keys, int64_t n, int64_t chunk,
                                    uint32_t *cursor, uint32_t *dest) {
    __shared__ uint32_t h[NK];
    grid_dep_wait();  // the keys (histogram pass) and the cursors (scan)
    grid_dep_trigger();
    for (int64_t c0 = blockIdx.x * chunk; c0 < n; c0 += (int64_t)gridDim.x * chunk) {
        const int64_t c1 = min(n, c0 + chunk);
        for (int i = threadIdx.x; i < NK; i += blockDim.x) h[i] = 0;
        __syncthreads();
        for (int64_t i = c0 + threadIdx.x; i < c1; i += blockDim.x) {
            const uint16_t k = __ldg(keys + i);
            if (k != kNoKey) atomicAdd(&h[k], 1u);
        }
        __syncthreads();
        for (int i = threadIdx.x; i < NK; i += blockDim.x)
            if (h[i]) h[i] = atomicAdd(&cursor[i], h[i]);
        __syncthreads();
        for (int64_t i = c0 + threadIdx.x; i < c1; i += blockDim.x) {
            const uint16_t k = __ldg(keys + i);
            dest[i] = k != kNoKey ? atomicAdd(&h[k], 1u) : kNoDest;
        }
        __syncthreads();
    }
}

// Decode pass.  Blocks take windows of `window` consecutive candidates:
// their records and sorted positions are read coalesced into shared memory,
// and each decoded 32-byte record is written to its sorted position.  The
// decode's cost grows with the number of unranking stages (S, or N*V for an
// interleaved record) and a window mixes them, so the block orders the
// window's candidates by that count (a counting sort over 16 buckets) and
// its warps then decode 32 consecutive entries of that order at a time:
// the lanes of a warp loop over (nearly) the same number of stages.
// LIM: only the binomials (the blob's first off_Pw bytes) and the
// memory-limit table are staged, the table right after the binomials.
constexpr int kDecodeThreads = 256;
constexpr int kDecodeWindowMax = 768;
constexpr int kDecodeBuckets = POS_MAX_STAGES + 1;  // stage counts 1..16 (0 unused)

__device__ __forceinline__ int decode_bucket(int sched, uint32_t w) {
    const int S = w & 0xff, V = (int)(w >> 24);
    const int J = (sched == POS_SCHED_INTERLEAVED_1F1B && V >= 2) ? S * V : S;
    return min(max(J, 1), POS_MAX_STAGES);  // records beyond are answered at once
}

// the two 16-byte words of a decoded record in one 32-byte store
__device__ __forceinline__ void store_decoded(uint4 *dst, const uint4 &a, const uint4 &b) {
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(dst),
                 "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b.x), "r"(b.y), "r"(b.z), "r"(b.w)
                 : "memory");
}

struct DecodeWindow {
    uint4 rec[kDecodeWindowMax];       // RecView::rec of each candidate
    uint32_t tpc[kDecodeWindowMax];    // RecView::tpc
    uint32_t dest[kDecodeWindowMax];   // sorted position (kNoDest: no key)
    uint16_t order[kDecodeWindowMax];  // window offsets in bucket order
    uint8_t bucket[kDecodeWindowMax];  // bucket of each candidate (0: no key)
    uint32_t slot[kDecodeBuckets + 1]; // bucket counts, then next free slots
    uint32_t n_valid;
};

template <bool LIM>
__global__ void __launch_bounds__(kDecodeThreads, 4) decode_kernel(EvalParams p, int window) {
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ DecodeWindow win;
    if constexpr (LIM) {
        stage_blob(sm, p.blob, p.lay.off_Pw);
        stage_blob(sm + p.lay.off_Pw, static_cast<const unsigned char *>(p.blob) + p.lim_off,
                   p.lim_bytes);
    } else {
        stage_blob(sm, p.blob, p.lay.bytes);
    }
    __syncthreads();
    grid_dep_wait();  // the sorted positions (scatter pass)
    grid_dep_trigger();
    const Tab t = tab_at(sm, p.lay);
    const uint8_t *lim = sm + p.lay.off_Pw;
    const int sched = p.lay.sched;
    const int lane = threadIdx.x & 31;
    for (int64_t w0 = blockIdx.x * (int64_t)window; w0 < p.n; w0 += (int64_t)gridDim.x * window) {
        const int wn = (int)min((int64_t)window, p.n - w0);
        // 1. the window's records and positions, and the candidates per
        // bucket (those without a key are already answered)
        if (threadIdx.x <= kDecodeBuckets) win.slot[threadIdx.x] = 0;
        __syncthreads();
#pragma unroll 4
        for (int li = threadIdx.x; li < wn; li += kDecodeThreads) {
            const uint32_t i = (uint32_t)(w0 + li);
            const RecView v = load_record(p, i);
            const uint32_t d = __ldg(p.dest + i);
            win.rec[li] = v.rec;
            win.tpc[li] = v.tpc;
            win.dest[li] = d;
            const int b = d != kNoDest ? decode_bucket(sched, v.rec.w) : 0;
            win.bucket[li] = (uint8_t)b;
            if (b) atomicAdd(&win.slot[b], 1u);
        }
        __syncthreads();
        // 2. exclusive prefix over the buckets (first warp)
        if (threadIdx.x < 32) {
            const uint32_t c = lane <= kDecodeBuckets ? win.slot[lane] : 0u;
            uint32_t incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += v;
            }
            if (lane <= kDecodeBuckets) win.slot[lane] = incl - c;
            if (lane == 31) win.n_valid = incl;
        }
        __syncthreads();
        // 3. the window's offsets in bucket order
        for (int li = threadIdx.x; li < wn; li += kDecodeThreads) {
            const int b = win.bucket[li];
            if (b) win.order[atomicAdd(&win.slot[b], 1u)] = (uint16_t)li;
        }
        __syncthreads();
        // 4. decode: each warp takes 32 consecutive entries of the order
        const int nv = (int)win.n_valid;
        for (int k = threadIdx.x; k < nv; k += kDecodeThreads) {
            const int li = win.order[k];
            const uint32_t i = (uint32_t)(w0 + li);
            const uint4 rec = win.rec[li];
            const uint32_t tpc = win.tpc[li];
            const uint4 out = decode_one<LIM>(t, rec, tpc, p, i, lim);
            store_decoded(p.cuts + 2 * (size_t)win.dest[li], out, make_uint4(i, rec.z, rec.w, tpc));
        }
        __syncthreads();  // the window's arrays are rewritten for the next one
    }
}

pos_status launch_decode(const EvalParams &p, cudaStream_t stream) {
    const bool lim = p.lim_bytes > 0;
    const void *kern = lim ? reinterpret_cast<const void *>(decode_kernel<true>)
                           : reinterpret_cast<const void *>(decode_kernel<false>);
    const int smem = lim ? p.lay.off_Pw + p.lim_bytes : p.lay.bytes;
    POS_TRY(ensure_smem(kern, smem));
    int per_sm = 0;
    POS_TRY(blocks_per_sm(kern, kDecodeThreads, smem, &per_sm));
    // blocks of at least 1024 candidates; the same number of windows for
    // every block (up to one), so that the blocks finish together
    const int64_t blocks = std::max<int64_t>(
        1, std::min<int64_t>((p.n + 1023) / 1024, (int64_t)std::max(per_sm, 1) * sm_count()));
    const int64_t rounds = (p.n + blocks * kDecodeWindowMax - 1) / (blocks * kDecodeWindowMax);
    const int window = (int)((p.n + blocks * rounds - 1) / (blocks * rounds));
    if (lim) POS_CUDA(launch_dependent(decode_kernel<true>, (int)blocks, kDecodeThreads, smem, stream, p, window));
    else POS_CUDA(launch_dependent(decode_kernel<false>, (int)blocks, kDecodeThreads, smem, stream, p, window));
    return POS_OK;
}

// Stream-ordered scratch comes from a library-owned pool per device that
// keeps its memory between calls (release threshold: unlimited).
static std::mutex g_pool_mutex;
static cudaMemPool_t g_pool[64];

static pos_status scratch_pool(cudaMemPool_t *out) {
    int dev = 0;
    POS_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= 64) return fail(POS_EINVAL, "device index above 63");
    std::lock_guard<std::mutex> lock(g_pool_mutex);
    if (!g_pool[dev]) {
        cudaMemPoolProps props = {};
        props.allocType = cudaMemAllocationTypePinned;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        cudaMemPool_t pool;
        POS_CUDA(cudaMemPoolCreate(&pool, &props));
        uint64_t keep = ~0ull;
        POS_CUDA(cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep));
        g_pool[dev] = pool;
    }
    *out = g_pool[dev];
    return POS_OK;
}

// A second stream per device for the short-path kernels (M < S under 1F1B,
// M < 2S-1 under Eager 1F1B) and then the smallest fast-path range (under
// Interleaved 1F1B: every 1F1B range, then the smallest interleaved range):
// every evaluation kernel depends only on the decode pass, and the short
// paths are bound by instruction fetch rather than by the ALU, so they run
// beside the other fast-path kernels instead of after them (measured: the
// side chain with the smallest fast range was faster than the short paths
// alone, two chains splitting the fast ranges slower).  The
// fork and join events are shared per device, so a call holds the device's
// side mutex from the fork to the join (two calls from different host
// threads must not interleave their record / wait pairs).
struct SideStream {
    cudaStream_t s = nullptr;
    cudaEvent_t fork = nullptr, join = nullptr;
    std::mutex mu;
};
static std::mutex g_side_mutex;
static SideStream g_side[64];

static pos_status side_stream(SideStream **out) {
    int dev = 0;
    POS_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= 64) return fail(POS_EINVAL, "device index above 63");
    std::lock_guard<std::mutex> lock(g_side_mutex);
    SideStream &ss = g_side[dev];
    if (!ss.s) {
        POS_CUDA(cudaEventCreateWithFlags(&ss.fork, cudaEventDisableTiming));
        POS_CUDA(cudaEventCreateWithFlags(&ss.join, cudaEventDisableTiming));
        POS_CUDA(cudaStreamCreateWithFlags(&ss.s, cudaStreamNonBlocking));
    }
    *out = &ss;
    return POS_OK;
}

// d_cands: 16-byte records, or 24-byte records when per_stage_tp.
pos_status launch_eval(Handle *h, const void *d_cands, bool per_stage_tp, int64_t n,
                       int32_t *d_T, uint8_t *d_F, cudaStream_t stream) {
    if (n == 0) return POS_OK;
    cudaMemPool_t pool;
    pos_status st = scratch_pool(&pool);
    if (st != POS_OK) return st;
    Programs pg;  // the schedule's level programs (Eager 1F1B, few micro-batches)
    if ((st = schedule_programs(h->lay.sched, &pg)) != POS_OK) return st;
    // batches above 2^24 candidates go in chunks of 2^24: a chunk's outputs
    // (5 bytes per candidate, 80 MB), written in sorted order and so
    // scattered over the output arrays, stay in L2 until whole sectors are
    // written back (the 32-bit sorted positions would allow 2^31)
    const int64_t chunk = (int64_t)1 << 24;
    for (int64_t base = 0; base < n; base += chunk) {
        const int64_t m = std::min(chunk, n - base);
        void *scratch = nullptr;
        const bool il = h->lay.sched == POS_SCHED_INTERLEAVED_1F1B;
        const int nk = il ? kKeysIl : kKeys;
        // scratch: decoded records (32 B per candidate), the sort arrays, the keys
        const size_t sbytes = 32 * (size_t)m + sizeof(uint32_t) * (3 * (size_t)nk + 1 + (size_t)m) +
                              sizeof(uint16_t) * (size_t)m;
        POS_CUDA(cudaMallocFromPoolAsync(&scratch, sbytes, pool, stream));
        uint4 *cuts = static_cast<uint4 *>(scratch);
        uint32_t *hist = reinterpret_cast<uint32_t *>(static_cast<char *>(scratch) + 32 * (size_t)m);
        uint32_t *offs = hist + nk;
        uint32_t *cursor = offs + nk + 1;
        uint32_t *dest = cursor + nk;
        uint16_t *keys = reinterpret_cast<uint16_t *>(dest + m);
        EvalParams p;
        p.per_stage_tp = per_stage_tp ? 1 : 0;
        p.cands = per_stage_tp ? nullptr : static_cast<const uint4 *>(d_cands) + base;
        p.cands_ex = per_stage_tp ? static_cast<const uint2 *>(d_cands) + 3 * base : nullptr;
        p.n = m;
        p.T = d_T + base;
        p.F = d_F + base;
        p.dest = dest;
        p.offs = offs;
        p.cuts = cuts;
        p.blob = h->d_blob;
        p.lay = h->lay;
        for (int J = 1; J <= POS_MAX_STAGES; ++J) {  // smallest tripping M, by bisection
            int lo = 1, hi = 256;
            while (lo < hi) {
                const int mid = (lo + hi) / 2;
                if (guard_trips(h->guard_A, h->guard_D, h->guard_P, J, mid)) hi = mid;
                else lo = mid + 1;
            }
            p.guard_m[J] = (uint16_t)lo;
        }
        p.guard_m[0] = 0;
        p.pg = pg;
        p.nkeys = nk;
        p.lim_off = h->lim_off;
        p.lim_w = h->lim_w;
        p.lim_bytes = h->lim_bytes;
        // histogram pass: 256 threads, four candidates per thread and round
        const int grid = (int)std::max<int64_t>(
            1, std::min<int64_t>((m + 1023) / 1024, 4LL * sm_count()));
        cudaError_t e = cudaMemsetAsync(hist, 0, sizeof(uint32_t) * nk, stream);
        if (e == cudaSuccess) {
            const int64_t chunk = scatter_chunk(m, sm_count());
            const int sgrid = (int)std::max<int64_t>(
                1, std::min<int64_t>((m + chunk - 1) / chunk, 8LL * sm_count()));
            // the histogram follows a memset; the kernels after it are chained
            // by programmatic dependent launch
            if (il) {
                sort_hist_kernel<kKeysIl><<<grid, 256, 0, stream>>>(p, m, hist, keys, p.T, p.F);
                e = cudaGetLastError();
                if (e == cudaSuccess)
                    e = launch_dependent(sort_scan_kernel<kKeysIl>, 1, 1024, 0, stream, hist, offs,
                                         cursor);
                if (e == cudaSuccess)
                    e = launch_dependent(sort_scatter_kernel<kKeysIl>, sgrid, 512, 0, stream, keys,
                                         m, chunk, cursor, dest);
            } else {
                sort_hist_kernel<kKeys><<<grid, 256, 0, stream>>>(p, m, hist, keys, p.T, p.F);
                e = cudaGetLastError();
                if (e == cudaSuccess)
                    e = launch_dependent(sort_scan_kernel<kKeys>, 1, 1024, 0, stream, hist, offs,
                                         cursor);
                if (e == cudaSuccess)
                    e = launch_dependent(sort_scatter_kernel<kKeys>, sgrid, 512, 0, stream, keys, m,
                                         chunk, cursor, dest);
            }
        }
        if (e == cudaSuccess) st = launch_decode(p, stream);
        if (e == cudaSuccess && st == POS_OK) {
            SideStream *ss = nullptr;
            st = side_stream(&ss);
            if (st == POS_OK) {
                std::lock_guard<std::mutex> lock(ss->mu);
                // fork: the side chain starts after the decode pass
                e = cudaEventRecord(ss->fork, stream);
                if (e == cudaSuccess) e = cudaStreamWaitEvent(ss->s, ss->fork, 0);
                if (e == cudaSuccess) {
                    const cudaStream_t side = ss->s;
                    if (p.lay.sched == POS_SCHED_EAGER_1F1B) {
                        if ((st = eval_eager_short_2_8(p, side)) == POS_OK &&
                            (st = eval_eager_short_9_10(p, side)) == POS_OK &&
                            (st = eval_eager_short_11_12(p, side)) == POS_OK &&
                            (st = eval_eager_short_13_13(p, side)) == POS_OK &&
                            (st = eval_eager_short_14_14(p, side)) == POS_OK &&
                            (st = eval_eager_short_15_15(p, side)) == POS_OK &&
                            (st = eval_eager_short_16_16(p, side)) == POS_OK &&
                            (st = eval_eager_1_6(p, side)) == POS_OK &&
                            (st = eval_eager_7_10(p, stream)) == POS_OK &&
                            (st = eval_eager_11_13(p, stream)) == POS_OK)
                            st = eval_eager_14_16(p, stream);
                    } else if (il) {
                        // interleaved handle: the 1F1B ranges (records with
                        // V < 2, usually none) and the smallest interleaved
                        // range on the side, the other interleaved ranges here
                        if ((st = eval_generic_2_8(p, side)) == POS_OK &&
                            (st = eval_generic_9_12(p, side)) == POS_OK &&
                            (st = eval_generic_13_14(p, side)) == POS_OK &&
                            (st = eval_generic_15_15(p, side)) == POS_OK &&
                            (st = eval_generic_16_16(p, side)) == POS_OK &&
                            (st = eval_fast_1_4(p, side)) == POS_OK &&
                            (st = eval_fast_5_8(p, side)) == POS_OK &&
                            (st = eval_fast_9_12(p, side)) == POS_OK &&
                            (st = eval_fast_13_16(p, side)) == POS_OK &&
                            (st = eval_il_30_31(p, side)) == POS_OK &&
                            (st = eval_il_0_11(p, stream)) == POS_OK &&
                            (st = eval_il_12_22(p, stream)) == POS_OK &&
                            (st = eval_il_23_29(p, stream)) == POS_OK)
                            st = eval_il_32_33(p, stream);
                    } else if ((st = eval_generic_2_8(p, side)) == POS_OK &&
                               (st = eval_generic_9_12(p, side)) == POS_OK &&
                               (st = eval_generic_13_14(p, side)) == POS_OK &&
                               (st = eval_generic_15_15(p, side)) == POS_OK &&
                               (st = eval_generic_16_16(p, side)) == POS_OK &&
                               (st = eval_fast_1_4(p, side)) == POS_OK &&
                               (st = eval_fast_5_8(p, stream)) == POS_OK &&
                               (st = eval_fast_9_12(p, stream)) == POS_OK) {
                        st = eval_fast_13_16(p, stream);
                    }
                    // join, also after a failed launch (the side stream's
                    // queued work stays ordered before the scratch is freed)
                    cudaError_t ej = cudaEventRecord(ss->join, side);
                    if (ej == cudaSuccess) ej = cudaStreamWaitEvent(stream, ss->join, 0);
                    if (e == cudaSuccess) e = ej;
                }
            }
        }
        const cudaError_t e2 = cudaFreeAsync(scratch, stream);
        if (e != cudaSuccess) return cuda_fail(e, "eval sort launch");
        if (st != POS_OK) return st;
        if (e2 != cudaSuccess) return cuda_fail(e2, "eval scratch free");
    }
    return POS_OK;
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
    return pos::launch_eval(static_cast<pos::Handle *>(handle), d_cands, false, n, d_makespan,
                            d_feasible, static_cast<cudaStream_t>(stream));
}

pos_status poseidon_eval_batch_ex(void *handle, const pos_candidate_ex *d_cands, int64_t n,
                                  int32_t *d_makespan, uint8_t *d_feasible, void *stream) {
    if (!handle) return pos::fail(POS_EINVAL, "handle is NULL");
    if (n < 0) return pos::fail(POS_EINVAL, "n < 0");
    if (n > 0 && (!d_cands || !d_makespan || !d_feasible))
        return pos::fail(POS_EINVAL, "NULL buffer");
    if ((reinterpret_cast<uintptr_t>(d_cands) & 7) != 0)
        return pos::fail(POS_EINVAL, "candidates must be 8-byte aligned");
    pos::Handle *h = static_cast<pos::Handle *>(handle);
    if (h->lay.n_tp > 4)
        return pos::fail(POS_EINVAL, "per-stage TP records need n_tp <= 4 (2-bit TP fields)");
    return pos::launch_eval(h, d_cands, true, n, d_makespan, d_feasible,
                            static_cast<cudaStream_t>(stream));
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
        st = pos::launch_eval(static_cast<pos::Handle *>(handle), dc, false, n, dt, df, 0);
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
        1, std::min<int64_t>((n + pos::kArgminThreads - 1) / pos::kArgminThreads,
                             4LL * pos::sm_count()));
    void *scratch = nullptr;
    POS_CUDA(cudaMallocAsync(&scratch, (size_t)parts * 16, s));
    int32_t *pt = static_cast<int32_t *>(scratch);
    long long *pi = reinterpret_cast<long long *>(static_cast<char *>(scratch) + parts * 8);
    pos::argmin_partial<<<parts, pos::kArgminThreads, 0, s>>>(d_makespan, d_feasible, n, pt, pi);
    pos::argmin_final<<<1, 32, 0, s>>>(pt, pi, parts, d_out);
    const cudaError_t e = cudaGetLastError();
    const cudaError_t e2 = cudaFreeAsync(scratch, s);
    if (e != cudaSuccess) return pos::cuda_fail(e, "argmin launch");
    if (e2 != cudaSuccess) return pos::cuda_fail(e2, "argmin free");
    return POS_OK;
}

}  // extern "C"
