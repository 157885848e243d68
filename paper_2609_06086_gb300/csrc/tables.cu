// Handle life cycle, error state and the cost-table kernel (hot-path step
// a1: per-class exclusive prefix sums of the Sec. 4.1.3 weights and the
// Sec. 3.2 memory footprints).
#include <algorithm>
#include <atomic>
#include <cstring>
#include <map>
#include <tuple>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "common.cuh"

namespace pos {

static thread_local std::string g_last_error;

void set_error(const std::string &msg) { g_last_error = msg; }

pos_status fail(pos_status st, const std::string &msg) {
    g_last_error = msg;
    return st;
}

pos_status cuda_fail(cudaError_t e, const char *what) {
    g_last_error = std::string("CUDA error in ") + what + ": " + cudaGetErrorString(e);
    return e == cudaErrorMemoryAllocation ? POS_ENOMEM : POS_ECUDA;
}

const char *last_error() { return g_last_error.c_str(); }

pos_status ensure_smem(const void *kernel, int smem) {
    static std::mutex mu;
    static std::map<std::pair<int, const void *>, int> set;  // (device, kernel) -> limit
    int dev = 0;
    POS_CUDA(cudaGetDevice(&dev));
    std::lock_guard<std::mutex> lock(mu);
    int &cur = set[{dev, kernel}];
    if (smem <= cur) return POS_OK;
    POS_CUDA(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    cur = smem;
    return POS_OK;
}

pos_status blocks_per_sm(const void *kernel, int threads, int smem, int *out) {
    static std::mutex mu;
    // (device, kernel, threads, shared bytes) -> resident blocks per SM
    static std::map<std::tuple<int, const void *, int, int>, int> known;
    int dev = 0;
    POS_CUDA(cudaGetDevice(&dev));
    std::lock_guard<std::mutex> lock(mu);
    const auto key = std::make_tuple(dev, kernel, threads, smem);
    const auto it = known.find(key);
    if (it != known.end()) {
        *out = it->second;
        return POS_OK;
    }
    int n = 0;
    POS_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, smem));
    known[key] = n;
    *out = n;
    return POS_OK;
}

int sm_count() {
    static std::atomic<int> known[64];  // per device, 0 = not queried yet
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && (n = known[dev].load(std::memory_order_relaxed)) > 0) return n;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) return 1;
    if (dev >= 0 && dev < 64) known[dev].store(n, std::memory_order_relaxed);
    return n;
}

static int align16(int x) { return (x + 15) & ~15; }

BlobLayout make_layout(int L, int n_types, int n_tp) {
    BlobLayout ly;
    ly.L = L;
    ly.n_types = n_types;
    ly.n_tp = n_tp;
    ly.K = n_types * n_tp;
    ly.sched = POS_SCHED_1F1B;
    const int K = ly.K, Lp1 = L + 1;
    int off = 0;
    ly.off_binom = off;
    off = align16(off + kBinomN * kBinomK * 8);
    ly.off_Pw = off;
    off = align16(off + K * Lp1 * 8);
    ly.off_Pa = off;
    off = align16(off + K * Lp1 * 8);
    ly.off_cap = off;
    off = align16(off + K * 8);
    ly.off_Pf = off;
    off = align16(off + K * Lp1 * 4);
    ly.off_Pb = off;
    off = align16(off + K * Lp1 * 4);
    ly.off_Pd = off;
    off = align16(off + K * Lp1 * 4);
    ly.off_p2f = off;
    off = align16(off + K * K * 4);
    ly.off_p2b = off;
    off = align16(off + K * K * 4);
    ly.bytes = off;
    return ly;
}

BlobLayout timing_layout(const BlobLayout &ly) {
    BlobLayout t = ly;
    const int base = ly.off_Pf;
    t.off_binom = t.off_Pw = t.off_Pa = t.off_cap = -1;  // not staged
    t.off_Pf -= base;
    t.off_Pb -= base;
    t.off_Pd -= base;
    t.off_p2f -= base;
    t.off_p2b -= base;
    t.bytes = ly.bytes - base;
    return t;
}

BlobLayout memory_layout(const BlobLayout &ly) {
    BlobLayout t = ly;
    const int base = ly.off_Pw;
    t.off_binom = t.off_Pf = t.off_Pb = t.off_Pd = t.off_p2f = t.off_p2b = -1;  // not staged
    t.off_Pw -= base;
    t.off_Pa -= base;
    t.off_cap -= base;
    t.bytes = ly.off_Pf - base;
    return t;
}

// One thread per (table, class) row: the raw per-layer row sits at entries
// 1..L of the row; turn it into an exclusive prefix sum with P[0] = 0.
__global__ void prefix_rows_kernel(unsigned char *blob, BlobLayout ly) {
    const int K = ly.K, Lp1 = ly.L + 1;
    const int row = blockIdx.x * blockDim.x + threadIdx.x;
    if (row >= 5 * K) return;
    const int table = row / K, k = row % K;
    if (table < 2) {
        int64_t *P = reinterpret_cast<int64_t *>(blob + (table == 0 ? ly.off_Pw : ly.off_Pa)) +
                     (int64_t)k * Lp1;
        int64_t acc = 0;
        P[0] = 0;
        for (int l = 1; l <= ly.L; ++l) {
            acc += P[l];
            P[l] = acc;
        }
    } else {
        const int off = table == 2 ? ly.off_Pf : (table == 3 ? ly.off_Pb : ly.off_Pd);
        int32_t *P = reinterpret_cast<int32_t *>(blob + off) + (int64_t)k * Lp1;
        int32_t acc = 0;
        P[0] = 0;
        for (int l = 1; l <= ly.L; ++l) {
            acc += P[l];
            P[l] = acc;
        }
    }
}

// One block per (class, in-flight count w): lim[k][w-1][a] for every start
// a, by binary search (the memory need grows with the layer count, the
// tables being non-negative).
__global__ void lim_kernel(unsigned char *blob, BlobLayout ly, int wmax, int lim_off) {
    const int k = blockIdx.x / wmax, w = blockIdx.x % wmax + 1, L = ly.L;
    const int64_t *Pw = reinterpret_cast<const int64_t *>(blob + ly.off_Pw) + (int64_t)k * (L + 1);
    const int64_t *Pa = reinterpret_cast<const int64_t *>(blob + ly.off_Pa) + (int64_t)k * (L + 1);
    const int64_t cap = reinterpret_cast<const int64_t *>(blob + ly.off_cap)[k];
    uint8_t *out = blob + lim_off + (size_t)blockIdx.x * (L + 1);
    for (int a = threadIdx.x; a <= L; a += blockDim.x) {
        int lo = a, hi = L;
        while (lo < hi) {
            const int mid = (lo + hi + 1) / 2;
            const int64_t need = (Pw[mid] - Pw[a]) + (int64_t)w * (Pa[mid] - Pa[a]);
            if (need <= cap) lo = mid;
            else hi = mid - 1;
        }
        out[a] = (uint8_t)lo;
    }
}

pos_status validate_tables(const pos_tables *t) {
    if (!t) return fail(POS_EINVAL, "tables is NULL");
    if (t->L < 1 || t->L > POS_MAX_LAYERS) return fail(POS_EINVAL, "L must be in 1..127");
    if (t->n_types < 1 || t->n_types > POS_MAX_TYPES)
        return fail(POS_EINVAL, "n_types must be in 1..4");
    if (t->n_tp < 1 || t->n_tp > POS_MAX_TP) return fail(POS_EINVAL, "n_tp must be in 1..8");
    if (!t->fwd || !t->bwd || !t->dsync || !t->p2p_f || !t->p2p_b || !t->mem_w || !t->mem_a ||
        !t->cap)
        return fail(POS_EINVAL, "a table pointer is NULL");
    const int K = t->n_types * t->n_tp, L = t->L;
    for (int k = 0; k < K; ++k) {
        int64_t sfb = 0, sd = 0, smw = 0, sma = 0;
        for (int l = 0; l < L; ++l) {
            const int64_t i = (int64_t)k * L + l;
            if (t->fwd[i] < 0 || t->bwd[i] < 0 || t->dsync[i] < 0 || t->mem_w[i] < 0 ||
                t->mem_a[i] < 0)
                return fail(POS_EINVAL, "negative cost or memory entry");
            sfb += (int64_t)t->fwd[i] + t->bwd[i];
            sd += t->dsync[i];
            smw += t->mem_w[i];
            sma += t->mem_a[i];
            if (smw > ((int64_t)1 << 52) || sma > ((int64_t)1 << 52))
                return fail(POS_EOVERFLOW, "per-class summed memory above 2^52 bytes");
        }
        if (sfb >= ((int64_t)1 << 31) || sd >= ((int64_t)1 << 31))
            return fail(POS_EOVERFLOW, "per-class summed costs reach 2^31");
        if (t->cap[k] < 0) return fail(POS_EINVAL, "negative capacity");
    }
    for (int i = 0; i < K * K; ++i)
        if (t->p2p_f[i] < 0 || t->p2p_b[i] < 0) return fail(POS_EINVAL, "negative transfer time");
    return POS_OK;
}

pos_status build_blob(const pos_tables *t, int sched, std::vector<unsigned char> &host,
                      BlobLayout &ly, int64_t &guard_A, int64_t &guard_D, int64_t &guard_P) {
    pos_status st = validate_tables(t);
    if (st != POS_OK) return st;
    const int L = t->L, K = t->n_types * t->n_tp, Lp1 = L + 1;
    ly = make_layout(L, t->n_types, t->n_tp);
    ly.sched = sched;
    host.assign(ly.bytes, 0);
    // binomials by Pascal's rule (k <= 15 is exact in 64 bits for n <= 127),
    // one 64-bit word each, [k][n]
    uint64_t *bn = reinterpret_cast<uint64_t *>(host.data() + ly.off_binom);
    for (int n = 0; n < kBinomN; ++n)
        for (int k = 0; k < kBinomK; ++k)
            bn[k * kBinomN + n] =
                k == 0 ? 1 : (n == 0 ? 0 : bn[(k - 1) * kBinomN + n - 1] + bn[k * kBinomN + n - 1]);
    // raw rows at entries 1..L; prefix_rows_kernel turns them into sums
    int64_t *Pw_ = reinterpret_cast<int64_t *>(host.data() + ly.off_Pw);
    int64_t *Pa_ = reinterpret_cast<int64_t *>(host.data() + ly.off_Pa);
    int32_t *Pf_ = reinterpret_cast<int32_t *>(host.data() + ly.off_Pf);
    int32_t *Pb_ = reinterpret_cast<int32_t *>(host.data() + ly.off_Pb);
    int32_t *Pd_ = reinterpret_cast<int32_t *>(host.data() + ly.off_Pd);
    for (int k = 0; k < K; ++k)
        for (int l = 0; l < L; ++l) {
            const int64_t src = (int64_t)k * L + l, dst = (int64_t)k * Lp1 + l + 1;
            Pw_[dst] = t->mem_w[src];
            Pa_[dst] = t->mem_a[src];
            Pf_[dst] = t->fwd[src];
            Pb_[dst] = t->bwd[src];
            Pd_[dst] = t->dsync[src];
        }
    std::memcpy(host.data() + ly.off_cap, t->cap, sizeof(int64_t) * K);
    std::memcpy(host.data() + ly.off_p2f, t->p2p_f, sizeof(int32_t) * K * K);
    std::memcpy(host.data() + ly.off_p2b, t->p2p_b, sizeof(int32_t) * K * K);
    int64_t A = 0, D = 0, P = 0;
    for (int l = 0; l < L; ++l) {
        int64_t mfb = 0, md = 0;
        for (int k = 0; k < K; ++k) {
            const int64_t i = (int64_t)k * L + l;
            mfb = std::max<int64_t>(mfb, (int64_t)t->fwd[i] + t->bwd[i]);
            md = std::max<int64_t>(md, t->dsync[i]);
        }
        A += mfb;
        D += md;
    }
    for (int i = 0; i < K * K; ++i)
        P = std::max<int64_t>(P, std::max(t->p2p_f[i], t->p2p_b[i]));
    guard_A = A;
    guard_D = D;
    guard_P = P;
    return POS_OK;
}

pos_status launch_prefix_rows(void *d_blob, const BlobLayout &ly, cudaStream_t stream) {
    const int rows = 5 * ly.K;
    prefix_rows_kernel<<<(rows + 127) / 128, 128, 0, stream>>>(
        static_cast<unsigned char *>(d_blob), ly);
    POS_CUDA(cudaGetLastError());
    return POS_OK;
}

pos_status create_handle(const pos_tables *t, int sched, Handle **out) {
    std::vector<unsigned char> host;
    BlobLayout ly;
    int64_t A, D, P;
    pos_status st = build_blob(t, sched, host, ly, A, D, P);
    if (st != POS_OK) return st;
    Handle *h = new (std::nothrow) Handle();
    if (!h) return fail(POS_ENOMEM, "host allocation failed");
    h->lay = ly;
    h->d_blob = nullptr;
    h->guard_A = A;
    h->guard_D = D;
    h->guard_P = P;
    // in-flight micro-batches of a stage: at most 16 (1F1B), 31 (Eager 1F1B)
    h->lim_w = sched == POS_SCHED_EAGER_1F1B ? 2 * POS_MAX_STAGES - 1 : POS_MAX_STAGES;
    h->lim_off = ly.bytes;
    const long long lb = (long long)ly.K * h->lim_w * (ly.L + 1);
    h->lim_bytes = lb <= kLimMaxBytes ? (int)((lb + 15) & ~15ll) : 0;
    cudaError_t e = cudaGetDevice(&h->device);
    if (e == cudaSuccess) e = cudaMalloc(&h->d_blob, (size_t)ly.bytes + h->lim_bytes);
    if (e == cudaSuccess) e = cudaMemcpy(h->d_blob, host.data(), ly.bytes, cudaMemcpyHostToDevice);
    if (e == cudaSuccess && launch_prefix_rows(h->d_blob, ly, 0) != POS_OK) e = cudaErrorLaunchFailure;
    if (e == cudaSuccess && h->lim_bytes > 0) {
        lim_kernel<<<ly.K * h->lim_w, 128>>>(static_cast<unsigned char *>(h->d_blob), ly,
                                            h->lim_w, h->lim_off);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(0);
    if (e != cudaSuccess) {
        if (h->d_blob) cudaFree(h->d_blob);
        delete h;
        return cuda_fail(e, "tables upload");
    }
    *out = h;
    return POS_OK;
}

void destroy_handle(Handle *h) {
    if (!h) return;
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != h->device) cudaSetDevice(h->device);
    cudaFree(h->d_blob);
    if (cur != h->device && cur >= 0) cudaSetDevice(cur);
    delete h;
}

}  // namespace pos

extern "C" {

pos_status poseidon_tables_create(const pos_tables *tables, int32_t schedule, void **handle) {
    if (!handle) return pos::fail(POS_EINVAL, "handle out-pointer is NULL");
    *handle = nullptr;
    if (schedule != POS_SCHED_1F1B && schedule != POS_SCHED_EAGER_1F1B &&
        schedule != POS_SCHED_INTERLEAVED_1F1B)
        return pos::fail(POS_ENOTIMPL, "schedule must be POS_SCHED_1F1B, POS_SCHED_EAGER_1F1B "
                                       "or POS_SCHED_INTERLEAVED_1F1B");
    pos::Handle *h = nullptr;
    const pos_status st = pos::create_handle(tables, schedule, &h);
    if (st == POS_OK) *handle = h;
    return st;
}

pos_status poseidon_tables_destroy(void *handle) {
    if (!handle) return pos::fail(POS_EINVAL, "handle is NULL");
    pos::destroy_handle(static_cast<pos::Handle *>(handle));
    return POS_OK;
}

const char *poseidon_last_error(void) { return pos::last_error(); }

}  // extern "C"
