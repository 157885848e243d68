// Level programs for the schedules whose short case (few micro-batches) has
// no closed-form level order: Eager 1F1B with M < 2S-1.  For each (S, M)
// the unit-weight ASAP level of every op is computed from the stage chains
// (an op runs one level after the later of its stage's previous op and its
// inter-stage predecessor), and each level becomes one 64-bit word of
// forward / backward / lag-2 stage masks (see makespan_program).
#include <mutex>
#include <vector>

#include "common.cuh"

namespace pos {

namespace {

constexpr int kMaxDevices = 64;

struct DevicePrograms {
    uint64_t *words = nullptr;
    uint2 *index = nullptr;
};

std::mutex g_mutex;
DevicePrograms g_eager[kMaxDevices];

// Chain of 0-based stage s: W forwards, then (B_i, F_{W+i}), then the rest
// of the backwards; entries encode (is_backward << 8) | micro-batch.
std::vector<int> stage_chain(int sched, int S, int M, int s) {
    const int W = inflight(sched, S, M, s);
    std::vector<int> c;
    for (int m = 0; m < W; ++m) c.push_back(m);
    for (int i = 0; i < M - W; ++i) {
        c.push_back(256 | i);
        c.push_back(W + i);
    }
    for (int m = M - W; m < M; ++m) c.push_back(256 | m);
    return c;
}

// Program of (sched, S, M) appended to words; returns the level count or
// -1 if the level order needs a forward history deeper than two.
int build_program(int sched, int S, int M, std::vector<uint64_t> &words) {
    std::vector<std::vector<int>> chain(S);
    for (int s = 0; s < S; ++s) chain[s] = stage_chain(sched, S, M, s);
    std::vector<int> lf(S * M, 0), lb(S * M, 0);  // ASAP levels of F_{s,m}, B_{s,m}
    for (bool changed = true; changed;) {
        changed = false;
        for (int s = 0; s < S; ++s) {
            int prev = 0;
            for (int e : chain[s]) {
                const int m = e & 255;
                int p = prev;
                if (e & 256) {
                    if (s + 1 < S) p = std::max(p, lb[(s + 1) * M + m]);
                } else if (s > 0) {
                    p = std::max(p, lf[(s - 1) * M + m]);
                }
                int &v = (e & 256) ? lb[s * M + m] : lf[s * M + m];
                if (v != p + 1) {
                    v = p + 1;
                    changed = true;
                }
                prev = p + 1;
            }
        }
    }
    int n_levels = 0;
    for (int i = 0; i < S * M; ++i) n_levels = std::max(n_levels, std::max(lf[i], lb[i]));
    for (int l = 1; l <= n_levels; ++l) {
        uint64_t fm = 0, bm = 0, lm = 0;
        for (int s = S - 1; s >= 0; --s) {  // the kernel's visiting order
            for (int m = 0; m < M; ++m) {
                if (lf[s * M + m] == l) {
                    if ((fm | bm) >> s & 1) return -1;  // two ops of one stage in a level
                    fm |= 1ull << s;
                    if (s > 0) {
                        // forwards stage s-1 is ahead (its ops of this level come later)
                        int ahead = 0;
                        for (int u = 0; u < M; ++u) ahead += lf[(s - 1) * M + u] < l;
                        const int lag = ahead - m;
                        if (lag == 2) lm |= 1ull << s;
                        else if (lag != 1) return -1;
                    }
                }
                if (lb[s * M + m] == l) {
                    if ((fm | bm) >> s & 1) return -1;
                    bm |= 1ull << s;
                }
            }
        }
        words.push_back(fm | (bm << 16) | (lm << 32));
    }
    return n_levels;
}

}  // namespace

pos_status schedule_programs(int sched, Programs *out) {
    out->words = nullptr;
    out->index = nullptr;
    if (sched != POS_SCHED_EAGER_1F1B) return POS_OK;
    int dev = 0;
    POS_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kMaxDevices) return fail(POS_EINVAL, "device index above 63");
    std::lock_guard<std::mutex> lock(g_mutex);
    DevicePrograms &dp = g_eager[dev];
    if (!dp.words) {
        std::vector<uint64_t> words;
        std::vector<uint2> index(POS_MAX_STAGES * 32, make_uint2(0, 0));
        for (int S = 1; S <= POS_MAX_STAGES; ++S)
            for (int M = 1; M < fast_min_m(sched, S); ++M) {
                const size_t first = words.size();
                const int n = build_program(sched, S, M, words);
                if (n < 0) return fail(POS_EINVAL, "schedule needs a deeper forward history");
                index[(S - 1) * 32 + M] = make_uint2((uint32_t)first, (uint32_t)n);
            }
        uint64_t *w = nullptr;
        uint2 *ix = nullptr;
        cudaError_t e = cudaMalloc(&w, sizeof(uint64_t) * words.size());
        if (e == cudaSuccess) e = cudaMalloc(&ix, sizeof(uint2) * index.size());
        if (e == cudaSuccess)
            e = cudaMemcpy(w, words.data(), sizeof(uint64_t) * words.size(),
                           cudaMemcpyHostToDevice);
        if (e == cudaSuccess)
            e = cudaMemcpy(ix, index.data(), sizeof(uint2) * index.size(), cudaMemcpyHostToDevice);
        if (e != cudaSuccess) {
            if (w) cudaFree(w);
            if (ix) cudaFree(ix);
            return cuda_fail(e, "schedule programs");
        }
        dp.words = w;
        dp.index = ix;
    }
    out->words = dp.words;
    out->index = dp.index;
    return POS_OK;
}

}  // namespace pos
