// Host side shared by the search drivers (search.cu: 1F1B and Eager 1F1B;
// search_il.cu: Interleaved 1F1B): the per-device workspace kept between
// calls, and host versions of the combinatorics.
#pragma once
#include <mutex>
#include <new>
#include <vector>

#include "search_kernels.cuh"

namespace pos {

inline uint64_t gcd64(uint64_t a, uint64_t b) {
    while (b) {
        const uint64_t r = a % b;
        a = b;
        b = r;
    }
    return a;
}

struct DevBuf {
    void *p = nullptr;
    size_t bytes = 0;
    DevBuf() = default;
    DevBuf(const DevBuf &) = delete;
    DevBuf &operator=(const DevBuf &) = delete;
    ~DevBuf() {
        if (p) cudaFree(p);
    }
    cudaError_t reserve(size_t b) {
        if (b <= bytes) return cudaSuccess;
        if (p) cudaFree(p);
        p = nullptr;
        bytes = 0;
        const cudaError_t e = cudaMalloc(&p, b);
        if (e == cudaSuccess) bytes = b;
        return e;
    }
};

// Device work buffers, stream and events of one GPU, kept between calls
// (grown on demand) so that a search allocates and frees nothing in the
// steady state.  Searches on the same device are serialised by `mu`.
struct Workspace {
    std::mutex mu;
    cudaStream_t stream = nullptr;
    cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};
    DevBuf blob, d_lim, d_vb, d_bctr, d_rows, d_greedy, d_wcnt, d_lb, d_slices, d_feas, d_batch, d_inc, d_ctr, d_best, d_feasible, d_leaves, d_roots,
        d_root;
    // Interleaved 1F1B search: decoded records of complete plans (two uint4
    // each), their slice, makespan and feasibility, and the key offsets of
    // the makespan kernels
    DevBuf il_rec, il_slice, il_T, il_F, il_offs;
    DevBuf d_front[POS_MAX_STAGES + 1];        // per depth: Prefix buffers
    DevBuf d_defer[2 * (POS_MAX_STAGES + 1)];  // per depth: two deferred group lists
    unsigned long long *h_cnt = nullptr;       // pinned host counters
    unsigned char *h_stage = nullptr;          // pinned staging area for uploads
    size_t h_stage_cap = 0;
    unsigned char *h_read = nullptr;           // pinned landing area for reads
    size_t h_read_cap = 0;
    unsigned long long *h_lb = nullptr;        // pinned landing area of the root bounds
    size_t h_lb_cap = 0;                       // (elements)
    cudaEvent_t ev_lb = nullptr;               // recorded after their copy
    // second stream for the greedy plans' makespans (forked after the bound
    // kernel, joined before the enumeration), so that they run while the
    // host reads the root bounds and plans the batches
    cudaStream_t side = nullptr;
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
    std::vector<cudaEvent_t> evs;              // timing events of the batch pipelines
};

inline uint64_t host_binom(int n, int k) {
    if (k < 0 || k > n) return 0;
    uint64_t r = 1;
    for (int i = 1; i <= k; ++i) r = r * (uint64_t)(n - k + i) / (uint64_t)i;
    return r;
}

inline void host_unrank(int L, int S, uint64_t rank, int32_t *layers) {
    int rem = L;
    for (int s = 0; s < S - 1; ++s) {
        const int after = S - s - 1;
        int v = 1;
        for (; v <= rem - after; ++v) {
            const uint64_t cnt = host_binom(rem - v - 1, after - 1);
            if (rank < cnt) break;
            rank -= cnt;
        }
        layers[s] = v;
        rem -= v;
    }
    layers[S - 1] = rem;
}

// The slices of a search in global-index order (Sec. 4.2.3): the M value,
// then a group -- the TP index under POS_PLACE_FREE / POS_PLACE_EXACT
// (every stage on it), the data-parallel degree under POS_PLACE_DEVICES (a
// class per stage) -- then the group's allowed sequences in lexicographic
// order.  Built on the host before the device is touched.
struct SliceSpace {
    int units = 0;          // stages (devices under Interleaved 1F1B)
    bool per_stage = false; // POS_PLACE_DEVICES
    int n_grp = 0;          // TP indices, or D values
    // FREE / EXACT: one list of type sequences shared by the TP indices;
    // DEVICES: one list of class sequences per D value (units bytes each)
    std::vector<std::vector<uint8_t>> seqs;
    std::vector<uint64_t> grp_off;  // first slice of each group within one M value
    uint64_t per_m = 0;             // slices per M value
    std::vector<int32_t> D;         // data-parallel degree of each group

    uint64_t n_seq(int g) const { return seqs[per_stage ? g : 0].size() / units; }
    const uint8_t *seq(int g, uint64_t place_rank) const {
        return seqs[per_stage ? g : 0].data() + place_rank * units;
    }
    // (m_idx, group, place_rank) of a slice ordinal
    void decode(uint64_t ord, int *m_idx, int *grp, uint64_t *place_rank) const {
        *m_idx = (int)(ord / per_m);
        const uint64_t r = ord % per_m;
        int g = 0;
        while (g + 1 < n_grp && grp_off[g + 1] <= r) ++g;
        *grp = g;
        *place_rank = r - grp_off[g];
    }
    // class of unit u of the slice (group g, rank pr)
    int cls(int g, uint64_t pr, int u, int n_tp) const {
        const uint8_t v = seq(g, pr)[u];
        return per_stage ? v : v * n_tp + g;
    }
};

// Validates the placement fields of p and enumerates its slices for
// `units` stages: POS_EINVAL beyond 2^22 placements or slices.
pos_status build_slice_space(const pos_problem *p, int units, SliceSpace &sp);

// Writes the slice-identity fields of a found plan (m_idx, tp_idx, M, tp,
// D, d_idx, place_rank, type[], tp_stage[]) for slice ordinal `ord`.
void plan_slice_fields(const pos_problem *p, const SliceSpace &sp, uint64_t ord, pos_plan *out);

// The workspace of the current device, created on first use.
pos_status get_workspace(Workspace **out);

// poseidon_search under POS_SCHED_INTERLEAVED_1F1B (search_il.cu), for a
// validated problem; the caller holds the workspace's lock.
pos_status search_interleaved(Workspace &ws, const pos_problem *p, const SliceSpace &sp,
                              pos_plan *out, pos_search_stats *stats);

}  // namespace pos
