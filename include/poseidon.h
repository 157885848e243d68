/*
 * poseidon.h -- C ABI of libposeidon.so: batched evaluation of Poseidon's
 * DAG training-time model and the exact parallelism search built on it,
 * on one GB300 (sm_103a).
 *
 * Model (paper Sec. 4.1): for a pipeline of N = S stages and M micro-batches
 * the DAG has nodes F_{s,m}, B_{s,m} (Sec. 4.1.1), inter-stage edges
 * F_{s,m} -> F_{s+1,m} and B_{s+1,m} -> B_{s,m}, an intra-stage chain in 1F1B
 * order, B_{s,M} -> R_s and R_s -> E (Sec. 4.1.2).  Node weights are the
 * per-layer times summed over the stage's layers, inter-stage edges carry the
 * activation-transfer time, R_s the gradient all-reduce time (Sec. 4.1.3).
 * The makespan T is the longest path: T = max_s (finish(B_{s,M}) + d_s).
 *
 * Conventions shared by every entry point:
 *  - every call returns a pos_status; no C++ exception crosses the ABI;
 *    poseidon_last_error() describes the last failure of the calling thread;
 *  - the caller owns every buffer it passes; the library copies what it keeps;
 *  - costs are int32 microseconds, memory int64 bytes; all arithmetic is
 *    integer, so results are exact and reproducible;
 *  - class k = type * n_tp + tp_idx indexes every per-class table.
 */
#ifndef POSEIDON_H
#define POSEIDON_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t pos_status;
#define POS_OK 0
#define POS_EINVAL 1        /* bad argument, table or problem */
#define POS_EOVERFLOW 2     /* a makespan could exceed int32 (guard below) */
#define POS_ENOMEM 3        /* device or host allocation failed */
#define POS_ECUDA 4         /* a CUDA runtime call failed */
#define POS_ETIMEOUT 5      /* a bounded device loop hit its iteration limit */
#define POS_EINFEASIBLE 6   /* the search space has no memory-feasible plan */
#define POS_ENOTIMPL 7

/* Pipeline schedules (the intra-stage order of Sec. 4.1.2).  Stage s
 * (1-based) of N runs W_s forwards, then (B_i, F_{W_s+i}) for
 * i = 1..M-W_s, then the remaining backwards, and holds the activations of
 * W_s micro-batches at once:
 *   POS_SCHED_1F1B        W_s = min(N-s+1, M)
 *   POS_SCHED_EAGER_1F1B  W_s = min(2(N-s)+1, M)   (Eager 1F1B, App. B)
 *   POS_SCHED_INTERLEAVED_1F1B  Interleaved 1F1B (Sec. 4.1.4) for candidates
 *       whose V field is >= 2, 1F1B for the others.  The S = N devices each
 *       hold V model chunks; the L layers are split over the J = N*V
 *       virtual stages in order, virtual stage j (0-based) being chunk j / N
 *       on device j % N, so the DAG has 2VNM compute nodes, 2(NV-1)M
 *       inter-stage and N(2VM-1) intra-stage edges.  M must be a multiple
 *       of N.  Device d (0-based) runs the interleaved order of Narayanan et
 *       al. (2021), which the paper cites: its k-th forward (k = 0..VM-1)
 *       is chunk (k mod NV) / N of micro-batch (k / NV)*N + k mod N, its
 *       k-th backward chunk V-1 - (k mod NV) / N of the same micro-batch;
 *       it runs w_d = min(2(N-d-1) + (V-1)N, VM) forwards (all VM when
 *       M = N), then alternates one forward and one backward, then runs
 *       the remaining backwards.  Memory: the largest sum of activations
 *       the device holds along that order (a forward of chunk c adds its
 *       mem_a, the matching backward releases it) plus the mem_w of all its
 *       chunks must fit cap of its class.  The edge between virtual stages
 *       j and j+1 uses the classes of their devices (p2p_f[k_{j%N}][k_{(j+1)%N}],
 *       p2p_b[k_{(j+1)%N}][k_{j%N}]); R_d sums dsync over the device's chunks
 *       and follows its last op.  poseidon_eval_batch evaluates such
 *       records; poseidon_search searches over them (pos_problem.V). */
#define POS_SCHED_1F1B 0
#define POS_SCHED_EAGER_1F1B 1
#define POS_SCHED_INTERLEAVED_1F1B 2

#define POS_PLACE_FREE 0    /* any device type on any stage */
#define POS_PLACE_EXACT 1   /* exactly type_counts[t] stages of type t */
#define POS_PLACE_DEVICES 2 /* a (device type, TP index) per stage; the stages of
                               type t use exactly type_counts[t] devices: the sum
                               over them of D * tp_list[tp index] (per-stage TP) */

#define POS_MAX_STAGES 16
#define POS_MAX_LAYERS 127
#define POS_MAX_TYPES 4
#define POS_MAX_TP 8

/*
 * Profiled cost tables (Sec. 3.2 and Sec. 4.1.3), host pointers, row-major:
 *   fwd, bwd, dsync [K][L]   per-layer forward, backward and DP all-reduce
 *                            time in us (>= 0);
 *   p2p_f, p2p_b    [K][K]   activation / gradient transfer time per
 *                            micro-batch, indexed [sending class][receiving
 *                            class]; the F edge s->s+1 uses p2p_f[k_s][k_s+1],
 *                            the B edge s+1->s uses p2p_b[k_s+1][k_s];
 *   mem_w, mem_a    [K][L]   bytes per layer: resident (weights, optimizer)
 *                            and activations per in-flight micro-batch (>= 0);
 *   cap             [K]      device memory per class, bytes.
 * A stage s (1-based) holding layers [a, b) on class k fits when
 *   sum mem_w + W_s * sum mem_a <= cap[k],   W_s = min(S - s + 1, M),
 * W_s being the 1F1B in-flight micro-batches of that stage.
 * Limits: 1 <= L <= 127, 1 <= n_types <= 4, 1 <= n_tp <= 8, and per class
 * sum_l (fwd + bwd) and sum_l dsync below 2^31.
 */
typedef struct pos_tables {
    int32_t L, n_types, n_tp;
    const int32_t *fwd, *bwd, *dsync;
    const int32_t *p2p_f, *p2p_b;
    const int64_t *mem_w, *mem_a;
    const int64_t *cap;
} pos_tables;

/*
 * One encoded candidate plan, 16 bytes:
 *   map_rank   lexicographic rank of the layer composition (l_1..l_S) among
 *              all C(L-1, S-1) compositions of L into S non-empty stages;
 *              rank 0 = (1, ..., 1, L-S+1);
 *   type_code  device type of stage s (0-based) in bits [2s, 2s+2);
 *   S          stages (1..16), M micro-batches (1..255), tp_idx < n_tp;
 *   V          model chunks per device under POS_SCHED_INTERLEAVED_1F1B
 *              (V >= 2: S is the device count N, map_rank ranks the
 *              composition of L into the J = S*V virtual stages among
 *              C(L-1, J-1), J <= 16, and M must be a multiple of S);
 *              ignored by the other schedules and when V < 2.
 */
typedef struct pos_candidate {
    uint64_t map_rank;
    uint32_t type_code;
    uint8_t S, M, tp_idx, V;
} pos_candidate;

/*
 * A candidate whose stages may use different TP indices (the per-stage
 * heterogeneous TP of the Metis and HexiScale plans in the paper's Table 1),
 * 24 bytes:
 *   map_rank, type_code, S, M, V   as in pos_candidate;
 *   tp_code    TP index of stage s (0-based; of device s for interleaved
 *              records) in bits [2s, 2s+2), so the class of stage s is
 *              type_s * n_tp + tp_s; needs n_tp <= 4.
 * The tables' TP axis may stand for any per-stage parallel setting (TP
 * degree, and the data-parallel degree of the stage's all-reduce and
 * memory); every stage still runs the pipeline's M micro-batches.
 */
typedef struct pos_candidate_ex {
    uint64_t map_rank;
    uint32_t type_code;
    uint32_t tp_code;
    uint8_t S, M, V, pad0;
    uint32_t pad1;
} pos_candidate_ex;

/* feasible[] codes written by poseidon_eval_batch */
#define POS_FEAS_NO 0        /* some stage exceeds its memory capacity */
#define POS_FEAS_YES 1
#define POS_FEAS_INVALID 2   /* a field is out of range; makespan = -1 */
#define POS_FEAS_OVERFLOW 3  /* guard U(S,M) >= 2^31; makespan = -1 */

/*
 * Overflow guard: every DAG path visits each node once, so
 *   T <= U(S,M) = M * sum_l max_k (fwd + bwd) + sum_l max_k dsync
 *                 + 2 M (S-1) max_{k,k'} max(p2p_f, p2p_b).
 * Candidates with U(S,M) >= 2^31 are not evaluated.
 */

/*
 * Copy the tables to the current CUDA device and build the per-class
 * exclusive prefix sums used by every kernel (hot-path step a1, Sec. 4.1.3)
 * and, when it takes at most 32 KB, a byte table of each class's largest
 * memory-feasible stage end per start layer and in-flight count (the
 * evaluator's memory check).
 * *handle owns the device copies until poseidon_tables_destroy.  schedule
 * (POS_SCHED_1F1B, POS_SCHED_EAGER_1F1B or POS_SCHED_INTERLEAVED_1F1B)
 * applies to every evaluation through the handle.
 * Errors: POS_EINVAL (null pointer, limits, negative cost or memory),
 * POS_EOVERFLOW (a class's summed costs reach 2^31), POS_ENOTIMPL (schedule),
 * POS_ENOMEM, POS_ECUDA.
 */
pos_status poseidon_tables_create(const pos_tables *tables, int32_t schedule, void **handle);
pos_status poseidon_tables_destroy(void *handle);

/*
 * Evaluate n candidates: makespan (Sec. 4.1) and memory feasibility
 * (Sec. 3.2).  d_cands (16-byte aligned), d_makespan (int32[n]) and
 * d_feasible (uint8[n]) are DEVICE pointers on the handle's device; outputs
 * are in input order; the call is asynchronous on `stream` (a cudaStream_t,
 * NULL = legacy default stream) and returns after the launches.  Part of the
 * work runs on a library-owned second stream of the device, forked from
 * `stream` after the sort and joined back into it before the call's last
 * operation, so every effect is still ordered after earlier work on
 * `stream` and before later work on it.  Infeasible
 * plans still get their makespan.  Scratch: the batch is counting-sorted by
 * (S, M) (and by (N, V, M/N) for interleaved records) and decoded into a
 * 38*n + 56 KB (Interleaved 1F1B: 38*n + 121 KB) stream-ordered allocation
 * (decoded record 32 B, sorted position 4 B and sort key 2 B per candidate,
 * key histograms) from a library-owned memory pool (per device, kept
 * between calls); batches above 2^24 candidates go in chunks of 2^24, one
 * after another.
 * Errors: POS_EINVAL (null handle or pointers, n < 0, misaligned
 * candidates), POS_ENOMEM, POS_ECUDA (launch failure).
 */
pos_status poseidon_eval_batch(void *handle, const pos_candidate *d_cands, int64_t n,
                               int32_t *d_makespan, uint8_t *d_feasible, void *stream);

/*
 * poseidon_eval_batch for 24-byte pos_candidate_ex records (a TP index per
 * stage): same outputs, flags, schedules, scratch and stream semantics;
 * a record whose TP field of some stage s < S is >= n_tp is flagged
 * POS_FEAS_INVALID.  d_cands must be 8-byte aligned.
 * Errors: those of poseidon_eval_batch, and POS_EINVAL when the handle's
 * tables have n_tp > 4.
 */
pos_status poseidon_eval_batch_ex(void *handle, const pos_candidate_ex *d_cands, int64_t n,
                                  int32_t *d_makespan, uint8_t *d_feasible, void *stream);

/*
 * Same as poseidon_eval_batch but with HOST buffers: copies the candidates
 * to the device, evaluates, copies the results back and synchronises.
 * Allocates n*21 bytes of device memory for the duration of the call.
 */
pos_status poseidon_eval_batch_host(void *handle, const pos_candidate *cands, int64_t n,
                                    int32_t *makespan, uint8_t *feasible);

/*
 * Deterministic argmin over eval_batch outputs (hot-path step a9): the
 * smallest makespan among entries with feasible == 1, ties broken to the
 * lowest index.  Device pointers; *d_out (int64, device) receives the index
 * or -1 when no entry is feasible.  Asynchronous on `stream`; uses a
 * stream-ordered scratch allocation of at most 16 bytes per SM * 4.
 */
pos_status poseidon_argmin(const int32_t *d_makespan, const uint8_t *d_feasible, int64_t n,
                           int64_t *d_out, void *stream);

/*
 * poseidon_argmin_noalloc: same inputs, output and result as poseidon_argmin,
 * for callers that cannot allocate device memory during a call -- a process
 * whose device memory belongs to another allocator (a framework's caching
 * allocator holding the free memory, or a service that reserves everything
 * at start-up and forbids allocation afterwards).  The paper has no
 * counterpart; this is a library convenience.
 * It allocates nothing: its per-block partial results live in a fixed
 * 64 KB array of device global memory (4096 partial results) that every GPU
 * loading the library holds until the process exits.  The first call on a
 * device looks up that array's device address (cudaGetSymbolAddress) with
 * the device current; make that first call before any stream capture.
 * That address is kept for the life of the process: do not use the
 * library across a cudaDeviceReset (the array may move when the module is
 * loaded again).
 * All calls on a device share the array and it keeps the last call's
 * contents (every slot a call reads is written earlier in the same call, so
 * nothing needs clearing); calls that overlap on the GPU, e.g. on two
 * streams at once, race on it.  Errors: POS_EINVAL for bad arguments or
 * when the GPU would need more than 4096 partial results (more than 1024
 * SMs), POS_ECUDA for a failed address lookup or launch.
 */
pos_status poseidon_argmin_noalloc(const int32_t *d_makespan, const uint8_t *d_feasible,
                                   int64_t n, int64_t *d_out, void *stream);

/*
 * Search problem (Sec. 4.2.3): choose M from M_list, a TP index, a
 * device-type-to-stage placement and a layer composition for S stages.
 * Slices are (m_idx, tp_idx, placement) in this nesting order; placements
 * are the allowed type sequences in lexicographic order.  Global index of a
 * plan = (((m_idx*n_tp + tp_idx)*n_place + place_rank)*n_map + map_rank),
 * n_map = C(L-1, S-1).  Objective: time per sample T/(D*M), compared exactly;
 * ties go to the lowest global index.
 * POS_PLACE_DEVICES (per-stage TP, as in the mixed-TP plans of the paper's
 * Table 1): slices are (m_idx, d_idx, class sequence), the classes
 * k_s = type_s * n_tp + tp_s of the S stages chosen freely among those whose
 * stages of every type t use exactly type_counts[t] devices (sum of
 * D_list[d_idx] * tp_list[tp_s]); the sequences of one D in lexicographic
 * order of (k_1, ..., k_S); slice ordinal = m_idx * P + (sequences of
 * D_list[0..d_idx-1]) + place_rank, P = the sequences of every D; global
 * index = ordinal * n_map + map_rank.  The tables must hold every class's
 * costs for each D tried; ridge pruning is not available (POS_EINVAL);
 * under POS_SCHED_INTERLEAVED_1F1B the sequence is over the S devices and
 * needs n_tp <= 4 (POS_EINVAL).
 */
/* Stage-level pruning (Sec. 4.2.1).  Every mode returns the same plan.
 *   POS_PRUNE_NONE   exhaustive enumeration (memory cut only).
 *   POS_PRUNE_EQ2    cut a prefix S_x when g(S_x) > T_min, g of Eq. 2 as
 *                    printed (Theorem 1).
 *   POS_PRUNE_TIGHT  a larger valid bound, not in the paper: Eq. 2 with the
 *                    inter-stage F and B edges on its path added, and the
 *                    largest of two bounds over the stages not yet placed.
 *                    For a complete plan and 1-based stages i <= y, the path
 *                    through the first micro-batch's forwards up to y, stage
 *                    y's whole chain, the last micro-batch's backwards down
 *                    to i and R_i has length
 *                      P(y, i) = sum_{j<y} (F_j + pf_j) + M (F_y + B_y)
 *                                + sum_{j=i}^{y-1} (B_j + pb_j) + d_i <= T;
 *                    the prefix bound is max( max_{i<=x} P(x, i),
 *                    min over memory-feasible completions of max_{y>x} P(y, y),
 *                    min over them of max_{y>x, i<=x} P(y, i) ), the minima
 *                    taken from per-slice tables built by a dynamic program
 *                    over (stage, first layer). */
#define POS_PRUNE_NONE 0
#define POS_PRUNE_EQ2 1
#define POS_PRUNE_TIGHT 2

typedef struct pos_problem {
    pos_tables tables;
    int32_t S;
    int32_t n_M;
    const int32_t *M_list;      /* [n_M], 1..255 */
    const int32_t *tp_list;     /* [n_tp] TP degree of each TP index (reported) */
    const int32_t *dp_list;     /* [n_tp] data-parallel degree D of each TP index */
    int32_t placement;          /* POS_PLACE_FREE or POS_PLACE_EXACT */
    const int32_t *type_counts; /* [n_types] stages per type (POS_PLACE_EXACT) */
    int32_t warmup;             /* random feasible samples seeding T_min (paper: 500) */
    int32_t prune;              /* POS_PRUNE_NONE, POS_PRUNE_EQ2 or POS_PRUNE_TIGHT */
    uint64_t seed;              /* warm-up sampling seed */
    int32_t schedule;           /* POS_SCHED_1F1B, POS_SCHED_EAGER_1F1B or
                                   POS_SCHED_INTERLEAVED_1F1B (with V below) */
    int64_t frontier_cap;       /* entries per frontier buffer; 0 = default 2^24;
                                   raised to at least 32*L */
    int32_t profile;            /* 1: device time per kernel kind in the stats (CUDA
                                   events around every launch); 0: those fields are 0 */
    int32_t ridge;              /* 1: layer-level pruning (Theorem 2): only plans whose
                                   layer counts over the stages of each device type rise,
                                   then fall ("ridge-like") are enumerated or returned.
                                   Theorem 2 guarantees a ridge-like optimum only under
                                   its assumptions: the result may be worse than the
                                   exact optimum (never better); 0: exact search */
    int32_t V;                  /* POS_SCHED_INTERLEAVED_1F1B: model chunks per device
                                   (>= 2, S*V <= 16); ignored by the other schedules */
    int32_t cas_limit;          /* rounds of the incumbent's compare-and-swap loop before
                                   the search gives up with POS_ETIMEOUT: 0 = default
                                   (2^20); < 0 = no round, so every update that would
                                   lower the incumbent gives up (tests the time-out path) */
    int32_t n_D;                /* POS_PLACE_DEVICES: data-parallel degrees tried */
    const int32_t *D_list;      /* [n_D] (>= 1); dp_list is not read there */
} pos_problem;

typedef struct pos_plan {
    int32_t found;
    int32_t m_idx, tp_idx, M, tp, D, S;  /* tp_idx, tp: -1 under POS_PLACE_DEVICES */
    int32_t makespan;           /* T in us */
    int32_t type[POS_MAX_STAGES];    /* device type per stage (per device, interleaved) */
    int32_t layers[POS_MAX_STAGES];  /* layers per stage (per virtual stage, interleaved) */
    uint64_t place_rank, map_rank, global_index;
    int32_t tp_stage[POS_MAX_STAGES];  /* TP index per stage (per device); -1 past S */
    int32_t d_idx;              /* POS_PLACE_DEVICES: index of D in D_list; else -1 */
} pos_plan;

typedef struct pos_search_stats {
    uint64_t evaluated;         /* complete plans whose makespan was computed */
    uint64_t warmup_evaluated;  /* of which in the warm-up */
    uint64_t prefixes;          /* partial plans generated (all depths) */
    uint64_t pruned_bound;      /* children cut by g(S_x) > T_min */
    uint64_t pruned_memory;     /* children cut by memory feasibility */
    uint64_t relaxations;       /* DAG node relaxations (2*S*M per evaluation) */
    uint64_t slices, slices_feasible;
    uint64_t launches;          /* kernel launches */
    double ms_setup, ms_warmup, ms_search, ms_total;  /* host wall clock */
    /* device time per kernel kind, CUDA events on the search's stream */
    double ms_expand, ms_complete, ms_leaf;
    uint64_t expand_launches, complete_launches, leaf_launches;
    /* frontier entries read by the expansion / completion kernels, and
       complete plans written by the completion kernel */
    uint64_t parents_expand, parents_complete, leaves;
    /* POS_PRUNE_TIGHT: device time and launches of the completion-bound
       tables (one launch per batch of slices) */
    double ms_bound;
    uint64_t bound_launches;
    /* batches of slices run a second time, host-driven, because a frontier
       of their pipelined pass overflowed frontier_cap */
    uint64_t reruns;
    /* per parent depth x (stages 0..x-1 placed; x = S-2 is the completion):
       device time of its level kernels (profile only), their launches, the
       frontier entries they read and the children (plans) they wrote */
    double ms_depth[POS_MAX_STAGES];
    uint64_t launches_depth[POS_MAX_STAGES];
    uint64_t parents_depth[POS_MAX_STAGES];
    uint64_t children_depth[POS_MAX_STAGES];
    uint64_t pruned_ridge;      /* children cut by the layer-level (ridge) rule */
} pos_search_stats;

/*
 * Exact search (Sec. 4.2.3) on the current CUDA device: warm-up sampling,
 * then enumeration of every slice's layer compositions with the memory cut
 * and the stage-level prune chosen by problem->prune (Eq. 2 / Theorem 1, or
 * the tighter bound); the result equals the exhaustive optimum.  Host pointers in, host plan out;
 * synchronous.  stats may be NULL.
 * Under POS_SCHED_INTERLEAVED_1F1B the S = N devices hold problem->V chunks
 * each: a plan is a slice (M, TP index, type placement over the N devices)
 * and a composition of L into the N*V virtual stages (C(L-1, NV-1) per
 * slice in the global index); M values that are not multiples of N are
 * skipped (their indices still count).  Prune modes there: POS_PRUNE_EQ2
 * cuts a prefix when some device's serial work over its placed chunks,
 * M * sum (F + B) + sum dsync, is already worse than the incumbent;
 * POS_PRUNE_TIGHT adds, per device whose first chunk is placed, the path
 * through the fill forwards, its chain and the drain backwards.  Layer-level
 * (ridge) pruning is not defined there (POS_EINVAL).
 * Errors: POS_EINVAL, POS_EOVERFLOW (guard fails for some M), POS_ENOMEM,
 * POS_ECUDA, POS_ETIMEOUT, POS_EINFEASIBLE (no memory-feasible plan; *out
 * has found = 0).
 * Limits (checked on the host before the device is touched; POS_EINVAL):
 * at most 2^22 slices (M values x TP indices x placements; M values x
 * class sequences of every D under POS_PLACE_DEVICES) and 2^22 placements;
 * under POS_PLACE_DEVICES at most 65536 devices per type; the global index
 * (slices x compositions) must fit in 64 bits; the lcm of all D*M must be
 * below 2^32.  Memory-feasible slices are
 * enumerated in batches of at most 65535 slices, one after another.
 * Memory: the work buffers (one frontier of frontier_cap 32-byte entries per
 * depth, a leaf buffer of the same length, slice and feasibility tables,
 * and with POS_PRUNE_TIGHT 1 KB of bound tables per stage and slice of a
 * batch),
 * a stream and pinned counters are kept per device between calls, grown on
 * demand and released at process exit; concurrent searches on one device
 * are serialised.
 */
pos_status poseidon_search(const pos_problem *problem, pos_plan *out, pos_search_stats *stats);

/* Message describing the last error of the calling thread ("" if none). */
const char *poseidon_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* POSEIDON_H */
