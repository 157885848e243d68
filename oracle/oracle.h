/*
 * Poseidon CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded C implementation of what the search hot
 * path computes, written from the paper's definitions:
 *   - the DAG cost model of Sec. 4.1 (nodes Sec. 4.1.1, edges Sec. 4.1.2,
 *     weights Sec. 4.1.3) with the 1F1B intra-stage order, evaluated as the
 *     longest path through an explicitly built graph (Kahn order + DP);
 *   - per-stage memory feasibility (Sec. 3.2, Sec. 4.2.3, Lemma "memlimit"
 *     of App. B.3);
 *   - the stage-level lower bound g(S_x) of Eq. 2 and the search of
 *     Sec. 4.2.3 (depth-first over slices and layer allocations, prune when
 *     g(S_x) > T_min, Theorem 1).
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's CPU baseline may load
 * this library.  It shares no code, header or table with the CUDA path.
 */
#ifndef POSEIDON_ORACLE_H
#define POSEIDON_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ORC_MAX_S 16

typedef struct {
    int32_t L, n_types, n_tp;            /* K = n_types * n_tp classes, k = type*n_tp + tp_idx */
    const int32_t *fwd, *bwd, *dsync;    /* [K][L] microseconds per layer */
    const int32_t *p2p_f, *p2p_b;        /* [K][K] microseconds, [src class][dst class] */
    const int64_t *mem_w, *mem_a;        /* [K][L] bytes; mem_a per in-flight micro-batch */
    const int64_t *cap;                  /* [K] bytes */
    int32_t schedule;                    /* ORC_SCHED_1F1B or ORC_SCHED_EAGER_1F1B */
} orc_tables;

/* Pipeline schedules: the order of each stage's chain and its in-flight
 * micro-batches.  Stage s (1-based) of N runs W_s forwards, then
 * (B_i, F_{W_s+i}) for i = 1..M-W_s, then the remaining backwards, with
 *   1F1B:        W_s = min(N-s+1, M)
 *   Eager 1F1B:  W_s = min(2(N-s)+1, M)     (App. B: warm-up of 2(N-i)+1
 *                forwards, steady B-F groups, cool-down backwards). */
#define ORC_SCHED_1F1B 0
#define ORC_SCHED_EAGER_1F1B 1
#define ORC_SCHED_INTERLEAVED_1F1B 2  /* candidates carry V; V <= 1 runs 1F1B */

/* 16-byte candidate record (same field meaning as the library's). */
typedef struct {
    uint64_t map_rank;
    uint32_t type_code;
    uint8_t S, M, tp_idx, pad;
} orc_candidate;

/* 24-byte record with a TP index per stage (same field meaning as the
 * library's pos_candidate_ex): TP index of stage s in bits [2s, 2s+2) of
 * tp_code, so n_tp <= 4. */
typedef struct {
    uint64_t map_rank;
    uint32_t type_code;
    uint32_t tp_code;
    uint8_t S, M, V, pad0;
    uint32_t pad1;
} orc_candidate_ex;

typedef struct {
    orc_tables tab;
    int32_t S;
    int32_t n_M;
    const int32_t *M_list;      /* [n_M] ascending */
    const int32_t *dp_list;     /* [n_tp] data-parallel degree D per TP index */
    int32_t placement;          /* 0 = any type per stage, 1 = exact per-type stage counts,
                                   2 = a (type, TP index) per stage using exactly the
                                   devices of each type (per-stage TP, see below) */
    const int32_t *type_counts; /* [n_types] stages per type (placement 1), devices per
                                   type (placement 2) */
    int32_t ridge;              /* 1: layer-level pruning (Theorem 2): only plans whose
                                   layer counts over the stages of each device type
                                   rise, then fall ("ridge-like"); placements 0 and 1 */
    /* placement 2 only: slices are (M, D, class sequence k_1..k_S) with
     * k = type * n_tp + tp_idx chosen per stage, allowed when for every type
     * sum over its stages of D * tp_list[tp_idx] == type_counts[type]; the
     * class sequences of one D in lexicographic order. */
    const int32_t *tp_list;     /* [n_tp] TP degree of each TP index */
    int32_t n_D;                /* data-parallel degrees tried */
    const int32_t *D_list;      /* [n_D] */
} orc_problem;

typedef struct {
    int32_t found;
    int32_t m_idx, tp_idx, M, D;
    int32_t T;                  /* makespan (us) */
    uint64_t place_rank, map_rank, global_index;
    int32_t types[ORC_MAX_S], layers[ORC_MAX_S];
    int32_t tps[ORC_MAX_S];     /* TP index of each stage (device, interleaved) */
    int32_t d_idx;              /* placement 2: index into D_list (tp_idx is -1) */
} orc_plan;

typedef struct {
    uint64_t leaves_evaluated;  /* complete configurations whose DAG was evaluated */
    uint64_t prefixes_pruned;   /* partial configurations cut by g(S_x) > T_min */
    uint64_t prefixes_memory;   /* partial configurations cut by memory */
    uint64_t warmup_evaluated;
    uint64_t prefixes_ridge;    /* partial configurations cut by the ridge rule */
} orc_stats;

typedef struct {
    int64_t nodes, compute_nodes, allreduce_nodes, control_nodes;
    int64_t inter_edges, intra_edges, allreduce_edges, aux_edges;
} orc_dag_counts;

/* C(n, k) from Pascal's rule; 0 when k < 0 or k > n.  n <= 127, k <= 15
 * (exact in 64 bits there; S <= 16 stages never needs more). */
uint64_t orc_binom(int n, int k);
/* Lexicographic (ascending l_1, l_2, ...) rank <-> composition of L into S parts. */
int orc_unrank(int L, int S, uint64_t rank, int32_t *layers);
uint64_t orc_rank(int L, int S, const int32_t *layers);

/* Evaluate one configuration: stage s (0-based) holds layers[s] consecutive
 * layers and runs on class cls[s].  Writes the makespan (longest path) and
 * the memory-feasibility flag.  Returns 0, or -1 on invalid input. */
int orc_eval(const orc_tables *t, int S, int M, const int32_t *cls, const int32_t *layers,
             int32_t *T, int32_t *feasible, orc_dag_counts *counts);
/* Same DAG, but also returns every node's finish time (F then B, stage-major,
 * [s][m]); finish must hold 2*S*M values. */
int orc_eval_finish(const orc_tables *t, int S, int M, const int32_t *cls, const int32_t *layers,
                    int32_t *finish);
/* g(S_x) of Eq. 2 for the prefix of stages 1..x (1 <= x <= S). */
int64_t orc_lower_bound(const orc_tables *t, int S, int M, const int32_t *cls,
                        const int32_t *layers, int x);
/* Tightened lower bound for the prefix of stages 1..x (only layers[0..x-1]
 * are read).  With the path lengths
 *   P(y, i) = sum_{j<y} (F_j + pf_j) + M (F_y + B_y) + sum_{j=i}^{y-1} (B_j + pb_j) + d_i
 * of a complete configuration (1 <= i <= y <= S), it is the largest of
 *   max_{i<=x} P(x, i)                        (Eq. 2 with the P2P edges),
 *   min over completions of max_{y>x} P(y, y),
 *   min over completions of max_{y>x, i<=x} P(y, i),
 * the minima taken over the memory-feasible completions of stages x+1..S,
 * enumerated one by one.  Each P(y, i) is a path of the DAG, so the bound
 * never exceeds the makespan of a feasible completion.  Returns -1 on
 * invalid input and -2 when no completion fits in memory. */
int64_t orc_lower_bound_tight(const orc_tables *t, int S, int M, const int32_t *cls,
                              const int32_t *layers, int x);
/* Interleaved 1F1B (Sec. 4.1.4): N devices of classes cls[0..N-1], each
 * holding V >= 2 model chunks; layers[0..NV-1] are the layer counts of the
 * NV virtual stages in model order (virtual stage j is chunk j / N on
 * device j % N).  Device order and memory: see oracle.c.  M must be a
 * multiple of N.  Returns 0, or -1 on invalid input. */
int orc_eval_interleaved(const orc_tables *t, int N, int V, int M, const int32_t *cls,
                         const int32_t *layers, int32_t *T, int32_t *feasible,
                         orc_dag_counts *counts);
/* orc_eval_interleaved with the finish time of every compute node
 * (finish[j*M + m] for F_{j,m}, finish[NV*M + j*M + m] for B_{j,m}; 2NVM
 * entries) and each device's largest activation footprint along its order
 * (peak[0..N-1], bytes, without its weights). */
int orc_eval_interleaved_detail(const orc_tables *t, int N, int V, int M, const int32_t *cls,
                                const int32_t *layers, int32_t *T, int32_t *feasible,
                                int32_t *finish, int64_t *peak);
/* Decode and evaluate n candidate records.  feasible: 1 ok, 0 memory
 * infeasible, 2 invalid record, 3 overflow guard tripped. */
int orc_eval_batch(const orc_tables *t, const orc_candidate *c, int64_t n, int32_t *T,
                   uint8_t *feasible);
/* Same with a TP index per stage (per device for interleaved records): the
 * class of stage s is type_s * n_tp + tp_s.  Returns -1 when n_tp > 4. */
int orc_eval_batch_ex(const orc_tables *t, const orc_candidate_ex *c, int64_t n, int32_t *T,
                      uint8_t *feasible);
/* Exact search of Sec. 4.2.3.  prune=0 disables the g(S_x) prune (memory
 * infeasible prefixes are still skipped).  warmup = number of random feasible
 * samples evaluated first (Sec. 4.2.3); it never changes the result.
 * Slice order and global index: placements 0 and 1 take (m_idx, tp_idx,
 * type sequence), ordinal (m_idx * n_tp + tp_idx) * n_place + place_rank;
 * placement 2 takes (m_idx, d_idx, class sequence), ordinal
 * m_idx * P + (sequences of D_list[0..d_idx-1]) + place_rank, P = the
 * sequences of all D; global index = ordinal * C(L-1, S-1) + map_rank.
 * Returns 0 (plan->found tells whether a feasible plan exists) or -1. */
int orc_search(const orc_problem *p, int prune, int warmup, uint64_t seed, orc_plan *plan,
               orc_stats *stats);
/* orc_search over the slices whose index in the global order is
 * part (mod n_parts) only (warm-up samples too): a driver that runs the
 * parts in separate processes and keeps the best plan by (T/(D*M), global
 * index) obtains orc_search's plan. */
int orc_search_part(const orc_problem *p, int prune, int warmup, uint64_t seed, int part,
                    int n_parts, orc_plan *plan, orc_stats *stats);

/* Search over Interleaved 1F1B plans with V chunks per device: the slices
 * of orc_search over the N = p->S devices (M values that are not multiples
 * of N skipped), every composition of L into the N*V virtual stages,
 * evaluated by orc_eval_interleaved; objective, global index (with
 * C(L-1, N*V-1) compositions per slice) and ties as in orc_search.  Cuts:
 * memory (a device's placed chunk weights exceed its capacity) and, when
 * prune != 0, the per-device serial-work bound (see oracle.c).  Returns 0,
 * -1 on invalid input, -2 when the overflow guard trips. */
int orc_search_interleaved(const orc_problem *p, int V, int prune, orc_plan *plan,
                           orc_stats *stats);

#ifdef __cplusplus
}
#endif
#endif
