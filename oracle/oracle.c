/*
 * Poseidon CPU oracle -- TEST INFRASTRUCTURE ONLY (see oracle.h).
 *
 * Everything here follows the paper's definitions literally and is meant to
 * be checked by eye against it:
 *   Sec. 4.1.1  nodes: F_{s,m}, B_{s,m} (2NM), R_s (N), control nodes S, E
 *   Sec. 4.1.2  edges: inter-stage F_{s,m}->F_{s+1,m}, B_{s,m}->B_{s-1,m};
 *               intra-stage chain given by the schedule (2M-1 per stage);
 *               B_{s,M}->R_s; S->F_{1,1}; R_s->E
 *   Sec. 4.1.3  weights: F/B = per-layer time summed over the stage's layers,
 *               inter-stage edge = activation transfer time, intra-stage
 *               edges 0, R_s = all-reduce time summed over the stage's
 *               layers, control nodes and auxiliary edges 0
 *   Sec. 4.1    T = longest path (node + edge weights), computed by DP
 *   Eq. 2       g(S_x), Theorem 1: prune when g(S_x) > T_min
 *   Sec. 4.2.3  warm-up sampling, then enumeration of 3D configurations,
 *               device-to-stage assignments and layer allocations with
 *               memory constraints
 *
 * Readings where the paper is silent (the library documents the same ones):
 *   - 1F1B order of stage s (1-based) with W_s = min(N-s+1, M) warm-up
 *     forwards: F_1..F_W, then (B_i, F_{W+i}) for i = 1..M-W, then the
 *     remaining backwards.  Eager 1F1B (App. B): the same with
 *     W_s = min(2(N-s)+1, M).
 *   - weights use per-layer tables summed over the stage's layers (reduces to
 *     the paper's product for identical layers).
 *   - inter-stage edge weights come from a table indexed by the ordered
 *     (sending class, receiving class) pair.
 *   - memory of stage s: sum(mem_w) + W_s * sum(mem_a) <= cap.
 *   - one pipeline is modelled: all D pipelines are identical (Sec. 4.2.3),
 *     so the D edges into R_s carry the same value.
 *   - objective across slices: T / (D*M) (time per sample), compared exactly
 *     by cross-multiplication; ties go to the lowest global index.
 */
#include "oracle.h"

#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------ */
/* Binomial coefficients by Pascal's rule.                             */
/* ------------------------------------------------------------------ */
static uint64_t binom_tab[128][16];
static int binom_ready = 0;

static void binom_init(void) {
    if (binom_ready) return;
    for (int n = 0; n < 128; ++n) {
        for (int k = 0; k <= 15; ++k) {
            if (k == 0) binom_tab[n][k] = 1;
            else if (n == 0) binom_tab[n][k] = 0;
            else binom_tab[n][k] = binom_tab[n - 1][k - 1] + binom_tab[n - 1][k];
        }
    }
    binom_ready = 1;
}

uint64_t orc_binom(int n, int k) {
    binom_init();
    if (n < 0 || k < 0 || k > n || n > 127 || k > 15) return 0;
    return binom_tab[n][k];
}

/* Number of compositions of r layers into p non-empty stages. */
static uint64_t n_comp(int r, int p) {
    if (p == 0) return r == 0 ? 1 : 0;
    if (r < p) return 0;
    return orc_binom(r - 1, p - 1);
}

/* Lexicographic order on (l_1, ..., l_S): the rank of a composition is the
 * number of compositions that are lexicographically smaller. */
uint64_t orc_rank(int L, int S, const int32_t *layers) {
    uint64_t r = 0;
    int rem = L;
    for (int s = 0; s < S - 1; ++s) {
        int after = S - s - 1;
        for (int v = 1; v < layers[s]; ++v) r += n_comp(rem - v, after);
        rem -= layers[s];
    }
    return r;
}

int orc_unrank(int L, int S, uint64_t rank, int32_t *layers) {
    if (S < 1 || S > ORC_MAX_S || S > L || L > 127) return -1;
    if (rank >= n_comp(L, S)) return -1;
    int rem = L;
    for (int s = 0; s < S - 1; ++s) {
        int after = S - s - 1;
        int v;
        for (v = 1; v <= rem - after; ++v) {
            uint64_t cnt = n_comp(rem - v, after);
            if (rank < cnt) break;
            rank -= cnt;
        }
        layers[s] = v;
        rem -= v;
    }
    layers[S - 1] = rem;
    return 0;
}

/* ------------------------------------------------------------------ */
/* Stage weights (Sec. 4.1.3) and memory (Sec. 3.2).                   */
/* ------------------------------------------------------------------ */
typedef struct {
    int64_t F[ORC_MAX_S], B[ORC_MAX_S], d[ORC_MAX_S];
    int64_t pf[ORC_MAX_S], pb[ORC_MAX_S]; /* pf[s]: F edge s->s+1, pb[s]: B edge s+1->s */
} stage_w;

/* Forwards before the first backward of stage s (0-based), which is also
 * the number of micro-batches whose activations the stage holds at once:
 * N - s + 1 (1F1B) or 2(N - s) + 1 (Eager 1F1B) in 1-based numbering. */
static int warmup_count(int sched, int S, int M, int s /* 0-based */) {
    int w = sched == ORC_SCHED_EAGER_1F1B ? 2 * (S - 1 - s) + 1 : S - s;
    return w < M ? w : M;
}

static void stage_weights(const orc_tables *t, int S, const int32_t *cls, const int32_t *layers,
                          stage_w *w) {
    int L = t->L;
    int first = 0;
    for (int s = 0; s < S; ++s) {
        const int32_t *f = t->fwd + (int64_t)cls[s] * L;
        const int32_t *b = t->bwd + (int64_t)cls[s] * L;
        const int32_t *d = t->dsync + (int64_t)cls[s] * L;
        int64_t sf = 0, sb = 0, sd = 0;
        for (int l = first; l < first + layers[s]; ++l) {
            sf += f[l];
            sb += b[l];
            sd += d[l];
        }
        w->F[s] = sf;
        w->B[s] = sb;
        w->d[s] = sd;
        first += layers[s];
    }
    int K = t->n_types * t->n_tp;
    for (int s = 0; s + 1 < S; ++s) {
        w->pf[s] = t->p2p_f[(int64_t)cls[s] * K + cls[s + 1]];
        w->pb[s] = t->p2p_b[(int64_t)cls[s + 1] * K + cls[s]];
    }
}

/* Memory of stage s holding layers [first, first+l): weights plus W_s
 * in-flight micro-batches of activations must fit the device capacity. */
static int stage_memory_ok(const orc_tables *t, int S, int M, int s, int cls, int first, int l) {
    int L = t->L;
    const int64_t *mw = t->mem_w + (int64_t)cls * L;
    const int64_t *ma = t->mem_a + (int64_t)cls * L;
    int64_t sw = 0, sa = 0;
    for (int i = first; i < first + l; ++i) {
        sw += mw[i];
        sa += ma[i];
    }
    const int sched = t->schedule == ORC_SCHED_INTERLEAVED_1F1B ? ORC_SCHED_1F1B : t->schedule;
    int64_t need = sw + (int64_t)warmup_count(sched, S, M, s) * sa;
    return need <= t->cap[cls];
}

static int config_memory_ok(const orc_tables *t, int S, int M, const int32_t *cls,
                            const int32_t *layers) {
    int first = 0;
    for (int s = 0; s < S; ++s) {
        if (!stage_memory_ok(t, S, M, s, cls[s], first, layers[s])) return 0;
        first += layers[s];
    }
    return 1;
}

/* Overflow guard: every path visits each node at most once, so its length is
 * at most M*sum_l max_k(fwd+bwd) + sum_l max_k dsync + 2M(S-1)*max p2p. */
static int64_t overflow_bound(const orc_tables *t, int S, int M) {
    int K = t->n_types * t->n_tp, L = t->L;
    int64_t A = 0, Dm = 0, P = 0;
    for (int l = 0; l < L; ++l) {
        int64_t mfb = 0, md = 0;
        for (int k = 0; k < K; ++k) {
            int64_t fb = (int64_t)t->fwd[(int64_t)k * L + l] + t->bwd[(int64_t)k * L + l];
            if (fb > mfb) mfb = fb;
            if (t->dsync[(int64_t)k * L + l] > md) md = t->dsync[(int64_t)k * L + l];
        }
        A += mfb;
        Dm += md;
    }
    for (int i = 0; i < K * K; ++i) {
        if (t->p2p_f[i] > P) P = t->p2p_f[i];
        if (t->p2p_b[i] > P) P = t->p2p_b[i];
    }
    return (int64_t)M * A + Dm + 2 * (int64_t)M * (S - 1) * P;
}

/* ------------------------------------------------------------------ */
/* The explicit DAG (Sec. 4.1) and its longest path.                   */
/* ------------------------------------------------------------------ */
typedef struct {
    int n_nodes, n_edges;
    int64_t *w;          /* node weights */
    int *esrc, *edst;    /* edge list */
    int64_t *ew;         /* edge weights */
    int *indeg, *head, *next_e, *queue;
    int64_t *start, *fin;
    int cap_nodes, cap_edges;
} dag;

static void dag_free(dag *g) {
    free(g->w); free(g->esrc); free(g->edst); free(g->ew); free(g->indeg); free(g->head);
    free(g->next_e); free(g->queue); free(g->start); free(g->fin);
    memset(g, 0, sizeof(*g));
}

static int dag_reserve(dag *g, int nodes, int edges) {
    if (nodes <= g->cap_nodes && edges <= g->cap_edges) return 0;
    dag_free(g);
    g->w = malloc(sizeof(int64_t) * nodes);
    g->indeg = malloc(sizeof(int) * nodes);
    g->head = malloc(sizeof(int) * nodes);
    g->queue = malloc(sizeof(int) * nodes);
    g->start = malloc(sizeof(int64_t) * nodes);
    g->fin = malloc(sizeof(int64_t) * nodes);
    g->esrc = malloc(sizeof(int) * edges);
    g->edst = malloc(sizeof(int) * edges);
    g->ew = malloc(sizeof(int64_t) * edges);
    g->next_e = malloc(sizeof(int) * edges);
    if (!g->w || !g->indeg || !g->head || !g->queue || !g->start || !g->fin || !g->esrc ||
        !g->edst || !g->ew || !g->next_e) {
        dag_free(g);
        return -1;
    }
    g->cap_nodes = nodes;
    g->cap_edges = edges;
    return 0;
}

static void add_edge(dag *g, int a, int b, int64_t w) {
    int e = g->n_edges++;
    g->esrc[e] = a;
    g->edst[e] = b;
    g->ew[e] = w;
}

/* node numbering: 0 = start S; F(s,m), B(s,m) compute nodes; R(s); E last */
#define NODE_F(s, m) (1 + 2 * ((s) * M + (m)))
#define NODE_B(s, m) (2 + 2 * ((s) * M + (m)))
#define NODE_R(s) (1 + 2 * S * M + (s))

/* Kahn topological order; longest path where a node finishes at its
 * latest predecessor finish (+ edge weight) plus its own weight. */
static int solve_longest(dag *g, int n_nodes, int node_E, int64_t *T_out) {
    for (int i = 0; i < n_nodes; ++i) {
        g->indeg[i] = 0;
        g->head[i] = -1;
        g->start[i] = 0;
    }
    for (int e = 0; e < g->n_edges; ++e) {
        g->indeg[g->edst[e]]++;
        g->next_e[e] = g->head[g->esrc[e]];
        g->head[g->esrc[e]] = e;
    }
    int qh = 0, qt = 0;
    for (int i = 0; i < n_nodes; ++i)
        if (g->indeg[i] == 0) g->queue[qt++] = i;
    while (qh < qt) {
        int u = g->queue[qh++];
        g->fin[u] = g->start[u] + g->w[u];
        for (int e = g->head[u]; e >= 0; e = g->next_e[e]) {
            int v = g->edst[e];
            int64_t cand = g->fin[u] + g->ew[e];
            if (cand > g->start[v]) g->start[v] = cand;
            if (--g->indeg[v] == 0) g->queue[qt++] = v;
        }
    }
    if (qt != n_nodes) return -1; /* not a DAG */
    *T_out = g->fin[node_E];
    return 0;
}

static int build_and_solve(dag *g, int sched, int S, int M, const stage_w *sw,
                           orc_dag_counts *counts, int64_t *T_out) {
    int n_nodes = 2 + 2 * S * M + S;
    int n_edges_max = 2 * (S - 1) * M + S * (2 * M - 1) + S + 1 + S;
    if (dag_reserve(g, n_nodes, n_edges_max)) return -1;
    g->n_nodes = n_nodes;
    g->n_edges = 0;
    int node_E = n_nodes - 1;

    /* nodes and weights (Sec. 4.1.1, 4.1.3) */
    g->w[0] = 0;
    g->w[node_E] = 0;
    for (int s = 0; s < S; ++s) {
        for (int m = 0; m < M; ++m) {
            g->w[NODE_F(s, m)] = sw->F[s];
            g->w[NODE_B(s, m)] = sw->B[s];
        }
        g->w[NODE_R(s)] = sw->d[s];
    }
    int64_t c_inter = 0, c_intra = 0, c_ar = 0, c_aux = 0;

    /* inter-stage edges: activations forward, gradients backward */
    for (int m = 0; m < M; ++m) {
        for (int s = 0; s + 1 < S; ++s) {
            add_edge(g, NODE_F(s, m), NODE_F(s + 1, m), sw->pf[s]);
            add_edge(g, NODE_B(s + 1, m), NODE_B(s, m), sw->pb[s]);
            c_inter += 2;
        }
    }
    /* intra-stage edges: the schedule's order of each stage, weight 0 */
    int order_node[2 * 255];
    for (int s = 0; s < S; ++s) {
        int W = warmup_count(sched, S, M, s), n = 0;
        for (int m = 0; m < W; ++m) order_node[n++] = NODE_F(s, m);
        for (int i = 0; i < M - W; ++i) {
            order_node[n++] = NODE_B(s, i);
            order_node[n++] = NODE_F(s, W + i);
        }
        for (int m = M - W; m < M; ++m) order_node[n++] = NODE_B(s, m);
        if (n != 2 * M) return -1;
        /* F_{s,m} must come before B_{s,m} in the chain */
        for (int m = 0; m < M; ++m) {
            int pf_ = -1, pb_ = -1;
            for (int i = 0; i < n; ++i) {
                if (order_node[i] == NODE_F(s, m)) pf_ = i;
                if (order_node[i] == NODE_B(s, m)) pb_ = i;
            }
            if (!(pf_ >= 0 && pb_ > pf_)) return -1;
        }
        for (int i = 0; i + 1 < n; ++i) {
            add_edge(g, order_node[i], order_node[i + 1], 0);
            c_intra += 1;
        }
    }
    /* all-reduce edges B_{s,M} -> R_s and auxiliary edges */
    for (int s = 0; s < S; ++s) {
        add_edge(g, NODE_B(s, M - 1), NODE_R(s), 0);
        c_ar += 1;
    }
    add_edge(g, 0, NODE_F(0, 0), 0);
    c_aux += 1;
    for (int s = 0; s < S; ++s) {
        add_edge(g, NODE_R(s), node_E, 0);
        c_aux += 1;
    }
    if (counts) {
        counts->nodes = n_nodes;
        counts->compute_nodes = 2 * (int64_t)S * M;
        counts->allreduce_nodes = S;
        counts->control_nodes = 2;
        counts->inter_edges = c_inter;
        counts->intra_edges = c_intra;
        counts->allreduce_edges = c_ar;
        counts->aux_edges = c_aux;
    }

    return solve_longest(g, n_nodes, node_E, T_out);
}

static int check_inputs(const orc_tables *t, int S, int M, const int32_t *cls,
                        const int32_t *layers) {
    int K = t->n_types * t->n_tp;
    if (S < 1 || S > ORC_MAX_S || M < 1 || M > 255 || S > t->L || t->L > 127) return -1;
    int sum = 0;
    for (int s = 0; s < S; ++s) {
        if (cls[s] < 0 || cls[s] >= K || layers[s] < 1) return -1;
        sum += layers[s];
    }
    return sum == t->L ? 0 : -1;
}

int orc_eval(const orc_tables *t, int S, int M, const int32_t *cls, const int32_t *layers,
             int32_t *T, int32_t *feasible, orc_dag_counts *counts) {
    if (check_inputs(t, S, M, cls, layers)) return -1;
    stage_w sw;
    stage_weights(t, S, cls, layers, &sw);
    dag g;
    memset(&g, 0, sizeof(g));
    int64_t T64;
    int rc = build_and_solve(&g, t->schedule, S, M, &sw, counts, &T64);
    dag_free(&g);
    if (rc) return -1;
    if (T64 >= ((int64_t)1 << 31)) return -1;
    *T = (int32_t)T64;
    *feasible = config_memory_ok(t, S, M, cls, layers);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Interleaved 1F1B (Sec. 4.1.4).                                      */
/* ------------------------------------------------------------------ */
/* N devices (physical stages) each hold V model chunks: virtual stage j
 * (0-based, j < NV) is chunk j / N on device j % N, and the L layers are
 * split over the NV virtual stages in order.  The paper fixes the node and
 * edge counts (2VNM compute nodes, 2(NV-1)M inter-stage edges, N(2VM-1)
 * intra-stage edges) but not the order of a device's 2VM ops; the order
 * taken is the interleaved schedule the paper cites (Narayanan et al.
 * 2021): forward number k (k = 0..VM-1) of a device runs chunk
 * (k mod NV) div N on micro-batch (k div NV) N + k mod N, backward number k
 * the chunk V-1-((k mod NV) div N) on the same micro-batch; the device runs
 * w = min((N-d-1)*2 + (V-1)*N, VM) warm-up forwards (w = VM when M = N),
 * then alternates one forward and one backward, then runs the remaining
 * backwards.  M must be a multiple of N. */
typedef struct {
    int c, m, is_b;
} il_op;

static void interleaved_chain(int N, int V, int M, int d, il_op *ops) {
    int total = M * V;
    int warm = M == N ? total : (N - d - 1) * 2 + (V - 1) * N;
    if (warm > total) warm = total;
    /* forwards 0..warm-1, then (F, B) pairs, then the remaining backwards */
    int f = 0, b = 0, n = 0;
    while (f < warm) {
        int p = f % (N * V);
        ops[n].c = p / N;
        ops[n].m = (f / (N * V)) * N + p % N;
        ops[n].is_b = 0;
        ++n;
        ++f;
    }
    while (f < total) {
        int p = f % (N * V);
        ops[n].c = p / N;
        ops[n].m = (f / (N * V)) * N + p % N;
        ops[n].is_b = 0;
        ++n;
        ++f;
        p = b % (N * V);
        ops[n].c = V - 1 - p / N;
        ops[n].m = (b / (N * V)) * N + p % N;
        ops[n].is_b = 1;
        ++n;
        ++b;
    }
    while (b < total) {
        int p = b % (N * V);
        ops[n].c = V - 1 - p / N;
        ops[n].m = (b / (N * V)) * N + p % N;
        ops[n].is_b = 1;
        ++n;
        ++b;
    }
}

/* The interleaved DAG of one plan and its longest path; optionally the
 * finish time of every compute node (finish[j*M + m] for F_{j,m},
 * finish[J*M + j*M + m] for B_{j,m}) and each device's activation peak. */
static int il_eval(const orc_tables *t, int N, int V, int M, const int32_t *cls,
                   const int32_t *layers, int32_t *T, int32_t *feasible, orc_dag_counts *counts,
                   int32_t *finish, int64_t *peak_out) {
    const int J = N * V, L = t->L, K = t->n_types * t->n_tp;
    if (N < 1 || V < 2 || J > ORC_MAX_S || M < 1 || M % N != 0) return -1;
    int sum = 0;
    for (int j = 0; j < J; ++j) {
        if (layers[j] < 1) return -1;
        sum += layers[j];
    }
    if (sum != L) return -1;
    for (int d = 0; d < N; ++d)
        if (cls[d] < 0 || cls[d] >= K) return -1;
    /* virtual-stage weights (Sec. 4.1.3): F_j, B_j over chunk j's layers on
       its device's class; all-reduce per device over all its chunks */
    int64_t F[ORC_MAX_S], B[ORC_MAX_S], dsum[ORC_MAX_S], act[ORC_MAX_S], wsum[ORC_MAX_S];
    for (int d = 0; d < N; ++d) dsum[d] = wsum[d] = 0;
    int first = 0;
    for (int j = 0; j < J; ++j) {
        const int k = cls[j % N];
        int64_t f = 0, b = 0, dd = 0, a = 0, w = 0;
        for (int l = first; l < first + layers[j]; ++l) {
            f += t->fwd[(int64_t)k * L + l];
            b += t->bwd[(int64_t)k * L + l];
            dd += t->dsync[(int64_t)k * L + l];
            a += t->mem_a[(int64_t)k * L + l];
            w += t->mem_w[(int64_t)k * L + l];
        }
        F[j] = f;
        B[j] = b;
        act[j] = a;
        dsum[j % N] += dd;
        wsum[j % N] += w;
        first += layers[j];
    }
    /* nodes: S (0), F_{j,m} and B_{j,m}, R_d, E */
    const int n_nodes = 2 + 2 * J * M + N, node_E = n_nodes - 1;
    const int n_edges_max = 2 * (J - 1) * M + N * (2 * V * M - 1) + N + 1 + N + 1;
    dag g;
    memset(&g, 0, sizeof(g));
    il_op *ops = malloc(sizeof(il_op) * 2 * V * M);
    if (!ops || dag_reserve(&g, n_nodes, n_edges_max)) {
        free(ops);
        dag_free(&g);
        return -1;
    }
#define IL_F(j, m) (1 + 2 * ((j) * M + (m)))
#define IL_B(j, m) (2 + 2 * ((j) * M + (m)))
#define IL_R(d) (1 + 2 * J * M + (d))
    g.n_nodes = n_nodes;
    g.n_edges = 0;
    g.w[0] = 0;
    g.w[node_E] = 0;
    for (int j = 0; j < J; ++j)
        for (int m = 0; m < M; ++m) {
            g.w[IL_F(j, m)] = F[j];
            g.w[IL_B(j, m)] = B[j];
        }
    for (int d = 0; d < N; ++d) g.w[IL_R(d)] = dsum[d];
    int64_t c_inter = 0, c_intra = 0;
    /* inter-stage edges between consecutive virtual stages (their devices) */
    for (int m = 0; m < M; ++m)
        for (int j = 0; j + 1 < J; ++j) {
            const int ka = cls[j % N], kb = cls[(j + 1) % N];
            add_edge(&g, IL_F(j, m), IL_F(j + 1, m), t->p2p_f[(int64_t)ka * K + kb]);
            add_edge(&g, IL_B(j + 1, m), IL_B(j, m), t->p2p_b[(int64_t)kb * K + ka]);
            c_inter += 2;
        }
    /* intra-device chains and the peak of the activations each device holds */
    int ok = 1;
    *feasible = 1;
    for (int d = 0; d < N && ok; ++d) {
        interleaved_chain(N, V, M, d, ops);
        int64_t held = 0, peak = 0;
        for (int i = 0; i < 2 * V * M; ++i) {
            const int j = ops[i].c * N + d;
            held += ops[i].is_b ? -act[j] : act[j];
            if (held > peak) peak = held;
            if (i > 0) {
                const int a = ops[i - 1].c * N + d;
                add_edge(&g, ops[i - 1].is_b ? IL_B(a, ops[i - 1].m) : IL_F(a, ops[i - 1].m),
                         ops[i].is_b ? IL_B(j, ops[i].m) : IL_F(j, ops[i].m), 0);
                c_intra += 1;
            }
        }
        /* each forward precedes its backward on the device */
        for (int i = 0; i < 2 * V * M && ok; ++i) {
            if (!ops[i].is_b) continue;
            int seen = 0;
            for (int u = 0; u < i; ++u)
                seen |= !ops[u].is_b && ops[u].c == ops[i].c && ops[u].m == ops[i].m;
            ok = seen;
        }
        const int lc = ops[2 * V * M - 1].c * N + d;
        add_edge(&g, IL_B(lc, ops[2 * V * M - 1].m), IL_R(d), 0);
        add_edge(&g, IL_R(d), node_E, 0);
        if (peak_out) peak_out[d] = peak;
        if (peak + wsum[d] > t->cap[cls[d]]) *feasible = 0;
    }
    add_edge(&g, 0, IL_F(0, 0), 0);
    int64_t T64 = 0;
    int rc = ok ? solve_longest(&g, n_nodes, node_E, &T64) : -1;
    if (counts) {
        counts->nodes = n_nodes;
        counts->compute_nodes = 2 * (int64_t)J * M;
        counts->allreduce_nodes = N;
        counts->control_nodes = 2;
        counts->inter_edges = c_inter;
        counts->intra_edges = c_intra;
        counts->allreduce_edges = N;
        counts->aux_edges = N + 1;
    }
    if (!rc && finish)
        for (int j = 0; j < J; ++j)
            for (int m = 0; m < M; ++m) {
                finish[j * M + m] = (int32_t)g.fin[IL_F(j, m)];
                finish[J * M + j * M + m] = (int32_t)g.fin[IL_B(j, m)];
            }
#undef IL_F
#undef IL_B
#undef IL_R
    free(ops);
    dag_free(&g);
    if (rc || T64 >= ((int64_t)1 << 31)) return -1;
    *T = (int32_t)T64;
    return 0;
}

int orc_eval_interleaved(const orc_tables *t, int N, int V, int M, const int32_t *cls,
                         const int32_t *layers, int32_t *T, int32_t *feasible,
                         orc_dag_counts *counts) {
    return il_eval(t, N, V, M, cls, layers, T, feasible, counts, NULL, NULL);
}

int orc_eval_interleaved_detail(const orc_tables *t, int N, int V, int M, const int32_t *cls,
                                const int32_t *layers, int32_t *T, int32_t *feasible,
                                int32_t *finish, int64_t *peak) {
    return il_eval(t, N, V, M, cls, layers, T, feasible, NULL, finish, peak);
}

int orc_eval_finish(const orc_tables *t, int S, int M, const int32_t *cls, const int32_t *layers,
                    int32_t *finish) {
    if (check_inputs(t, S, M, cls, layers)) return -1;
    stage_w sw;
    stage_weights(t, S, cls, layers, &sw);
    dag g;
    memset(&g, 0, sizeof(g));
    int64_t T64;
    int rc = build_and_solve(&g, t->schedule, S, M, &sw, NULL, &T64);
    if (!rc) {
        for (int s = 0; s < S; ++s)
            for (int m = 0; m < M; ++m) {
                finish[(s * M + m)] = (int32_t)g.fin[NODE_F(s, m)];
                finish[S * M + (s * M + m)] = (int32_t)g.fin[NODE_B(s, m)];
            }
    }
    dag_free(&g);
    return rc;
}

/* Eq. 2 with stage totals (1-based x):
 *   g(S_x) = sum_{i<x} F_i + M (F_x + B_x) + max_{1<=i<=x} ( sum_{j=i}^{x-1} B_j + d_i ) */
static int64_t lower_bound_w(const stage_w *w, int M, int x) {
    int64_t g = 0;
    for (int i = 1; i <= x - 1; ++i) g += w->F[i - 1];
    g += (int64_t)M * (w->F[x - 1] + w->B[x - 1]);
    int64_t best = 0;
    for (int i = 1; i <= x; ++i) {
        int64_t v = w->d[i - 1];
        for (int j = i; j <= x - 1; ++j) v += w->B[j - 1];
        if (i == 1 || v > best) best = v;
    }
    return g + best;
}

int64_t orc_lower_bound(const orc_tables *t, int S, int M, const int32_t *cls,
                        const int32_t *layers, int x) {
    if (check_inputs(t, S, M, cls, layers) || x < 1 || x > S) return -1;
    stage_w sw;
    stage_weights(t, S, cls, layers, &sw);
    return lower_bound_w(&sw, M, x);
}

/* ------------------------------------------------------------------ */
/* Tightened stage-level bound (the P2P-inclusive form of Eq. 2 plus a   */
/* bound over the unplaced stages).  Not in the paper: a library option. */
/* ------------------------------------------------------------------ */
/* Length of one S -> E path of the DAG of a complete configuration, for
 * 1 <= i <= y <= S (1-based): the first micro-batch's forwards and their
 * F edges up to stage y, stage y's whole chain (M forwards and M
 * backwards, first op F_{y,1}, last op B_{y,M}), the last micro-batch's
 * backwards and B edges from stage y down to stage i, and R_i:
 *   P(y, i) = sum_{j<y} (F_j + pf_j) + M (F_y + B_y)
 *             + sum_{j=i}^{y-1} (B_j + pb_j) + d_i.
 * Every such path exists (Sec. 4.1.2), so P(y, i) <= T. */
static int64_t path_len(const stage_w *w, int M, int y, int i) {
    int64_t v = 0;
    for (int j = 1; j <= y - 1; ++j) v += w->F[j - 1] + w->pf[j - 1];
    v += (int64_t)M * (w->F[y - 1] + w->B[y - 1]);
    for (int j = i; j <= y - 1; ++j) v += w->B[j - 1] + w->pb[j - 1];
    return v + w->d[i - 1];
}

typedef struct {
    const orc_tables *t;
    int S, M, x;
    const int32_t *cls;
    int32_t layers[ORC_MAX_S];
    int64_t best2, best3; /* minima over the completions seen so far */
    int any;
} tight_ctx;

/* Every memory-feasible completion of stages x+1..S: the two completion
 * terms of the bound, each minimised over completions separately. */
static void tight_completions(tight_ctx *q, int s /* 0-based next stage */, int first) {
    const int L = q->t->L, S = q->S;
    if (s == S) {
        if (first != L) return;
        stage_w w;
        stage_weights(q->t, S, q->cls, q->layers, &w);
        int64_t v2 = INT64_MIN, v3 = INT64_MIN;
        for (int y = q->x + 1; y <= S; ++y) {
            const int64_t a = path_len(&w, q->M, y, y);
            if (a > v2) v2 = a;
            for (int i = 1; i <= q->x; ++i) {
                const int64_t b = path_len(&w, q->M, y, i);
                if (b > v3) v3 = b;
            }
        }
        if (!q->any || v2 < q->best2) q->best2 = v2;
        if (!q->any || v3 < q->best3) q->best3 = v3;
        q->any = 1;
        return;
    }
    for (int l = 1; first + l <= L - (S - s - 1); ++l) {
        if (!stage_memory_ok(q->t, S, q->M, s, q->cls[s], first, l)) continue;
        q->layers[s] = l;
        tight_completions(q, s + 1, first + l);
    }
}

int64_t orc_lower_bound_tight(const orc_tables *t, int S, int M, const int32_t *cls,
                              const int32_t *layers, int x) {
    if (x < 1 || x > S || S > ORC_MAX_S || M < 1) return -1;
    int first = 0;
    for (int s = 0; s < x; ++s) {
        if (layers[s] < 1) return -1;
        first += layers[s];
    }
    if (first > t->L - (S - x)) return -1;
    tight_ctx q;
    memset(&q, 0, sizeof(q));
    q.t = t;
    q.S = S;
    q.M = M;
    q.x = x;
    q.cls = cls;
    for (int s = 0; s < x; ++s) q.layers[s] = layers[s];
    /* term 1: the paths through stage x itself, which the prefix fixes
       (Eq. 2 with the F and B edges on the path added) */
    stage_w w;
    for (int s = x; s < S; ++s) q.layers[s] = 1; /* placeholder: only stages <= x are read */
    stage_weights(t, S, cls, q.layers, &w);
    int64_t lb = INT64_MIN;
    for (int i = 1; i <= x; ++i) {
        const int64_t v = path_len(&w, M, x, i);
        if (v > lb) lb = v;
    }
    if (x == S) return lb;
    tight_completions(&q, x, first);
    if (!q.any) return -2; /* no memory-feasible completion */
    if (q.best2 > lb) lb = q.best2;
    if (q.best3 > lb) lb = q.best3;
    return lb;
}

/* Decode and evaluate one record: stage (device) s has type
 * (tcode >> 2s) & 3 and TP index tp[s]; V >= 2 under the interleaved
 * schedule makes it an interleaved record.  Returns -1 on an internal
 * failure, else 0 with T and the flag written. */
static int eval_record(const orc_tables *t, dag *g, uint64_t rank, uint32_t tcode,
                       const int *tp, int S, int M, int Vbyte, int32_t *T, uint8_t *feasible) {
    int32_t layers[ORC_MAX_S], cls[ORC_MAX_S];
    /* Interleaved 1F1B: V model chunks per device; the composition is over
       the S*V virtual stages */
    const int V = t->schedule == ORC_SCHED_INTERLEAVED_1F1B && Vbyte >= 2 ? Vbyte : 1;
    const int J = S * V;
    int ok = S >= 1 && J <= ORC_MAX_S && J <= t->L && M >= 1 && (V == 1 || M % S == 0);
    if (ok) ok = orc_unrank(t->L, J, rank, layers) == 0;
    for (int s = 0; ok && s < S; ++s) {
        const int ty = (tcode >> (2 * s)) & 3;
        if (ty >= t->n_types || tp[s] < 0 || tp[s] >= t->n_tp) ok = 0;
        cls[s] = ty * t->n_tp + tp[s];
    }
    if (!ok) {
        *T = -1;
        *feasible = 2;
        return 0;
    }
    if (overflow_bound(t, J, M) >= ((int64_t)1 << 31)) {
        *T = -1;
        *feasible = 3;
        return 0;
    }
    if (V >= 2) {
        int32_t Ti, Fi;
        if (orc_eval_interleaved(t, S, V, M, cls, layers, &Ti, &Fi, NULL)) return -1;
        *T = Ti;
        *feasible = (uint8_t)Fi;
        return 0;
    }
    stage_w sw;
    stage_weights(t, S, cls, layers, &sw);
    int64_t T64;
    const int sched = t->schedule == ORC_SCHED_INTERLEAVED_1F1B ? ORC_SCHED_1F1B : t->schedule;
    if (build_and_solve(g, sched, S, M, &sw, NULL, &T64)) return -1;
    *T = (int32_t)T64;
    *feasible = (uint8_t)config_memory_ok(t, S, M, cls, layers);
    return 0;
}

int orc_eval_batch(const orc_tables *t, const orc_candidate *c, int64_t n, int32_t *T,
                   uint8_t *feasible) {
    dag g;
    memset(&g, 0, sizeof(g));
    for (int64_t i = 0; i < n; ++i) {
        int tp[ORC_MAX_S];
        for (int s = 0; s < ORC_MAX_S; ++s) tp[s] = c[i].tp_idx;
        if (eval_record(t, &g, c[i].map_rank, c[i].type_code, tp, c[i].S, c[i].M, c[i].pad,
                        &T[i], &feasible[i])) {
            dag_free(&g);
            return -1;
        }
    }
    dag_free(&g);
    return 0;
}

int orc_eval_batch_ex(const orc_tables *t, const orc_candidate_ex *c, int64_t n, int32_t *T,
                      uint8_t *feasible) {
    if (t->n_tp > 4) return -1;
    dag g;
    memset(&g, 0, sizeof(g));
    for (int64_t i = 0; i < n; ++i) {
        int tp[ORC_MAX_S];
        for (int s = 0; s < ORC_MAX_S; ++s) tp[s] = (int)((c[i].tp_code >> (2 * s)) & 3);
        if (eval_record(t, &g, c[i].map_rank, c[i].type_code, tp, c[i].S, c[i].M, c[i].V,
                        &T[i], &feasible[i])) {
            dag_free(&g);
            return -1;
        }
    }
    dag_free(&g);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Search (Sec. 4.2.3).                                                */
/* ------------------------------------------------------------------ */
typedef struct {
    const orc_problem *p;
    int S, L, M, D, m_idx, tp_idx, d_idx, prune, ridge;
    uint64_t place_rank, ordinal, n_map;
    int32_t cls[ORC_MAX_S], types[ORC_MAX_S], tps[ORC_MAX_S], layers[ORC_MAX_S];
    unsigned char *feas; /* feas[x*(L+1)+c]: layers [c, L) fit stages x..S-1 */
    orc_plan *best;
    orc_stats *st;
    dag g;
    int err;
} search_ctx;

/* The searches' cuts assume non-negative weights: a lower bound from a
 * partial plan (Theorem 1, the per-device serial work) only grows as
 * stages are added, and so does the memory of a stage as it takes more
 * layers.  Tables with a negative cost, transfer or memory entry are
 * rejected by both searches. */
static int tables_nonnegative(const orc_tables *t) {
    const int64_t K = (int64_t)t->n_types * t->n_tp, L = t->L;
    for (int64_t i = 0; i < K * L; ++i)
        if (t->fwd[i] < 0 || t->bwd[i] < 0 || t->dsync[i] < 0 || t->mem_w[i] < 0 ||
            t->mem_a[i] < 0)
            return 0;
    for (int64_t i = 0; i < K * K; ++i)
        if (t->p2p_f[i] < 0 || t->p2p_b[i] < 0) return 0;
    return 1;
}

/* a strictly better than the incumbent: smaller T/(D*M), then smaller index */
static int better(int64_t T, int D, int M, uint64_t idx, const orc_plan *b) {
    if (!b->found) return 1;
    int64_t lhs = T * (int64_t)b->D * b->M, rhs = (int64_t)b->T * D * M;
    if (lhs != rhs) return lhs < rhs;
    return idx < b->global_index;
}

static void consider_leaf(search_ctx *cx) {
    stage_w sw;
    stage_weights(&cx->p->tab, cx->S, cx->cls, cx->layers, &sw);
    int64_t T64;
    if (build_and_solve(&cx->g, cx->p->tab.schedule, cx->S, cx->M, &sw, NULL, &T64)) {
        cx->err = 1;
        return;
    }
    uint64_t map_rank = orc_rank(cx->L, cx->S, cx->layers);
    uint64_t idx = cx->ordinal * cx->n_map + map_rank;
    if (better(T64, cx->D, cx->M, idx, cx->best)) {
        orc_plan *b = cx->best;
        b->found = 1;
        b->m_idx = cx->m_idx;
        b->tp_idx = cx->tp_idx;
        b->d_idx = cx->d_idx;
        b->M = cx->M;
        b->D = cx->D;
        b->T = (int32_t)T64;
        b->place_rank = cx->place_rank;
        b->map_rank = map_rank;
        b->global_index = idx;
        for (int s = 0; s < ORC_MAX_S; ++s) {
            b->types[s] = s < cx->S ? cx->types[s] : -1;
            b->tps[s] = s < cx->S ? cx->tps[s] : -1;
            b->layers[s] = s < cx->S ? cx->layers[s] : 0;
        }
    }
}

/* Layer-level pruning (Theorem 2): among the stages 0..x (0-based) placed so
 * far, the layer counts of the stages of each device type, in stage order,
 * must never rise again after they have fallen (a ridge: non-decreasing,
 * then non-increasing).  A prefix that breaks this has no ridge completion. */
static int ridge_ok(const int32_t *types, const int32_t *layers, int n) {
    for (int a = 0; a < n; ++a) {
        int fallen = 0, prev = -1;
        for (int s = 0; s < n; ++s) {
            if (types[s] != types[a]) continue;
            if (prev >= 0 && layers[s] < prev) fallen = 1;
            if (prev >= 0 && layers[s] > prev && fallen) return 0;
            prev = layers[s];
        }
    }
    return 1;
}

/* Prefix S_x (stages 0..x-1 placed, 1-based x) is cut when its lower bound
 * exceeds the incumbent: g(S_x)/(D M) > T_inc/(D_inc M_inc), i.e. it is strictly worse. */
static int pruned_by_bound(search_ctx *cx, int x) {
    if (!cx->prune || !cx->best->found) return 0;
    stage_w sw;
    stage_weights(&cx->p->tab, x, cx->cls, cx->layers, &sw);
    int64_t g = lower_bound_w(&sw, cx->M, x);
    const orc_plan *b = cx->best;
    return g * (int64_t)b->D * b->M > (int64_t)b->T * cx->D * cx->M;
}

static void dfs(search_ctx *cx, int x, int used) {
    if (cx->err) return;
    int S = cx->S, L = cx->L;
    int lo = 1, hi = L - used - (S - x - 1);
    if (x == S - 1) lo = hi; /* the last stage takes the remaining layers */
    for (int l = lo; l <= hi; ++l) {
        cx->layers[x] = l;
        if (!stage_memory_ok(&cx->p->tab, S, cx->M, x, cx->cls[x], used, l) ||
            !cx->feas[(x + 1) * (L + 1) + used + l]) {
            cx->st->prefixes_memory++;
            continue;
        }
        if (cx->ridge && !ridge_ok(cx->types, cx->layers, x + 1)) {
            cx->st->prefixes_ridge++;
            continue;
        }
        /* the stage-x bound uses only stages 0..x, which are all fixed now */
        if (pruned_by_bound(cx, x + 1)) {
            cx->st->prefixes_pruned++;
            continue;
        }
        if (x == S - 1) {
            cx->st->leaves_evaluated++;
            consider_leaf(cx);
        } else {
            dfs(cx, x + 1, used + l);
        }
    }
}

/* feas[x][c] = the layers [c, L) can be split over stages x..S-1 within memory */
static void suffix_feasibility(search_ctx *cx) {
    int S = cx->S, L = cx->L;
    for (int x = 0; x <= S; ++x)
        for (int c = 0; c <= L; ++c) cx->feas[x * (L + 1) + c] = 0;
    cx->feas[S * (L + 1) + L] = 1;
    for (int x = S - 1; x >= 0; --x)
        for (int c = 0; c < L; ++c)
            for (int l = 1; c + l <= L; ++l)
                if (cx->feas[(x + 1) * (L + 1) + c + l] &&
                    stage_memory_ok(&cx->p->tab, S, cx->M, x, cx->cls[x], c, l)) {
                    cx->feas[x * (L + 1) + c] = 1;
                    break;
                }
}

/* ------------------------------------------------------------------ */
/* Slices of the search space in global-index order (Sec. 4.2.3): the  */
/* M value, then the TP index (placements 0, 1) or the data-parallel   */
/* degree (placement 2), then the allowed stage sequences in           */
/* lexicographic order.                                                */
/* ------------------------------------------------------------------ */
typedef struct {
    int m_idx, grp;          /* grp: TP index (placements 0, 1), D index (placement 2) */
    int M, D;
    uint64_t place_rank;     /* rank among the allowed sequences of this grp */
    uint64_t ordinal;        /* global index = ordinal * n_map + map_rank */
    int32_t cls[ORC_MAX_S], types[ORC_MAX_S], tps[ORC_MAX_S];
} orc_slice;

/* Is the sequence seq[0..S-1] allowed?  Placements 0 and 1: seq holds
 * device types (1: exactly type_counts[t] stages of type t).  Placement 2:
 * seq holds classes k = type * n_tp + tp_idx, and the stages of each type
 * use D * tp_list[tp_idx] devices each, type_counts[type] in total. */
static int sequence_allowed(const orc_problem *p, const int32_t *seq, int S, int D) {
    int T = p->tab.n_types, n_tp = p->tab.n_tp;
    if (p->placement == 0) return 1;
    for (int ty = 0; ty < T; ++ty) {
        int64_t cnt = 0;
        for (int s = 0; s < S; ++s) {
            if (p->placement == 1) cnt += seq[s] == ty;
            else if (seq[s] / n_tp == ty) cnt += (int64_t)D * p->tp_list[seq[s] % n_tp];
        }
        if (cnt != p->type_counts[ty]) return 0;
    }
    return 1;
}

/* Every slice of p for S stages (devices), in order; NULL on failure. */
static orc_slice *list_slices(const orc_problem *p, int S, uint64_t *count) {
    const int n_tp = p->tab.n_tp, per_stage = p->placement == 2;
    const int alpha = per_stage ? p->tab.n_types * n_tp : p->tab.n_types;
    const int n_grp = per_stage ? p->n_D : n_tp;
    /* allowed sequences per group (one list shared by every TP index when
       the rule does not depend on it), each in lexicographic order */
    int32_t **seqs = calloc((size_t)n_grp, sizeof(int32_t *));
    uint64_t *n_seq = calloc((size_t)n_grp, sizeof(uint64_t));
    orc_slice *out = NULL;
    *count = 0;
    if (!seqs || !n_seq) goto done;
    for (int g = 0; g < n_grp; ++g) {
        if (!per_stage && g > 0) break;
        const int D = per_stage ? p->D_list[g] : 1;
        uint64_t cap = 0;
        int32_t seq[ORC_MAX_S];
        for (int s = 0; s < S; ++s) seq[s] = 0;
        for (;;) {  /* odometer over alpha^S, last stage fastest */
            if (sequence_allowed(p, seq, S, D)) {
                if (n_seq[g] == cap) {
                    cap = cap ? 2 * cap : 64;
                    int32_t *grown = realloc(seqs[g], sizeof(int32_t) * S * cap);
                    if (!grown) goto done;
                    seqs[g] = grown;
                }
                memcpy(seqs[g] + n_seq[g] * S, seq, sizeof(int32_t) * S);
                n_seq[g]++;
            }
            int s = S - 1;
            while (s >= 0 && seq[s] == alpha - 1) seq[s--] = 0;
            if (s < 0) break;
            seq[s]++;
        }
    }
    uint64_t per_m = 0;
    for (int g = 0; g < n_grp; ++g) per_m += n_seq[per_stage ? g : 0];
    out = malloc(sizeof(orc_slice) * (per_m * p->n_M > 0 ? per_m * p->n_M : 1));
    if (!out) goto done;
    uint64_t o = 0;
    for (int mi = 0; mi < p->n_M; ++mi)
        for (int g = 0; g < n_grp; ++g) {
            const int q = per_stage ? g : 0;
            for (uint64_t pr = 0; pr < n_seq[q]; ++pr, ++o) {
                orc_slice *sl = &out[o];
                const int32_t *seq = seqs[q] + pr * S;
                sl->m_idx = mi;
                sl->grp = g;
                sl->M = p->M_list[mi];
                sl->D = per_stage ? p->D_list[g] : p->dp_list[g];
                sl->place_rank = pr;
                sl->ordinal = o;
                for (int s = 0; s < ORC_MAX_S; ++s) {
                    const int k = s < S ? (per_stage ? seq[s] : seq[s] * n_tp + g) : 0;
                    sl->cls[s] = k;
                    sl->types[s] = k / n_tp;
                    sl->tps[s] = k % n_tp;
                }
            }
        }
    *count = o;
done:
    if (seqs)
        for (int g = 0; g < n_grp; ++g) free(seqs[g]);
    free(seqs);
    free(n_seq);
    return out;
}

/* Checks shared by both searches on the slice-space fields of p. */
static int slice_space_valid(const orc_problem *p) {
    if (p->placement < 0 || p->placement > 2) return 0;
    if (p->placement >= 1 && !p->type_counts) return 0;
    if (p->placement == 2) {
        if (p->ridge || !p->tp_list || !p->D_list || p->n_D < 1) return 0;
        for (int i = 0; i < p->tab.n_tp; ++i)
            if (p->tp_list[i] < 1) return 0;
        for (int i = 0; i < p->n_D; ++i)
            if (p->D_list[i] < 1) return 0;
        for (int ty = 0; ty < p->tab.n_types; ++ty)
            if (p->type_counts[ty] < 0) return 0;
    } else {
        if (!p->dp_list) return 0;
        for (int i = 0; i < p->tab.n_tp; ++i)
            if (p->dp_list[i] < 1) return 0;
    }
    return 1;
}

/* splitmix64 (Steele, Lea & Flood, OOPSLA 2014) for warm-up sampling */
static uint64_t splitmix64(uint64_t *state) {
    uint64_t z = (*state += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static void set_slice(search_ctx *cx, const orc_slice *sl) {
    cx->m_idx = sl->m_idx;
    cx->tp_idx = cx->p->placement == 2 ? -1 : sl->grp;
    cx->d_idx = cx->p->placement == 2 ? sl->grp : -1;
    cx->M = sl->M;
    cx->D = sl->D;
    cx->place_rank = sl->place_rank;
    cx->ordinal = sl->ordinal;
    for (int s = 0; s < cx->S; ++s) {
        cx->types[s] = sl->types[s];
        cx->tps[s] = sl->tps[s];
        cx->cls[s] = sl->cls[s];
    }
    suffix_feasibility(cx);
}

int orc_search(const orc_problem *p, int prune, int warmup, uint64_t seed, orc_plan *plan,
               orc_stats *stats) {
    return orc_search_part(p, prune, warmup, seed, 0, 1, plan, stats);
}

int orc_search_part(const orc_problem *p, int prune, int warmup, uint64_t seed, int part,
                    int n_parts, orc_plan *plan, orc_stats *stats) {
    int S = p->S, L = p->tab.L;
    if (n_parts < 1 || part < 0 || part >= n_parts) return -1;
    if (S < 1 || S > ORC_MAX_S || S > L || L > 127 || p->n_M < 1 || p->tab.n_types < 1 ||
        p->tab.n_types > 4 || p->tab.n_tp < 1 || !tables_nonnegative(&p->tab) ||
        !slice_space_valid(p))
        return -1;
    for (int i = 0; i < p->n_M; ++i)
        if (p->M_list[i] < 1 || p->M_list[i] > 255) return -1;
    for (int i = 0; i < p->n_M; ++i)
        if (overflow_bound(&p->tab, S, p->M_list[i]) >= ((int64_t)1 << 31)) return -2;

    memset(plan, 0, sizeof(*plan));
    memset(stats, 0, sizeof(*stats));
    search_ctx cx;
    memset(&cx, 0, sizeof(cx));
    cx.p = p;
    cx.S = S;
    cx.L = L;
    cx.prune = prune;
    cx.ridge = p->ridge;
    cx.best = plan;
    cx.st = stats;
    cx.n_map = n_comp(L, S);
    cx.feas = malloc((size_t)(S + 1) * (L + 1));
    uint64_t n_slices = 0;
    orc_slice *slices = list_slices(p, S, &n_slices);
    if (!cx.feas || !slices) {
        free(cx.feas);
        free(slices);
        return -1;
    }

    /* warm-up: random feasible configurations seed T_min (Sec. 4.2.3) */
    if (warmup > 0 && n_slices > 0) {
        uint64_t rs = seed;
        for (int w = 0; w < warmup; ++w) {
            uint64_t pick = splitmix64(&rs) % n_slices;
            if (n_parts > 1) {  /* a slice of this part */
                uint64_t in_part = (uint64_t)part < n_slices
                                       ? (n_slices - (uint64_t)part + n_parts - 1) / n_parts : 0;
                if (in_part == 0) break;
                pick = (pick % in_part) * n_parts + part;
            }
            set_slice(&cx, &slices[pick]);
            if (!cx.feas[0]) continue;
            int used = 0;
            for (int x = 0; x < S; ++x) {
                int opts[128], n = 0;
                int hi = L - used - (S - x - 1), lo = x == S - 1 ? hi : 1;
                for (int l = lo; l <= hi; ++l)
                    if (stage_memory_ok(&p->tab, S, cx.M, x, cx.cls[x], used, l) &&
                        cx.feas[(x + 1) * (L + 1) + used + l])
                        opts[n++] = l;
                cx.layers[x] = opts[splitmix64(&rs) % (uint64_t)n];
                used += cx.layers[x];
            }
            stats->warmup_evaluated++;
            /* with layer-level pruning only ridge-like plans can be the result */
            if (!cx.ridge || ridge_ok(cx.types, cx.layers, cx.S)) consider_leaf(&cx);
        }
    }

    /* exhaustive enumeration in global-index order with the two cuts */
    for (uint64_t i = (uint64_t)part; i < n_slices && !cx.err; i += (uint64_t)n_parts) {
        set_slice(&cx, &slices[i]);
        if (!cx.feas[0]) continue;
        dfs(&cx, 0, 0);
    }
    free(slices);
    free(cx.feas);
    dag_free(&cx.g);
    return cx.err ? -1 : 0;
}

/* ------------------------------------------------------------------ */
/* Search over Interleaved 1F1B plans (Sec. 4.1.4 model, Sec. 4.2.3    */
/* search order).                                                      */
/* ------------------------------------------------------------------ */
/* Slices (M, TP index, placement of types over the N = p->S devices) in
 * the order of orc_search; per slice, every composition of the L layers
 * into the J = N*V virtual stages in lexicographic order, evaluated by
 * orc_eval_interleaved.  M values that are not multiples of N are skipped.
 * Cuts (both only remove plans that cannot be feasible or better):
 *   memory: the weights of a device's chunks placed so far already exceed
 *     its capacity (activations only add to them);
 *   bound (prune != 0): for a device d, the chain of its 2VM ops runs one
 *     op at a time and R_d follows its last op, so
 *       T >= M * sum over its chunks of (F + B) + its all-reduce time;
 *     summed over the chunks placed so far this is a lower bound of every
 *     completion; a prefix whose largest such bound is worse than the
 *     incumbent (objective T/(D*M), strictly) is cut. */
typedef struct {
    const orc_problem *p;
    int N, V, J, L, M, D, m_idx, tp_idx, d_idx, prune;
    uint64_t place_rank, ordinal, n_map;
    int32_t cls[ORC_MAX_S], types[ORC_MAX_S], tps[ORC_MAX_S], layers[ORC_MAX_S];
    int64_t wsum[ORC_MAX_S], work[ORC_MAX_S];
    orc_plan *best;
    orc_stats *st;
    int err;
} il_ctx;

static void il_leaf(il_ctx *cx) {
    int32_t T, F;
    if (orc_eval_interleaved(&cx->p->tab, cx->N, cx->V, cx->M, cx->cls, cx->layers, &T, &F,
                             NULL)) {
        cx->err = 1;
        return;
    }
    cx->st->leaves_evaluated++;
    if (!F) return;
    const uint64_t map_rank = orc_rank(cx->L, cx->J, cx->layers);
    const uint64_t idx = cx->ordinal * cx->n_map + map_rank;
    if (!better(T, cx->D, cx->M, idx, cx->best)) return;
    orc_plan *b = cx->best;
    b->found = 1;
    b->m_idx = cx->m_idx;
    b->tp_idx = cx->tp_idx;
    b->d_idx = cx->d_idx;
    b->M = cx->M;
    b->D = cx->D;
    b->T = T;
    b->place_rank = cx->place_rank;
    b->map_rank = map_rank;
    b->global_index = idx;
    for (int s = 0; s < ORC_MAX_S; ++s) {
        b->types[s] = s < cx->N ? cx->types[s] : 0;
        b->tps[s] = s < cx->N ? cx->tps[s] : -1;
        b->layers[s] = s < cx->J ? cx->layers[s] : 0;
    }
}

static void il_dfs(il_ctx *cx, int j, int used) {
    const orc_tables *t = &cx->p->tab;
    const int L = cx->L, d = j % cx->N, k = cx->cls[d];
    const int hi = L - used - (cx->J - j - 1), lo = j == cx->J - 1 ? hi : 1;
    int64_t w = 0, work = 0;
    for (int l = 1; l <= hi && !cx->err; ++l) {
        const int at = used + l - 1;  /* the layer this step adds */
        w += t->mem_w[(int64_t)k * L + at];
        work += (int64_t)cx->M * (t->fwd[(int64_t)k * L + at] + t->bwd[(int64_t)k * L + at]) +
                t->dsync[(int64_t)k * L + at];
        if (l < lo) continue;
        if (cx->wsum[d] + w > t->cap[k]) {  /* more layers only add weights */
            cx->st->prefixes_memory++;
            break;
        }
        cx->wsum[d] += w;
        cx->work[d] += work;
        cx->layers[j] = l;
        int cut = 0;
        if (cx->prune && cx->best->found) {
            int64_t lb = 0;
            for (int e = 0; e < cx->N; ++e)
                if (cx->work[e] > lb) lb = cx->work[e];
            /* lb / (D M) > T_min / (D_min M_min) */
            cut = lb * (int64_t)cx->best->D * cx->best->M >
                  (int64_t)cx->best->T * cx->D * cx->M;
        }
        if (cut) {
            cx->st->prefixes_pruned++;
        } else if (j == cx->J - 1) {
            il_leaf(cx);
        } else {
            il_dfs(cx, j + 1, used + l);
        }
        cx->wsum[d] -= w;
        cx->work[d] -= work;
        if (cut) break;  /* the bound only grows with the stage's layers */
    }
}

int orc_search_interleaved(const orc_problem *p, int V, int prune, orc_plan *plan,
                           orc_stats *stats) {
    const int N = p->S, L = p->tab.L, J = N * V;
    if (N < 1 || V < 2 || J > ORC_MAX_S || J > L || L > 127 || p->n_M < 1 ||
        p->tab.n_types < 1 || p->tab.n_types > 4 || p->tab.n_tp < 1 ||
        !tables_nonnegative(&p->tab) || !slice_space_valid(p) || p->ridge)
        return -1;
    for (int i = 0; i < p->n_M; ++i)
        if (p->M_list[i] < 1 || p->M_list[i] > 255) return -1;
    for (int i = 0; i < p->n_M; ++i)
        if (p->M_list[i] % N == 0 && overflow_bound(&p->tab, J, p->M_list[i]) >= ((int64_t)1 << 31))
            return -2;
    memset(plan, 0, sizeof(*plan));
    memset(stats, 0, sizeof(*stats));
    il_ctx cx;
    memset(&cx, 0, sizeof(cx));
    cx.p = p;
    cx.N = N;
    cx.V = V;
    cx.J = J;
    cx.L = L;
    cx.prune = prune;
    cx.best = plan;
    cx.st = stats;
    cx.n_map = n_comp(L, J);
    uint64_t n_slices = 0;
    orc_slice *slices = list_slices(p, N, &n_slices);
    if (!slices) return -1;
    for (uint64_t i = 0; i < n_slices && !cx.err; ++i) {
        const orc_slice *sl = &slices[i];
        if (sl->M % N != 0) continue;  /* no interleaved schedule; its indices still count */
        cx.m_idx = sl->m_idx;
        cx.tp_idx = p->placement == 2 ? -1 : sl->grp;
        cx.d_idx = p->placement == 2 ? sl->grp : -1;
        cx.M = sl->M;
        cx.D = sl->D;
        cx.place_rank = sl->place_rank;
        cx.ordinal = sl->ordinal;
        for (int s = 0; s < N; ++s) {
            cx.types[s] = sl->types[s];
            cx.tps[s] = sl->tps[s];
            cx.cls[s] = sl->cls[s];
            cx.wsum[s] = 0;
            cx.work[s] = 0;
        }
        il_dfs(&cx, 0, 0);
    }
    free(slices);
    return cx.err ? -1 : 0;
}
