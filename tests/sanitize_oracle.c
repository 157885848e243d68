/*
 * Drives every entry point of the CPU oracle (oracle/oracle.c) on seeded
 * random small problems, for a build with AddressSanitizer and
 * UndefinedBehaviorSanitizer (tests/test_sanitizers.py compiles and runs
 * it).  It checks memory safety and the absence of undefined behaviour, not
 * results: the other oracle tests pin those.  Exit status 0 = clean run.
 */
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "../oracle/oracle.h"

static uint64_t rng_state = 0x9e3779b97f4a7c15ull;

/* xorshift64* (Vigna 2016): inputs only */
static uint64_t next_u64(void) {
    rng_state ^= rng_state >> 12;
    rng_state ^= rng_state << 25;
    rng_state ^= rng_state >> 27;
    return rng_state * 0x2545f4914f6cdd1dull;
}

static int uniform(int lo, int hi) { return lo + (int)(next_u64() % (uint64_t)(hi - lo + 1)); }

typedef struct {
    int32_t fwd[8 * 16], bwd[8 * 16], dsync[8 * 16], p2p_f[64], p2p_b[64];
    int64_t mem_w[8 * 16], mem_a[8 * 16], cap[8];
} store;

static void fill(store *s, orc_tables *t, int L, int n_types, int n_tp, int sched) {
    const int K = n_types * n_tp;
    for (int i = 0; i < K * L; ++i) {
        s->fwd[i] = uniform(1, 60);
        s->bwd[i] = uniform(1, 90);
        s->dsync[i] = uniform(0, 30);
        s->mem_w[i] = uniform(0, 5);
        s->mem_a[i] = uniform(0, 3);
    }
    for (int i = 0; i < K * K; ++i) {
        s->p2p_f[i] = uniform(0, 20);
        s->p2p_b[i] = uniform(0, 20);
    }
    for (int k = 0; k < K; ++k) s->cap[k] = uniform(10, 80);
    t->L = L;
    t->n_types = n_types;
    t->n_tp = n_tp;
    t->fwd = s->fwd;
    t->bwd = s->bwd;
    t->dsync = s->dsync;
    t->p2p_f = s->p2p_f;
    t->p2p_b = s->p2p_b;
    t->mem_w = s->mem_w;
    t->mem_a = s->mem_a;
    t->cap = s->cap;
    t->schedule = sched;
}

int main(void) {
    store st;
    orc_tables t;
    for (int iter = 0; iter < 60; ++iter) {
        const int sched = iter % 3;
        const int n_types = uniform(1, 2), n_tp = uniform(1, 2), L = uniform(4, 10);
        fill(&st, &t, L, n_types, n_tp, sched == 2 ? 2 : sched);
        const int K = n_types * n_tp;
        int32_t cls[ORC_MAX_S], layers[ORC_MAX_S], T = 0, F = 0;
        /* single evaluations, finish times, bounds */
        const int S = uniform(1, L < 4 ? L : 4), M = uniform(1, 6);
        for (int s = 0; s < S; ++s) cls[s] = uniform(0, K - 1);
        if (orc_unrank(L, S, next_u64() % orc_binom(L - 1, S - 1), layers)) return 2;
        t.schedule = sched == 2 ? 0 : sched;
        orc_dag_counts dc;
        if (orc_eval(&t, S, M, cls, layers, &T, &F, &dc)) return 3;
        int32_t *fin = malloc(sizeof(int32_t) * 2 * S * M);
        if (!fin || orc_eval_finish(&t, S, M, cls, layers, fin)) return 4;
        free(fin);
        for (int x = 1; x <= S; ++x) {
            if (orc_lower_bound(&t, S, M, cls, layers, x) < 0) return 5;
            (void)orc_lower_bound_tight(&t, S, M, cls, layers, x);
        }
        (void)orc_rank(L, S, layers);
        /* interleaved evaluations */
        const int N = uniform(1, 2), V = uniform(2, 3);
        if (N * V <= L) {
            t.schedule = 2;
            const int Mi = N * uniform(1, 3);
            for (int d = 0; d < N; ++d) cls[d] = uniform(0, K - 1);
            if (orc_unrank(L, N * V, next_u64() % orc_binom(L - 1, N * V - 1), layers)) return 6;
            if (orc_eval_interleaved(&t, N, V, Mi, cls, layers, &T, &F, &dc)) return 7;
            int32_t *fi = malloc(sizeof(int32_t) * 2 * N * V * Mi);
            int64_t peak[ORC_MAX_S];
            if (!fi || orc_eval_interleaved_detail(&t, N, V, Mi, cls, layers, &T, &F, fi, peak))
                return 8;
            free(fi);
        }
        /* batches, with invalid records mixed in */
        t.schedule = sched;
        orc_candidate c[16];
        orc_candidate_ex cx[16];
        int32_t Tb[16];
        uint8_t Fb[16];
        for (int i = 0; i < 16; ++i) {
            const int Si = uniform(1, L < 17 ? L : 16);
            memset(&c[i], 0, sizeof(c[i]));
            memset(&cx[i], 0, sizeof(cx[i]));
            c[i].S = cx[i].S = (uint8_t)(i == 3 ? 0 : Si);
            c[i].M = cx[i].M = (uint8_t)uniform(0, 8);
            c[i].map_rank = cx[i].map_rank = next_u64() % (orc_binom(L - 1, Si - 1) + 1);
            c[i].type_code = cx[i].type_code = (uint32_t)next_u64();
            c[i].tp_idx = (uint8_t)uniform(0, n_tp);
            c[i].pad = (uint8_t)(sched == 2 ? uniform(0, 3) : 0);
            cx[i].V = c[i].pad;
            cx[i].tp_code = (uint32_t)next_u64();
        }
        if (orc_eval_batch(&t, c, 16, Tb, Fb)) return 9;
        (void)orc_eval_batch_ex(&t, cx, 16, Tb, Fb);
        /* searches */
        orc_problem p;
        memset(&p, 0, sizeof(p));
        int32_t Ms[2] = {uniform(1, 4), uniform(5, 8)}, dp[2] = {1, uniform(1, 3)};
        int32_t counts[2] = {0, 0};
        p.tab = t;
        p.tab.schedule = sched == 2 ? 0 : sched;
        p.S = uniform(1, L < 4 ? L : 4);
        p.n_M = 2;
        p.M_list = Ms;
        p.dp_list = dp;
        p.placement = 0;
        p.type_counts = counts;
        p.ridge = iter % 2;
        orc_plan plan;
        orc_stats ss;
        if (orc_search(&p, 1, 20, (uint64_t)iter, &plan, &ss) < -1) return 10;
        /* per-stage TP: a (type, TP index) per stage under per-type device counts */
        int32_t tps[4] = {1, 2, 4, 8}, Ds[2] = {1, 2}, devs[2] = {uniform(0, 6), uniform(1, 6)};
        p.placement = 2;
        p.ridge = 0;
        p.tp_list = tps;
        p.n_D = 2;
        p.D_list = Ds;
        p.type_counts = devs;
        if (orc_search(&p, 1, 20, (uint64_t)iter, &plan, &ss) < -1) return 12;
        p.placement = 0;
        p.type_counts = counts;
        p.S = N;
        p.ridge = 0;
        p.tab.schedule = 2;
        Ms[0] = N;
        Ms[1] = 2 * N;
        if (N * V <= L && orc_search_interleaved(&p, V, 1, &plan, &ss) < -1) return 11;
    }
    printf("sanitized oracle run: ok\n");
    return 0;
}
