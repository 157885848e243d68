"""Pins for the oracle's Eager-1F1B schedule (App. B): stage i of N runs a
warm-up of 2(N-i)+1 forwards, steady backward-forward groups and a
cool-down of backwards; it holds up to 2(N-i)+1 micro-batches of
activations.  Checked against the independent event-driven simulator, the
paper's critical-path characterisation K(x, y, w), closed forms, the memory
rule and brute-force search."""
import itertools
import random
from fractions import Fraction

import numpy as np

import gen
from tests._event_sim import simulate, stage_program
from tests.test_oracle import _brute_force_plan, _random_problem, rand_stages, stage_tables

EAGER = 1


def test_event_simulator_program_is_eager():
    # N = 4, stage 1: 2(N-1)+1 = 7 warm-up forwards (capped at M = 9), then
    # B-F groups, then backwards; the last stage alternates from the start
    assert stage_program(4, 9, 0, eager=True) == (
        [("F", m) for m in range(7)] + [("B", 0), ("F", 7), ("B", 1), ("F", 8)] +
        [("B", m) for m in range(2, 9)])
    assert stage_program(4, 9, 3, eager=True)[:4] == [("F", 0), ("B", 0), ("F", 1), ("B", 1)]
    assert stage_program(4, 9, 1, eager=True)[:6] == [("F", m) for m in range(5)] + [("B", 0)]


def test_eager_matches_event_simulator(orc):
    rng = random.Random(41)
    for _ in range(600):
        S, M = rng.randint(1, 6), rng.randint(1, 13)
        F, B, d, pf, pb = rand_stages(rng, S)
        tab, cls, lay = stage_tables(orc, F, B, d, pf, pb, schedule=EAGER)
        T_sim, fF_sim, fB_sim = simulate(S, M, F, B, pf, pb, d, eager=True)
        fF, fB = orc.finish_times(tab, S, M, cls, lay)
        assert fF.tolist() == fF_sim and fB.tolist() == fB_sim, (S, M)
        assert orc.evaluate(tab, S, M, cls, lay)[0] == T_sim


def _K(N, M, F, B, t_down, t_up, x, y, w):
    """Cost of the path K(x, y, w) of App. B (1-based stages): the
    downward and upward steps through stages 1..x, 2(N-x) forwards and
    2(N-y) backwards of stage w, and M - 2(N-y) - 1 forward-backward pairs of
    stage y.  t_down[i] / t_up[i]: transfers between stages i+1 and i+2."""
    c = sum(F[i] + B[i] + t_down[i] + t_up[i] for i in range(x - 1)) + F[x - 1] + B[x - 1]
    c += 2 * (N - x) * F[w - 1] + 2 * (N - y) * B[w - 1]
    c += (M - 2 * (N - y) - 1) * (F[y - 1] + B[y - 1])
    return c


def test_eager_critical_path_is_K_under_assumptions(orc):
    """Under Assumptions 1-4 (B_i = r F_i, transfers at most (r-1)/2 F_k,
    M >= 2N, F_min >= max(2/3, r/(1+r)) F_max) a critical path has the form
    K(x, y, w); with no all-reduce time the makespan is the largest
    C(K(x, y, w)) over 1 <= w <= y <= x <= N."""
    rng = random.Random(42)
    n = 0
    for _ in range(400):
        N = rng.randint(1, 6)
        M = rng.randint(2 * N, 2 * N + 9)
        r = rng.choice([Fraction(3, 2), Fraction(2), Fraction(5, 2), Fraction(3)])
        alpha = max(Fraction(2, 3), r / (1 + r))
        Fmax = 2 * rng.randint(60, 500)
        F = [2 * rng.randint(int(alpha * Fmax / 2) + 1, Fmax // 2) for _ in range(N)]
        B = [int(r * f) for f in F]
        assert all(b == r * f for b, f in zip(B, F))
        tmax = int((r - 1) / 2 * min(F))
        pf = [rng.randint(0, tmax) for _ in range(N - 1)]
        pb = [rng.randint(0, tmax) for _ in range(N - 1)]
        tab, cls, lay = stage_tables(orc, F, B, [0] * N, pf, pb, schedule=EAGER)
        T = orc.evaluate(tab, N, M, cls, lay)[0]
        best = max(_K(N, M, F, B, pf, pb, x, y, w)
                   for x in range(1, N + 1) for y in range(1, x + 1) for w in range(1, y + 1))
        assert T == best, (N, M, F, B, pf, pb)
        n += 1
    assert n == 400


def test_eager_K_paths_never_exceed_the_makespan(orc):
    """Without the assumptions every K(x, y, w) is still a path of the DAG
    (for M >= 2(N-y)+1), so its cost is at most the makespan."""
    rng = random.Random(43)
    for _ in range(300):
        N, M = rng.randint(1, 6), rng.randint(1, 16)
        F, B, _, pf, pb = rand_stages(rng, N)
        tab, cls, lay = stage_tables(orc, F, B, [0] * N, pf, pb, schedule=EAGER)
        T = orc.evaluate(tab, N, M, cls, lay)[0]
        for x, y, w in itertools.product(range(1, N + 1), repeat=3):
            if w <= y <= x and M >= 2 * (N - y) + 1:
                assert _K(N, M, F, B, pf, pb, x, y, w) <= T


def test_eager_closed_forms(orc):
    rng = random.Random(44)
    for _ in range(100):
        S = rng.randint(1, 8)
        F, B, d, pf, pb = rand_stages(rng, S)
        tab1, cls, lay = stage_tables(orc, F, B, d, pf, pb)
        tabE, _, _ = stage_tables(orc, F, B, d, pf, pb, schedule=EAGER)
        # M = 1: one micro-batch, every warm-up is capped at 1: the same chain
        assert orc.evaluate(tabE, S, 1, cls, lay)[0] == orc.evaluate(tab1, S, 1, cls, lay)[0]
        # a single stage: M (F + B) + d whatever the schedule
        tabS, c1, l1 = stage_tables(orc, F[:1], B[:1], d[:1], [], [], schedule=EAGER)
        M = rng.randint(1, 20)
        assert orc.evaluate(tabS, 1, M, c1, l1)[0] == M * (F[0] + B[0]) + d[0]


def test_eager_uniform_pipeline(orc):
    """Identical stages and no transfers: the pipeline is limited by the
    first forward wave and the last backward wave, (M + N - 1)(F + B) for
    M >= 2N - 1 (the extra warm-up forwards only fill bubbles)."""
    for N in range(1, 7):
        for M in range(2 * N - 1, 2 * N + 6):
            for f, b in ((3, 5), (7, 2), (4, 4)):
                tab, cls, lay = stage_tables(orc, [f] * N, [b] * N, [0] * N, [0] * (N - 1),
                                             [0] * (N - 1), schedule=EAGER)
                assert orc.evaluate(tab, N, M, cls, lay)[0] == (M + N - 1) * (f + b), (N, M)


def test_eager_memory_holds_more_micro_batches(orc):
    """Stage 1 of N holds 2N-1 micro-batches under Eager 1F1B, N under 1F1B."""
    N, M = 4, 12
    a = 1000
    for held, fits_1f1b, fits_eager in ((N, True, False), (2 * N - 1, True, True)):
        cap = np.full(N, held * a, np.int64)
        tabs = []
        for sched in (0, EAGER):
            t = orc.OracleTables(L=N, n_types=N, n_tp=1, fwd=np.eye(N, dtype=np.int32) * 5,
                                 bwd=np.eye(N, dtype=np.int32) * 9, dsync=np.zeros((N, N)),
                                 p2p_f=np.zeros((N, N)), p2p_b=np.zeros((N, N)),
                                 mem_w=np.zeros((N, N)), mem_a=np.eye(N, dtype=np.int64) * a,
                                 cap=cap, schedule=sched)
            tabs.append(orc.evaluate(t, N, M, list(range(N)), [1] * N)[1])
        assert tabs == [fits_1f1b, fits_eager]


def test_eager_search_equals_brute_force(orc):
    """Eq. 2 bounds every schedule whose stage chains start with F_{s,1} and
    end with B_{s,M}, so the pruned Eager search is exact."""
    rng = random.Random(45)
    n_found = 0
    for seed in range(80):
        w = _random_problem(rng, seed)
        best = _brute_force_plan(orc, w, schedule=EAGER)
        for prune, warm in ((False, 0), (True, 0), (True, 20)):
            plan, _ = orc.search(w, prune=prune, warmup=warm, seed=seed, schedule=EAGER)
            if best is None:
                assert not plan["found"]
                continue
            n_found += 1
            assert plan["global_index"] == best[1], (seed, prune, warm)
            assert Fraction(plan["T"], plan["D"] * plan["M"]) == best[0]
    assert n_found > 80
