"""Pins for the CPU oracle: each test checks it against something other than
itself -- hand-worked finish times, closed forms, an independent event-driven
simulator, brute-force enumeration, structural counts and invariants."""
import itertools
import math
import os
import random
from fractions import Fraction

import numpy as np
import pytest

import gen
from tests._event_sim import simulate, stage_program

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "two_stage_1f1b.txt")


def stage_tables(orc, F, B, d, pf, pb, schedule=0):
    """Tables where stage s holds layer s of its own class s."""
    S = len(F)
    fwd = np.zeros((S, S), np.int32)
    bwd = np.zeros((S, S), np.int32)
    ds = np.zeros((S, S), np.int32)
    p2f = np.zeros((S, S), np.int32)
    p2b = np.zeros((S, S), np.int32)
    for s in range(S):
        fwd[s, s], bwd[s, s], ds[s, s] = F[s], B[s], d[s]
    for s in range(S - 1):
        p2f[s, s + 1] = pf[s]
        p2b[s + 1, s] = pb[s]
    tab = orc.OracleTables(L=S, n_types=S, n_tp=1, fwd=fwd, bwd=bwd, dsync=ds, p2p_f=p2f,
                           p2p_b=p2b, mem_w=np.zeros((S, S)), mem_a=np.zeros((S, S)),
                           cap=np.ones(S), schedule=schedule)
    return tab, list(range(S)), [1] * S


def rand_stages(rng, S, comm=True):
    F = [rng.randint(1, 400) for _ in range(S)]
    B = [rng.randint(1, 800) for _ in range(S)]
    d = [rng.randint(0, 900) for _ in range(S)]
    pf = [rng.randint(0, 150) if comm else 0 for _ in range(S - 1)]
    pb = [rng.randint(0, 150) if comm else 0 for _ in range(S - 1)]
    return F, B, d, pf, pb


def read_golden():
    cases, cur = [], None
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        if line.startswith("case"):
            parts = [p.split() for p in line[4:].split("|")]
            S, M = map(int, parts[0])
            cur = dict(S=S, M=M, F=list(map(int, parts[1])), B=list(map(int, parts[2])),
                       pf=list(map(int, parts[3])), pb=list(map(int, parts[4])),
                       d=list(map(int, parts[5])), T=int(parts[6][0]), fF=[], fB=[])
            cases.append(cur)
        elif line[0] in "FB":
            cur["f" + line[0]].append(list(map(int, line[1:].split())))
    return cases


# -- hand-worked pipelines (Sec. 4.1) ---------------------------------------

@pytest.mark.parametrize("case", read_golden(), ids=lambda c: f"S{c['S']}M{c['M']}")
def test_hand_worked_finish_times(orc, case):
    tab, cls, lay = stage_tables(orc, case["F"], case["B"], case["d"], case["pf"], case["pb"])
    fF, fB = orc.finish_times(tab, case["S"], case["M"], cls, lay)
    assert fF.tolist() == case["fF"]
    assert fB.tolist() == case["fB"]
    T, feas = orc.evaluate(tab, case["S"], case["M"], cls, lay)
    assert T == case["T"]


# -- closed forms -------------------------------------------------------------

def test_single_stage_closed_form(orc):
    """One stage: its 2M ops run back to back, then R_1: T = M(F+B) + d."""
    rng = random.Random(11)
    for _ in range(200):
        M = rng.randint(1, 40)
        F, B, d, _, _ = rand_stages(rng, 1)
        tab, cls, lay = stage_tables(orc, F, B, d, [], [])
        assert orc.evaluate(tab, 1, M, cls, lay)[0] == M * (F[0] + B[0]) + d[0]


def test_uniform_pipeline_closed_form(orc):
    """Identical stages, no communication, no all-reduce: the textbook 1F1B
    makespan (M + N - 1)(F + B), for M >= N and M < N alike."""
    rng = random.Random(12)
    for S in range(1, 7):
        for M in range(1, 11):
            f, b = rng.randint(1, 50), rng.randint(1, 90)
            tab, cls, lay = stage_tables(orc, [f] * S, [b] * S, [0] * S, [0] * (S - 1),
                                         [0] * (S - 1))
            assert orc.evaluate(tab, S, M, cls, lay)[0] == (M + S - 1) * (f + b), (S, M)


def test_single_microbatch_chain(orc):
    """M = 1: the DAG is the chain F_1..F_N, B_N..B_1 with R_s hanging off B_s."""
    rng = random.Random(13)
    for _ in range(200):
        S = rng.randint(1, 10)
        F, B, d, pf, pb = rand_stages(rng, S)
        tab, cls, lay = stage_tables(orc, F, B, d, pf, pb)
        down = sum(F) + sum(pf)
        want = max(down + sum(B[s:]) + sum(pb[s:]) + d[s] for s in range(S))
        assert orc.evaluate(tab, S, 1, cls, lay)[0] == want


# -- independent formulation ---------------------------------------------------

def test_event_simulator_program_is_1f1b():
    # the in-flight rule reproduces the warm-up / steady / cool-down shape
    assert stage_program(4, 6, 0) == [("F", 0), ("F", 1), ("F", 2), ("F", 3), ("B", 0), ("F", 4),
                                      ("B", 1), ("F", 5), ("B", 2), ("B", 3), ("B", 4), ("B", 5)]
    assert stage_program(4, 6, 3)[:4] == [("F", 0), ("B", 0), ("F", 1), ("B", 1)]


def test_matches_event_simulator(orc):
    rng = random.Random(14)
    for _ in range(600):
        S, M = rng.randint(1, 6), rng.randint(1, 9)
        F, B, d, pf, pb = rand_stages(rng, S)
        tab, cls, lay = stage_tables(orc, F, B, d, pf, pb)
        T_sim, fF_sim, fB_sim = simulate(S, M, F, B, pf, pb, d)
        fF, fB = orc.finish_times(tab, S, M, cls, lay)
        assert fF.tolist() == fF_sim and fB.tolist() == fB_sim, (S, M)
        assert orc.evaluate(tab, S, M, cls, lay)[0] == T_sim


# -- structure (Sec. 4.1.1, 4.1.2) ----------------------------------------------

@pytest.mark.parametrize("S,M", [(1, 1), (1, 5), (2, 4), (4, 2), (8, 32), (16, 8)])
def test_node_and_edge_counts(orc, S, M):
    rng = random.Random(S * 100 + M)
    tab, cls, lay = stage_tables(orc, *rand_stages(rng, S))
    _, _, c = orc.evaluate(tab, S, M, cls, lay, counts=True)
    D = 1  # one pipeline is modelled; all D pipelines are identical
    assert c["compute_nodes"] == 2 * S * M
    assert c["allreduce_nodes"] == S
    assert c["control_nodes"] == 2
    assert c["nodes"] == 2 * S * M + S + 2
    assert c["inter_edges"] == 2 * (S - 1) * M
    assert c["intra_edges"] == S * (2 * M - 1)
    assert c["allreduce_edges"] == S * D
    assert c["aux_edges"] == D + S


# -- invariants ------------------------------------------------------------------

def _random_config(rng, w, S):
    L = w.L
    cuts = sorted(rng.sample(range(1, L), S - 1))
    lay = [b - a for a, b in zip([0] + cuts, cuts + [L])]
    cls = [rng.randrange(w.K) for _ in range(S)]
    return cls, lay


def _stage_totals(w, cls, lay):
    out, first = [], 0
    for k, l in zip(cls, lay):
        out.append((int(w.fwd[k, first:first + l].sum()), int(w.bwd[k, first:first + l].sum()),
                    int(w.dsync[k, first:first + l].sum())))
        first += l
    return out


def test_lower_bound_and_bottleneck(orc):
    """Theorem 1 needs T >= g(S_x) for every prefix; and no stage can finish
    faster than its own serialized work M(F_s + B_s) followed by R_s."""
    rng = random.Random(15)
    for cfg in (2, 4, 5):
        w = gen.get_config(cfg)
        tab = orc.OracleTables.from_workload(w)
        for _ in range(150):
            S, M = rng.randint(1, 12), rng.randint(1, 64)
            cls, lay = _random_config(rng, w, S)
            T, _ = orc.evaluate(tab, S, M, cls, lay)
            for x in range(1, S + 1):
                assert orc.lower_bound(tab, S, M, cls, lay, x) <= T
            for F, B, d in _stage_totals(w, cls, lay):
                assert T >= M * (F + B) + d


def test_lower_bound_value(orc):
    """g(S_x) of Eq. 2 on a hand-sized prefix: stages (F, B, d) =
    (2,5,10), (3,6,0), (4,7,4), M = 2, x = 3:
    sum_{i<3} F_i = 5, M(F_3+B_3) = 22, max(B_1+B_2+d_1, B_2+d_2, d_3) = 21."""
    tab, cls, lay = stage_tables(orc, [2, 3, 4], [5, 6, 7], [10, 0, 4], [1, 2], [3, 1])
    assert orc.lower_bound(tab, 3, 2, cls, lay, 3) == 5 + 22 + 21
    assert orc.lower_bound(tab, 3, 2, cls, lay, 1) == 0 + 2 * 7 + 10


def test_tight_bound_hand_value(orc):
    """Tightened bound on the same three stages, pf = (1, 2), pb = (3, 1),
    M = 2 (one layer per stage, so the completion is unique).  Path lengths
    P(y, i) = sum_{j<y}(F_j+pf_j) + M(F_y+B_y) + sum_{j=i}^{y-1}(B_j+pb_j) + d_i:
    P(1,1) = 24, P(2,1) = 3+18+8+10 = 39, P(2,2) = 21, P(3,1) = 8+22+15+10 = 55,
    P(3,2) = 37, P(3,3) = 34.  Every prefix of this plan is bounded by 55,
    where Eq. 2 gives 24 at x = 1 and 48 at x = 3."""
    tab, cls, lay = stage_tables(orc, [2, 3, 4], [5, 6, 7], [10, 0, 4], [1, 2], [3, 1])
    for x in (1, 2, 3):
        assert orc.lower_bound_tight(tab, 3, 2, cls, lay, x) == 55
    # a large d_3 makes the completion term P(3,3) the largest
    tab, cls, lay = stage_tables(orc, [2, 3, 4], [5, 6, 7], [10, 0, 40], [1, 2], [3, 1])
    assert orc.lower_bound_tight(tab, 3, 2, cls, lay, 1) == 8 + 22 + 40
    assert orc.lower_bound_tight(tab, 3, 2, cls, lay, 3) == 8 + 22 + 40


def test_tight_bound_is_the_makespan_of_a_chain(orc):
    """M = 1: the DAG is a chain, and max_i P(S, i) is exactly its longest
    path (the closed form of test_single_microbatch_chain)."""
    rng = random.Random(31)
    for _ in range(200):
        S = rng.randint(1, 9)
        F, B, d, pf, pb = rand_stages(rng, S)
        tab, cls, lay = stage_tables(orc, F, B, d, pf, pb)
        T, _ = orc.evaluate(tab, S, 1, cls, lay)
        assert orc.lower_bound_tight(tab, S, 1, cls, lay, S) == T


def test_tight_bound_valid_and_tighter(orc):
    """Brute force over every plan of small random problems: for each prefix,
    the tightened bound never exceeds the best makespan among the prefix's
    memory-feasible completions (so pruning with it is exact), is at least
    Eq. 2, and is strictly larger than Eq. 2 for a good share of prefixes."""
    rng = random.Random(32)
    n_pref = n_strict = 0
    for seed in range(60):
        w = _random_problem(rng, seed)
        tab = orc.OracleTables.from_workload(w)
        S, L = w.S, w.L
        for tp in range(w.n_tp):
            for seq in gen.workloads.place_list(w)[:6]:
                cls = [t * w.n_tp + tp for t in seq]
                for M in w.M_list:
                    best = {}  # prefix -> min T over feasible completions
                    for r in range(orc.binom(L - 1, S - 1)):
                        lay = orc.unrank(L, S, r)
                        T, feas = orc.evaluate(tab, S, M, cls, lay)
                        if not feas:
                            continue
                        for x in range(1, S + 1):
                            key = tuple(lay[:x])
                            if key not in best or T < best[key][0]:
                                best[key] = (T, lay)
                    for key, (tmin, lay) in best.items():
                        x = len(key)
                        lb = orc.lower_bound_tight(tab, S, M, cls, lay, x)
                        g = orc.lower_bound(tab, S, M, cls, lay, x)
                        assert lb is not None and g <= lb <= tmin, (seed, key, g, lb, tmin)
                        n_pref += 1
                        n_strict += lb > g
    assert n_pref > 2000 and n_strict > n_pref // 4, (n_pref, n_strict)


def test_tight_bound_without_feasible_completion(orc):
    """A prefix that leaves no memory-feasible completion has no bound."""
    tab, cls, lay = stage_tables(orc, [2, 3], [5, 6], [0, 0], [1], [1])
    # stage 2 holds the only layer of class 1; give it a weight that cannot fit
    tab2 = orc.OracleTables(L=2, n_types=2, n_tp=1, fwd=np.array([[2, 2], [3, 3]]),
                            bwd=np.array([[5, 5], [6, 6]]), dsync=np.zeros((2, 2)),
                            p2p_f=np.zeros((2, 2)), p2p_b=np.zeros((2, 2)),
                            mem_w=np.array([[0, 0], [9, 9]]), mem_a=np.zeros((2, 2)),
                            cap=np.array([1, 1]))
    assert orc.lower_bound_tight(tab2, 2, 1, [0, 1], [1, 1], 1) is None
    assert orc.lower_bound_tight(tab, 2, 1, [0, 1], [1, 1], 1) is not None


def test_monotone_in_weights(orc):
    rng = random.Random(16)
    for _ in range(300):
        S, M = rng.randint(1, 6), rng.randint(1, 9)
        F, B, d, pf, pb = rand_stages(rng, S)
        tab, cls, lay = stage_tables(orc, F, B, d, pf, pb)
        T0 = orc.evaluate(tab, S, M, cls, lay)[0]
        arrs = [F, B, d, pf, pb]
        which = rng.choice([i for i, a in enumerate(arrs) if a])
        arrs[which][rng.randrange(len(arrs[which]))] += rng.randint(1, 100)
        tab2, _, _ = stage_tables(orc, *arrs)
        assert orc.evaluate(tab2, S, M, cls, lay)[0] >= T0
        tab3, _, _ = stage_tables(orc, F, B, d, [0] * (S - 1), [0] * (S - 1))
        assert orc.evaluate(tab3, S, M, cls, lay)[0] <= orc.evaluate(tab2, S, M, cls, lay)[0]


def test_memory_limit_non_decreasing_in_stage(orc):
    """Lemma memlimit (App. B.3): with fewer in-flight micro-batches later in
    the pipeline, the largest layer count a device type can hold never
    shrinks with the stage index.  The oracle's feasibility flag decides
    each case: stage s runs on the class under test and every other stage
    on a memory-free copy of it, so the flag is stage s's own fit."""
    w = gen.config4()
    S, M = 8, 32
    K = w.n_types * w.n_tp
    for k in range(K):
        z64 = np.zeros((1, w.L), np.int64)
        tab = orc.OracleTables(
            L=w.L, n_types=2, n_tp=1,
            fwd=np.vstack([w.fwd[k], w.fwd[k]]), bwd=np.vstack([w.bwd[k], w.bwd[k]]),
            dsync=np.vstack([w.dsync[k], w.dsync[k]]),
            p2p_f=np.zeros((2, 2), np.int32), p2p_b=np.zeros((2, 2), np.int32),
            mem_w=np.vstack([w.mem_w[k:k + 1], z64]), mem_a=np.vstack([w.mem_a[k:k + 1], z64]),
            cap=np.array([w.cap[k], 1], np.int64))
        limits = []
        for s in range(S):
            best = 0
            for l in range(1, w.L - S + 2):
                lay = [1] * S
                lay[s] = l
                lay[(s + 1) % S] = w.L - l - (S - 2)
                cls = [1] * S
                cls[s] = 0
                if orc.evaluate(tab, S, M, cls, lay)[1]:
                    best = l
            limits.append(best)
        assert limits == sorted(limits), (k, limits)
        assert any(limits), k  # some class-k stage fits: the check is not vacuous


# -- combinatorics ---------------------------------------------------------------

@pytest.mark.parametrize("L,S", [(1, 1), (5, 1), (5, 5), (8, 2), (9, 4), (12, 6), (10, 3)])
def test_rank_unrank_lexicographic(orc, L, S):
    comps = sorted(c for c in itertools.product(range(1, L + 1), repeat=S) if sum(c) == L)
    assert len(comps) == math.comb(L - 1, S - 1)
    for r, c in enumerate(comps):
        assert orc.unrank(L, S, r) == list(c)
        assert orc.rank(L, S, c) == r
    with pytest.raises(ValueError):
        orc.unrank(L, S, len(comps))


def test_binomials(orc):
    for n in range(0, 128):
        for k in range(0, 16):
            assert orc.binom(n, k) == (math.comb(n, k) if k <= n else 0)


# -- memory feasibility (Sec. 3.2) -------------------------------------------------

def test_config1_feasibility(orc):
    """Only B-first with 7 layers on B fails: 7 x (1.5 + 2 x 0.4) GB > 16 GB."""
    w = gen.config1()
    tab = orc.OracleTables.from_workload(w)
    T, F = orc.eval_batch(tab, gen.all_candidates(w))
    assert F.tolist() == [1] * 13 + [0]


def test_eval_batch_flags(orc):
    w = gen.config5_tables()
    tab = orc.OracleTables.from_workload(w)
    c = gen.config5_candidates(4)
    c[0]["S"] = 17
    c[1]["M"] = 0
    c[2]["map_rank"] = math.comb(63, int(c[2]["S"]) - 1)
    c[3]["tp_idx"] = 1
    T, F = orc.eval_batch(tab, c)
    assert F.tolist() == [2, 2, 2, 2] and T.tolist() == [-1] * 4
    big = orc.OracleTables(L=2, n_types=1, n_tp=1, fwd=[[2 ** 29, 1]], bwd=[[2 ** 29, 1]],
                           dsync=[[0, 0]], p2p_f=[[0]], p2p_b=[[0]], mem_w=[[0, 0]],
                           mem_a=[[0, 0]], cap=[1])
    c = np.zeros(2, gen.CANDIDATE_DTYPE)
    c["S"], c["M"] = 1, [1, 2]
    T, F = orc.eval_batch(big, c)
    assert F.tolist() == [1, 3] and T[0] == 2 ** 30 + 2


# -- search (Sec. 4.2) --------------------------------------------------------------

def _brute_force_plan(orc, w, schedule=0):
    """Every candidate through eval_batch; argmin of T/(D M), then global index."""
    cands = gen.all_candidates(w)
    tab = orc.OracleTables.from_workload(w, schedule)
    T, F = orc.eval_batch(tab, cands)
    best = None
    n_place = len(gen.place_list(w))
    n_map = gen.n_compositions(w.L, w.S)
    for i in np.flatnonzero(F == 1):
        c = cands[i]
        m_idx = w.M_list.index(int(c["M"]))
        D = w.dp_list[int(c["tp_idx"])]
        key = (Fraction(int(T[i]), D * int(c["M"])), int(i))
        if best is None or key < best:
            best = key
    assert len(cands) == len(w.M_list) * w.n_tp * n_place * n_map
    return best


@pytest.mark.parametrize("cfg", [1, 2])
def test_search_equals_brute_force(orc, cfg):
    w = gen.get_config(cfg)
    best = _brute_force_plan(orc, w)
    for prune, warm in ((False, 0), (True, 0), (True, 500)):
        plan, _ = orc.search(w, prune=prune, warmup=warm, seed=3)
        assert plan["found"]
        assert plan["global_index"] == best[1]
        assert Fraction(plan["T"], plan["D"] * plan["M"]) == best[0]


def _random_problem(rng, seed):
    T_ = rng.randint(1, 3)
    n_tp = rng.randint(1, 2)
    L = rng.randint(3, 9)
    S = rng.randint(1, min(4, L))
    K = T_ * n_tp
    w = gen.Workload(name="random", L=L, n_types=T_, n_tp=n_tp,
                     fwd=np.array([[rng.randint(1, 60) for _ in range(L)] for _ in range(K)],
                                  np.int32),
                     bwd=np.array([[rng.randint(1, 90) for _ in range(L)] for _ in range(K)],
                                  np.int32),
                     dsync=np.array([[rng.randint(0, 40) for _ in range(L)] for _ in range(K)],
                                    np.int32),
                     p2p_f=np.array([[rng.randint(0, 30) for _ in range(K)] for _ in range(K)],
                                    np.int32),
                     p2p_b=np.array([[rng.randint(0, 30) for _ in range(K)] for _ in range(K)],
                                    np.int32),
                     mem_w=np.array([[rng.randint(0, 5) for _ in range(L)] for _ in range(K)],
                                    np.int64),
                     mem_a=np.array([[rng.randint(0, 3) for _ in range(L)] for _ in range(K)],
                                    np.int64),
                     cap=np.array([rng.randint(8, 40) for _ in range(K)], np.int64),
                     S=S, M_list=sorted(rng.sample(range(1, 9), rng.randint(1, 2))),
                     tp_list=list(range(1, n_tp + 1)),
                     dp_list=[rng.randint(1, 3) for _ in range(n_tp)], seed=seed)
    if rng.random() < 0.5 and S >= T_:
        w.placement = gen.workloads.PLACE_EXACT
        counts = [1] * T_
        for _ in range(S - T_):
            counts[rng.randrange(T_)] += 1
        w.type_counts = counts
    return w


def test_search_random_problems_equal_brute_force(orc):
    rng = random.Random(17)
    n_found = 0
    for seed in range(150):
        w = _random_problem(rng, seed)
        best = _brute_force_plan(orc, w)
        for prune, warm in ((False, 0), (True, 0), (True, 20)):
            plan, _ = orc.search(w, prune=prune, warmup=warm, seed=seed)
            if best is None:
                assert not plan["found"]
                continue
            n_found += 1
            assert plan["global_index"] == best[1], (seed, prune, warm)
            assert Fraction(plan["T"], plan["D"] * plan["M"]) == best[0]
    assert n_found > 150


def test_search_config3_pruned_equals_exhaustive(orc):
    w = gen.config3()
    a, sa = orc.search(w, prune=False)
    b, sb = orc.search(w, prune=True, warmup=500, seed=1)
    assert a == b
    assert sb["leaves_evaluated"] < sa["leaves_evaluated"]
