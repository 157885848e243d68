"""Pins for the oracle's layer-level pruning (Theorem 2, App. B): the search
restricted to ridge-like plans -- for every device type, the layer counts of
its stages, in stage order, rise and then fall.  Theorem 2 only asserts that
some optimal plan is ridge-like (under Assumptions 1-4, proved for Eager
1F1B), so the pins are: the restricted search returns exactly the best
ridge-like plan (brute force), it is never better than the exact optimum,
and it reaches the exact optimum on instances shaped like the assumptions
under Eager 1F1B."""
import random
from fractions import Fraction

import numpy as np

import gen
from tests.test_oracle import _random_problem


def _ridge(types, layers):
    """Definition: a sequence is ridge-like when it is non-decreasing up to
    some position and non-increasing after it."""
    for t in set(types):
        seq = [l for ty, l in zip(types, layers) if ty == t]
        if not any(all(a <= b for a, b in zip(seq[:p], seq[1:p + 1])) and
                   all(a >= b for a, b in zip(seq[p:], seq[p + 1:])) for p in range(len(seq))):
            return False
    return True


def _best(orc, w, schedule, ridge):
    """Brute force: every plan through eval_batch, argmin of T/(D M) then
    global index, over all feasible plans or the ridge-like ones."""
    cands = gen.all_candidates(w)
    T, F = orc.eval_batch(orc.OracleTables.from_workload(w, schedule), cands)
    places = gen.place_list(w)
    n_map = gen.n_compositions(w.L, w.S)
    best = None
    for i in np.flatnonzero(F == 1):
        c = cands[i]
        if ridge and not _ridge(places[(i // n_map) % len(places)],
                                orc.unrank(w.L, w.S, int(c["map_rank"]))):
            continue
        key = (Fraction(int(T[i]), w.dp_list[int(c["tp_idx"])] * int(c["M"])), int(i))
        if best is None or key < best:
            best = key
    return best


def test_ridge_definition_examples():
    assert _ridge([0, 0, 0, 0], [1, 3, 3, 2])
    assert _ridge([0, 1, 0, 1, 0], [5, 1, 4, 9, 2])      # type 0: 5,4,2; type 1: 1,9
    assert not _ridge([0, 0, 0], [3, 1, 2])
    assert not _ridge([1, 0, 1, 0, 1], [4, 1, 2, 1, 5])  # type 1: 4,2,5
    assert _ridge([2], [7])


def test_ridge_search_is_the_best_ridge_plan(orc):
    rng = random.Random(51)
    n = 0
    for seed in range(120):
        w = _random_problem(rng, seed)
        for schedule in (0, 1):
            best = _best(orc, w, schedule, ridge=True)
            for prune, warm in ((False, 0), (True, 0), (True, 30)):
                plan, st = orc.search(w, prune=prune, warmup=warm, seed=seed, schedule=schedule,
                                      ridge=True)
                if best is None:
                    assert not plan["found"]
                    continue
                assert plan["global_index"] == best[1], (seed, schedule, prune, warm)
                n += 1
    assert n > 500


def test_ridge_never_beats_the_exact_optimum(orc):
    rng = random.Random(52)
    worse = 0
    for seed in range(120):
        w = _random_problem(rng, seed)
        for schedule in (0, 1):
            exact, _ = orc.search(w, prune=True, schedule=schedule)
            ridge, _ = orc.search(w, prune=True, schedule=schedule, ridge=True)
            if not exact["found"]:
                assert not ridge["found"]
                continue
            if not ridge["found"]:
                continue
            a = Fraction(exact["T"], exact["D"] * exact["M"])
            b = Fraction(ridge["T"], ridge["D"] * ridge["M"])
            assert b >= a
            worse += b > a
    assert worse < 40  # usually the same value, sometimes worse (no guarantee here)


def _assumption_like(rng, seed):
    """Identical layers per type, B = r F, transfers at most (r-1)/2 of the
    smallest layer's forward, M >= 2N, no all-reduce, no memory limit."""
    T_ = rng.randint(1, 3)
    L = rng.randint(4, 10)
    S = rng.randint(2, min(5, L))
    r = rng.choice([2, 3])
    f = [rng.randint(20, 60) for _ in range(T_)]
    fwd = np.array([[f[k]] * L for k in range(T_)], np.int32)
    tmax = (r - 1) * min(f) // 2
    return gen.Workload(
        name="assumption-like", L=L, n_types=T_, n_tp=1, fwd=fwd, bwd=fwd * r,
        dsync=np.zeros((T_, L), np.int32),
        p2p_f=np.array([[rng.randint(0, tmax) for _ in range(T_)] for _ in range(T_)], np.int32),
        p2p_b=np.array([[rng.randint(0, tmax) for _ in range(T_)] for _ in range(T_)], np.int32),
        mem_w=np.zeros((T_, L), np.int64), mem_a=np.zeros((T_, L), np.int64),
        cap=np.ones(T_, np.int64), S=S, M_list=[2 * S + rng.randint(0, 4)], tp_list=[1],
        dp_list=[1], seed=seed)


def test_ridge_reaches_the_optimum_under_the_assumptions_eager(orc):
    rng = random.Random(53)
    for seed in range(150):
        w = _assumption_like(rng, seed)
        exact, _ = orc.search(w, prune=True, schedule=1)
        ridge, _ = orc.search(w, prune=True, schedule=1, ridge=True)
        assert ridge["T"] == exact["T"], (seed, exact, ridge)


def test_ridge_cuts_prefixes_on_config3(orc):
    w = gen.config3()
    exact, se = orc.search(w, prune=True, warmup=500, seed=1)
    ridge, sr = orc.search(w, prune=True, warmup=500, seed=1, ridge=True)
    assert sr["prefixes_ridge"] > 0
    assert sr["leaves_evaluated"] < se["leaves_evaluated"]
    assert ridge["T"] >= exact["T"]
