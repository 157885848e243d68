"""Pins for the oracle's search over Interleaved 1F1B plans: on small random
problems its result equals a brute force written here from the problem's
definition (every slice, every composition of L into the N*V virtual
stages, each evaluated by the oracle's interleaved DAG, the smallest time
per sample with ties to the lowest global index), with and without the
per-device serial-work bound; the bound never exceeds a plan's makespan."""
import itertools
import math
import random
from fractions import Fraction

import numpy as np
import pytest

import gen

IL = 2


def _problem(rng, seed):
    T_ = rng.randint(1, 2)
    n_tp = rng.randint(1, 2)
    N = rng.randint(1, 3)
    V = rng.randint(2, 3)
    L = rng.randint(N * V, min(N * V + 4, 9))
    K = T_ * n_tp
    r = lambda lo, hi, shape: np.array([[rng.randint(lo, hi) for _ in range(shape[1])]  # noqa: E731
                                        for _ in range(shape[0])])
    w = gen.Workload(name="random-il", L=L, n_types=T_, n_tp=n_tp,
                     fwd=r(1, 60, (K, L)).astype(np.int32), bwd=r(1, 90, (K, L)).astype(np.int32),
                     dsync=r(0, 40, (K, L)).astype(np.int32),
                     p2p_f=r(0, 30, (K, K)).astype(np.int32), p2p_b=r(0, 30, (K, K)).astype(np.int32),
                     mem_w=r(0, 5, (K, L)).astype(np.int64), mem_a=r(0, 3, (K, L)).astype(np.int64),
                     cap=np.array([rng.randint(8, 70) for _ in range(K)], np.int64),
                     S=N, M_list=sorted(rng.sample(range(1, 3 * N + 2), rng.randint(1, 3))),
                     tp_list=list(range(1, n_tp + 1)),
                     dp_list=[rng.randint(1, 3) for _ in range(n_tp)], seed=seed)
    if rng.random() < 0.5 and N >= T_:
        w.placement = gen.workloads.PLACE_EXACT
        counts = [1] * T_
        for _ in range(N - T_):
            counts[rng.randrange(T_)] += 1
        w.type_counts = counts
    return w, V


def _brute_force(orc, w, V):
    tab = orc.OracleTables.from_workload(w, schedule=IL)
    N, L = w.S, w.L
    J = N * V
    places = gen.place_list(w)
    n_map = math.comb(L - 1, J - 1)
    best = None
    for mi, M in enumerate(w.M_list):
        if M % N:
            continue
        for tp in range(w.n_tp):
            D = w.dp_list[tp]
            for pr, seq in enumerate(places):
                cls = [t * w.n_tp + tp for t in seq]
                for cuts in itertools.combinations(range(1, L), J - 1):
                    b = (0,) + cuts + (L,)
                    layers = [b[i + 1] - b[i] for i in range(J)]
                    T, fits = orc.evaluate_interleaved(tab, N, V, M, cls, layers)
                    if not fits:
                        continue
                    idx = ((mi * w.n_tp + tp) * len(places) + pr) * n_map + orc.rank(L, J, layers)
                    key = (Fraction(T, D * M), idx)
                    if best is None or key < best[0]:
                        best = (key, T, idx, layers, list(seq))
    return best


def test_search_equals_brute_force(orc):
    rng = random.Random(29)
    found = pruned = 0
    for seed in range(100):
        w, V = _problem(rng, seed)
        ref = _brute_force(orc, w, V)
        for prune in (False, True):
            plan, st = orc.search_interleaved(w, V, prune=prune)
            if ref is None:
                assert not plan["found"], seed
                continue
            _, T, idx, layers, types = ref
            assert plan["found"] and plan["T"] == T and plan["global_index"] == idx, (seed, prune)
            assert plan["layers"] == layers and plan["types"] == types
            pruned += st["prefixes_pruned"] if prune else 0
        found += ref is not None
    assert found > 50 and pruned > 0


def test_bound_is_below_every_makespan(orc):
    """The cut's bound for a complete plan: max over devices of M * (F + B)
    over its chunks plus their all-reduce time, never above the makespan."""
    rng = random.Random(31)
    for seed in range(40):
        w, V = _problem(rng, seed)
        tab = orc.OracleTables.from_workload(w, schedule=IL)
        N, L, J = w.S, w.L, w.S * V
        fwd, bwd, ds = (np.asarray(x, np.int64) for x in (w.fwd, w.bwd, w.dsync))
        M = N * rng.randint(1, 3)
        for _ in range(10):
            cuts = sorted(rng.sample(range(1, L), J - 1))
            b = [0] + cuts + [L]
            layers = [b[i + 1] - b[i] for i in range(J)]
            cls = [rng.randrange(w.n_types) * w.n_tp for _ in range(N)]
            T, _ = orc.evaluate_interleaved(tab, N, V, M, cls, layers)
            lb = 0
            for d in range(N):
                k = cls[d]
                work = sum(M * int(fwd[k, b[j]:b[j + 1]].sum() + bwd[k, b[j]:b[j + 1]].sum()) +
                           int(ds[k, b[j]:b[j + 1]].sum()) for j in range(d, J, N))
                lb = max(lb, work)
            assert lb <= T, seed


@pytest.mark.parametrize("field", ["fwd", "bwd", "dsync", "mem_w", "mem_a", "p2p_f", "p2p_b"])
def test_negative_tables_are_rejected(orc, field):
    """The cuts assume non-negative weights (a partial plan's bound and a
    stage's memory only grow as layers are added), so both searches refuse
    a table with a negative entry instead of silently cutting plans."""
    w, V = _problem(random.Random(7), 0)
    arr = np.array(getattr(w, field))
    arr.flat[0] = -1
    setattr(w, field, arr)
    with pytest.raises(RuntimeError):
        orc.search_interleaved(w, V, prune=True)
    w.S = 2 if w.L >= 2 else 1
    with pytest.raises(RuntimeError):
        orc.search(w, prune=True)
