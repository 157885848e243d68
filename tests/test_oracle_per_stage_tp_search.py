"""Pins for the oracle's search with a TP index per stage (placement 2: the
per-stage heterogeneous TP of Table 1's Metis and HexiScale plans, searched
under the per-type device counts of Sec. 4.2.3).

A slice is (M, D, class sequence k_1..k_S), k = type * n_tp + tp_idx, and it
is allowed when the stages of every type use exactly that type's devices:
sum over its stages of D * tp_degree = devices of the type.  The brute force
below is written from that definition alone (itertools over every class
sequence and every composition, each plan evaluated by the oracle's DAG,
the smallest time per sample T/(D*M), ties to the lowest global index), and
the search must return its plan with and without the Eq. 2 prune and the
warm-up.  With one TP index and one D the rule is the exact-count placement,
so the result must equal the fixed-TP search's."""
import itertools
import math
import random
from fractions import Fraction

import numpy as np
import pytest

import gen

DEV = gen.workloads.PLACE_DEVICES


def _tables(rng, L, T_, n_tp, tight_memory):
    K = T_ * n_tp
    r = lambda lo, hi, shape: np.array([[rng.randint(lo, hi) for _ in range(shape[1])]  # noqa: E731
                                        for _ in range(shape[0])])
    cap_hi = 40 if tight_memory else 400
    return dict(L=L, n_types=T_, n_tp=n_tp,
                fwd=r(1, 60, (K, L)).astype(np.int32), bwd=r(1, 90, (K, L)).astype(np.int32),
                dsync=r(0, 40, (K, L)).astype(np.int32),
                p2p_f=r(0, 30, (K, K)).astype(np.int32), p2p_b=r(0, 30, (K, K)).astype(np.int32),
                mem_w=r(0, 5, (K, L)).astype(np.int64), mem_a=r(0, 3, (K, L)).astype(np.int64),
                cap=np.array([rng.randint(8, cap_hi) for _ in range(K)], np.int64))


def _problem(rng, seed, S=None, L=None):
    T_ = rng.randint(1, 2)
    n_tp = rng.randint(1, 3)
    S = S or rng.randint(1, 4)
    L = L or rng.randint(S, min(S + 4, 8))
    tp_deg = sorted(rng.sample([1, 2, 4], n_tp))
    D_list = sorted(rng.sample([1, 2, 3], rng.randint(1, 2)))
    # device counts that some (D, TP degrees) split can use up exactly: draw
    # one plan's stage classes and sum its devices per type
    D0 = rng.choice(D_list)
    devices = [0] * T_
    for _ in range(S):
        devices[rng.randrange(T_)] += D0 * rng.choice(tp_deg)
    w = gen.Workload(name="random-pstp", **_tables(rng, L, T_, n_tp, rng.random() < 0.5),
                     S=S, M_list=sorted(rng.sample(range(1, 9), rng.randint(1, 2))),
                     tp_list=tp_deg, dp_list=[1] * n_tp, placement=DEV, type_counts=devices,
                     D_list=D_list, seed=seed)
    return w


def _allowed(w, seq, D):
    use = [0] * w.n_types
    for k in seq:
        use[k // w.n_tp] += D * w.tp_list[k % w.n_tp]
    return use == list(w.type_counts)


def _brute_force(orc, w):
    tab = orc.OracleTables.from_workload(w)
    S, L, K = w.S, w.L, w.n_types * w.n_tp
    n_map = math.comb(L - 1, S - 1)
    per_D = [[seq for seq in itertools.product(range(K), repeat=S) if _allowed(w, seq, D)]
             for D in w.D_list]
    P = sum(len(x) for x in per_D)
    comps = []
    for cuts in itertools.combinations(range(1, L), S - 1):
        b = (0,) + cuts + (L,)
        comps.append([b[i + 1] - b[i] for i in range(S)])  # lexicographic order
    best = None
    for mi, M in enumerate(w.M_list):
        off = 0
        for di, D in enumerate(w.D_list):
            for pr, seq in enumerate(per_D[di]):
                for r, layers in enumerate(comps):
                    T, fits = orc.evaluate(tab, S, M, list(seq), layers)
                    if not fits:
                        continue
                    idx = (mi * P + off + pr) * n_map + r
                    key = (Fraction(T, D * M), idx)
                    if best is None or key < best[0]:
                        best = (key, T, idx, layers, list(seq), D, M)
            off += len(per_D[di])
    return best


def _check(ref, plan, w):
    if ref is None:
        assert not plan["found"]
        return
    _, T, idx, layers, seq, D, M = ref
    assert plan["found"]
    assert (plan["T"], plan["global_index"], plan["layers"], plan["D"], plan["M"]) == \
        (T, idx, layers, D, M)
    assert [t * w.n_tp + p for t, p in zip(plan["types"], plan["tps"])] == seq
    assert plan["tp_idx"] == -1 and w.D_list[plan["d_idx"]] == D


def test_search_equals_brute_force(orc):
    rng = random.Random(61)
    found = mixed = 0
    for seed in range(120):
        w = _problem(rng, seed)
        ref = _brute_force(orc, w)
        for prune, warmup in ((False, 0), (True, 0), (True, 25)):
            plan, _ = orc.search(w, prune=prune, warmup=warmup, seed=seed)
            _check(ref, plan, w)
        found += ref is not None
        if ref is not None:
            mixed += len({k % w.n_tp for k in ref[4]}) > 1
    assert found > 60 and mixed > 5  # many feasible problems, some optima mix TP degrees


def test_interleaved_search_equals_brute_force(orc):
    """Placement 2 under Interleaved 1F1B: the class sequence is over the N
    devices, the composition over the N*V virtual stages."""
    rng = random.Random(67)
    found = 0
    for seed in range(40):
        N, V = rng.randint(1, 2), 2
        L = rng.randint(N * V, N * V + 3)
        w = _problem(rng, seed, S=N, L=L)
        w.M_list = sorted({N * rng.randint(1, 3) for _ in range(2)})
        tab = orc.OracleTables.from_workload(w, schedule=2)
        K, J = w.n_types * w.n_tp, N * V
        n_map = math.comb(L - 1, J - 1)
        per_D = [[s for s in itertools.product(range(K), repeat=N) if _allowed(w, s, D)]
                 for D in w.D_list]
        P = sum(len(x) for x in per_D)
        best = None
        for mi, M in enumerate(w.M_list):
            off = 0
            for di, D in enumerate(w.D_list):
                for pr, seq in enumerate(per_D[di]):
                    for cuts in itertools.combinations(range(1, L), J - 1):
                        b = (0,) + cuts + (L,)
                        layers = [b[i + 1] - b[i] for i in range(J)]
                        T, fits = orc.evaluate_interleaved(tab, N, V, M, list(seq), layers)
                        if not fits:
                            continue
                        idx = (mi * P + off + pr) * n_map + orc.rank(L, J, layers)
                        key = (Fraction(T, D * M), idx)
                        if best is None or key < best[0]:
                            best = (key, T, idx)
                off += len(per_D[di])
        for prune in (False, True):
            plan, _ = orc.search_interleaved(w, V, prune=prune)
            if best is None:
                assert not plan["found"]
            else:
                assert plan["found"] and (plan["T"], plan["global_index"]) == best[1:]
        found += best is not None
    assert found > 15


def test_one_tp_and_one_D_reduce_to_exact_counts(orc):
    """One TP index (degree t) and one D: a class sequence is a type
    sequence and the device rule says type u has devices_u / (D t) stages,
    the exact-count placement; the plan and its global index must equal the
    fixed-TP search's on config 3 (L=48, S=8, 4 + 4 stages)."""
    w = gen.config3()
    ref, _ = orc.search(w, prune=True)
    w2 = gen.config3()
    w2.placement, w2.D_list, w2.tp_list = DEV, [1], [1]
    w2.type_counts = [4, 4]  # devices: 4 stages x D=1 x t=1 per type
    plan, _ = orc.search(w2, prune=True)
    for key in ("found", "T", "global_index", "layers", "types", "M", "D", "place_rank"):
        assert plan[key] == ref[key], key
    assert plan["tps"] == [0] * w.S


def test_devices_rule_examples():
    """The device rule on hand-checked sequences: 2 types, TP degrees
    {1, 2}, D = 2, 6 devices of type 0 and 2 of type 1; classes
    0 = (type 0, t=1), 1 = (type 0, t=2), 2 = (type 1, t=1), 3 = (type 1, t=2)."""
    w = gen.Workload(name="rule", L=4, n_types=2, n_tp=2, fwd=None, bwd=None, dsync=None,
                     p2p_f=None, p2p_b=None, mem_w=None, mem_a=None, cap=None, S=3,
                     tp_list=[1, 2], type_counts=[6, 2], placement=DEV, D_list=[2])
    assert _allowed(w, (0, 1, 2), 2)        # 2*1 + 2*2 = 6 on type 0, 2*1 on type 1
    assert _allowed(w, (1, 2, 0), 2)
    assert not _allowed(w, (1, 1, 2), 2)    # 8 devices of type 0
    assert not _allowed(w, (0, 1, 3), 2)    # 4 devices of type 1
    assert not _allowed(w, (0, 1, 2), 1)    # D = 1 uses only 3 + 1


@pytest.mark.parametrize("bad", ["ridge", "zero_tp", "zero_D"])
def test_invalid_problems_are_rejected(orc, bad):
    w = _problem(random.Random(5), 0)
    if bad == "zero_tp":
        w.tp_list = [0] + list(w.tp_list[1:])
    elif bad == "zero_D":
        w.D_list = [0]
    with pytest.raises(RuntimeError):
        orc.search(w, ridge=bad == "ridge")


def test_empty_D_list_is_rejected(orc):
    w = _problem(random.Random(5), 0)
    p, keep = orc._problem(w, orc.OracleTables.from_workload(w), False)
    p.n_D = 0
    plan, st = orc.Plan(), orc.Stats()
    assert orc.lib().orc_search(orc.C.byref(p), 1, 0, orc.C.c_uint64(0), orc.C.byref(plan),
                                orc.C.byref(st)) == -1


def test_partitioned_search_keeps_the_plan(orc):
    """orc_search_part over slice index classes mod n, best of the parts by
    (T/(D*M), global index) = the whole search's plan (config 2, and random
    per-stage-TP problems); a part index outside 0..n-1 is rejected."""
    cases = [gen.config2()] + [_problem(random.Random(71), s) for s in range(30)]
    for w in cases:
        ref, _ = orc.search(w, prune=True, warmup=20, seed=1)
        for n in (2, 3, 7):
            best = None
            for part in range(n):
                plan, _ = orc.search(w, prune=True, warmup=20, seed=1, part=part, n_parts=n)
                if plan["found"]:
                    key = (Fraction(plan["T"], plan["D"] * plan["M"]), plan["global_index"])
                    if best is None or key < best[0]:
                        best = (key, plan)
            if not ref["found"]:
                assert best is None
            else:
                assert best[1] == ref
    with pytest.raises(RuntimeError):
        orc.search(cases[0], part=3, n_parts=3)
