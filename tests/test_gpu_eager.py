"""Eager 1F1B on the GPU (App. B: warm-up of 2(N-i)+1 forwards) against the
oracle with the same schedule: makespans and feasibility flags bit-exact,
search plans identical.  Covers both GPU paths: M >= 2S-1 (compile-time
ramps and a steady loop) and M < 2S-1 (level programs)."""
import json
import os
import random

import numpy as np
import pytest

import gen
from tests.gpu_util import eval_device
from tests.test_oracle import _random_problem

pytestmark = pytest.mark.gpu

EAGER = 1
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "search_plans.json")


@pytest.fixture(scope="module")
def P():
    import torch
    assert torch.cuda.is_available()
    import paper_2609_06086_gb300 as P
    P.lib()
    return P


def _both(P, orc, w, cands):
    h = P.Handle(P.Tables.from_workload(w), schedule=EAGER)
    T, F = eval_device(P, h, cands)
    Tr, Fr = orc.eval_batch(orc.OracleTables.from_workload(w, EAGER), cands)
    return T, F, Tr, Fr


@pytest.mark.parametrize("cfg", [1, 2])
def test_eager_all_plans(P, orc, cfg):
    w = gen.get_config(cfg)
    T, F, Tr, Fr = _both(P, orc, w, gen.all_candidates(w))
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_eager_config5_sample(P, orc):
    w = gen.config5_tables()
    c = gen.config5_candidates(200_000, seed=7)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (c["M"] < 2 * c["S"].astype(int) - 1).sum() > 1000  # both paths ran


def test_eager_every_stage_count_around_the_path_switch(P, orc):
    """S = 1..16 with M = 1..40: every (S, M) of the level programs and the
    first M values of the fast path."""
    w = gen.config5_tables()
    rng = np.random.default_rng(11)
    cs = []
    for S in range(1, 17):
        for M in range(1, 41):
            c = gen.random_candidates(6, L=w.L, n_types=2, S_range=(S, S), M_range=(M, M),
                                      seed=int(rng.integers(1 << 30)))
            cs.append(c)
    c = np.concatenate(cs)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_eager_config4_tables(P, orc):
    w = gen.config4()
    c = gen.random_candidates(50_000, L=w.L, n_types=3, S_range=(2, 12), M_range=(1, 64), seed=13)
    c["tp_idx"] = np.random.default_rng(13).integers(0, 4, len(c))
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_schedules_differ(P):
    """The two handles give different makespans and feasibility on the same
    candidates (Eager holds more micro-batches in flight)."""
    w = gen.config2()
    c = gen.all_candidates(w)
    T1, F1 = eval_device(P, P.Handle(P.Tables.from_workload(w)), c)
    T2, F2 = eval_device(P, P.Handle(P.Tables.from_workload(w), schedule=EAGER), c)
    assert (T1 != T2).any() and (F1 != F2).any()


def gpu_search(P, w, **kw):
    prob, keep = P.make_problem(w, schedule=EAGER, **kw)
    return P.poseidon_search(prob)


def same_plan(a, b):
    return all(a[k] == b[k] for k in ("global_index", "T", "M", "D", "types", "layers"))


@pytest.mark.parametrize("cfg", [1, 2, 3])
@pytest.mark.parametrize("prune", [0, 1, 2])
def test_eager_search_configs(P, orc, cfg, prune):
    w = gen.get_config(cfg)
    ref, _ = orc.search(w, prune=True, warmup=0, schedule=EAGER)
    plan, st = gpu_search(P, w, prune=prune, warmup=300, seed=cfg)
    assert same_plan(plan, ref), (plan, ref)


def test_eager_search_random_problems(P, orc):
    rng = random.Random(47)
    n = 0
    for seed in range(100):
        w = _random_problem(rng, seed)
        ref, _ = orc.search(w, prune=False, schedule=EAGER)
        try:
            plan, _ = gpu_search(P, w, prune=seed % 3, warmup=seed % 5, seed=seed)
        except P.PoseidonError as e:
            assert e.status == P.binding.POS_EINFEASIBLE and not ref["found"], (seed, e)
            continue
        assert ref["found"] and same_plan(plan, ref), (seed, plan, ref)
        n += 1
    assert n > 50


@pytest.mark.parametrize("cap", [1, 5000])
def test_eager_search_tiny_frontiers(P, orc, cap):
    w = gen.config3()
    ref, _ = orc.search(w, prune=True, warmup=0, schedule=EAGER)
    for prune in (1, 2):
        plan, _ = gpu_search(P, w, prune=prune, warmup=50, frontier_cap=cap)
        assert same_plan(plan, ref), (cap, prune)


def test_eager_config4_matches_stored_oracle_plan(P):
    ref = json.load(open(GOLDEN))["config4_eager"]["plan"]
    plan, st = gpu_search(P, gen.config4(), prune=2, warmup=65536, seed=0)
    assert same_plan(plan, ref), (plan, ref)
