"""Layer-level (ridge) pruning on the GPU (Theorem 2) against the oracle's
ridge-restricted search: the same plan, for both schedules and every
stage-level prune mode; on config 4 the ridge optimum is compared with the
exact one (Theorem 2 guarantees equality only under its assumptions)."""
import json
import os
import random
from fractions import Fraction

import pytest

import gen
from tests.test_oracle import _random_problem

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "search_plans.json")


@pytest.fixture(scope="module")
def P():
    import torch
    assert torch.cuda.is_available()
    import paper_2609_06086_gb300 as P
    P.lib()
    return P


def gpu_search(P, w, **kw):
    prob, keep = P.make_problem(w, ridge=True, **kw)
    return P.poseidon_search(prob)


def same_plan(a, b):
    return all(a[k] == b[k] for k in ("global_index", "T", "M", "D", "types", "layers"))


@pytest.mark.parametrize("cfg", [1, 2, 3])
@pytest.mark.parametrize("schedule", [0, 1])
@pytest.mark.parametrize("prune", [1, 2])
def test_ridge_configs(P, orc, cfg, schedule, prune):
    w = gen.get_config(cfg)
    ref, _ = orc.search(w, prune=True, warmup=0, schedule=schedule, ridge=True)
    plan, st = gpu_search(P, w, prune=prune, warmup=400, seed=cfg, schedule=schedule)
    assert same_plan(plan, ref), (plan, ref)
    if cfg == 3 and schedule == 0:
        # (under Eager the bounds cut everything before any type's counts fall)
        assert st["pruned_ridge"] > 0


def test_ridge_random_problems(P, orc):
    rng = random.Random(57)
    n = 0
    for seed in range(100):
        w = _random_problem(rng, seed)
        schedule = seed % 2
        ref, _ = orc.search(w, prune=False, schedule=schedule, ridge=True)
        try:
            plan, _ = gpu_search(P, w, prune=1 + seed % 2, warmup=seed % 7, seed=seed,
                                 schedule=schedule)
        except P.PoseidonError as e:
            assert e.status == P.binding.POS_EINFEASIBLE and not ref["found"], (seed, e)
            continue
        assert ref["found"] and same_plan(plan, ref), (seed, plan, ref)
        n += 1
    assert n > 50


def test_ridge_tiny_frontiers(P, orc):
    w = gen.config2()
    ref, _ = orc.search(w, prune=True, warmup=0, ridge=True)
    for cap in (1, 3000):
        plan, _ = gpu_search(P, w, prune=2, warmup=20, frontier_cap=cap)
        assert same_plan(plan, ref), cap


@pytest.mark.parametrize("key,schedule", [("config4", 0), ("config4_eager", 1)])
def test_ridge_config4_against_exact_and_oracle(P, key, schedule):
    gold = json.load(open(GOLDEN))
    exact = gold[key]["plan"]
    plan, st = gpu_search(P, gen.config4(), prune=2, warmup=65536, seed=0, schedule=schedule)
    assert Fraction(plan["T"], plan["D"] * plan["M"]) >= Fraction(exact["T"], exact["D"] * exact["M"])
    if key + "_ridge" in gold:
        assert same_plan(plan, gold[key + "_ridge"]["plan"])
