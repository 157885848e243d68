"""poseidon_search on the GPU against the oracle's exact search.  The plan
(global index, makespan, placement, layers) must be identical."""
import json
import os
import random

import numpy as np
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
    prob, keep = P.make_problem(w, **kw)
    return P.poseidon_search(prob)


def same_plan(a, b):
    keys = ("global_index", "T", "m_idx", "tp_idx", "M", "D", "place_rank", "map_rank",
            "types", "layers")
    return all(a[k] == b[k] for k in keys)


@pytest.mark.parametrize("cfg", [1, 2, 3])
@pytest.mark.parametrize("prune", [0, 1, 2])
def test_configs_match_oracle(P, orc, cfg, prune):
    w = gen.get_config(cfg)
    ref, _ = orc.search(w, prune=True, warmup=0)
    plan, st = gpu_search(P, w, prune=prune, warmup=500, seed=cfg)
    assert same_plan(plan, ref), (plan, ref)
    assert st["evaluated"] >= 1


@pytest.mark.parametrize("prune", [1, 2])
def test_config4_matches_stored_oracle_plan(P, prune):
    """The bench's workload and launch configuration (warm-up 65536 samples;
    the bench times both prune modes); expected plan written by
    tests/golden/make_search_plans.py."""
    ref = json.load(open(GOLDEN))["config4"]["plan"]
    plan, st = gpu_search(P, gen.config4(), prune=prune, warmup=65536, seed=0)
    assert same_plan(plan, ref), (plan, ref)
    assert st["slices_feasible"] == 420


def test_tight_bound_cuts_more(P):
    """The tightened bound removes prefixes that Eq. 2 keeps: on config 3
    it generates fewer prefixes and evaluates no more plans."""
    w = gen.config3()
    _, s1 = gpu_search(P, w, prune=1, warmup=500, seed=0)
    _, s2 = gpu_search(P, w, prune=2, warmup=500, seed=0)
    assert s2["prefixes"] < s1["prefixes"]
    assert s2["evaluated"] <= s1["evaluated"]


@pytest.mark.parametrize("warmup", [0, 1, 500, 100_000])
def test_warmup_never_changes_the_plan(P, orc, warmup):
    w = gen.config2()
    ref, _ = orc.search(w, prune=False)
    for prune in (1, 2):
        plan, _ = gpu_search(P, w, prune=prune, warmup=warmup, seed=warmup)
        assert same_plan(plan, ref), prune


@pytest.mark.parametrize("cap", [1, 3000, 20_000])
def test_tiny_frontiers_defer_and_still_match(P, orc, cap):
    """Capacities far below the frontier sizes force many deferral passes
    (a capacity below 32*L is raised to 32*L)."""
    for cfg in (2, 3):
        w = gen.get_config(cfg)
        ref, _ = orc.search(w, prune=True, warmup=0)
        for prune in (1, 2):
            plan, _ = gpu_search(P, w, prune=prune, warmup=50, frontier_cap=cap)
            assert same_plan(plan, ref), (cfg, cap, prune)


def test_random_small_problems(P, orc):
    rng = random.Random(23)
    n_found = 0
    for seed in range(120):
        w = _random_problem(rng, seed)
        ref, _ = orc.search(w, prune=False)
        try:
            plan, _ = gpu_search(P, w, prune=seed % 3, warmup=seed % 7, seed=seed)
        except P.PoseidonError as e:
            assert e.status == P.binding.POS_EINFEASIBLE and not ref["found"], (seed, e)
            continue
        assert ref["found"]
        assert same_plan(plan, ref), (seed, plan, ref)
        n_found += 1
    assert n_found > 60


def test_single_stage_and_two_stage(P, orc):
    w = gen.config1()
    for S, counts in ((1, None), (2, [1, 1])):
        w.S = S
        w.placement = gen.workloads.PLACE_FREE if counts is None else gen.workloads.PLACE_EXACT
        w.type_counts = counts or []
        ref, _ = orc.search(w, prune=False)
        for prune in (1, 2):
            plan, _ = gpu_search(P, w, prune=prune, warmup=3)
            assert same_plan(plan, ref), (S, prune)


def test_infeasible_and_overflow(P):
    w = gen.config1()
    w.cap = np.array([1, 1], np.int64)
    with pytest.raises(P.PoseidonError) as e:
        gpu_search(P, w)
    assert e.value.status == P.binding.POS_EINFEASIBLE
    w = gen.config1()
    w.M_list = [255]
    w.fwd = np.full_like(w.fwd, 600_000)
    w.bwd = np.full_like(w.bwd, 600_000)
    with pytest.raises(P.PoseidonError) as e:
        gpu_search(P, w)
    assert e.value.status == P.binding.POS_EOVERFLOW


def _limits_problem(seed, S, L, n_types, placement, counts, M_list):
    rng = np.random.default_rng(seed)
    K = n_types
    w = gen.Workload(name="limits", L=L, n_types=n_types, n_tp=1,
                     fwd=rng.integers(1, 500, (K, L)).astype(np.int32),
                     bwd=rng.integers(1, 900, (K, L)).astype(np.int32),
                     dsync=rng.integers(0, 200, (K, L)).astype(np.int32),
                     p2p_f=rng.integers(0, 100, (K, K)).astype(np.int32),
                     p2p_b=rng.integers(0, 100, (K, K)).astype(np.int32),
                     mem_w=rng.integers(0, 4, (K, L)).astype(np.int64),
                     mem_a=rng.integers(0, 2, (K, L)).astype(np.int64),
                     cap=(rng.integers(20, 60, K) * L // 10).astype(np.int64),
                     S=S, M_list=M_list, tp_list=[1], dp_list=[1], placement=placement,
                     type_counts=counts, seed=seed)
    return w


@pytest.mark.parametrize("S,L,types,placement,counts,M_list", [
    (16, 19, 1, 0, [], [16, 40]),          # 16 stages, M = S and M > S
    (16, 18, 2, 1, [8, 8], [5]),           # M < S with 16 stages, exact placement
    (12, 16, 4, 1, [3, 3, 3, 3], [12]),    # 4 device types
    (3, 127, 2, 0, [], [255]),             # the longest model, the most micro-batches
])
def test_search_at_the_limits(P, orc, S, L, types, placement, counts, M_list):
    w = _limits_problem(S * 31 + L, S, L, types, placement, counts, M_list)
    ref, _ = orc.search(w, prune=True, warmup=0)
    for prune in (1, 2):
        try:
            plan, _ = gpu_search(P, w, prune=prune, warmup=200, seed=1)
        except P.PoseidonError as e:
            assert e.status == P.binding.POS_EINFEASIBLE and not ref["found"]
            continue
        assert same_plan(plan, ref), (prune, plan, ref)


def test_incumbent_cas_limit_times_out_and_the_next_search_recovers(P, orc):
    """The incumbent's compare-and-swap loop is bounded.  With no round
    allowed (cas_limit < 0) every update that would lower the incumbent
    gives up, the search returns POS_ETIMEOUT with a message naming that
    loop, and the device stays usable: the next search on the same
    workspace returns the oracle's plan."""
    w = gen.config2()
    prob, keep = P.make_problem(w, warmup=64, prune=2, cas_limit=-1)
    with pytest.raises(P.PoseidonError) as err:
        P.poseidon_search(prob)
    assert err.value.status == P.binding.POS_ETIMEOUT
    assert "compare-and-swap" in str(err.value)
    plan, _ = gpu_search(P, w, warmup=64, prune=2)
    ref, _ = orc.search(w, prune=True)
    assert plan["global_index"] == ref["global_index"] and plan["T"] == ref["T"]
