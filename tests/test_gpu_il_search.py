"""poseidon_search over Interleaved 1F1B plans on the GPU against the
oracle's interleaved search: the same plan (global index, makespan,
placement, virtual-stage layers) on random small problems under every
prune mode, on the config-2 tables with V = 2, 3, 4 chunks per device, and
with a frontier so small that most groups are deferred."""
import json
import os
import random

import pytest

import gen
from tests.test_oracle_interleaved_search import _problem

pytestmark = pytest.mark.gpu

IL = 2
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "search_plans.json")
KEYS = ("global_index", "T", "m_idx", "tp_idx", "M", "D", "place_rank", "map_rank", "types",
        "layers")


@pytest.fixture(scope="module")
def P():
    import torch
    assert torch.cuda.is_available()
    import paper_2609_06086_gb300 as P
    P.lib()
    return P


def gpu_search(P, w, V, **kw):
    prob, keep = P.make_problem(w, schedule=IL, V=V, **kw)
    return P.poseidon_search(prob)


def check(P, w, V, ref, **kw):
    if not ref["found"]:
        with pytest.raises(P.PoseidonError) as err:
            gpu_search(P, w, V, **kw)
        assert err.value.status == P.binding.POS_EINFEASIBLE
        return None
    plan, st = gpu_search(P, w, V, **kw)
    assert all(plan[k] == ref[k] for k in KEYS), (plan, ref, kw)
    return st


def test_random_problems_match_oracle(P, orc):
    rng = random.Random(29)
    found = 0
    for seed in range(100):
        w, V = _problem(rng, seed)
        ref, _ = orc.search_interleaved(w, V, prune=True)
        for prune in (0, 1, 2):
            check(P, w, V, ref, prune=prune, warmup=0)
        found += ref["found"]
    assert found > 50


def test_config2_v2_matches_oracle_live(P, orc):
    w = gen.config2()
    ref, _ = orc.search_interleaved(w, 2, prune=True)
    for prune in (1, 2):
        st = check(P, w, 2, ref, prune=prune)
        assert st["evaluated"] > 0 and st["relaxations"] > 0


@pytest.mark.parametrize("V", [2, 3])
def test_config2_matches_stored_oracle_plan(P, V):
    """Stored oracle plans (V = 4 would make the oracle enumerate 16 virtual
    stages over 32 layers, C(31, 15) compositions per slice: not stored)."""
    data = json.load(open(GOLDEN))
    ref = data[f"config2_il_v{V}"]["plan"]
    for prune in (1, 2):
        check(P, gen.config2(), V, ref, prune=prune)


def test_small_frontier_defers_and_matches(P, orc):
    """frontier_cap at its floor (32 L entries): most 32-parent groups are
    deferred and re-expanded after the part that fit; same plan."""
    w = gen.config2()
    ref, _ = orc.search_interleaved(w, 2, prune=True)
    check(P, w, 2, ref, prune=1, frontier_cap=1)
