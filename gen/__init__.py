"""Seeded synthetic workloads shared by the oracle tests, the GPU tests and the bench.

This package only draws inputs (cost tables, search problems, candidate
batches).  It holds none of the method's arithmetic: no DAG, no makespan,
no lower bound, no search.
"""
from .workloads import (  # noqa: F401
    CANDIDATE_DTYPE, CANDIDATE_EX_DTYPE, Workload, config1, config2, config3, config4,
    config4_per_stage_tp,
    config5_tables, config5_candidates, all_candidates, random_candidates,
    interleaved_candidates, per_stage_tp_candidates, search_space_sample, get_config,
    n_compositions, place_list,
)
