"""Poseidon's search hot path on one GB300: batched DAG-makespan evaluation,
memory feasibility, the stage-level prune and the exact search, in CUDA
kernels behind the C ABI of include/poseidon.h (libposeidon.so).

The Python side is the ctypes binding in ``binding``; it loads the in-tree
library and never computes anything itself.
"""
from .binding import (  # noqa: F401
    EXPORTS, Handle, PoseidonError, Tables, lib, make_problem, poseidon_argmin,
    poseidon_eval_batch, poseidon_eval_batch_ex, poseidon_eval_batch_host, poseidon_search,
)
