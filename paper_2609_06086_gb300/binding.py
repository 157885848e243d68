"""Thin ctypes binding of libposeidon.so (include/poseidon.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  Device buffers are passed as raw pointers (e.g. a torch tensor's
``data_ptr()``); there is no CPU fallback, and loading fails loudly when the
library has not been built.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libposeidon.so")

POS_OK, POS_EINVAL, POS_EOVERFLOW, POS_ENOMEM, POS_ECUDA, POS_ETIMEOUT, POS_EINFEASIBLE, \
    POS_ENOTIMPL = range(8)
STATUS_NAMES = ["POS_OK", "POS_EINVAL", "POS_EOVERFLOW", "POS_ENOMEM", "POS_ECUDA",
                "POS_ETIMEOUT", "POS_EINFEASIBLE", "POS_ENOTIMPL"]
POS_SCHED_1F1B = 0
POS_SCHED_EAGER_1F1B = 1
POS_SCHED_INTERLEAVED_1F1B = 2
POS_PLACE_FREE, POS_PLACE_EXACT, POS_PLACE_DEVICES = 0, 1, 2
MAX_STAGES = 16

# the exported entry points, as declared in include/poseidon.h
EXPORTS = ["poseidon_tables_create", "poseidon_tables_destroy", "poseidon_eval_batch",
           "poseidon_eval_batch_ex", "poseidon_eval_batch_host", "poseidon_argmin",
           "poseidon_argmin_noalloc", "poseidon_search", "poseidon_last_error"]


class pos_tables(C.Structure):
    _fields_ = [("L", C.c_int32), ("n_types", C.c_int32), ("n_tp", C.c_int32),
                ("fwd", C.c_void_p), ("bwd", C.c_void_p), ("dsync", C.c_void_p),
                ("p2p_f", C.c_void_p), ("p2p_b", C.c_void_p),
                ("mem_w", C.c_void_p), ("mem_a", C.c_void_p), ("cap", C.c_void_p)]


class pos_problem(C.Structure):
    _fields_ = [("tables", pos_tables), ("S", C.c_int32), ("n_M", C.c_int32),
                ("M_list", C.c_void_p), ("tp_list", C.c_void_p), ("dp_list", C.c_void_p),
                ("placement", C.c_int32), ("type_counts", C.c_void_p), ("warmup", C.c_int32),
                ("prune", C.c_int32), ("seed", C.c_uint64), ("schedule", C.c_int32),
                ("frontier_cap", C.c_int64), ("profile", C.c_int32), ("ridge", C.c_int32),
                ("V", C.c_int32), ("cas_limit", C.c_int32), ("n_D", C.c_int32),
                ("D_list", C.c_void_p)]


class pos_plan(C.Structure):
    _fields_ = [("found", C.c_int32), ("m_idx", C.c_int32), ("tp_idx", C.c_int32),
                ("M", C.c_int32), ("tp", C.c_int32), ("D", C.c_int32), ("S", C.c_int32),
                ("makespan", C.c_int32), ("type", C.c_int32 * MAX_STAGES),
                ("layers", C.c_int32 * MAX_STAGES), ("place_rank", C.c_uint64),
                ("map_rank", C.c_uint64), ("global_index", C.c_uint64),
                ("tp_stage", C.c_int32 * MAX_STAGES), ("d_idx", C.c_int32)]


class pos_search_stats(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in ("evaluated", "warmup_evaluated", "prefixes",
                                          "pruned_bound", "pruned_memory", "relaxations",
                                          "slices", "slices_feasible", "launches")] + \
               [(n, C.c_double) for n in ("ms_setup", "ms_warmup", "ms_search", "ms_total",
                                          "ms_expand", "ms_complete", "ms_leaf")] + \
               [(n, C.c_uint64) for n in ("expand_launches", "complete_launches",
                                          "leaf_launches", "parents_expand", "parents_complete",
                                          "leaves")] + \
               [("ms_bound", C.c_double), ("bound_launches", C.c_uint64), ("reruns", C.c_uint64),
                ("ms_depth", C.c_double * 16), ("launches_depth", C.c_uint64 * 16),
                ("parents_depth", C.c_uint64 * 16), ("children_depth", C.c_uint64 * 16),
                ("pruned_ridge", C.c_uint64)]


class PoseidonError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS_NAMES[status] if 0 <= status < 8 else status}: {msg}")
        self.status = status


_lib = None


def lib():
    """Load libposeidon.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: run __graft_entry__.build() first")
        L = C.CDLL(LIB_PATH)
        vp, i64, i32 = C.c_void_p, C.c_int64, C.c_int32
        L.poseidon_tables_create.argtypes = [C.POINTER(pos_tables), i32, C.POINTER(vp)]
        L.poseidon_tables_destroy.argtypes = [vp]
        L.poseidon_eval_batch.argtypes = [vp, vp, i64, vp, vp, vp]
        L.poseidon_eval_batch_ex.argtypes = [vp, vp, i64, vp, vp, vp]
        L.poseidon_eval_batch_host.argtypes = [vp, vp, i64, vp, vp]
        L.poseidon_argmin.argtypes = [vp, vp, i64, vp, vp]
        L.poseidon_argmin_noalloc.argtypes = [vp, vp, i64, vp, vp]
        L.poseidon_search.argtypes = [C.POINTER(pos_problem), C.POINTER(pos_plan),
                                      C.POINTER(pos_search_stats)]
        L.poseidon_last_error.restype = C.c_char_p
        L.poseidon_last_error.argtypes = []
        for name in EXPORTS[:-1]:
            getattr(L, name).restype = i32
        _lib = L
    return _lib


def _check(status):
    if status != POS_OK:
        raise PoseidonError(status, lib().poseidon_last_error().decode())


class Tables:
    """Host copies of a cost table set plus the pos_tables struct pointing at them."""

    def __init__(self, L, n_types, n_tp, fwd, bwd, dsync, p2p_f, p2p_b, mem_w, mem_a, cap):
        K = n_types * n_tp
        i32 = lambda a, s: np.ascontiguousarray(np.asarray(a, np.int32).reshape(s))  # noqa: E731
        i64 = lambda a, s: np.ascontiguousarray(np.asarray(a, np.int64).reshape(s))  # noqa: E731
        self.arrays = dict(fwd=i32(fwd, (K, L)), bwd=i32(bwd, (K, L)), dsync=i32(dsync, (K, L)),
                           p2p_f=i32(p2p_f, (K, K)), p2p_b=i32(p2p_b, (K, K)),
                           mem_w=i64(mem_w, (K, L)), mem_a=i64(mem_a, (K, L)),
                           cap=i64(cap, (K,)))
        a = self.arrays
        self.c = pos_tables(L, n_types, n_tp, *(a[n].ctypes.data for n in (
            "fwd", "bwd", "dsync", "p2p_f", "p2p_b", "mem_w", "mem_a", "cap")))

    @classmethod
    def from_workload(cls, w):
        return cls(**w.tables_dict())


class Handle:
    """poseidon_tables_create / poseidon_tables_destroy."""

    def __init__(self, tables: Tables, schedule: int = POS_SCHED_1F1B):
        self.tables = tables
        h = C.c_void_p()
        _check(lib().poseidon_tables_create(C.byref(tables.c), schedule, C.byref(h)))
        self.ptr = h

    def close(self):
        if self.ptr:
            _check(lib().poseidon_tables_destroy(self.ptr))
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def poseidon_eval_batch(handle: Handle, d_cands: int, n: int, d_makespan: int, d_feasible: int,
                        stream: int = 0):
    """Device pointers in and out (asynchronous on `stream`)."""
    _check(lib().poseidon_eval_batch(handle.ptr, d_cands, n, d_makespan, d_feasible, stream))


def poseidon_eval_batch_ex(handle: Handle, d_cands: int, n: int, d_makespan: int,
                           d_feasible: int, stream: int = 0):
    """24-byte records with a TP index per stage; device pointers in and out
    (asynchronous on `stream`)."""
    _check(lib().poseidon_eval_batch_ex(handle.ptr, d_cands, n, d_makespan, d_feasible, stream))


_probe = None


def poseidon_int32_probe(stream: int = 0):
    """(int32 ops, ms) of the relaxation microbenchmark in the measurement
    library libposeidon_probe.so (include/poseidon_probe.h)."""
    global _probe
    if _probe is None:
        path = os.path.join(os.path.dirname(LIB_PATH), "libposeidon_probe.so")
        if not os.path.exists(path):
            raise ImportError(f"{path} is missing: run __graft_entry__.build() first")
        P = C.CDLL(path)
        P.poseidon_probe_int32.restype = C.c_int
        P.poseidon_probe_int32.argtypes = [C.c_void_p, C.POINTER(C.c_int64),
                                           C.POINTER(C.c_double)]
        _probe = P
    ops, ms = C.c_int64(), C.c_double()
    rc = _probe.poseidon_probe_int32(stream, C.byref(ops), C.byref(ms))
    if rc != 0:
        raise RuntimeError(f"INT32 probe failed: cudaError {rc}")
    return ops.value, ms.value


def poseidon_eval_batch_host(handle: Handle, cands: np.ndarray):
    """Host candidates in, host (makespan, feasible) out."""
    cands = np.ascontiguousarray(cands)
    assert cands.dtype.itemsize == 16
    n = len(cands)
    T = np.zeros(n, np.int32)
    F = np.zeros(n, np.uint8)
    _check(lib().poseidon_eval_batch_host(handle.ptr, cands.ctypes.data, n, T.ctypes.data,
                                          F.ctypes.data))
    return T, F


def poseidon_argmin(d_makespan: int, d_feasible: int, n: int, d_out: int, stream: int = 0):
    _check(lib().poseidon_argmin(d_makespan, d_feasible, n, d_out, stream))


def poseidon_argmin_noalloc(d_makespan: int, d_feasible: int, n: int, d_out: int,
                            stream: int = 0):
    """poseidon_argmin without device allocation (fixed scratch in the library)."""
    _check(lib().poseidon_argmin_noalloc(d_makespan, d_feasible, n, d_out, stream))


POS_PRUNE_NONE, POS_PRUNE_EQ2, POS_PRUNE_TIGHT = 0, 1, 2


def _prune_mode(prune):
    """False/True map to POS_PRUNE_NONE/POS_PRUNE_EQ2; 0, 1, 2 pass through."""
    if isinstance(prune, bool):
        return POS_PRUNE_EQ2 if prune else POS_PRUNE_NONE
    return int(prune)


def make_problem(w, warmup=500, prune=True, seed=0, frontier_cap=0, profile=False,
                 schedule=POS_SCHED_1F1B, ridge=False, V=0, cas_limit=0):
    """pos_problem for a gen.Workload search; returns (problem, keep-alive list).
    V: model chunks per device under POS_SCHED_INTERLEAVED_1F1B; cas_limit:
    rounds of the incumbent's compare-and-swap loop (0 = the library's
    default, < 0 = none)."""
    tab = Tables.from_workload(w)
    keep = [tab]

    def arr(x):
        a = np.ascontiguousarray(np.asarray(x, np.int32))
        keep.append(a)
        return a.ctypes.data

    D_list = list(getattr(w, "D_list", None) or [])
    p = pos_problem(tab.c, w.S, len(w.M_list), arr(w.M_list), arr(w.tp_list),
                    arr(w.dp_list if w.dp_list else [1] * w.n_tp),
                    w.placement, arr(w.type_counts if w.type_counts else [0] * w.n_types),
                    int(warmup), _prune_mode(prune), int(seed), int(schedule), int(frontier_cap),
                    int(bool(profile)), int(bool(ridge)), int(V), int(cas_limit), len(D_list),
                    arr(D_list if D_list else [1]))
    return p, keep


def plan_dict(problem: pos_problem, plan: pos_plan):
    """The fields of a pos_plan as a dict (layers of the S stages, or of the
    S*V virtual stages under Interleaved 1F1B)."""
    S = problem.S
    J = S * problem.V if problem.schedule == POS_SCHED_INTERLEAVED_1F1B else S
    return dict(found=bool(plan.found), m_idx=plan.m_idx, tp_idx=plan.tp_idx, M=plan.M,
                tp=plan.tp, D=plan.D, d_idx=plan.d_idx, T=plan.makespan,
                place_rank=plan.place_rank, map_rank=plan.map_rank,
                global_index=plan.global_index, types=list(plan.type)[:S],
                tps=list(plan.tp_stage)[:S], layers=list(plan.layers)[:J])


def stats_dict(st: pos_search_stats):
    return {n: (list(getattr(st, n)) if n.endswith("_depth") else getattr(st, n))
            for n, _ in pos_search_stats._fields_}


def poseidon_search(problem: pos_problem):
    """Returns (plan dict, stats dict); raises PoseidonError on failure
    (POS_EINFEASIBLE included)."""
    plan, st = pos_plan(), pos_search_stats()
    _check(lib().poseidon_search(C.byref(problem), C.byref(plan), C.byref(st)))
    return plan_dict(problem, plan), stats_dict(st)
