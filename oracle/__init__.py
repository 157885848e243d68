"""ctypes binding of the CPU oracle (oracle.c) -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU baseline
may import this module.  It builds ``liboracle.so`` with gcc on first use and
never touches the CUDA library.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_SO = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

MAX_S = 16


SCHED_1F1B, SCHED_EAGER_1F1B, SCHED_INTERLEAVED_1F1B = 0, 1, 2


class Tables(C.Structure):
    _fields_ = [("L", C.c_int32), ("n_types", C.c_int32), ("n_tp", C.c_int32),
                ("fwd", C.c_void_p), ("bwd", C.c_void_p), ("dsync", C.c_void_p),
                ("p2p_f", C.c_void_p), ("p2p_b", C.c_void_p),
                ("mem_w", C.c_void_p), ("mem_a", C.c_void_p), ("cap", C.c_void_p),
                ("schedule", C.c_int32)]


class Problem(C.Structure):
    _fields_ = [("tab", Tables), ("S", C.c_int32), ("n_M", C.c_int32), ("M_list", C.c_void_p),
                ("dp_list", C.c_void_p), ("placement", C.c_int32), ("type_counts", C.c_void_p),
                ("ridge", C.c_int32), ("tp_list", C.c_void_p), ("n_D", C.c_int32),
                ("D_list", C.c_void_p)]


class Plan(C.Structure):
    _fields_ = [("found", C.c_int32), ("m_idx", C.c_int32), ("tp_idx", C.c_int32),
                ("M", C.c_int32), ("D", C.c_int32), ("T", C.c_int32),
                ("place_rank", C.c_uint64), ("map_rank", C.c_uint64),
                ("global_index", C.c_uint64),
                ("types", C.c_int32 * MAX_S), ("layers", C.c_int32 * MAX_S),
                ("tps", C.c_int32 * MAX_S), ("d_idx", C.c_int32)]


class Stats(C.Structure):
    _fields_ = [("leaves_evaluated", C.c_uint64), ("prefixes_pruned", C.c_uint64),
                ("prefixes_memory", C.c_uint64), ("warmup_evaluated", C.c_uint64),
                ("prefixes_ridge", C.c_uint64)]


class DagCounts(C.Structure):
    _fields_ = [(n, C.c_int64) for n in ("nodes", "compute_nodes", "allreduce_nodes",
                                         "control_nodes", "inter_edges", "intra_edges",
                                         "allreduce_edges", "aux_edges")]


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (plain C99, -O2)."""
    with _lock:
        if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < max(
                os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "oracle.h"))):
            tmp = _SO + f".tmp{os.getpid()}"
            subprocess.check_call(["gcc", "-std=c99", "-O2", "-Wall", "-Wextra", "-shared", "-fPIC",
                                   "-o", tmp, _SRC])
            os.replace(tmp, _SO)
    return _SO


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(_SO)
        L.orc_binom.restype = C.c_uint64
        L.orc_binom.argtypes = [C.c_int, C.c_int]
        L.orc_unrank.restype = C.c_int
        L.orc_unrank.argtypes = [C.c_int, C.c_int, C.c_uint64, C.c_void_p]
        L.orc_rank.restype = C.c_uint64
        L.orc_rank.argtypes = [C.c_int, C.c_int, C.c_void_p]
        L.orc_eval.restype = C.c_int
        L.orc_eval.argtypes = [C.POINTER(Tables), C.c_int, C.c_int, C.c_void_p, C.c_void_p,
                               C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.POINTER(DagCounts)]
        L.orc_eval_finish.restype = C.c_int
        L.orc_eval_finish.argtypes = [C.POINTER(Tables), C.c_int, C.c_int, C.c_void_p,
                                      C.c_void_p, C.c_void_p]
        L.orc_lower_bound.restype = C.c_int64
        L.orc_lower_bound.argtypes = [C.POINTER(Tables), C.c_int, C.c_int, C.c_void_p,
                                      C.c_void_p, C.c_int]
        L.orc_lower_bound_tight.restype = C.c_int64
        L.orc_lower_bound_tight.argtypes = [C.POINTER(Tables), C.c_int, C.c_int, C.c_void_p,
                                            C.c_void_p, C.c_int]
        L.orc_eval_interleaved.restype = C.c_int
        L.orc_eval_interleaved.argtypes = [C.POINTER(Tables), C.c_int, C.c_int, C.c_int,
                                           C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                           C.c_void_p]
        L.orc_eval_interleaved_detail.restype = C.c_int
        L.orc_eval_interleaved_detail.argtypes = [C.POINTER(Tables), C.c_int, C.c_int, C.c_int,
                                                  C.c_void_p, C.c_void_p, C.c_void_p,
                                                  C.c_void_p, C.c_void_p, C.c_void_p]
        L.orc_search_interleaved.restype = C.c_int
        L.orc_search_interleaved.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_void_p,
                                             C.c_void_p]
        L.orc_eval_batch_ex.restype = C.c_int
        L.orc_eval_batch_ex.argtypes = [C.POINTER(Tables), C.c_void_p, C.c_int64, C.c_void_p,
                                        C.c_void_p]
        L.orc_eval_batch.restype = C.c_int
        L.orc_eval_batch.argtypes = [C.POINTER(Tables), C.c_void_p, C.c_int64, C.c_void_p,
                                     C.c_void_p]
        L.orc_search.restype = C.c_int
        L.orc_search.argtypes = [C.POINTER(Problem), C.c_int, C.c_int, C.c_uint64,
                                 C.POINTER(Plan), C.POINTER(Stats)]
        L.orc_search_part.restype = C.c_int
        L.orc_search_part.argtypes = [C.POINTER(Problem), C.c_int, C.c_int, C.c_uint64,
                                      C.c_int, C.c_int, C.POINTER(Plan), C.POINTER(Stats)]
        _lib = L
    return _lib


class OracleTables:
    """Holds contiguous copies of a workload's tables and the ctypes struct."""

    def __init__(self, L, n_types, n_tp, fwd, bwd, dsync, p2p_f, p2p_b, mem_w, mem_a, cap,
                 schedule=SCHED_1F1B):
        K = n_types * n_tp
        i32 = lambda a, shp: np.ascontiguousarray(np.asarray(a, np.int32).reshape(shp))  # noqa: E731
        i64 = lambda a, shp: np.ascontiguousarray(np.asarray(a, np.int64).reshape(shp))  # noqa: E731
        self.arrays = dict(fwd=i32(fwd, (K, L)), bwd=i32(bwd, (K, L)), dsync=i32(dsync, (K, L)),
                           p2p_f=i32(p2p_f, (K, K)), p2p_b=i32(p2p_b, (K, K)),
                           mem_w=i64(mem_w, (K, L)), mem_a=i64(mem_a, (K, L)), cap=i64(cap, (K,)))
        self.L, self.n_types, self.n_tp, self.schedule = L, n_types, n_tp, schedule
        a = self.arrays
        self.c = Tables(L, n_types, n_tp, *(a[n].ctypes.data for n in
                                            ("fwd", "bwd", "dsync", "p2p_f", "p2p_b", "mem_w",
                                             "mem_a", "cap")), schedule)

    @classmethod
    def from_workload(cls, w, schedule=SCHED_1F1B):
        return cls(**w.tables_dict(), schedule=schedule)


def _i32(x, n=None):
    a = np.ascontiguousarray(np.asarray(x, np.int32))
    assert n is None or a.size == n
    return a


def binom(n, k):
    return int(lib().orc_binom(n, k))


def unrank(L, S, rank):
    out = np.zeros(S, np.int32)
    rc = lib().orc_unrank(L, S, C.c_uint64(rank), out.ctypes.data)
    if rc:
        raise ValueError("rank out of range")
    return out.tolist()


def rank(L, S, layers):
    a = _i32(layers, S)
    return int(lib().orc_rank(L, S, a.ctypes.data))


def evaluate(tab: OracleTables, S, M, cls, layers, counts=False):
    """Makespan (us) and memory feasibility of one configuration."""
    c, l = _i32(cls, S), _i32(layers, S)
    T, F = C.c_int32(), C.c_int32()
    dc = DagCounts()
    rc = lib().orc_eval(C.byref(tab.c), S, M, c.ctypes.data, l.ctypes.data, C.byref(T),
                        C.byref(F), C.byref(dc))
    if rc:
        raise ValueError("invalid configuration")
    if counts:
        return T.value, bool(F.value), {n: getattr(dc, n) for n, _ in DagCounts._fields_}
    return T.value, bool(F.value)


def finish_times(tab: OracleTables, S, M, cls, layers):
    """Finish times of every F_{s,m} and B_{s,m}: arrays [S][M] (0-based)."""
    c, l = _i32(cls, S), _i32(layers, S)
    out = np.zeros(2 * S * M, np.int32)
    if lib().orc_eval_finish(C.byref(tab.c), S, M, c.ctypes.data, l.ctypes.data,
                             out.ctypes.data):
        raise ValueError("invalid configuration")
    return out[:S * M].reshape(S, M), out[S * M:].reshape(S, M)


def lower_bound(tab: OracleTables, S, M, cls, layers, x):
    c, l = _i32(cls, S), _i32(layers, S)
    g = lib().orc_lower_bound(C.byref(tab.c), S, M, c.ctypes.data, l.ctypes.data, x)
    if g < 0:
        raise ValueError("invalid configuration")
    return int(g)


def evaluate_interleaved(tab: OracleTables, N, V, M, cls, layers, counts=False):
    """Interleaved 1F1B: makespan and memory feasibility of N devices with
    V chunks each; layers has N*V entries (virtual stages in model order)."""
    c, l = _i32(cls, N), _i32(layers, N * V)
    T, F = C.c_int32(), C.c_int32()
    dc = DagCounts()
    rc = lib().orc_eval_interleaved(C.byref(tab.c), N, V, M, c.ctypes.data, l.ctypes.data,
                                    C.byref(T), C.byref(F), C.byref(dc))
    if rc:
        raise ValueError("invalid configuration")
    if counts:
        return T.value, bool(F.value), {n: getattr(dc, n) for n, _ in DagCounts._fields_}
    return T.value, bool(F.value)


def interleaved_detail(tab: OracleTables, N, V, M, cls, layers):
    """Interleaved 1F1B with every compute node's finish time and each
    device's activation peak: (T, feasible, F finish [NV][M], B finish
    [NV][M], peak [N])."""
    J = N * V
    c, l = _i32(cls, N), _i32(layers, J)
    T, F = C.c_int32(), C.c_int32()
    fin = np.zeros(2 * J * M, np.int32)
    peak = np.zeros(N, np.int64)
    rc = lib().orc_eval_interleaved_detail(C.byref(tab.c), N, V, M, c.ctypes.data, l.ctypes.data,
                                           C.byref(T), C.byref(F), fin.ctypes.data,
                                           peak.ctypes.data)
    if rc:
        raise ValueError("invalid configuration")
    return (T.value, bool(F.value), fin[:J * M].reshape(J, M), fin[J * M:].reshape(J, M),
            peak.tolist())


def lower_bound_tight(tab: OracleTables, S, M, cls, layers, x):
    """Tightened prefix bound (P2P-inclusive Eq. 2 plus the completion
    terms); None when no memory-feasible completion exists."""
    c, l = _i32(cls, S), _i32(layers, S)
    g = lib().orc_lower_bound_tight(C.byref(tab.c), S, M, c.ctypes.data, l.ctypes.data, x)
    if g == -2:
        return None
    if g < 0:
        raise ValueError("invalid configuration")
    return int(g)


def eval_batch(tab: OracleTables, cands: np.ndarray):
    """Evaluate a structured array of 16-byte candidate records."""
    cands = np.ascontiguousarray(cands)
    assert cands.dtype.itemsize == 16
    n = len(cands)
    T = np.zeros(n, np.int32)
    F = np.zeros(n, np.uint8)
    if lib().orc_eval_batch(C.byref(tab.c), cands.ctypes.data, n, T.ctypes.data, F.ctypes.data):
        raise RuntimeError("oracle eval_batch failed")
    return T, F


def eval_batch_ex(tab: OracleTables, cands: np.ndarray):
    """Evaluate a structured array of 24-byte records with a TP index per
    stage (bits [2s, 2s+2) of tp_code)."""
    cands = np.ascontiguousarray(cands)
    assert cands.dtype.itemsize == 24
    n = len(cands)
    T = np.zeros(n, np.int32)
    F = np.zeros(n, np.uint8)
    if lib().orc_eval_batch_ex(C.byref(tab.c), cands.ctypes.data, n, T.ctypes.data,
                               F.ctypes.data):
        raise RuntimeError("oracle eval_batch_ex failed (n_tp > 4?)")
    return T, F


def _problem(w, tab, ridge):
    """Problem struct for a gen.Workload and the arrays it points into."""
    keep = [_i32(w.M_list), _i32(w.dp_list if w.dp_list else [1] * w.n_tp),
            _i32(w.type_counts if w.type_counts else [0] * w.n_types),
            _i32(w.tp_list if w.tp_list else [1] * w.n_tp),
            _i32(w.D_list if w.D_list else [1])]
    M_list, dp, tc, tpl, Dl = keep
    p = Problem(tab.c, w.S, len(M_list), M_list.ctypes.data, dp.ctypes.data, w.placement,
                tc.ctypes.data, int(bool(ridge)), tpl.ctypes.data, len(Dl), Dl.ctypes.data)
    return p, keep


def _plan_dict(plan, n_units, n_layers):
    return dict(found=bool(plan.found), m_idx=plan.m_idx, tp_idx=plan.tp_idx,
                d_idx=plan.d_idx, M=plan.M, D=plan.D, T=plan.T, place_rank=plan.place_rank,
                map_rank=plan.map_rank, global_index=plan.global_index,
                types=list(plan.types)[:n_units], tps=list(plan.tps)[:n_units],
                layers=list(plan.layers)[:n_layers])


def search(w, prune=True, warmup=0, seed=0, tab: OracleTables | None = None,
           schedule=SCHED_1F1B, ridge=False, part=0, n_parts=1):
    """Exact search over a gen.Workload search problem.  Returns (plan dict, stats dict).
    With n_parts > 1 only the slices whose global-order index is part
    (mod n_parts) are searched (orc_search_part)."""
    tab = tab or OracleTables.from_workload(w, schedule)
    p, keep = _problem(w, tab, ridge)
    plan, st = Plan(), Stats()
    rc = lib().orc_search_part(C.byref(p), int(prune), int(warmup), C.c_uint64(seed), int(part),
                               int(n_parts), C.byref(plan), C.byref(st))
    if rc == -2:
        raise OverflowError("overflow guard")
    if rc:
        raise RuntimeError("oracle search failed")
    out = _plan_dict(plan, w.S, w.S)
    stats = {n: getattr(st, n) for n, _ in Stats._fields_}
    return out, stats


def search_interleaved(w, V, prune=True, tab: OracleTables | None = None):
    """Search over Interleaved 1F1B plans with V chunks per device (w.S
    devices).  Returns (plan dict, stats dict); layers has N*V entries."""
    tab = tab or OracleTables.from_workload(w, SCHED_INTERLEAVED_1F1B)
    p, keep = _problem(w, tab, False)
    plan, st = Plan(), Stats()
    rc = lib().orc_search_interleaved(C.byref(p), int(V), int(prune), C.byref(plan),
                                      C.byref(st))
    if rc == -2:
        raise OverflowError("overflow guard")
    if rc:
        raise RuntimeError("oracle interleaved search failed")
    out = _plan_dict(plan, w.S, w.S * V)
    return out, {n: getattr(st, n) for n, _ in Stats._fields_}

