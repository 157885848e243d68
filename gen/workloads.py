"""Seeded synthetic cost tables and candidate batches.

The paper's inputs are profiled per-layer forward/backward/all-reduce times,
activation-transfer times and memory footprints per (device type, TP degree)
(Sec. 4.1.3 and Sec. 3.2).  Those profiles, models and clusters are not
available, so every workload here is synthetic, drawn with numpy's PCG64
``default_rng(seed)`` in the order documented in each function.  The shapes
follow the paper's settings (7B/13B/70B-class models, 2-3 device types,
Sec. 6.1 and Sec. 6.5.3).

Common formulas (documented once, used by configs 2-5):

* layer forward FLOPs (micro-batch 1)  = 24*s*h^2 + 4*s^2*h
* compute_us = FLOPs / (TFLOPS*1e12*t) * 1e6 * exp(0.1*z), z ~ N(0,1) per
  (type, layer), shared across TP degrees t
* fwd = compute_us (+ 2 TP all-reduces), bwd = 2*compute_us (+ 2 TP all-reduces)
* TP all-reduce of s*h*2 bytes: ring time 2(t-1)/t * bytes / 300 GB/s
* dsync per layer = 2 * (12*h^2 * 2 / t bytes) / 100 GB/s
* P2P per micro-batch = s*h*2 bytes at 25 GB/s between stages of the same
  device type, 9.375 GB/s across types (the paper's 200 / 75 Gbps links)
* mem_w per layer = 16 * 12*h^2 / t bytes (bf16 weights, fp32 master, Adam)
* mem_a per layer per micro-batch = 34*s*h / t bytes
* cap = GB * 1e9
* rounding: us = floor(x + 0.5); max(1, .) for compute, max(0, .) for comm

Class index k = type * n_tp + tp_idx.  Tables are [K][L] (int32 us or int64
bytes), [K][K] for P2P (indexed src class, dst class) and [K] for capacity.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from itertools import permutations, product

import numpy as np

# pos_candidate layout (16 bytes): u64 map_rank, u32 type_code (2 bits per
# stage, stage 1 in the low bits), u8 S, u8 M, u8 tp_idx, u8 V (model chunks
# per device under Interleaved 1F1B; 0 otherwise).
CANDIDATE_DTYPE = np.dtype([("map_rank", "<u8"), ("type_code", "<u4"), ("S", "u1"),
                            ("M", "u1"), ("tp_idx", "u1"), ("V", "u1")])
assert CANDIDATE_DTYPE.itemsize == 16

# pos_candidate_ex layout (24 bytes): u64 map_rank, u32 type_code, u32 tp_code
# (TP index of stage s in bits [2s, 2s+2)), u8 S, u8 M, u8 V, u8 pad, u32 pad.
CANDIDATE_EX_DTYPE = np.dtype([("map_rank", "<u8"), ("type_code", "<u4"), ("tp_code", "<u4"),
                               ("S", "u1"), ("M", "u1"), ("V", "u1"), ("pad0", "u1"),
                               ("pad1", "<u4")])
assert CANDIDATE_EX_DTYPE.itemsize == 24

PLACE_FREE = 0
PLACE_EXACT = 1
PLACE_DEVICES = 2  # a (type, TP index) per stage; type_counts = devices per type


@dataclass
class Workload:
    name: str
    L: int
    n_types: int
    n_tp: int
    fwd: np.ndarray          # [K][L] int32 us
    bwd: np.ndarray          # [K][L] int32 us
    dsync: np.ndarray        # [K][L] int32 us
    p2p_f: np.ndarray        # [K][K] int32 us, src class -> dst class
    p2p_b: np.ndarray        # [K][K] int32 us, src class -> dst class
    mem_w: np.ndarray        # [K][L] int64 bytes
    mem_a: np.ndarray        # [K][L] int64 bytes per in-flight micro-batch
    cap: np.ndarray          # [K] int64 bytes
    # search problem (configs 1-4); S=0 for evaluator-only tables
    S: int = 0
    M_list: list = field(default_factory=list)
    tp_list: list = field(default_factory=list)
    dp_list: list = field(default_factory=list)
    placement: int = PLACE_FREE
    type_counts: list = field(default_factory=list)   # stages (EXACT) / devices (DEVICES) per type
    D_list: list = field(default_factory=list)        # data-parallel degrees (DEVICES)
    seed: int = 0

    @property
    def K(self) -> int:
        return self.n_types * self.n_tp

    def tables_dict(self):
        return dict(L=self.L, n_types=self.n_types, n_tp=self.n_tp, fwd=self.fwd, bwd=self.bwd,
                    dsync=self.dsync, p2p_f=self.p2p_f, p2p_b=self.p2p_b, mem_w=self.mem_w,
                    mem_a=self.mem_a, cap=self.cap)


def n_compositions(L: int, S: int) -> int:
    """Number of compositions of L layers into S non-empty stages."""
    if S < 1 or S > L:
        return 0
    return math.comb(L - 1, S - 1)


def _round_us(x, lo):
    return np.maximum(lo, np.floor(np.asarray(x, dtype=np.float64) + 0.5)).astype(np.int64)


def _as_i32(a):
    a = np.asarray(a, dtype=np.int64)
    assert a.min() >= -(2 ** 31) and a.max() < 2 ** 31
    return np.ascontiguousarray(a.astype(np.int32))


def _layer_flops(s, h):
    return 24.0 * s * h * h + 4.0 * s * s * h


def _llm_tables(rng, *, L, h, seq, tflops, gbs, tp_list, tp_comm, name, seed):
    """Tables for configs 2-5.  Draw order: z[type][layer] ~ N(0,1)."""
    T = len(tflops)
    n_tp = len(tp_list)
    K = T * n_tp
    z = rng.standard_normal((T, L))
    flops = _layer_flops(seq, h)
    fwd = np.zeros((K, L), np.int64)
    bwd = np.zeros((K, L), np.int64)
    dsync = np.zeros((K, L), np.int64)
    mem_w = np.zeros((K, L), np.int64)
    mem_a = np.zeros((K, L), np.int64)
    cap = np.zeros(K, np.int64)
    act_bytes = seq * h * 2.0
    for ty in range(T):
        for j, t in enumerate(tp_list):
            k = ty * n_tp + j
            comp = flops / (tflops[ty] * 1e12 * t) * 1e6 * np.exp(0.1 * z[ty])
            ar = 0.0
            if tp_comm and t > 1:
                ar = 2.0 * (t - 1) / t * act_bytes / 300e9 * 1e6
            fwd[k] = _round_us(comp + 2 * ar, 1)
            bwd[k] = _round_us(2 * comp + 2 * ar, 1)
            dsync[k] = _round_us(np.full(L, 2.0 * (12.0 * h * h * 2.0 / t) / 100e9 * 1e6), 0)
            mem_w[k] = int(16 * 12 * h * h // t)
            mem_a[k] = int(34 * seq * h // t)
            cap[k] = int(gbs[ty] * 1e9)
    p2p = np.zeros((K, K), np.int64)
    same = act_bytes / 25e9 * 1e6
    cross = act_bytes / 9.375e9 * 1e6
    for a in range(K):
        for b in range(K):
            p2p[a, b] = _round_us(same if a // n_tp == b // n_tp else cross, 0)
    return Workload(name=name, L=L, n_types=T, n_tp=n_tp, fwd=_as_i32(fwd), bwd=_as_i32(bwd),
                    dsync=_as_i32(dsync), p2p_f=_as_i32(p2p), p2p_b=_as_i32(p2p.copy()),
                    mem_w=mem_w, mem_a=mem_a, cap=cap, tp_list=list(tp_list), seed=seed)


def config1(seed: int = 0) -> Workload:
    """Tiny search: L=8, S=2, M=4, D=t=1, types A (40 GB) and B (16 GB).

    Draw order: fwd_A ~ U{800..1200}[L]; mult ~ U[1.5,2.5)[L];
    noise ~ U{-50..50}[2][L]; p2p_f ~ U{50..200}[2][2]; p2p_b ~ U{50..200}[2][2].
    """
    rng = np.random.default_rng(seed)
    L = 8
    fa = rng.integers(800, 1201, size=L).astype(np.int64)
    mult = rng.uniform(1.5, 2.5, size=L)
    fb = np.floor(fa * mult + 0.5).astype(np.int64)
    noise = rng.integers(-50, 51, size=(2, L)).astype(np.int64)
    fwd = np.stack([fa, fb])
    bwd = 2 * fwd + noise
    p2p_f = rng.integers(50, 201, size=(2, 2)).astype(np.int64)
    p2p_b = rng.integers(50, 201, size=(2, 2)).astype(np.int64)
    mem_w = np.full((2, L), 1_500_000_000, np.int64)
    mem_a = np.full((2, L), 400_000_000, np.int64)
    cap = np.array([40_000_000_000, 16_000_000_000], np.int64)
    return Workload(name="tiny L=8 S=2 M=4 (2 types, 14 candidates)", L=L, n_types=2, n_tp=1,
                    fwd=_as_i32(fwd), bwd=_as_i32(bwd), dsync=_as_i32(np.zeros((2, L))),
                    p2p_f=_as_i32(p2p_f), p2p_b=_as_i32(p2p_b), mem_w=mem_w, mem_a=mem_a, cap=cap,
                    S=2, M_list=[4], tp_list=[1], dp_list=[1], placement=PLACE_EXACT,
                    type_counts=[1, 1], seed=seed)


def config2(seed: int = 0) -> Workload:
    """7B-like: L=32, h=4096, S=4, M in {8,16,32}, D=t=1, free placement (2^4)."""
    rng = np.random.default_rng(seed)
    w = _llm_tables(rng, L=32, h=4096, seq=4096, tflops=[312, 125], gbs=[80, 32], tp_list=[1],
                    tp_comm=False, name="7B-like L=32 S=4 M={8,16,32} (2 types, free placement)",
                    seed=seed)
    w.S, w.M_list, w.dp_list, w.placement, w.type_counts = 4, [8, 16, 32], [1], PLACE_FREE, []
    return w


def config3(seed: int = 0) -> Workload:
    """Deep pipeline: L=48, h=5120, S=8, M=64, D=t=1, exactly 4 A + 4 B stages."""
    rng = np.random.default_rng(seed)
    w = _llm_tables(rng, L=48, h=5120, seq=4096, tflops=[312, 125], gbs=[80, 32], tp_list=[1],
                    tp_comm=False, name="deep L=48 S=8 M=64 (4 A + 4 B stages)", seed=seed)
    w.S, w.M_list, w.dp_list, w.placement, w.type_counts = 8, [64], [1], PLACE_EXACT, [4, 4]
    return w


def config4(seed: int = 0) -> Workload:
    """70B-like heterogeneous search: L=80, h=8192, S=8, M=32, 3 device types
    (312/125/65 TFLOPS, 80/32/16 GB, 32/32/64 devices), t in {1,2,4,8}, D=16/t,
    stage-type counts (2,2,4) so that n_type * D * t = devices_type."""
    rng = np.random.default_rng(seed)
    tps = [1, 2, 4, 8]
    w = _llm_tables(rng, L=80, h=8192, seq=4096, tflops=[312, 125, 65], gbs=[80, 32, 16],
                    tp_list=tps, tp_comm=True,
                    name="70B-like L=80 S=8 M=32 (3 types, t in {1,2,4,8}, D=16/t)", seed=seed)
    w.S, w.M_list, w.dp_list = 8, [32], [16 // t for t in tps]
    w.placement, w.type_counts = PLACE_EXACT, [2, 2, 4]
    return w


def config4_per_stage_tp(seed: int = 0) -> Workload:
    """Config 4's tables and cluster with a TP degree chosen per stage:
    D in {2, 4, 8, 16}, and the stages of each type use exactly its devices
    (32/32/64): sum over its stages of D * t = devices (PLACE_DEVICES)."""
    w = config4(seed)
    w.name = "70B-like L=80 S=8 M=32 (3 types, per-stage t in {1,2,4,8}, D in {2,4,8,16})"
    w.placement, w.type_counts, w.D_list = PLACE_DEVICES, [32, 32, 64], [2, 4, 8, 16]
    return w


def config5_tables(seed: int = 0) -> Workload:
    """Evaluator sweep tables: L=64, 7B-like costs (h=4096), 2 types, t=1."""
    rng = np.random.default_rng(seed)
    return _llm_tables(rng, L=64, h=4096, seq=4096, tflops=[312, 125], gbs=[80, 32], tp_list=[1],
                       tp_comm=False, name="sweep L=64 (7B-like costs, 2 types)", seed=seed)


def random_candidates(n: int, *, L: int, n_types: int, S_range=(2, 16), M_range=(8, 128),
                      seed: int = 0, chunk: int = 1 << 20) -> np.ndarray:
    """n random pre-encoded candidates: S ~ U{S_range}, M ~ U{M_range}, stage
    types i.i.d. uniform over n_types, map_rank ~ U[0, C(L-1, S-1)).

    Generated in chunks of ``chunk`` records; chunk i uses
    ``default_rng(SeedSequence(seed).spawn(...)[i])`` and draws, in order,
    S[n], M[n], raw type bits u32[n] and map_rank[n].
    """
    out = np.empty(n, CANDIDATE_DTYPE)
    n_chunks = max(1, (n + chunk - 1) // chunk)
    children = np.random.SeedSequence(seed).spawn(n_chunks)
    highs = np.zeros(17, np.uint64)
    for S in range(1, 17):
        highs[S] = max(1, n_compositions(L, S))
    for i in range(n_chunks):
        lo, hi = i * chunk, min(n, (i + 1) * chunk)
        m = hi - lo
        if m <= 0:
            break
        rng = np.random.default_rng(children[i])
        S = rng.integers(S_range[0], S_range[1] + 1, size=m)
        M = rng.integers(M_range[0], M_range[1] + 1, size=m)
        if n_types <= 2:
            bits = rng.integers(0, 2 ** 32, size=m, dtype=np.uint64).astype(np.uint32)
            tc = bits & np.uint32(0x55555555 if n_types == 2 else 0)
        else:
            ty = rng.integers(0, n_types, size=(m, 16)).astype(np.uint32)
            tc = np.zeros(m, np.uint32)
            for s in range(16):
                tc |= ty[:, s] << np.uint32(2 * s)
        mask = np.where(S >= 16, np.uint64(0xFFFFFFFF),
                        (np.uint64(1) << (2 * S).astype(np.uint64)) - np.uint64(1)).astype(np.uint32)
        tc = tc & mask
        rank = rng.integers(0, highs[S], size=m, dtype=np.uint64)
        o = out[lo:hi]
        o["map_rank"] = rank
        o["type_code"] = tc
        o["S"] = S.astype(np.uint8)
        o["M"] = M.astype(np.uint8)
        o["tp_idx"] = 0
        o["V"] = 0
    return out


def per_stage_tp_candidates(n: int, L: int, n_types: int, n_tp: int, seed: int = 0,
                            S_range=(1, 16), M_range=(1, 64)) -> np.ndarray:
    """Records with a TP index per stage, drawn in this order: S ~ U{S_range},
    M ~ U{M_range}, 16 types and 16 TP indices i.i.d. uniform (fields beyond
    S cleared), and the composition rank uniform in [0, C(L-1, S-1)) from a
    64-bit draw."""
    rng = np.random.default_rng(seed)
    S = rng.integers(S_range[0], S_range[1] + 1, size=n)
    S = np.minimum(S, L)
    M = rng.integers(M_range[0], M_range[1] + 1, size=n)
    ty = rng.integers(0, n_types, size=(n, 16)).astype(np.uint32)
    tp = rng.integers(0, n_tp, size=(n, 16)).astype(np.uint32)
    tc = np.zeros(n, np.uint32)
    pc = np.zeros(n, np.uint32)
    for s in range(16):
        keep = s < S
        tc |= np.where(keep, ty[:, s] << np.uint32(2 * s), 0).astype(np.uint32)
        pc |= np.where(keep, tp[:, s] << np.uint32(2 * s), 0).astype(np.uint32)
    u = rng.integers(0, np.iinfo(np.uint64).max, size=n, dtype=np.uint64, endpoint=True)
    highs = np.array([math.comb(L - 1, k - 1) if 1 <= k <= L else 1 for k in range(17)],
                     dtype=np.uint64)  # C(126, 15) < 2^64
    rank = u % highs[S]
    out = np.zeros(n, dtype=CANDIDATE_EX_DTYPE)
    out["map_rank"] = rank
    out["type_code"] = tc
    out["tp_code"] = pc
    out["S"] = S.astype(np.uint8)
    out["M"] = M.astype(np.uint8)
    return out


def search_space_sample(w: Workload, n: int, seed: int = 0) -> np.ndarray:
    """n plans drawn uniformly from a search workload's whole space (every
    slice and composition, memory-feasible or not), in this order: the
    M index, the TP index, the placement rank, then the composition rank
    from a 64-bit draw."""
    rng = np.random.default_rng(seed)
    places = np.array([type_code_of(p) for p in place_list(w)], dtype=np.uint32)
    mi = rng.integers(0, len(w.M_list), size=n)
    ti = rng.integers(0, w.n_tp, size=n)
    pi = rng.integers(0, len(places), size=n)
    u = rng.integers(0, np.iinfo(np.uint64).max, size=n, dtype=np.uint64, endpoint=True)
    out = np.zeros(n, dtype=CANDIDATE_DTYPE)
    out["map_rank"] = u % np.uint64(math.comb(w.L - 1, w.S - 1))
    out["type_code"] = places[pi]
    out["S"] = w.S
    out["M"] = np.asarray(w.M_list, np.uint8)[mi]
    out["tp_idx"] = ti.astype(np.uint8)
    return out


def interleaved_candidates(n: int, L: int = 64, n_types: int = 2, seed: int = 0,
                           m_lo: int = 8, m_hi: int = 128) -> np.ndarray:
    """Interleaved 1F1B batch (Sec. 4.1.4): per record, in this draw order,
    N ~ U{1..8} devices, V ~ U{2..16//N} chunks per device, M ~ U{m_lo..m_hi}
    rounded down to a multiple of N (at least N), the N device types i.i.d.
    uniform, and the rank of the composition of L into the N*V virtual
    stages uniform in [0, C(L-1, N*V-1)) from a 64-bit draw."""
    rng = np.random.default_rng(seed)
    N = rng.integers(1, 9, size=n)
    V = 2 + (rng.random(n) * (16 // N - 1)).astype(np.int64)
    M = rng.integers(m_lo, m_hi + 1, size=n)
    M = np.maximum(N, (M // N) * N)
    ty = rng.integers(0, n_types, size=(n, 8)).astype(np.uint32)
    tc = np.zeros(n, np.uint32)
    for s in range(8):
        tc |= np.where(s < N, ty[:, s] << np.uint32(2 * s), 0).astype(np.uint32)
    u = rng.integers(0, np.iinfo(np.uint64).max, size=n, dtype=np.uint64, endpoint=True)
    J = N * V
    highs = np.array([math.comb(L - 1, j - 1) if 1 <= j <= L else 1 for j in range(17)],
                     dtype=np.uint64)  # C(126, 15) < 2^64
    rank = u % highs[J]
    out = np.zeros(n, dtype=CANDIDATE_DTYPE)
    out["map_rank"] = rank
    out["type_code"] = tc
    out["S"] = N.astype(np.uint8)
    out["M"] = M.astype(np.uint8)
    out["V"] = V.astype(np.uint8)
    return out


def config5_candidates(n: int, seed: int = 0) -> np.ndarray:
    """Config-5 batch: L=64, S ~ U{2..16}, M ~ U{8..128}, 2 types."""
    return random_candidates(n, L=64, n_types=2, seed=seed)


def place_list(w: Workload):
    """Allowed stage-type sequences in lexicographic order (type ids 0..T-1).

    FREE: every sequence in T^S.  EXACT: sequences whose type counts equal
    ``w.type_counts``.  The position in this list is the placement rank.
    """
    seqs = []
    for seq in product(range(w.n_types), repeat=w.S):
        if w.placement == PLACE_EXACT:
            if any(seq.count(t) != w.type_counts[t] for t in range(w.n_types)):
                continue
        seqs.append(seq)
    return seqs


def type_code_of(seq) -> int:
    code = 0
    for s, t in enumerate(seq):
        code |= int(t) << (2 * s)
    return code


def all_candidates(w: Workload) -> np.ndarray:
    """Every (M, tp, placement, map_rank) of a search workload, in global-index
    order: (((m_idx*n_tp + tp_idx)*n_place + place_rank)*n_map + map_rank)."""
    places = place_list(w)
    n_map = n_compositions(w.L, w.S)
    n = len(w.M_list) * w.n_tp * len(places) * n_map
    out = np.zeros(n, CANDIDATE_DTYPE)
    i = 0
    for M in w.M_list:
        for tp_idx in range(w.n_tp):
            for seq in places:
                o = out[i:i + n_map]
                o["map_rank"] = np.arange(n_map, dtype=np.uint64)
                o["type_code"] = type_code_of(seq)
                o["S"] = w.S
                o["M"] = M
                o["tp_idx"] = tp_idx
                i += n_map
    return out


def get_config(i: int, seed: int = 0) -> Workload:
    return {1: config1, 2: config2, 3: config3, 4: config4, 5: config5_tables}[i](seed)
