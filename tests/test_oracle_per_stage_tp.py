"""Pins for the oracle's records with a TP index per stage (the per-stage
heterogeneous TP of Table 1's Metis and HexiScale plans): stage s runs on
class type_s * n_tp + tp_s, so its node weights (Sec. 4.1.3), its
transfers (indexed by the two stages' classes), its all-reduce and its
memory (Sec. 3.2) all come from that class."""
import math

import numpy as np
import pytest

import gen


def _ex(rows):
    return np.array([r + (0, 0) for r in rows], dtype=gen.CANDIDATE_EX_DTYPE)


def test_uniform_tp_code_equals_the_standard_record(orc):
    """A tp_code that repeats one TP index in every field gives exactly the
    result of the 16-byte record with that tp_idx."""
    w = gen.config4()
    tab = orc.OracleTables.from_workload(w)
    c = gen.random_candidates(3000, L=w.L, n_types=3, S_range=(1, 16), M_range=(1, 40), seed=4)
    tp = np.random.default_rng(4).integers(0, 4, len(c))
    c["tp_idx"] = tp
    ex = np.zeros(len(c), dtype=gen.CANDIDATE_EX_DTYPE)
    for f in ("map_rank", "type_code", "S", "M"):
        ex[f] = c[f]
    rep = np.zeros(len(c), np.uint32)
    for s in range(16):
        rep |= (tp.astype(np.uint32) << np.uint32(2 * s))
    ex["tp_code"] = rep  # fields beyond S are ignored
    T, F = orc.eval_batch(tab, c)
    Te, Fe = orc.eval_batch_ex(tab, ex)
    assert np.array_equal(T, Te) and np.array_equal(F, Fe)


def test_records_decode_to_per_stage_classes(orc):
    """Each record equals the evaluation of its unranked layers with class
    type_s * n_tp + tp_s on stage s."""
    w = gen.config4()
    tab = orc.OracleTables.from_workload(w)
    c = gen.per_stage_tp_candidates(400, L=w.L, n_types=3, n_tp=4, seed=7, M_range=(1, 24))
    T, F = orc.eval_batch_ex(tab, c)
    for r, t, f in zip(c, T, F):
        S, M = int(r["S"]), int(r["M"])
        layers = orc.unrank(w.L, S, int(r["map_rank"]))
        cls = [((int(r["type_code"]) >> (2 * s)) & 3) * w.n_tp + ((int(r["tp_code"]) >> (2 * s)) & 3)
               for s in range(S)]
        assert (t, bool(f)) == orc.evaluate(tab, S, M, cls, layers)
    mixed = [len({(int(r["tp_code"]) >> (2 * s)) & 3 for s in range(int(r["S"]))}) > 1 for r in c]
    assert sum(mixed) > 300


def test_single_micro_batch_chain_by_hand(orc):
    """M = 1 is a chain (the closed form of Sec. 4.1 for one micro-batch):
    T = max_s (sum_i F_i + sum_{i<N} pf_i + sum_{i>=s} B_i + sum_{s<=i<N} pb_i + d_s),
    computed here from the raw per-layer rows of each stage's own class."""
    w = gen.config4()
    tab = orc.OracleTables.from_workload(w)
    fwd, bwd, ds = (np.asarray(x, np.int64) for x in (w.fwd, w.bwd, w.dsync))
    p2f, p2b = np.asarray(w.p2p_f, np.int64), np.asarray(w.p2p_b, np.int64)
    rng = np.random.default_rng(3)
    for _ in range(40):
        S = int(rng.integers(2, 7))
        layers = [int(x) for x in rng.multinomial(w.L - S, [1 / S] * S) + 1]
        types = [int(x) for x in rng.integers(0, 3, S)]
        tps = [int(x) for x in rng.integers(0, 4, S)]
        cls = [ty * w.n_tp + tp for ty, tp in zip(types, tps)]
        bounds = np.cumsum([0] + layers)
        F = [int(fwd[k, bounds[s]:bounds[s + 1]].sum()) for s, k in enumerate(cls)]
        B = [int(bwd[k, bounds[s]:bounds[s + 1]].sum()) for s, k in enumerate(cls)]
        d = [int(ds[k, bounds[s]:bounds[s + 1]].sum()) for s, k in enumerate(cls)]
        pf = [int(p2f[cls[s], cls[s + 1]]) for s in range(S - 1)]
        pb = [int(p2b[cls[s + 1], cls[s]]) for s in range(S - 1)]
        expect = max(sum(F) + sum(pf) + sum(B[s:]) + sum(pb[s:]) + d[s] for s in range(S))
        tc = sum(t << (2 * s) for s, t in enumerate(types))
        pc = sum(t << (2 * s) for s, t in enumerate(tps))
        rank = orc.rank(w.L, S, layers)
        T, F_ = orc.eval_batch_ex(tab, _ex([(rank, tc, pc, S, 1, 0)]))
        assert T[0] == expect


def test_invalid_tp_fields_and_too_many_tp_indices(orc):
    w = gen.config1()  # n_tp = 1: every field must be 0
    tab = orc.OracleTables.from_workload(w)
    T, F = orc.eval_batch_ex(tab, _ex([(0, 0, 1 << 2, 2, 4, 0), (0, 0, 0, 2, 4, 0),
                                       (0, 0, 1 << 4, 2, 4, 0)]))
    assert list(F[:1]) == [2] and F[1] != 2 and F[2] != 2  # stage 2 does not exist
    w8 = gen.config4()
    w8.n_tp = 8
    K = w8.n_types * 8
    for name in ("fwd", "bwd", "dsync", "mem_w", "mem_a"):
        a = np.asarray(getattr(w8, name))
        setattr(w8, name, np.concatenate([a, a])[:K])
    w8.p2p_f = np.ones((K, K), np.int32)
    w8.p2p_b = np.ones((K, K), np.int32)
    w8.cap = np.concatenate([np.asarray(w8.cap)] * 2)[:K]
    with pytest.raises(RuntimeError):
        orc.eval_batch_ex(orc.OracleTables.from_workload(w8), _ex([(0, 0, 0, 2, 4, 0)]))


def test_interleaved_records_take_a_tp_index_per_device(orc):
    w = gen.config4()
    tab = orc.OracleTables.from_workload(w, schedule=2)
    rng = np.random.default_rng(9)
    rows = []
    for _ in range(60):
        N = int(rng.integers(1, 5))
        V = int(rng.integers(2, 16 // N + 1))
        M = N * int(rng.integers(1, 4))
        rank = int(rng.integers(0, math.comb(w.L - 1, N * V - 1)))
        tc = sum(int(rng.integers(0, 3)) << (2 * s) for s in range(N))
        pc = sum(int(rng.integers(0, 4)) << (2 * s) for s in range(N))
        rows.append((rank, tc, pc, N, M, V))
    T, F = orc.eval_batch_ex(tab, _ex(rows))
    for (rank, tc, pc, N, M, V), t, f in zip(rows, T, F):
        layers = orc.unrank(w.L, N * V, rank)
        cls = [((tc >> (2 * s)) & 3) * w.n_tp + ((pc >> (2 * s)) & 3) for s in range(N)]
        assert (t, bool(f)) == orc.evaluate_interleaved(tab, N, V, M, cls, layers)
