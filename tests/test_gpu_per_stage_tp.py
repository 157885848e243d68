"""poseidon_eval_batch_ex (a TP index per stage) on the GPU against the
oracle, element by element, under the three schedules: makespans and flags
are integers, so the bar is bit-exact."""
import math

import numpy as np
import pytest

import gen
from tests.gpu_util import eval_device, eval_device_ex

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch
    assert torch.cuda.is_available()
    import paper_2609_06086_gb300 as P
    P.lib()
    return P


def _both(P, orc, w, cands, schedule=0):
    h = P.Handle(P.Tables.from_workload(w), schedule)
    T, F = eval_device_ex(P, h, cands)
    Tr, Fr = orc.eval_batch_ex(orc.OracleTables.from_workload(w, schedule=schedule), cands)
    return T, F, Tr, Fr


@pytest.mark.parametrize("schedule", [0, 1])
def test_random_per_stage_tp(P, orc, schedule):
    w = gen.config4()  # 3 device types x TP in {1, 2, 4, 8}
    w.cap = (np.asarray(w.cap) * 8).astype(np.int64)  # about half of the plans fit
    c = gen.per_stage_tp_candidates(40_000, L=w.L, n_types=3, n_tp=4, seed=50 + schedule,
                                    M_range=(1, 64))
    T, F, Tr, Fr = _both(P, orc, w, c, schedule)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (F == 1).sum() > 100 and (F == 0).sum() > 100


def test_interleaved_per_device_tp(P, orc):
    w = gen.config4()
    rng = np.random.default_rng(51)
    n = 8000
    c = np.zeros(n, dtype=gen.CANDIDATE_EX_DTYPE)
    base = gen.interleaved_candidates(n, L=w.L, n_types=3, seed=51, m_lo=1, m_hi=48)
    for f in ("map_rank", "type_code", "S", "M", "V"):
        c[f] = base[f]
    pc = rng.integers(0, 1 << 16, n).astype(np.uint32)
    mask = ((np.uint64(1) << (2 * base["S"].astype(np.uint64))) - np.uint64(1)).astype(np.uint32)
    c["tp_code"] = pc & mask
    T, F, Tr, Fr = _both(P, orc, w, c, 2)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_uniform_tp_code_equals_eval_batch(P):
    """The same plans as 16-byte records (one tp_idx) and as 24-byte records
    repeating it give identical outputs on the GPU."""
    w = gen.config4()
    c = gen.random_candidates(30_000, L=w.L, n_types=3, S_range=(1, 16), M_range=(1, 64), seed=52)
    tp = np.random.default_rng(52).integers(0, 4, len(c)).astype(np.uint32)
    c["tp_idx"] = tp
    ex = np.zeros(len(c), dtype=gen.CANDIDATE_EX_DTYPE)
    for f in ("map_rank", "type_code", "S", "M"):
        ex[f] = c[f]
    rep = np.zeros(len(c), np.uint32)
    for s in range(16):
        rep |= tp << np.uint32(2 * s)
    ex["tp_code"] = rep
    h = P.Handle(P.Tables.from_workload(w))
    assert all(np.array_equal(a, b) for a, b in zip(eval_device(P, h, c), eval_device_ex(P, h, ex)))


@pytest.mark.parametrize("n", [0, 1, 33, 4097])
def test_ragged_sizes(P, orc, n):
    w = gen.config4()
    c = gen.per_stage_tp_candidates(n, L=w.L, n_types=3, n_tp=4, seed=n)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_invalid_fields_and_too_many_tp_indices(P, orc):
    w = gen.config1()  # n_tp = 1
    rows = [(0, 0, 1 << 2, 2, 4, 0, 0, 0), (0, 0, 0, 2, 4, 0, 0, 0), (0, 0, 1 << 4, 2, 4, 0, 0, 0),
            (0, 2 << 2, 0, 2, 4, 0, 0, 0), (math.comb(w.L - 1, 1), 0, 0, 2, 4, 0, 0, 0)]
    c = np.array(rows, dtype=gen.CANDIDATE_EX_DTYPE)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert list(F) == [2, F[1], F[2], 2, 2] and F[1] != 2 and F[2] != 2
    w8 = gen.config4()
    w8.n_tp = 8
    K = w8.n_types * 8
    for name in ("fwd", "bwd", "dsync", "mem_w", "mem_a"):
        a = np.asarray(getattr(w8, name))
        setattr(w8, name, np.concatenate([a, a])[:K])
    w8.p2p_f = np.ones((K, K), np.int32)
    w8.p2p_b = np.ones((K, K), np.int32)
    w8.cap = np.concatenate([np.asarray(w8.cap)] * 2)[:K]
    h = P.Handle(P.Tables.from_workload(w8))
    with pytest.raises(P.PoseidonError) as e:
        eval_device_ex(P, h, c)
    assert e.value.status == P.binding.POS_EINVAL


@pytest.mark.parametrize("schedule", [0, 1, 2])
def test_limits_L127_four_types_four_tp(P, orc, schedule):
    """L = 127 with 4 types x 4 TP indices (every 2-bit TP field used), S up
    to 16 and M up to 255 (guard permitting), under each schedule."""
    from tests.test_gpu_eval import _max_tables
    tab = _max_tables(127, 4, 4, 7 + schedule)
    h = P.Handle(P.Tables(**tab), schedule)
    if schedule == 2:
        base = gen.interleaved_candidates(10_000, L=127, n_types=4, seed=8, m_lo=1, m_hi=255)
        c = np.zeros(len(base), dtype=gen.CANDIDATE_EX_DTYPE)
        for f in ("map_rank", "type_code", "S", "M", "V"):
            c[f] = base[f]
        pc = np.random.default_rng(8).integers(0, 1 << 16, len(c)).astype(np.uint32)
        mask = ((np.uint64(1) << (2 * base["S"].astype(np.uint64))) - np.uint64(1))
        c["tp_code"] = pc & mask.astype(np.uint32)
    else:
        c = gen.per_stage_tp_candidates(20_000, L=127, n_types=4, n_tp=4, seed=8,
                                        M_range=(1, 255))
        c["map_rank"][:30] = math.comb(126, 15) - 1 - np.arange(30, dtype=np.uint64)
        c["S"][:30] = 16
        c["type_code"][:30] = 0xffffffff
        c["tp_code"][:30] = 0xffffffff
    T, F = eval_device_ex(P, h, c)
    Tr, Fr = orc.eval_batch_ex(orc.OracleTables(**tab, schedule=schedule), c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (F == 1).sum() > 0
