"""poseidon_eval_batch under Interleaved 1F1B (Sec. 4.1.4) on the GPU against
the oracle, element by element: makespans and feasibility flags are
integers, so the bar is bit-exact."""
import math

import numpy as np
import pytest

import gen
from tests.gpu_util import eval_device

pytestmark = pytest.mark.gpu

IL = 2  # POS_SCHED_INTERLEAVED_1F1B


@pytest.fixture(scope="module")
def P():
    import torch
    assert torch.cuda.is_available()
    import paper_2609_06086_gb300 as P
    P.lib()
    return P


def _both(P, orc, w, cands, tab=None):
    h = P.Handle(P.Tables.from_workload(w) if tab is None else tab, IL)
    T, F = eval_device(P, h, cands)
    Tr, Fr = orc.eval_batch(orc.OracleTables.from_workload(w, schedule=IL), cands)
    return T, F, Tr, Fr


def _pairs():
    return [(N, V) for N in range(1, 9) for V in range(2, 17) if N * V <= 16]


def _records(rng, L, n_types, N, V, M, k):
    J = N * V
    rows = []
    for _ in range(k):
        rank = int(rng.integers(0, math.comb(L - 1, J - 1)))
        tc = 0
        for s in range(N):
            tc |= int(rng.integers(0, n_types)) << (2 * s)
        rows.append((rank, tc, N, M, 0, V))
    return rows


def test_random_interleaved_batch(P, orc):
    """Mixed N, V and M (the interleaved sweep recipe) on the config-5 tables,
    with 1F1B records (V = 0 and V = 1) mixed in."""
    w = gen.config5_tables()
    c = gen.interleaved_candidates(30_000, L=w.L, seed=11)
    c1 = gen.config5_candidates(6_000, seed=12)
    c1["V"][::2] = 1
    c = np.concatenate([c, c1])
    np.random.default_rng(13).shuffle(c)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (F[c["V"] >= 2] != 2).all() and (T > 0).all()


def test_every_pair_and_group_count(P, orc):
    """Every (N, V) with N*V <= 16, at q = M/N = 1 (all forwards first), 2
    and 3 (the periodic order's first cases), 5, and the largest q with
    M <= 255: the short list, the prologue/epilogue and repeated bodies."""
    w = gen.config5_tables()
    rng = np.random.default_rng(21)
    rows = []
    for N, V in _pairs():
        for q in sorted({1, 2, 3, 5, 255 // N}):
            rows += _records(rng, w.L, 2, N, V, q * N, 6)
    c = np.array(rows, dtype=gen.CANDIDATE_DTYPE)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_memory_flags_near_capacity(P, orc):
    """Capacities raised 4x so that about half of the plans fit: the
    per-device activation peak decides the flag."""
    w = gen.config5_tables()
    w.cap = (np.asarray(w.cap) * 4).astype(np.int64)
    c = gen.interleaved_candidates(20_000, L=w.L, seed=31, m_lo=2, m_hi=64)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    frac = (F == 0).mean()
    assert 0.1 < frac < 0.9, frac


def test_three_types_and_tp(P, orc):
    w = gen.config4()
    c = gen.interleaved_candidates(12_000, L=w.L, n_types=3, seed=41, m_lo=1, m_hi=48)
    c["tp_idx"] = np.random.default_rng(41).integers(0, 4, len(c))
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


@pytest.mark.parametrize("n", [1, 31, 33, 4097])
def test_ragged_sizes(P, orc, n):
    w = gen.config2()
    c = gen.interleaved_candidates(n, L=w.L, seed=n)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_invalid_and_overflow_records(P, orc):
    w = gen.config5_tables()
    good = _records(np.random.default_rng(5), w.L, 2, 4, 2, 8, 1)[0]
    rows = [
        (0, 0, 4, 6, 0, 2),        # M not a multiple of N
        (0, 0, 4, 8, 0, 5),        # N*V = 20 > 16 virtual stages
        (0, 0, 0, 8, 0, 2),        # no device
        (0, 0, 2, 0, 0, 2),        # M = 0
        (math.comb(w.L - 1, 7), 0, 4, 8, 0, 2),  # rank beyond C(L-1, J-1)
        (0, 3 << 2, 4, 8, 0, 2),   # type 3 of 2
        (0, 0, 4, 8, 1, 2),        # tp_idx beyond n_tp
        good,
    ]
    c = np.array(rows, dtype=gen.CANDIDATE_DTYPE)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert list(F[:7]) == [2] * 7 and F[7] in (0, 1)

    # more virtual stages than layers
    ws = gen.config1()  # L = 8
    c = np.array([(0, 0, 2, 4, 0, 4), (0, 0, 2, 4, 0, 5), (0, 0, 1, 3, 0, 8)],
                 dtype=gen.CANDIDATE_DTYPE)
    T, F, Tr, Fr = _both(P, orc, ws, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert F[1] == 2 and F[0] != 2 and F[2] != 2

    # overflow guard over the N*V virtual stages
    wo = gen.config5_tables()
    wo.fwd = (np.asarray(wo.fwd) * 40).astype(np.int32)
    wo.bwd = (np.asarray(wo.bwd) * 40).astype(np.int32)
    c = np.array(_records(np.random.default_rng(6), wo.L, 2, 2, 4, 200, 4) +
                 _records(np.random.default_rng(7), wo.L, 2, 2, 4, 2, 4),
                 dtype=gen.CANDIDATE_DTYPE)
    T, F, Tr, Fr = _both(P, orc, wo, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (F == 3).sum() == 4


def test_one_device_is_sequential(P, orc):
    """N = 1 with free transfers: one device runs every chunk in sequence, so
    T = M (sum F + sum B) + d."""
    w = gen.config5_tables()
    w.p2p_f = np.zeros_like(w.p2p_f)
    w.p2p_b = np.zeros_like(w.p2p_b)
    rng = np.random.default_rng(8)
    rows = []
    for V in (2, 5, 16):
        rows += _records(rng, w.L, 2, 1, V, 7, 3)
    c = np.array(rows, dtype=gen.CANDIDATE_DTYPE)
    T, F, _, _ = _both(P, orc, w, c)
    fwd, bwd, ds = (np.asarray(x, np.int64) for x in (w.fwd, w.bwd, w.dsync))
    for (rank, tc, N, M, _, V), t in zip(rows, T):
        k = tc & 3
        assert t == M * int(fwd[k].sum() + bwd[k].sum()) + int(ds[k].sum())


def test_limits_L127_four_types_eight_tp(P, orc):
    """The largest tables the ABI accepts under Interleaved 1F1B: L = 127,
    4 types x 8 TP degrees, N*V up to 16 (ranks near C(126, 15)), M up to 255."""
    from tests.test_gpu_eval import _max_tables
    tab = _max_tables(127, 4, 8, 5)
    h = P.Handle(P.Tables(**tab), IL)
    c = gen.interleaved_candidates(20_000, L=127, n_types=4, seed=6, m_lo=1, m_hi=255)
    c["tp_idx"] = np.random.default_rng(6).integers(0, 8, len(c))
    J = c["S"].astype(np.int64) * c["V"].astype(np.int64)
    top = np.nonzero(J == 16)[0][:40]
    c["map_rank"][top] = math.comb(126, 15) - 1 - np.arange(len(top), dtype=np.uint64)
    T, F = eval_device(P, h, c)
    Tr, Fr = orc.eval_batch(orc.OracleTables(**tab, schedule=IL), c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (F == 3).sum() > 0 and (F == 1).sum() > 0


def test_bench_size_sampled(P, orc):
    """The bench's interleaved batch (1e7 records, one call); 20,000 sampled
    outputs checked against the oracle."""
    import torch
    w = gen.config5_tables()
    n = 10_000_000
    c = gen.interleaved_candidates(n, L=w.L, seed=0)
    h = P.Handle(P.Tables.from_workload(w), IL)
    d_c = torch.from_numpy(c.view(np.uint8)).cuda()
    d_T = torch.empty(n, dtype=torch.int32, device="cuda")
    d_F = torch.empty(n, dtype=torch.uint8, device="cuda")
    P.poseidon_eval_batch(h, d_c.data_ptr(), n, d_T.data_ptr(), d_F.data_ptr(),
                          torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    idx = np.sort(np.random.default_rng(5).choice(n, 20_000, replace=False))
    idx = np.concatenate([idx, [0, n - 1]])
    Tr, Fr = orc.eval_batch(orc.OracleTables.from_workload(w, schedule=IL), c[idx])
    ti = torch.from_numpy(idx).cuda()
    assert np.array_equal(d_T[ti].cpu().numpy(), Tr)
    assert np.array_equal(d_F[ti].cpu().numpy(), Fr)
