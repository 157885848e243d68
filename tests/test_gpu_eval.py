"""poseidon_eval_batch on the GPU against the oracle, element by element.
Makespans and feasibility flags are integers: the bar is bit-exact."""
import math

import numpy as np
import pytest

import gen
from tests.gpu_util import eval_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch
    assert torch.cuda.is_available()
    import paper_2609_06086_gb300 as P
    P.lib()
    return P


def _both(P, orc, w, cands):
    h = P.Handle(P.Tables.from_workload(w))
    T, F = eval_device(P, h, cands)
    Tr, Fr = orc.eval_batch(orc.OracleTables.from_workload(w), cands)
    return T, F, Tr, Fr


def test_config1_all_plans(P, orc):
    w = gen.config1()
    T, F, Tr, Fr = _both(P, orc, w, gen.all_candidates(w))
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert F.tolist().count(0) == 1


def test_config2_all_plans(P, orc):
    w = gen.config2()
    T, F, Tr, Fr = _both(P, orc, w, gen.all_candidates(w))
    assert len(T) == 215_760
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_config5_random_sample(P, orc):
    w = gen.config5_tables()
    c = gen.config5_candidates(200_000, seed=3)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_all_stage_counts_and_short_pipelines(P, orc):
    """S = 1..16 with M from 1 to 80, so both M >= S and M < S paths run."""
    w = gen.config5_tables()
    c = gen.random_candidates(60_000, L=w.L, n_types=2, S_range=(1, 16), M_range=(1, 80), seed=5)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (c["M"] < c["S"]).sum() > 1000


def test_config4_tables_three_types_and_tp(P, orc):
    w = gen.config4()
    c = gen.random_candidates(50_000, L=w.L, n_types=3, S_range=(1, 16), M_range=(1, 64), seed=9)
    c["tp_idx"] = np.random.default_rng(9).integers(0, 4, len(c))
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


@pytest.mark.parametrize("n", [0, 1, 31, 33, 2047, 2049, 4097, 10_001])
def test_ragged_sizes(P, orc, n):
    w = gen.config2()
    c = gen.random_candidates(n, L=w.L, n_types=2, seed=n)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)


def test_invalid_records_flagged(P, orc):
    w = gen.config5_tables()
    c = gen.config5_candidates(64, seed=1)
    c[0]["S"] = 0
    c[1]["S"] = 17
    c[2]["M"] = 0
    c[3]["map_rank"] = math.comb(63, int(c[3]["S"]) - 1)
    c[4]["tp_idx"] = 1
    c[5]["type_code"] |= 2  # type 2 does not exist in a 2-type table
    c[6]["S"], c[6]["map_rank"] = 16, math.comb(63, 15) - 1
    c[7]["S"], c[7]["map_rank"] = 1, 0
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert F[:6].tolist() == [2] * 6 and (T[:6] == -1).all()


def test_invalid_records_scattered(P, orc):
    """Invalid records spread over a batch that takes several decode windows
    per block: records without a sort key (S = 0, S = 17, M = 0) and records
    the decode pass rejects (rank, type or TP index out of range) sit
    between valid ones, in every window."""
    w = gen.config5_tables()
    n = 200_000
    c = gen.config5_candidates(n, seed=11)
    rng = np.random.default_rng(11)
    bad = rng.choice(n, n // 7, replace=False)
    kinds = rng.integers(0, 6, len(bad))
    for i, k in zip(bad, kinds):
        if k == 0:
            c[i]["S"] = 0
        elif k == 1:
            c[i]["S"] = 17
        elif k == 2:
            c[i]["M"] = 0
        elif k == 3:
            c[i]["map_rank"] = math.comb(63, int(c[i]["S"]) - 1)
        elif k == 4:
            c[i]["type_code"] |= 2 << (2 * int(rng.integers(0, int(c[i]["S"]))))
        else:
            c[i]["tp_idx"] = 1
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (F[bad] == 2).all() and (T[bad] == -1).all()
    assert (F != 2).sum() == n - len(bad)


def test_overflow_guard_flagged(P, orc):
    big = dict(L=4, n_types=1, n_tp=1, fwd=[[2 ** 26] * 4], bwd=[[2 ** 26] * 4],
               dsync=[[0] * 4], p2p_f=[[0]], p2p_b=[[0]], mem_w=[[0] * 4], mem_a=[[0] * 4],
               cap=[1])
    h = P.Handle(P.Tables(**big))
    c = np.zeros(4, gen.CANDIDATE_DTYPE)
    c["S"], c["M"] = 2, [1, 3, 4, 200]
    T, F = eval_device(P, h, c)
    Tr, Fr = orc.eval_batch(orc.OracleTables(**big), c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    # U(2, M) = M * 2^29: evaluable up to M = 3, flagged from M = 4
    assert F.tolist() == [1, 1, 3, 3]


def test_nondefault_stream_and_host_variant(P, orc):
    import torch
    w = gen.config2()
    c = gen.random_candidates(30_000, L=w.L, n_types=2, seed=11)
    h = P.Handle(P.Tables.from_workload(w))
    s = torch.cuda.Stream()
    T1, F1 = eval_device(P, h, c, stream=s)
    T2, F2 = P.poseidon_eval_batch_host(h, c)
    Tr, Fr = orc.eval_batch(orc.OracleTables.from_workload(w), c)
    assert np.array_equal(T1, Tr) and np.array_equal(F1, Fr)
    assert np.array_equal(T2, Tr) and np.array_equal(F2, Fr)


def test_argmin_lowest_index_on_ties(P):
    import torch
    rng = np.random.default_rng(2)
    for n in (1, 100, 70_000):
        T = rng.integers(0, 50, n).astype(np.int32)
        F = rng.integers(0, 2, n).astype(np.uint8)
        dT, dF = torch.from_numpy(T).cuda(), torch.from_numpy(F).cuda()
        out = torch.full((1,), -5, dtype=torch.int64, device="cuda")
        P.poseidon_argmin(dT.data_ptr(), dF.data_ptr(), n, out.data_ptr(),
                          torch.cuda.current_stream().cuda_stream)
        idx = np.flatnonzero(F == 1)
        want = -1 if len(idx) == 0 else int(idx[np.argmin(T[idx])])
        assert out.item() == want
    dT = torch.zeros(10, dtype=torch.int32, device="cuda")
    dF = torch.zeros(10, dtype=torch.uint8, device="cuda")
    out = torch.zeros(1, dtype=torch.int64, device="cuda")
    P.poseidon_argmin(dT.data_ptr(), dF.data_ptr(), 10, out.data_ptr(), 0)
    assert out.item() == -1


def test_config5_full_size_sampled(P, orc):
    """1e8 candidates (the largest sweep batch) in one call; 20,000 sampled
    outputs checked against the oracle."""
    import torch
    w = gen.config5_tables()
    n = 100_000_000
    c = gen.config5_candidates(n, seed=0)
    h = P.Handle(P.Tables.from_workload(w))
    d_c = torch.from_numpy(c.view(np.uint8)).cuda()
    del c
    d_T = torch.empty(n, dtype=torch.int32, device="cuda")
    d_F = torch.empty(n, dtype=torch.uint8, device="cuda")
    P.poseidon_eval_batch(h, d_c.data_ptr(), n, d_T.data_ptr(), d_F.data_ptr(),
                          torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    idx = np.sort(np.random.default_rng(4).choice(n, 20_000, replace=False))
    idx = np.concatenate([idx, [0, n - 1]])
    sample = d_c.view(-1, 16)[torch.from_numpy(idx).cuda()].cpu().numpy().view(gen.CANDIDATE_DTYPE)
    sample = sample.reshape(-1)
    Tr, Fr = orc.eval_batch(orc.OracleTables.from_workload(w), sample)
    ti = torch.from_numpy(idx).cuda()
    assert np.array_equal(d_T[ti].cpu().numpy(), Tr)
    assert np.array_equal(d_F[ti].cpu().numpy(), Fr)


def _max_tables(L, n_types, n_tp, seed):
    rng = np.random.default_rng(seed)
    K = n_types * n_tp
    return dict(L=L, n_types=n_types, n_tp=n_tp,
                fwd=rng.integers(1, 40_000, (K, L)), bwd=rng.integers(1, 80_000, (K, L)),
                dsync=rng.integers(0, 500, (K, L)), p2p_f=rng.integers(0, 300, (K, K)),
                p2p_b=rng.integers(0, 300, (K, K)), mem_w=rng.integers(0, 10 ** 9, (K, L)),
                mem_a=rng.integers(0, 10 ** 8, (K, L)),
                cap=rng.integers(10 ** 9, 10 ** 11, K))


def test_limits_L127_four_types_eight_tp(P, orc):
    """The largest tables the ABI accepts: L = 127 (ranks up to C(126, 15) ~ 1.2e19),
    4 device types x 8 TP degrees, S up to 16 and M up to 255 (guard permitting)."""
    tab = _max_tables(127, 4, 8, 3)
    h = P.Handle(P.Tables(**tab))
    c = gen.random_candidates(40_000, L=127, n_types=4, S_range=(1, 16), M_range=(1, 255),
                              seed=3)
    c["tp_idx"] = np.random.default_rng(4).integers(0, 8, len(c))
    c[:100]["S"] = 16
    c[:50]["map_rank"] = math.comb(126, 15) - 1 - np.arange(50, dtype=np.uint64)
    T, F = eval_device(P, h, c)
    Tr, Fr = orc.eval_batch(orc.OracleTables(**tab), c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert (F == 3).sum() > 0 and (F == 1).sum() > 0


def test_int32_probe_runs_near_the_lane_count(P):
    """The relaxation microbenchmark executes its stated op count; its rate
    is within a plausible band of SMs x 128 lanes x the maximum clock."""
    import torch
    ops, ms = P.binding.poseidon_int32_probe(torch.cuda.current_stream().cuda_stream)
    props = torch.cuda.get_device_properties(0)
    nominal = props.multi_processor_count * 128 * 2.07e9
    rate = ops / (ms / 1e3)
    assert ops == props.multi_processor_count * 8 * 256 * 4096 * 8 * 6
    assert 0.2 * nominal < rate < 1.5 * nominal, rate / nominal


@pytest.mark.parametrize("schedule", [0, 1])
def test_memory_check_at_the_capacity_boundary(P, orc, schedule):
    """Unit memory rows (mem_w = 1, mem_a = 1 per layer) make a stage's need
    l + W*l exactly, so small integer capacities put many stages exactly on,
    one above and one below the limit: the byte table of the decode pass
    must agree with the oracle's direct check (need <= cap) everywhere."""
    w = gen.config5_tables()
    K = w.n_types * w.n_tp
    w.mem_w = np.ones((K, w.L), np.int64)
    w.mem_a = np.ones((K, w.L), np.int64)
    w.cap = np.array([90, 150], np.int64)[:K]
    c = gen.random_candidates(60_000, L=w.L, n_types=2, S_range=(2, 16), M_range=(1, 40),
                              seed=17)
    h = P.Handle(P.Tables.from_workload(w), schedule)
    T, F = eval_device(P, h, c)
    Tr, Fr = orc.eval_batch(orc.OracleTables.from_workload(w, schedule=schedule), c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
    assert 0.05 < (F == 1).mean() < 0.95


def test_config3_whole_space_sample(P, orc):
    """Plans drawn uniformly from config 3's whole space (the bench's
    config-3 evaluator line), memory-feasible or not."""
    w = gen.config3()
    c = gen.search_space_sample(w, 50_000, seed=7)
    T, F, Tr, Fr = _both(P, orc, w, c)
    assert np.array_equal(T, Tr) and np.array_equal(F, Fr)
