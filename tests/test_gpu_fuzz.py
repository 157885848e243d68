"""Randomised small tables and records under every schedule, GPU against
the oracle element by element: degenerate shapes (one layer, one type, one
TP index, S = L, M = 1), zero costs and transfers, zero or huge capacities,
and records of both formats mixed with invalid ones."""
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


def _tables(rng):
    L = int(rng.choice([1, 2, 3, 5, 8, 13, 16, 20]))
    n_types = int(rng.integers(1, 5))
    n_tp = int(rng.integers(1, 5))
    K = n_types * n_tp
    zero = rng.random() < 0.2

    def costs(hi, shape):
        a = rng.integers(0, hi, shape)
        if zero:
            a[rng.random(shape) < 0.5] = 0
        return a
    cap_kind = rng.integers(0, 3)
    cap = (np.zeros(K, np.int64) if cap_kind == 0 else
           np.full(K, 1 << 50, np.int64) if cap_kind == 1 else
           rng.integers(0, 2000, K))
    return dict(L=L, n_types=n_types, n_tp=n_tp, fwd=costs(500, (K, L)), bwd=costs(900, (K, L)),
                dsync=costs(300, (K, L)), p2p_f=costs(200, (K, K)), p2p_b=costs(200, (K, K)),
                mem_w=rng.integers(0, 100, (K, L)), mem_a=rng.integers(0, 60, (K, L)), cap=cap)


def _records(rng, tab, n, schedule):
    L, T_, n_tp = tab["L"], tab["n_types"], tab["n_tp"]
    rows = []
    for _ in range(n):
        if schedule == 2 and rng.random() < 0.6:
            N = int(rng.integers(1, 5))
            V = int(rng.integers(2, 6))
            M = N * int(rng.integers(1, 5))
            J = N * V
        else:
            N = int(rng.integers(1, min(L, 16) + 1))
            V = int(rng.integers(0, 2))
            M = int(rng.integers(1, 40))
            J = N
        rank = int(rng.integers(0, math.comb(L - 1, J - 1))) if J <= L else 0
        tc = sum(int(rng.integers(0, T_)) << (2 * s) for s in range(min(N, 16)))
        tp = int(rng.integers(0, n_tp))
        rows.append((rank, tc, N, M, tp, V))
    # a few invalid ones
    rows += [(0, 0, 0, 4, 0, 0), (0, 0, 1, 0, 0, 0), (math.comb(L - 1, 0), 0, 1, 3, 0, 0),
             (0, 0, 1, 3, n_tp, 0)]
    return np.array(rows, dtype=gen.CANDIDATE_DTYPE)


@pytest.mark.parametrize("schedule", [0, 1, 2])
def test_random_small_tables(P, orc, schedule):
    rng = np.random.default_rng(1000 + schedule)
    for trial in range(40):
        tab = _tables(rng)
        c = _records(rng, tab, 300, schedule)
        h = P.Handle(P.Tables(**tab), schedule)
        T, F = eval_device(P, h, c)
        Tr, Fr = orc.eval_batch(orc.OracleTables(**tab, schedule=schedule), c)
        assert np.array_equal(T, Tr) and np.array_equal(F, Fr), trial
        if tab["n_tp"] <= 4:
            ex = np.zeros(len(c), dtype=gen.CANDIDATE_EX_DTYPE)
            for f in ("map_rank", "type_code", "S", "M", "V"):
                ex[f] = c[f]
            ex["tp_code"] = [sum(int(rng.integers(0, tab["n_tp"])) << (2 * s)
                                 for s in range(min(int(n), 16))) for n in c["S"]]
            Te, Fe = eval_device_ex(P, h, ex)
            Tre, Fre = orc.eval_batch_ex(orc.OracleTables(**tab, schedule=schedule), ex)
            assert np.array_equal(Te, Tre) and np.array_equal(Fe, Fre), trial
        h.close()
