"""Pins for the oracle's Interleaved 1F1B (Sec. 4.1.4): a hand-worked
pipeline (every finish time, the makespan and two activation peaks, one of
them reached in the steady phase, in tests/golden/interleaved_n2_v2_m4.txt),
the node and edge counts the paper gives, the V-fold smaller pipeline
bubble of uniform stages, an event-driven simulator (same device order,
written in the test from the schedule's description; it checks the DAG
arithmetic, not the order), the serial-work bound, the memory rule at
M = N, and the batch decoding of interleaved candidates."""
import os
import random

import numpy as np
import pytest

import gen

IL = 2  # ORC_SCHED_INTERLEAVED_1F1B


def chunk_tables(orc, N, V, F, B, d=None, pf=None, pb=None, act=None, wts=None, cap=None):
    """One layer per virtual stage j (cost F[j], B[j]); device d has class d;
    transfers pf/pb[j] between virtual stages j and j+1 are put on the
    (class of j's device, class of j+1's device) entries, so they must agree
    for pairs of devices that meet more than once (uniform values do)."""
    J = N * V
    fwd = np.zeros((N, J), np.int32)
    bwd = np.zeros((N, J), np.int32)
    ds = np.zeros((N, J), np.int32)
    ma = np.zeros((N, J), np.int64)
    mw = np.zeros((N, J), np.int64)
    for j in range(J):
        fwd[j % N, j], bwd[j % N, j] = F[j], B[j]
        if act is not None:
            ma[j % N, j] = act[j]
        if wts is not None:
            mw[j % N, j] = wts[j]
    if d is not None:
        for dev in range(N):
            ds[dev, dev] = d[dev]  # the device's first chunk carries its all-reduce
    p2f = np.zeros((N, N), np.int32)
    p2b = np.zeros((N, N), np.int32)
    for j in range(J - 1):
        a, b = j % N, (j + 1) % N
        if pf is not None:
            p2f[a, b] = pf[j]
        if pb is not None:
            p2b[b, a] = pb[j]
    return orc.OracleTables(L=J, n_types=N, n_tp=1, fwd=fwd, bwd=bwd, dsync=ds, p2p_f=p2f,
                            p2p_b=p2b, mem_w=mw, mem_a=ma,
                            cap=np.full(N, 1 << 40) if cap is None else cap, schedule=IL)


GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "interleaved_n2_v2_m4.txt")


def _golden():
    rows = {}
    mem = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, rest = line.split(None, 1)
            if key == "mem":
                mem.append([[int(v) for v in part.split()] for part in rest.split("|")])
            else:
                rows.setdefault(key, []).append([int(v) for v in rest.split()])
    return rows, mem


def _golden_tables(orc, rows, act=(0, 0, 0, 0), wts=(0, 0, 0, 0), cap=(1 << 40, 1 << 40)):
    """L = 4 layers, one per virtual stage; device d has class d (two types,
    one TP index); layer j is read on the class of its device j mod 2."""
    F, B = rows["F"][0], rows["B"][0]
    pf, pb = rows["pf"][0], rows["pb"][0]
    fwd = np.zeros((2, 4), np.int32)
    bwd = np.zeros((2, 4), np.int32)
    ma = np.zeros((2, 4), np.int64)
    mw = np.zeros((2, 4), np.int64)
    for j in range(4):
        fwd[j % 2, j], bwd[j % 2, j] = F[j], B[j]
        ma[j % 2, j], mw[j % 2, j] = act[j], wts[j]
    ds = np.zeros((2, 4), np.int32)
    ds[0, 0], ds[0, 2], ds[1, 1] = 1, 2, 4  # device all-reduce 3 and 4
    # F edge j -> j+1 reads p2p_f[class of j][class of j+1]; B edge j+1 -> j
    # reads p2p_b[class of j+1][class of j]; both pairs (0,1) and (1,0) occur
    p2f = np.array([[0, pf[0]], [pf[1], 0]], np.int32)
    p2b = np.array([[0, pb[1]], [pb[0], 0]], np.int32)
    assert pf[2] == pf[0] and pb[2] == pb[0]  # the 2->3 crossing reuses the 0->1 entries
    return orc.OracleTables(L=4, n_types=2, n_tp=1, fwd=fwd, bwd=bwd, dsync=ds, p2p_f=p2f,
                            p2p_b=p2b, mem_w=mw, mem_a=ma, cap=np.array(cap, np.int64),
                            schedule=IL)


def test_hand_worked_pipeline(orc):
    """Every finish time and the makespan of the hand-worked N = 2, V = 2,
    M = 4 pipeline (distinct chunk weights, transfers in both directions,
    different all-reduce times)."""
    rows, _ = _golden()
    tab = _golden_tables(orc, rows)
    T, fits, f_fin, b_fin, _ = orc.interleaved_detail(tab, 2, 2, 4, [0, 1], [1, 1, 1, 1])
    assert f_fin.tolist() == rows["Ffin"]
    assert b_fin.tolist() == rows["Bfin"]
    assert T == rows["T"][0][0] and fits
    assert rows["d"][0] == [3, 4]


def test_hand_worked_memory_peaks(orc):
    """The activation peak of each device along its order, and the capacity
    boundary: a device fits at exactly peak + weights and not one byte
    below.  The second case peaks in the steady phase (M = 2N)."""
    rows, mem = _golden()
    for act, wts, peaks, need in mem:
        tab = _golden_tables(orc, rows, act=act, wts=wts)
        _, fits, _, _, peak = orc.interleaved_detail(tab, 2, 2, 4, [0, 1], [1, 1, 1, 1])
        assert peak == peaks and fits
        for dev in range(2):
            for slack, ok in ((0, True), (-1, False)):
                cap = list(need)
                cap[dev] += slack
                tab = _golden_tables(orc, rows, act=act, wts=wts, cap=cap)
                assert orc.evaluate_interleaved(tab, 2, 2, 4, [0, 1], [1, 1, 1, 1])[1] is ok


@pytest.mark.parametrize("N,V,M", [(2, 2, 2), (2, 3, 6), (4, 2, 8), (4, 4, 4), (8, 2, 16)])
def test_node_and_edge_counts(orc, N, V, M):
    """Sec. 4.1.4: 2VNM compute nodes, 2(NV-1)M inter-stage edges and
    N(2VM-1) intra-stage edges."""
    tab = chunk_tables(orc, N, V, [1] * (N * V), [1] * (N * V))
    _, _, c = orc.evaluate_interleaved(tab, N, V, M, list(range(N)), [1] * (N * V), counts=True)
    assert c["compute_nodes"] == 2 * V * N * M
    assert c["inter_edges"] == 2 * (N * V - 1) * M
    assert c["intra_edges"] == N * (2 * V * M - 1)


def test_uniform_bubble_shrinks_by_V(orc):
    """Identical chunks (f, b each) and no transfers: (VM + N - 1)(f + b),
    i.e. the bubble of the plain pipeline, (N-1)(Vf + Vb), divided by V."""
    for N in range(1, 9):
        for V in range(2, 16 // N + 1):
            for M in (N, 2 * N, 3 * N):
                for f, b in ((3, 5), (7, 2)):
                    tab = chunk_tables(orc, N, V, [f] * (N * V), [b] * (N * V))
                    T, _ = orc.evaluate_interleaved(tab, N, V, M, list(range(N)), [1] * (N * V))
                    assert T == (V * M + N - 1) * (f + b), (N, V, M)


def device_order(N, V, M, d):
    """The interleaved schedule's device order, written from its
    description: forward number k of a device is chunk (k mod NV) div N of
    micro-batch (k div NV) N + k mod N (backwards take the chunks in
    reverse); the device first runs (N-d-1)*2 + (V-1)*N forwards (all of
    them if M = N), then a forward and a backward at a time, then the rest.
    This restates the order the oracle builds, so the simulator below pins
    the DAG arithmetic (edges, weights, longest path), not the order; the
    hand-worked pipeline and the uniform-bubble closed form pin the order."""
    total = V * M
    group = N * V

    def op(kind, k):
        c = (k % group) // N
        return (kind, (c if kind == "F" else V - 1 - c) * N + d, (k // group) * N + k % N)

    warm = total if M == N else min((N - d - 1) * 2 + (V - 1) * N, total)
    seq = [op("F", k) for k in range(warm)]
    nb = 0
    for k in range(warm, total):
        seq += [op("F", k), op("B", nb)]
        nb += 1
    return seq + [op("B", k) for k in range(nb, total)]


def simulate(N, V, M, F, B, pf, pb, d):
    """Workers with in-order programs: an op starts when its device is free
    and its input has arrived (activation of virtual stage j-1, gradient of
    virtual stage j+1); the all-reduce of a device follows its last op."""
    J = N * V
    progs = [device_order(N, V, M, dev) for dev in range(N)]
    pos, free = [0] * N, [0] * N
    fin = {}
    left = sum(len(p) for p in progs)
    while left:
        moved = False
        for dev in range(N):
            while pos[dev] < len(progs[dev]):
                kind, j, m = progs[dev][pos[dev]]
                if kind == "F":
                    src = ("F", j - 1, m) if j > 0 else None
                    edge = pf[j - 1] if j > 0 else 0
                else:
                    src = ("B", j + 1, m) if j < J - 1 else None
                    edge = pb[j] if j < J - 1 else 0
                if src is not None and src not in fin:
                    break
                ready = fin[src] + edge if src is not None else 0
                fin[(kind, j, m)] = max(free[dev], ready) + (F[j] if kind == "F" else B[j])
                free[dev] = fin[(kind, j, m)]
                pos[dev] += 1
                left -= 1
                moved = True
        assert moved, "deadlock"
    return max(free[dev] + d[dev] for dev in range(N))


def test_matches_event_simulator(orc):
    rng = random.Random(61)
    for _ in range(200):
        N = rng.randint(1, 6)
        V = rng.randint(2, max(2, 16 // N))
        if N * V > 16:
            V = 16 // N
        M = N * rng.randint(1, 4)
        J = N * V
        F = [rng.randint(1, 500) for _ in range(J)]
        B = [rng.randint(1, 900) for _ in range(J)]
        d = [rng.randint(0, 300) for _ in range(N)]
        # per device-pair transfers (a table entry serves every crossing of that pair)
        t_f = {(a, b): rng.randint(0, 200) for a in range(N) for b in range(N)}
        t_b = {(a, b): rng.randint(0, 200) for a in range(N) for b in range(N)}
        pf = [t_f[(j % N, (j + 1) % N)] for j in range(J - 1)]
        pb = [t_b[((j + 1) % N, j % N)] for j in range(J - 1)]
        tab = chunk_tables(orc, N, V, F, B, d=d, pf=pf, pb=pb)
        T, _ = orc.evaluate_interleaved(tab, N, V, M, list(range(N)), [1] * J)
        assert T == simulate(N, V, M, F, B, pf, pb, d), (N, V, M)


def test_device_work_bound_and_monotone(orc):
    rng = random.Random(62)
    for _ in range(150):
        N = rng.randint(1, 5)
        V = rng.randint(2, 16 // max(N, 1) if N > 1 else 8)
        V = max(2, min(V, 16 // N))
        M = N * rng.randint(1, 3)
        J = N * V
        F = [rng.randint(1, 300) for _ in range(J)]
        B = [rng.randint(1, 600) for _ in range(J)]
        tab = chunk_tables(orc, N, V, F, B)
        T, _ = orc.evaluate_interleaved(tab, N, V, M, list(range(N)), [1] * J)
        for dev in range(N):  # a device runs its 2VM ops one after another
            assert T >= M * sum(F[j] + B[j] for j in range(dev, J, N))
        j = rng.randrange(J)
        F2 = list(F)
        F2[j] += rng.randint(1, 100)
        T2, _ = orc.evaluate_interleaved(chunk_tables(orc, N, V, F2, B), N, V, M,
                                         list(range(N)), [1] * J)
        assert T2 >= T


def test_memory_of_the_all_warm_up_case(orc):
    """N = M = 2, V = 2: each device runs all four forwards before any
    backward, so it holds 2 micro-batches of each of its two chunks."""
    N, V, M = 2, 2, 2
    act = [10, 20, 30, 40]  # virtual stages 0, 1 (chunk 0), 2, 3 (chunk 1)
    wts = [1, 2, 3, 4]
    need = [wts[0] + wts[2] + 2 * (act[0] + act[2]), wts[1] + wts[3] + 2 * (act[1] + act[3])]
    for slack, fits in ((0, True), (-1, False)):
        cap = np.array([need[0] + slack, need[1]], np.int64)
        tab = chunk_tables(orc, N, V, [1] * 4, [1] * 4, act=act, wts=wts, cap=cap)
        assert orc.evaluate_interleaved(tab, N, V, M, [0, 1], [1] * 4)[1] is fits


def test_batch_records(orc):
    """Candidates carry V in their last byte under the interleaved schedule;
    the composition is over the N*V virtual stages; M must be a multiple of
    N and N*V at most 16."""
    w = gen.config5_tables()
    tab = orc.OracleTables.from_workload(w, schedule=IL)
    rng = np.random.default_rng(63)
    rows = []
    for _ in range(300):
        N = int(rng.integers(2, 9))
        V = int(rng.integers(2, 16 // N + 1))
        M = N * int(rng.integers(1, 6))
        J = N * V
        rank = int(rng.integers(0, orc.binom(w.L - 1, J - 1)))
        tc = int(rng.integers(0, 1 << 16)) & ((1 << (2 * N)) - 1) & 0x5555
        rows.append((rank, tc, N, M, 0, V))
    c = np.array(rows, dtype=gen.CANDIDATE_DTYPE)
    T, Fe = orc.eval_batch(tab, c)
    for (rank, tc, N, M, _, V), t, f in zip(rows, T, Fe):
        layers = orc.unrank(w.L, N * V, rank)
        cls = [(tc >> (2 * s)) & 3 for s in range(N)]
        assert (t, bool(f)) == orc.evaluate_interleaved(tab, N, V, M, cls, layers)
    bad = np.array([(0, 0, 4, 6, 0, 2), (0, 0, 4, 8, 0, 5)], dtype=gen.CANDIDATE_DTYPE)
    T, Fe = orc.eval_batch(tab, bad)  # M not a multiple of N; N*V = 20 > 16
    assert list(Fe) == [2, 2] and list(T) == [-1, -1]
