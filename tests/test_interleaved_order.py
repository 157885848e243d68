"""Host-side checks of the Interleaved 1F1B visiting order that the GPU
makespan kernel unrolls (paper_2609_06086_gb300/csrc/interleaved_order.h):
the header is what its generator writes, and running its op lists with one
register per (virtual stage, kind) and one clock per device -- the kernel's
state -- reproduces the oracle's longest path (Sec. 4.1.4) for every (N, V)
and several group counts q = M/N.  The activation-peak rule of the kernel
(warm-up plus one steady period) is re-checked against the oracle's flag."""
import importlib.util
import os
import re

import numpy as np
import pytest

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_2609_06086_gb300", "csrc")
IL = 2


def _load_generator():
    spec = importlib.util.spec_from_file_location(
        "gen_interleaved_order", os.path.join(CSRC, "gen_interleaved_order.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _parse_header():
    text = open(os.path.join(CSRC, "interleaved_order.h")).read()
    out = {}
    for m in re.finditer(r"struct IlOrder<(\d+), (\d+)> \{(.*?)\n\};", text, re.S):
        N, V, body = int(m.group(1)), int(m.group(2)), m.group(3)
        d = {"q0": int(re.search(r"q0 = (\d+)", body).group(1))}
        for name in ("P", "Body", "E", "Short"):
            n = int(re.search(rf"int n{name} = (\d+);", body).group(1))
            vals = re.search(rf"uint8_t {name}\[\d+\] = \{{([^}}]*)\}}", body).group(1)
            d[name] = [int(x) for x in vals.split(",")][:n]
        out[(N, V)] = d
    return out


ORDERS = _parse_header()


@pytest.mark.slow
def test_header_matches_generator():
    assert _load_generator().render() == open(os.path.join(CSRC, "interleaved_order.h")).read()


def test_every_pair_present():
    assert sorted(ORDERS) == sorted((N, V) for N in range(1, 9) for V in range(2, 17)
                                    if N * V <= 16)


def _ops(N, V, q):
    o = ORDERS[(N, V)]
    if q < o["q0"]:
        return o["Short"]
    return o["P"] + o["Body"] * (q - o["q0"]) + o["E"]


def _emulate(N, V, q, F, B, pf, pb, dsum):
    """The kernel's register wavefront over the op list."""
    J = N * V
    Fo, Bo, clk = [0] * J, [0] * J, [0] * N
    ops = _ops(N, V, q)
    assert len(ops) == 2 * J * q * N
    for op in ops:
        j, d = op & 15, (op & 15) % N
        if op & 0x80:
            t = clk[d] if j + 1 == J else max(clk[d], Bo[j + 1] + pb[d])
            Bo[j] = clk[d] = t + B[j]
        else:
            t = clk[d] if j == 0 else max(clk[d], Fo[j - 1] + pf[(j - 1) % N])
            Fo[j] = clk[d] = t + F[j]
    return max(clk[d] + dsum[d] for d in range(N))


def _peak_rule(N, V, q, act):
    """The kernel's activation peak of every device: act[j] per virtual stage."""
    NV = N * V
    peaks = []
    for d in range(N):
        a = [act[c * N + d] for c in range(V)]
        if q == 1:
            peaks.append(N * sum(a))
            continue
        w = 2 * (N - d - 1) + (V - 1) * N
        held = sum(a[(k % NV) // N] for k in range(w))
        steps = NV if (q >= 3 or 2 * NV - w >= NV) else 2 * NV - w
        peak = 0
        for i in range(steps):
            held += a[((w + i) % NV) // N]
            peak = max(peak, held)
            held -= a[V - 1 - (i % NV) // N]
        peaks.append(peak)
    return peaks


def _peak_runs(N, V, q, act):
    """The kernel's computation of the same peaks: the warm-up sum from
    per-chunk forward counts, then the steady pairs in runs of a fixed
    (forward chunk, backward chunk), each run's extreme at one of its ends."""
    NV = N * V
    peaks = []
    for d in range(N):
        a = [act[c * N + d] for c in range(V)]
        if q == 1:
            peaks.append(N * sum(a))
            continue
        w = 2 * (N - d - 1) + (V - 1) * N

        def count(k, c):
            part = k % NV - c * N
            return (k // NV) * N + min(max(part, 0), N)
        held = sum(count(w, c) * a[c] for c in range(V))
        steps = NV if (q >= 3 or 2 * NV - w >= NV) else 2 * NV - w
        peak, h0, first = 0, 0, 0
        for i in range(steps):
            aF, aB = a[((w + i) % NV) // N], a[V - 1 - (i % NV) // N]
            if i == 0 or (w + i) % N == 0 or i % N == 0:
                h0, first = held + aF, i
            if i == steps - 1 or (w + i + 1) % N == 0 or (i + 1) % N == 0:
                span = (i - first) * (aF - aB)
                peak = max(peak, h0, h0 + span)
                held = h0 + span - aB
        peaks.append(peak)
    return peaks


@pytest.mark.parametrize("NV", sorted(ORDERS))
def test_peak_runs_equal_the_step_rule(NV):
    N, V = NV
    rng = np.random.default_rng(7 * N + V)
    for q in (1, 2, 3, 4):
        for _ in range(20):
            act = [int(x) for x in rng.integers(0, 10 ** 9, N * V)]
            assert _peak_runs(N, V, q, act) == _peak_rule(N, V, q, act)


@pytest.mark.parametrize("NV", sorted(ORDERS))
def test_emulated_kernel_matches_oracle(orc, NV):
    N, V = NV
    J = N * V
    rng = np.random.default_rng(100 * N + V)
    for q in sorted({1, 2, 3, 4, 255 // N if N > 2 else 9}):
        for _ in range(3):
            # one layer per virtual stage; device d has class d
            F = rng.integers(1, 400, J)
            B = rng.integers(1, 800, J)
            pf = rng.integers(0, 150, N)
            pb = rng.integers(0, 150, N)
            ds = rng.integers(0, 300, N)
            act = rng.integers(0, 1000, J)
            fwd = np.zeros((N, J), np.int32)
            bwd = np.zeros((N, J), np.int32)
            dsync = np.zeros((N, J), np.int32)
            ma = np.zeros((N, J), np.int64)
            for j in range(J):
                fwd[j % N, j], bwd[j % N, j], ma[j % N, j] = F[j], B[j], act[j]
            for d in range(N):
                dsync[d, d] = ds[d]
            p2f = np.zeros((N, N), np.int32)
            p2b = np.zeros((N, N), np.int32)
            for d in range(N):
                p2f[d, (d + 1) % N] = pf[d]
                p2b[(d + 1) % N, d] = pb[d]
            peaks = _peak_rule(N, V, q, act)
            cap = np.array(peaks, np.int64) + rng.integers(-1, 2, N)  # on, above or below
            tab = orc.OracleTables(L=J, n_types=N, n_tp=1, fwd=fwd, bwd=bwd, dsync=dsync,
                                   p2p_f=p2f, p2p_b=p2b, mem_w=np.zeros((N, J), np.int64),
                                   mem_a=ma, cap=cap, schedule=IL)
            T, fe = orc.evaluate_interleaved(tab, N, V, q * N, list(range(N)), [1] * J)
            assert T == _emulate(N, V, q, F, B, pf, pb, ds)
            assert fe == all(peaks[d] <= cap[d] for d in range(N))
