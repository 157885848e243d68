"""The C ABI without a GPU: the library loads, exports every entry point
that include/poseidon.h declares, the ctypes structs match the C layout, and
argument validation rejects bad input before touching the device."""
import ctypes as C
import os
import re
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "poseidon.h")


@pytest.fixture(scope="module")
def P():
    from paper_2609_06086_gb300 import build
    build.build()
    import paper_2609_06086_gb300 as P
    P.lib()
    return P


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:pos_status|const char \*)\s*(poseidon_\w+)\(", text,
                                 re.M)))


def test_header_declares_the_binding(P):
    assert declared_functions() == sorted(P.EXPORTS)


def test_every_declared_symbol_is_exported(P):
    out = subprocess.run(["nm", "-D", "--defined-only", P.binding.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    syms = set(re.findall(r"\bT (\w+)", out))
    for f in declared_functions():
        assert f in syms, f


def test_struct_layouts_match_the_header(P, tmp_path):
    prog = tmp_path / "layout.c"
    fields = {
        "pos_tables": [f[0] for f in P.binding.pos_tables._fields_],
        "pos_candidate": ["map_rank", "type_code", "S", "M", "tp_idx", "V"],
        "pos_candidate_ex": ["map_rank", "type_code", "tp_code", "S", "M", "V", "pad0", "pad1"],
        "pos_problem": [f[0] for f in P.binding.pos_problem._fields_],
        "pos_plan": [f[0] for f in P.binding.pos_plan._fields_],
        "pos_search_stats": [f[0] for f in P.binding.pos_search_stats._fields_],
    }
    lines = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HEADER}"',
             "int main(void) {"]
    for st, fs in fields.items():
        lines.append(f'printf("{st} %zu\\n", sizeof({st}));')
        for f in fs:
            lines.append(f'printf("{st}.{f} %zu\\n", offsetof({st}, {f}));')
    lines += ["return 0;", "}"]
    prog.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-o", str(exe), str(prog)], check=True)
    got = dict(l.split() for l in subprocess.run([str(exe)], capture_output=True, text=True,
                                                  check=True).stdout.splitlines())
    import gen
    py = {"pos_tables": P.binding.pos_tables, "pos_problem": P.binding.pos_problem,
          "pos_plan": P.binding.pos_plan, "pos_search_stats": P.binding.pos_search_stats}
    for st, cls in py.items():
        assert int(got[st]) == C.sizeof(cls), st
        for f in fields[st]:
            assert int(got[f"{st}.{f}"]) == getattr(cls, f).offset, (st, f)
    assert int(got["pos_candidate"]) == gen.CANDIDATE_DTYPE.itemsize
    for f in fields["pos_candidate"]:
        assert int(got[f"pos_candidate.{f}"]) == gen.CANDIDATE_DTYPE.fields[f][1], f
    assert int(got["pos_candidate_ex"]) == gen.CANDIDATE_EX_DTYPE.itemsize
    for f in fields["pos_candidate_ex"]:
        assert int(got[f"pos_candidate_ex.{f}"]) == gen.CANDIDATE_EX_DTYPE.fields[f][1], f


def test_invalid_arguments_rejected_before_the_device(P):
    L = P.lib()
    h = C.c_void_p()
    assert L.poseidon_tables_create(None, 0, C.byref(h)) == P.binding.POS_EINVAL
    assert b"NULL" in L.poseidon_last_error()
    import gen
    w = gen.config1()
    t = P.Tables.from_workload(w)
    assert L.poseidon_tables_create(C.byref(t.c), 3, C.byref(h)) == P.binding.POS_ENOTIMPL
    bad = P.Tables.from_workload(w)
    bad.arrays["fwd"][0, 0] = -5
    assert L.poseidon_tables_create(C.byref(bad.c), 0, C.byref(h)) == P.binding.POS_EINVAL
    big = P.Tables(L=2, n_types=1, n_tp=1, fwd=[[2 ** 30, 2 ** 30]], bwd=[[1, 1]], dsync=[[0, 0]],
                   p2p_f=[[0]], p2p_b=[[0]], mem_w=[[0, 0]], mem_a=[[0, 0]], cap=[1])
    assert L.poseidon_tables_create(C.byref(big.c), 0, C.byref(h)) == P.binding.POS_EOVERFLOW
    assert L.poseidon_eval_batch(None, None, 0, None, None, None) == P.binding.POS_EINVAL
    plan = P.binding.pos_plan()
    assert L.poseidon_search(None, C.byref(plan), None) == P.binding.POS_EINVAL
    prob, keep = P.make_problem(w)
    prob.S = 17
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    prob.S = 2
    prob.warmup = -1
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    prob.warmup = 0
    prob.schedule = 2  # Interleaved 1F1B needs V >= 2 and S*V <= 16 (S = 2 here)
    for V in (0, 1, 9):
        prob.V = V
        assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
        assert b"Interleaved" in L.poseidon_last_error()
    prob.V = 2
    prob.ridge = 1  # the ridge rule is defined for 1F1B and Eager 1F1B plans
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    prob.ridge = 0
    prob.schedule = 7
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_ENOTIMPL
    prob.schedule = 0
    for mode in (-1, 3):
        prob.prune = mode
        assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
        assert b"prune" in L.poseidon_last_error()
    with pytest.raises(P.PoseidonError):
        P.Handle(bad)


def test_search_space_limits_rejected_before_the_device(P):
    """poseidon_search checks its documented limits on the host: more than
    2^22 slices (here 4 types free over 12 stages: 4^12 placements), and an
    lcm of the D*M values reaching 2^32."""
    import gen
    L = P.lib()
    plan = P.binding.pos_plan()
    rng = np.random.default_rng(5)
    K, Lw = 4, 16
    w = gen.Workload(name="wide", L=Lw, n_types=4, n_tp=1,
                     fwd=rng.integers(1, 9, (K, Lw)).astype(np.int32),
                     bwd=rng.integers(1, 9, (K, Lw)).astype(np.int32),
                     dsync=np.zeros((K, Lw), np.int32), p2p_f=np.zeros((K, K), np.int32),
                     p2p_b=np.zeros((K, K), np.int32), mem_w=np.zeros((K, Lw), np.int64),
                     mem_a=np.zeros((K, Lw), np.int64), cap=np.full(K, 10, np.int64),
                     S=12, M_list=[4], tp_list=[1], dp_list=[1], seed=0)
    prob, keep = P.make_problem(w)
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    assert b"placements" in L.poseidon_last_error()
    w.S = 11  # 4^11 = 2^22 placements pass; with two M values there are 2^23 slices
    w.M_list = [4, 8]
    prob, keep = P.make_problem(w)
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    assert b"2^22 slices" in L.poseidon_last_error()
    w.S = 2
    w.M_list = [229, 233, 239, 241, 251]  # pairwise coprime: lcm = product > 2^32
    prob, keep = P.make_problem(w)
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    assert b"lcm" in L.poseidon_last_error()


def test_per_stage_tp_problems_checked_before_the_device(P):
    """POS_PLACE_DEVICES: the device counts, D values, the ridge option and
    the 2^22 limit on class sequences are checked on the host."""
    import gen
    L = P.lib()
    plan = P.binding.pos_plan()
    rng = np.random.default_rng(6)
    T_, n_tp, Lw = 4, 4, 16
    K = T_ * n_tp
    w = gen.Workload(name="wide-tp", L=Lw, n_types=T_, n_tp=n_tp,
                     fwd=rng.integers(1, 9, (K, Lw)).astype(np.int32),
                     bwd=rng.integers(1, 9, (K, Lw)).astype(np.int32),
                     dsync=np.zeros((K, Lw), np.int32), p2p_f=np.zeros((K, K), np.int32),
                     p2p_b=np.zeros((K, K), np.int32), mem_w=np.zeros((K, Lw), np.int64),
                     mem_a=np.zeros((K, Lw), np.int64), cap=np.full(K, 10, np.int64),
                     S=12, M_list=[4], tp_list=[1, 1, 1, 1], dp_list=[1] * n_tp,
                     placement=gen.workloads.PLACE_DEVICES, type_counts=[3, 3, 3, 3],
                     D_list=[1], seed=0)
    # 12!/(3!)^4 type orders x 4^12 TP choices: far above 2^22 sequences
    prob, keep = P.make_problem(w)
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    assert b"2^22 class sequences" in L.poseidon_last_error()
    for field, value, msg in (("type_counts", [3, 3, 3, 70000], b"device counts"),
                              ("D_list", [0], b"D must be"), ("tp_list", [1, 0, 1, 1], b"TP")):
        w2 = gen.Workload(**{**w.__dict__, field: value})
        prob, keep = P.make_problem(w2)
        assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
        assert msg in L.poseidon_last_error(), field
    prob, keep = P.make_problem(w, ridge=True)
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    assert b"ridge" in L.poseidon_last_error()
    w5 = gen.Workload(**{**w.__dict__, "n_tp": 5, "n_types": 3, "S": 2,
                         "tp_list": [1] * 5, "dp_list": [1] * 5,
                         "type_counts": [1, 1, 0]})
    K5 = 15
    for f in ("fwd", "bwd", "dsync", "mem_w", "mem_a"):
        setattr(w5, f, np.resize(getattr(w, f), (K5, Lw)))
    for f in ("p2p_f", "p2p_b"):
        setattr(w5, f, np.zeros((K5, K5), getattr(w, f).dtype))
    w5.cap = np.full(K5, 10, np.int64)
    prob, keep = P.make_problem(w5, schedule=2, V=2)
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    assert b"n_tp <= 4" in L.poseidon_last_error()
    prob, keep = P.make_problem(w)
    prob.n_D = 0
    assert L.poseidon_search(C.byref(prob), C.byref(plan), None) == P.binding.POS_EINVAL
    assert b"D_list" in L.poseidon_last_error()


def test_binding_refuses_to_run_without_the_library(tmp_path, monkeypatch):
    import paper_2609_06086_gb300.binding as b
    monkeypatch.setattr(b, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(b, "_lib", None)
    with pytest.raises(ImportError):
        b.lib()


def test_product_path_does_not_import_the_oracle():
    src = os.path.join(ROOT, "paper_2609_06086_gb300")
    for dirpath, _, files in os.walk(src):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert "oracle" not in text.lower(), f
